"""Seeded synthetic inputs for the coded matrix-multiplication workloads.

This module holds shapes, seeds and random generators only.  It contains no
step of the coded method: no encoding, block product, erasure ranking or
decoding.  The tests and the benchmark draw every input from here and hand the
same arrays to both the CUDA library and the CPU oracle.

Input recipe (the paper draws its test matrices at random, Sec. III-F):
  * data matrices and vectors: i.i.d. N(0,1) fp32 from a seeded
    ``torch.Generator`` (bf16 inputs are those fp32 draws rounded to nearest
    even by ``Tensor.to``);
  * parity coefficients of the systematic generator G = [I_k; P]: i.i.d.
    N(0,1) drawn in fp64 by ``numpy.random.default_rng(seed)`` and rounded
    once to fp32; the fp32 values are the code everywhere;
  * regression labels: y = A x* + 0.01 * N(0,1) noise.
"""
from __future__ import annotations

import dataclasses
import math

import numpy as np
import torch

DATA_SEED = 1512
CODE_SEED = 2673
ERASURE_SEED = 3
SHUFFLE_PARTITION_SEED = 4   # coded shuffling: partitions of [q]
SHUFFLE_CACHE_SEED = 5       # coded shuffling: cache refills
STRAGGLE_SHIFT = 1.0   # shifted-exponential model, Sec. III-D: shift 1
STRAGGLE_RATE = 1.0    # straggling parameter mu


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    m: int                 # rows of A
    d: int                 # columns of A
    b: int                 # vectors per product (columns of X)
    n: int                 # coded blocks (simulated workers)
    k: int                 # systematic blocks
    dtype: str = "f32"
    data_device: str = "cpu"
    repeats: int = 1
    gemm_n: int = 0        # columns of B for the matrix-matrix variant

    @property
    def L(self) -> int:
        return -(-self.m // self.k)


@dataclasses.dataclass(frozen=True)
class GDWorkload:
    name: str
    m: int
    d: int
    n: int
    k_a: int               # code of A (first product)
    k_at: int              # code of A^T (second product)
    iters: int
    data_device: str = "cpu"

    @property
    def eta(self) -> float:
        return 0.5 / (math.sqrt(self.m) + math.sqrt(self.d)) ** 2


TINY = Workload("tiny (6,3) 1200x500", m=1200, d=500, b=1, n=6, k=3)
MATVEC = Workload("coded mat-vec (10,5) 12000x10000", m=12000, d=10000, b=1,
                  n=10, k=5, repeats=100)
GD = GDWorkload("coded GD (20,10) 40000x8000", m=40000, d=8000, n=20,
                k_a=10, k_at=10, iters=50)
BANDWIDTH = Workload("coded mat-multi-vec (32,24) 65536x65536 b=8", m=65536,
                     d=65536, b=8, n=32, k=24, data_device="cuda")
GEMM = Workload("coded GEMM bf16 (16,12) 32768x8192x4096", m=32768, d=8192,
                b=0, n=16, k=12, dtype="bf16", gemm_n=4096)
# the matrix shapes of the paper's cluster experiments (Sec. III-F): a (25,23)
# code on square, fat and tall matrices times one vector, and (10,8) coded
# gradient descent (iteration count not given there: 50, as above)
PAPER_MATVEC = [Workload("paper (25,23) %dx%d" % (m, d), m=m, d=d, b=1, n=25, k=23,
                         repeats=20) for m, d in [(5750, 5750), (5750, 11500), (11500, 5750)]]
PAPER_GD = [GDWorkload("paper GD (10,8) %dx%d" % (m, d), m=m, d=d, n=10, k_a=8, k_at=8,
                       iters=50) for m, d in [(2000, 2000), (400, 10000), (10000, 400)]]


@dataclasses.dataclass(frozen=True)
class ShuffleWorkload:
    """Coded shuffling (Sec. IV): q data rows of r fp32 words, n workers with
    caches of s rows, `transitions` reshuffles."""
    name: str
    n: int
    q: int
    s: int
    r: int
    transitions: int = 1


# the setting of the rate figure of Sec. IV-D (n = 50, q = 1000, s/q = 0.1) is
# a rate example; the data-plane workload keeps rows of 1 KiB and fewer
# workers so that every block of Alg. 1 holds thousands of rows
SHUFFLE = ShuffleWorkload("coded shuffling n=8 q=2097152 s=q/4 r=256", n=8, q=1 << 21,
                          s=1 << 19, r=256, transitions=4)
SHUFFLE_SMALL = ShuffleWorkload("coded shuffling n=4 q=4000 s=1700 r=67", n=4, q=4000,
                                s=1700, r=67, transitions=3)


def shuffle_rows(w: ShuffleWorkload, device="cpu", seed: int = DATA_SEED + 7) -> torch.Tensor:
    """The q x r data rows (i.i.d. N(0,1) fp32)."""
    return gaussian((w.q, w.r), seed, device)


def parity_coefficients(n: int, k: int, seed: int = CODE_SEED) -> np.ndarray:
    """(n-k) x k parity block P of G = [I_k; P], fp32, C-contiguous."""
    rng = np.random.default_rng(seed)
    return np.ascontiguousarray(rng.standard_normal((n - k, k)).astype(np.float32))


def gaussian(shape, seed: int, device="cpu", dtype=torch.float32) -> torch.Tensor:
    """i.i.d. N(0,1) drawn in fp32 on ``device`` and cast to ``dtype``."""
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    t = torch.randn(shape, generator=g, device=device, dtype=torch.float32)
    return t if dtype == torch.float32 else t.to(dtype)


def small_integers(shape, lo: int, hi: int, seed: int) -> torch.Tensor:
    """i.i.d. integers uniform on [lo, hi], stored as fp32 (exactly)."""
    g = torch.Generator()
    g.manual_seed(seed)
    return torch.randint(lo, hi + 1, shape, generator=g).to(torch.float32)


def matvec_inputs(w: Workload, device=None, seed: int = DATA_SEED):
    """A (m x d) and X (d x b) for a mat-(multi-)vec workload."""
    dev = device or w.data_device
    A = gaussian((w.m, w.d), seed, dev)
    X = gaussian((w.d, w.b), seed + 1, dev)
    return A, X


def regression_inputs(w: GDWorkload, device=None, seed: int = DATA_SEED):
    """A, x*, y = A x* + 0.01 noise (Sec. III-E linear regression)."""
    dev = device or w.data_device
    A = gaussian((w.m, w.d), seed, dev)
    x_star = gaussian((w.d,), seed + 1, dev)
    noise = gaussian((w.m,), seed + 2, dev)
    y = (A.double() @ x_star.double() + 0.01 * noise.double()).float()
    return A, x_star, y


def gemm_inputs(w: Workload, device=None, seed: int = DATA_SEED):
    """bf16 A (m x d) and B (d x N)."""
    dev = device or w.data_device
    A = gaussian((w.m, w.d), seed, dev, torch.bfloat16)
    B = gaussian((w.d, w.gemm_n), seed + 1, dev, torch.bfloat16)
    return A, B
