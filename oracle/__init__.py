"""Plain fp64 CPU oracle for MDS-coded matrix multiplication (Sec. III).

TEST INFRASTRUCTURE.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may import this package.  The CUDA library
and its Python binding never import, link or call it, and the two share no
code.  The arithmetic lives in ``oracle.c`` (fp64 loops, one function per
step of the paper); this module only compiles it with gcc and marshals numpy
arrays.

Parity pins: every function here is checked by ``tests/test_oracle_pins.py``
against something other than itself (the paper's worked example, closed forms,
library routines, brute force, exact integer arithmetic).
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")

STATUS = {0: "ok", -1: "bad argument", -2: "not decodable", -3: "singular"}


class OracleError(RuntimeError):
    pass


def build(force: bool = False) -> str:
    """Compile oracle.c into liboracle.so next to it (gcc, fp64, OpenMP)."""
    if (not force and os.path.exists(_LIB)
            and os.path.getmtime(_LIB) >= os.path.getmtime(_SRC)):
        return _LIB
    tmp = _LIB + ".tmp%d" % os.getpid()
    cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fopenmp",
           "-ffp-contract=off", "-o", tmp, _SRC, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB)
    return _LIB


_lib = None


def _load():
    global _lib
    if _lib is None:
        build()
        lib = ctypes.CDLL(_LIB)
        i32, i64, u32, u64, f64 = (ctypes.c_int32, ctypes.c_int64, ctypes.c_uint32,
                                   ctypes.c_uint64, ctypes.c_double)
        vp = ctypes.c_void_p
        sig = {
            "or_num_threads": (ctypes.c_int, []),
            "or_set_threads": (None, [ctypes.c_int]),
            "or_block_rows": (i64, [i64, i32]),
            "or_encode": (ctypes.c_int, [i32, i32, i64, i64, vp, vp, i64, vp, vp]),
            "or_encode_bf16": (ctypes.c_int, [i32, i32, i64, i64, vp, vp, i64, vp, vp]),
            "or_matmul": (ctypes.c_int, [i64, i64, i32, vp, i64, vp, vp]),
            "or_worker_outputs": (ctypes.c_int, [i32, i32, i64, i64, i32, vp, i64, vp, i64,
                                                 vp, vp]),
            "or_worker_outputs_f64": (ctypes.c_int, [i32, i32, i64, i64, i32, vp, i64, vp,
                                                     i64, vp, vp]),
            "or_worker_outputs_bf16": (ctypes.c_int, [i32, i32, i64, i64, i32, vp, i64, vp,
                                                      i64, vp, vp]),
            "or_splitmix64": (u64, [u64, u64]),
            "or_draw_erasures": (ctypes.c_int, [u64, u64, i32, i32, f64, f64,
                                                ctypes.POINTER(u32), vp]),
            "or_decode": (ctypes.c_int, [i32, i32, i64, i64, vp, u32, vp, vp]),
            "or_generator_inverse": (ctypes.c_int, [i32, i32, vp, u32, vp]),
            "or_gd": (ctypes.c_int, [i64, i64, vp, i64, vp, f64, i32, vp]),
            "or_runtime_simulate": (ctypes.c_int, [i32, i32, i32, f64, f64, u64, u64, i64, vp]),
            "or_repetition_select": (ctypes.c_int, [i32, i32, u32, ctypes.POINTER(u32)]),
        }
        for name, (res, args) in sig.items():
            f = getattr(lib, name)
            f.restype = res
            f.argtypes = args
        _lib = lib
    return _lib


def _ptr(a: np.ndarray):
    return a.ctypes.data_as(ctypes.c_void_p)


def _f32(a) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(a, dtype=np.float32))


def _f64(a) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(a, dtype=np.float64))


def _u16(a) -> np.ndarray:
    a = np.asarray(a)
    if a.dtype != np.uint16:
        raise TypeError("bf16 data is passed as raw uint16 bits")
    return np.ascontiguousarray(a)


def _check(status: int):
    if status != 0:
        raise OracleError(STATUS.get(status, str(status)))


def num_threads() -> int:
    return int(_load().or_num_threads())


def set_threads(threads: int) -> None:
    """Threads of the OpenMP loops (timing only)."""
    _load().or_set_threads(threads)


def block_rows(m: int, k: int) -> int:
    return int(_load().or_block_rows(m, k))


def encode(n: int, k: int, A, P, with_bound: bool = False):
    """fp64 parity blocks ((n-k) L x d) of A (fp32 m x d) under G = [I_k; P]."""
    A = _f32(A)
    P = _f64(P)
    m, d = A.shape
    L = block_rows(m, k)
    par = np.empty(((n - k) * L, d), np.float64)
    bound = np.empty_like(par) if with_bound else None
    _check(_load().or_encode(n, k, m, d, _ptr(P), _ptr(A), d, _ptr(par),
                             _ptr(bound) if with_bound else None))
    return (par, bound) if with_bound else par


def encode_bf16(n: int, k: int, A_bits, P, with_bound: bool = False):
    """fp64 parity blocks of bf16 A (raw uint16 bits)."""
    A = _u16(A_bits)
    P = _f64(P)
    m, d = A.shape
    L = block_rows(m, k)
    par = np.empty(((n - k) * L, d), np.float64)
    bound = np.empty_like(par) if with_bound else None
    _check(_load().or_encode_bf16(n, k, m, d, _ptr(P), _ptr(A), d, _ptr(par),
                                  _ptr(bound) if with_bound else None))
    return (par, bound) if with_bound else par


def matmul(A, X) -> np.ndarray:
    """Y = A X in fp64 (A fp32 m x d, X fp32 d x b)."""
    A = _f32(A)
    X = _f32(X)
    m, d = A.shape
    b = X.shape[1]
    Y = np.empty((m, b), np.float64)
    _check(_load().or_matmul(m, d, b, _ptr(A), d, _ptr(X), _ptr(Y)))
    return Y


def worker_outputs(n: int, k: int, A, parity, X) -> np.ndarray:
    """All n worker products (n L x b, fp64) from A and the given fp32 parity."""
    A = _f32(A)
    parity = _f32(parity)
    X = _f32(X)
    m, d = A.shape
    b = X.shape[1]
    L = block_rows(m, k)
    assert parity.shape == ((n - k) * L, d)
    Yt = np.empty((n * L, b), np.float64)
    _check(_load().or_worker_outputs(n, k, m, d, b, _ptr(A), d, _ptr(parity), d,
                                     _ptr(X), _ptr(Yt)))
    return Yt


def worker_outputs_f64(n: int, k: int, A, parity, X) -> np.ndarray:
    """All n worker products from A and fp64 parity (the exact code)."""
    A = _f32(A)
    parity = _f64(parity)
    X = _f32(X)
    m, d = A.shape
    b = X.shape[1]
    L = block_rows(m, k)
    assert parity.shape == ((n - k) * L, d)
    Yt = np.empty((n * L, b), np.float64)
    _check(_load().or_worker_outputs_f64(n, k, m, d, b, _ptr(A), d, _ptr(parity), d,
                                         _ptr(X), _ptr(Yt)))
    return Yt


def worker_outputs_bf16(n: int, k: int, A_bits, parity_bits, B_bits) -> np.ndarray:
    """All n worker products C~_j = A~_j B (n L x N, fp64) on bf16 blocks."""
    A = _u16(A_bits)
    par = _u16(parity_bits)
    B = _u16(B_bits)
    m, d = A.shape
    N = B.shape[1]
    L = block_rows(m, k)
    assert par.shape == ((n - k) * L, d)
    Ct = np.empty((n * L, N), np.float64)
    _check(_load().or_worker_outputs_bf16(n, k, m, d, N, _ptr(A), d, _ptr(par), d,
                                          _ptr(B), _ptr(Ct)))
    return Ct


def splitmix64(seed: int, i: int) -> int:
    return int(_load().or_splitmix64(seed, i))


def draw_erasures(seed: int, counter: int, n: int, k: int, shift: float = 1.0,
                  rate: float = 1.0):
    """(survivor bitmask, n task times) of one straggler draw."""
    mask = ctypes.c_uint32(0)
    times = np.empty(n, np.float64)
    _check(_load().or_draw_erasures(seed, counter, n, k, shift, rate,
                                    ctypes.byref(mask), _ptr(times)))
    return int(mask.value), times


def decode(n: int, k: int, m: int, P, survivors: int, Yt) -> np.ndarray:
    """Y (m x b, fp64) from the surviving rows of the stacked results Yt."""
    P = _f64(P)
    Yt = _f64(Yt)
    b = Yt.shape[1]
    Y = np.empty((m, b), np.float64)
    _check(_load().or_decode(n, k, m, b, _ptr(P), survivors, _ptr(Yt), _ptr(Y)))
    return Y


def generator_inverse(n: int, k: int, P, survivors: int) -> np.ndarray:
    P = _f64(P)
    Ginv = np.empty((k, k), np.float64)
    _check(_load().or_generator_inverse(n, k, _ptr(P), survivors, _ptr(Ginv)))
    return Ginv


def gd(A, y, eta: float, iters: int, x0=None) -> np.ndarray:
    """x after `iters` exact-gradient steps on 0.5 ||A x - y||^2 (fp64)."""
    A = _f32(A)
    y = _f32(y)
    m, d = A.shape
    x = np.zeros(d, np.float64) if x0 is None else _f64(x0).copy()
    _check(_load().or_gd(m, d, _ptr(A), d, _ptr(y), eta, iters, _ptr(x)))
    return x


SCHEMES = {"uncoded": 0, "repetition": 1, "mds": 2}


def runtime_simulate(scheme: str, n: int, k: int, shift: float, rate: float, seed: int,
                     counter0: int, count: int) -> np.ndarray:
    """Monte-Carlo overall runtimes (Sec. III-B/C/D) from the straggler draws."""
    T = np.empty(count, np.float64)
    _check(_load().or_runtime_simulate(SCHEMES[scheme], n, k, shift, rate, seed, counter0,
                                       count, _ptr(T)))
    return T


def repetition_select(n: int, k: int, survivors: int) -> int:
    """Decodable set of an n/k-repetition code: lowest surviving replica per block."""
    sel = ctypes.c_uint32(0)
    _check(_load().or_repetition_select(n, k, survivors, ctypes.byref(sel)))
    return int(sel.value)


def repetition_parity(n: int, k: int) -> np.ndarray:
    """P of the n/k-repetition code in systematic form: worker k + p copies block p mod k."""
    P = np.zeros((n - k, k))
    for p in range(n - k):
        P[p, p % k] = 1.0
    return P
