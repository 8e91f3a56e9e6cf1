"""GPU parity of coded gradient descent (Sec. III-E) against the oracle.

The coded iteration decodes both products exactly (up to rounding), so its
iterates must follow the oracle's plain fp64 iteration x <- x - eta A^T(Ax - y)
whatever the erasure sets are: relative l2 error <= 1e-3 after the stated
number of iterations.
"""
import numpy as np
import pytest
import torch

import synth

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


@pytest.fixture(scope="module")
def cm():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import os
    import paper_1512_02673_gb300 as cm
    if not os.path.exists(cm.LIB_PATH):
        from paper_1512_02673_gb300 import build
        build.build()
    return cm


def with_ld16(t):
    """Device copy of a row-major matrix whose rows start on 16-byte boundaries."""
    rows, cols = t.shape
    ld = (cols + 3) // 4 * 4
    buf = torch.zeros((rows, ld), dtype=t.dtype, device=DEV)
    buf[:, :cols] = t.to(DEV)
    return buf[:, :cols]


def run_coded_gd(cm, A, y, n, k_a, k_at, iters, eta, seed=synth.ERASURE_SEED,
                 survivors_only=False):
    m, d = A.shape
    cA = cm.Code(n, k_a, m, d, synth.parity_coefficients(n, k_a))
    cAT = cm.Code(n, k_at, d, m, synth.parity_coefficients(n, k_at, seed=synth.CODE_SEED + 1))
    Ad = with_ld16(A)
    ATd = with_ld16(A.t())             # A^T: its row split is the column split of A
    PA = cm.encode(cA, Ad)
    PAT = cm.encode(cAT, ATd)
    yd = y.to(DEV)
    x = torch.zeros(d, device=DEV)
    ws = torch.empty(cm.gd_workspace_bytes(cA, cAT), dtype=torch.uint8, device=DEV)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    masks = []
    for t in range(iters):
        sA, _ = cm.draw_erasures(seed, 2 * t, n, k_a)
        sAT, _ = cm.draw_erasures(seed, 2 * t + 1, n, k_at)
        masks.append((sA, sAT))
        cm.gd_step(cA, Ad, PA, cAT, ATd, PAT, yd, x, eta, sA, sAT, ws, status,
                   survivors_only=survivors_only)
    torch.cuda.synchronize()
    assert status.item() == 0
    return x.double().cpu().numpy(), masks


@pytest.mark.parametrize("survivors_only", [False, True], ids=["all-workers", "survivors-only"])
@pytest.mark.parametrize("m,d,n,k", [(600, 120, 10, 8), (1001, 203, 20, 10), (96, 500, 6, 3)])
def test_small_gd_matches_oracle(cm, orc, m, d, n, k, survivors_only):
    A = synth.gaussian((m, d), 21)
    y = synth.gaussian((m,), 22)
    eta = 0.5 / (m ** 0.5 + d ** 0.5) ** 2
    x, masks = run_coded_gd(cm, A, y, n, k, k, 40, eta, survivors_only=survivors_only)
    for t, (sA, sAT) in enumerate(masks):
        assert sA == orc.draw_erasures(synth.ERASURE_SEED, 2 * t, n, k)[0]
        assert sAT == orc.draw_erasures(synth.ERASURE_SEED, 2 * t + 1, n, k)[0]
    want = orc.gd(A.numpy(), y.numpy(), eta, 40)
    err = np.linalg.norm(x - want) / np.linalg.norm(want)
    assert err <= 1e-3, err


@pytest.mark.parametrize("survivors_only", [False, True], ids=["all-workers", "survivors-only"])
def test_gd_config_50_iterations(cm, orc, survivors_only):
    w = synth.GD
    A, _, y = synth.regression_inputs(w, device="cpu")
    x, _ = run_coded_gd(cm, A, y, w.n, w.k_a, w.k_at, w.iters, w.eta,
                        survivors_only=survivors_only)
    want = orc.gd(A.numpy(), y.numpy(), w.eta, w.iters)
    err = np.linalg.norm(x - want) / np.linalg.norm(want)
    assert err <= 1e-3, err


@pytest.mark.parametrize("survivors_only", [False, True], ids=["all-workers", "survivors-only"])
@pytest.mark.parametrize("w", synth.PAPER_GD, ids=lambda w: "%dx%d" % (w.m, w.d))
def test_gd_paper_shapes(cm, orc, w, survivors_only):
    """(10,8) coded gradient descent on the square, fat and tall matrices of
    Sec. III-F, 50 iterations against the oracle's fp64 iteration."""
    A, _, y = synth.regression_inputs(w, device="cpu")
    x, _ = run_coded_gd(cm, A, y, w.n, w.k_a, w.k_at, w.iters, w.eta,
                        survivors_only=survivors_only)
    want = orc.gd(A.numpy(), y.numpy(), w.eta, w.iters)
    err = np.linalg.norm(x - want) / np.linalg.norm(want)
    assert err <= 1e-3, err
