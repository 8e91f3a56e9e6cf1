"""The allocation-free gradient step, checked against cm_gd_step.

cm_gd_step_noalloc is for callers that cannot allocate device memory (a
plug-in inside an application that owns all device memory, a loop that must
not call cudaMalloc because it can synchronize the device): it runs the same
step out of a fixed device scratch array in the library instead of a caller
workspace.  This file is named so that pytest collects it last.
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


def padded_copy(t):
    rows, cols = t.shape
    buf = torch.zeros((rows, (cols + 3) // 4 * 4), device=DEV)
    buf[:, :cols] = t.to(DEV)
    return buf[:, :cols]


def problem(cm, m, d, n, k):
    A = synth.gaussian((m, d), 41)
    y = synth.gaussian((m,), 42).to(DEV)
    cA = cm.Code(n, k, m, d, synth.parity_coefficients(n, k))
    cAT = cm.Code(n, k, d, m, synth.parity_coefficients(n, k, seed=synth.CODE_SEED + 1))
    Ad, ATd = padded_copy(A), padded_copy(A.t())
    return cA, cAT, Ad, cm.encode(cA, Ad), ATd, cm.encode(cAT, ATd), y


def test_noalloc_step_matches_workspace_step_on_two_calls(cm, orc):
    m, d, n, k = 1001, 203, 20, 10
    cA, cAT, A, PA, AT, PAT, y = problem(cm, m, d, n, k)
    assert cm.gd_workspace_bytes(cA, cAT) <= cm.GD_STATIC_SCRATCH_BYTES
    eta = 0.5 / (m ** 0.5 + d ** 0.5) ** 2
    ws = torch.empty(cm.gd_workspace_bytes(cA, cAT), dtype=torch.uint8, device=DEV)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    x_ws = torch.zeros(d, device=DEV)
    x_na = torch.zeros(d, device=DEV)
    steps = 2
    for t in range(steps):                   # two calls in a row
        sA = cm.draw_erasures(synth.ERASURE_SEED, 2 * t, n, k)[0]
        sAT = cm.draw_erasures(synth.ERASURE_SEED, 2 * t + 1, n, k)[0]
        cm.gd_step(cA, A, PA, cAT, AT, PAT, y, x_ws, eta, sA, sAT, ws, status)
        cm.gd_step_noalloc(cA, A, PA, cAT, AT, PAT, y, x_na, eta, sA, sAT, status)
        torch.cuda.synchronize()
        assert status.item() == 0
        # the same kernels on the same inputs in the same order: identical
        assert torch.equal(x_na, x_ws), t
        assert torch.linalg.norm(x_ws).item() > 0
    # and the iterate is the exact-gradient iterate (the oracle's fp64 GD)
    want = orc.gd(A.cpu().numpy(), y.cpu().numpy(), eta, steps)
    got = x_na.double().cpu().numpy()
    assert np.linalg.norm(got - want) <= 1e-3 * np.linalg.norm(want)


def test_noalloc_step_allocates_nothing(cm):
    m, d, n, k = 1001, 203, 20, 10
    cA, cAT, A, PA, AT, PAT, y = problem(cm, m, d, n, k)
    eta = 0.5 / (m ** 0.5 + d ** 0.5) ** 2
    x = torch.zeros(d, device=DEV)
    mask = cm.draw_erasures(synth.ERASURE_SEED, 0, n, k)[0]
    cm.gd_step_noalloc(cA, A, PA, cAT, AT, PAT, y, x, eta, mask, mask)   # warm-up
    torch.cuda.synchronize()
    free0, torch0 = torch.cuda.mem_get_info()[0], torch.cuda.memory_allocated()
    for t in range(5):
        cm.gd_step_noalloc(cA, A, PA, cAT, AT, PAT, y, x, eta, mask, mask)
    torch.cuda.synchronize()
    assert torch.cuda.mem_get_info()[0] == free0
    assert torch.cuda.memory_allocated() == torch0


def test_noalloc_step_rejects_problems_beyond_the_array(cm):
    m, d, n, k = 100000, 2000, 32, 4         # stacked results alone need 6.4 MB
    cA = cm.Code(n, k, m, d, synth.parity_coefficients(n, k))
    cAT = cm.Code(n, k, d, m, synth.parity_coefficients(n, k, seed=synth.CODE_SEED + 1))
    assert cm.gd_workspace_bytes(cA, cAT) > cm.GD_STATIC_SCRATCH_BYTES
    t = torch.zeros((8, 8), device=DEV)      # never touched: the call is rejected first
    v = torch.zeros(8, device=DEV)
    with pytest.raises(cm.CodedError) as e:
        cm.gd_step_noalloc(cA, t, t, cAT, t, t, v, v, 0.1, (1 << n) - 1, (1 << n) - 1)
    assert e.value.status == cm.CM_ENOMEM
