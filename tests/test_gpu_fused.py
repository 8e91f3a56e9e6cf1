"""GPU parity of the worker products and the decode in one call
(cm_matvec_decode, Sec. III-A: the master needs only k results).

The one call runs the operations of cm_matvec (or cm_matvec_survivors)
followed by cm_decode.  Its Y equals theirs bit for bit, except on small
problems whose products it splits into column segments: each segment then
flushes its short fp32 partial sums into fp64 at other columns, so the worker
results differ by their own rounding (about 1e-7 relative), which the decode
amplifies by up to the condition number of G_S (relative l2 <= 1e-5 per
vector between the two).  Y is also checked against the oracle's plain A X at
the contract's relative l2 tolerance (1e-4 per output vector).
"""
import numpy as np
import pytest
import torch

import synth
from test_gpu_matvec import SHAPES, padded, rel_l2_cols

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


def same_or_reordered(Y, Y_sep):
    """Bit-equal, or (column segments) within the products' rounding."""
    if torch.equal(Y, Y_sep):
        return True
    return rel_l2_cols(Y.cpu().numpy(), Y_sep.cpu().numpy()).max() <= 1e-5


def separate(cm, code, A, par, X, mask, only):
    if only:
        Yt = cm.matvec_survivors(code, A, par, X, mask)
    else:
        Yt = cm.matvec(code, A, par, X)
    return cm.decode(code, Yt, mask)


@pytest.mark.parametrize("only", [False, True], ids=["all-workers", "survivors-only"])
@pytest.mark.parametrize("n,k,m,d,b,lda", SHAPES)
def test_fused_equals_products_then_decode(cm, orc, n, k, m, d, b, lda, only):
    P = synth.parity_coefficients(n, k)
    code = cm.Code(n, k, m, d, P)
    A = padded(m, d, lda or d, 7)
    X_cpu = synth.gaussian((d, b), 8)
    X = X_cpu.to(DEV)
    par = cm.encode(code, A)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    ws = torch.empty(cm.matvec_decode_workspace_bytes(code, b), dtype=torch.uint8, device=DEV)
    want = orc.matmul(A.cpu().numpy(), X_cpu.numpy())
    for counter in range(3):                 # the same workspace, three straggler sets
        mask, _ = cm.draw_erasures(synth.ERASURE_SEED, counter, n, k)
        Y = cm.matvec_decode(code, A, par, X, mask, only_survivors=only, ws=ws, status=status)
        Y_sep = separate(cm, code, A, par, X, mask, only)
        torch.cuda.synchronize()
        assert status.item() == 0
        assert same_or_reordered(Y, Y_sep), counter
        assert rel_l2_cols(Y.cpu().numpy(), want).max() <= 1e-4


@pytest.mark.parametrize("only", [False, True], ids=["all-workers", "survivors-only"])
def test_fused_every_erasure_count(cm, orc, only):
    # every number of missing systematic blocks, e = 0 .. min(k, n - k)
    n, k, m, d, b = 32, 16, 3000, 700, 2
    P = synth.parity_coefficients(n, k)
    code = cm.Code(n, k, m, d, P)
    A = padded(m, d, 700, 9)
    X_cpu = synth.gaussian((d, b), 10)
    X = X_cpu.to(DEV)
    par = cm.encode(code, A)
    want = orc.matmul(A.cpu().numpy(), X_cpu.numpy())
    rng = np.random.default_rng(11)
    G = np.vstack([np.eye(k), P.astype(np.float64)])
    Yt = cm.matvec(code, A, par, X)           # the products the fused path computes
    for e in range(0, 17):
        miss = rng.choice(k, e, replace=False)
        par_surv = rng.choice(np.arange(k, n), e, replace=False)
        mask = sum(1 << j for j in range(k) if j not in miss) + sum(1 << int(j) for j in par_surv)
        Y = cm.matvec_decode(code, A, par, X, mask, only_survivors=only)
        Y_sep = separate(cm, code, A, par, X, mask, only)
        torch.cuda.synchronize()
        assert same_or_reordered(Y, Y_sep), e
        # the decode stage: the oracle's fp64 decode of the same products
        Yo = orc.decode(n, k, m, P.astype(np.float64), mask, Yt.cpu().numpy())
        assert rel_l2_cols(Y.cpu().numpy(), Yo).max() <= 1e-6, e
        # the plain A X: decoding amplifies the products' rounding (fp32
        # partials combined in fp64, about 1e-7 relative) by up to the
        # condition number of G_S, which random sets with 16 missing blocks
        # push past 1e3
        kappa = np.linalg.cond(G[[j for j in range(n) if mask >> j & 1]])
        tol = max(1e-4, 10 * kappa * 2.0 ** -24)
        assert rel_l2_cols(Y.cpu().numpy(), want).max() <= tol, (e, kappa)


def test_fused_singular_sets_status(cm):
    n, k, m, d = 6, 3, 90, 40
    P = synth.parity_coefficients(n, k)
    P[1] = P[0]                               # duplicated parity rows
    code = cm.Code(n, k, m, d, P)
    A = synth.gaussian((m, d), 3).to(DEV)
    X = synth.gaussian((d, 1), 4).to(DEV)
    par = cm.encode(code, A)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    Y = torch.full((m, 1), 7.0, device=DEV)
    L = code.L
    cm.matvec_decode(code, A, par, X, 0b011001, Y=Y, status=status)   # survivors {0, 3, 4}
    Yt = cm.matvec(code, A, par, X)
    torch.cuda.synchronize()
    assert status.item() == cm.CM_ESINGULAR
    assert torch.all(Y[L:] == 7.0)            # missing blocks 1, 2: not written
    assert torch.equal(Y[:L], Yt[:L].float()) # surviving block 0 passes through


def test_fused_rejects_bad_calls(cm):
    n, k, m, d = 6, 3, 90, 40
    code = cm.Code(n, k, m, d, synth.parity_coefficients(n, k))
    A = synth.gaussian((m, d), 3).to(DEV)
    X = synth.gaussian((d, 1), 4).to(DEV)
    par = cm.encode(code, A)
    small = torch.empty(cm.matvec_decode_workspace_bytes(code, 1) - 256, dtype=torch.uint8,
                        device=DEV)
    with pytest.raises(cm.CodedError) as e:
        cm.matvec_decode(code, A, par, X, 0b111, ws=small)
    assert e.value.status == cm.CM_ENOMEM
    with pytest.raises(cm.CodedError) as e:
        cm.matvec_decode(code, A, par, X, 0b000011)
    assert e.value.status == cm.CM_ENOTDECODABLE


def test_fused_repetition_code(cm, orc):
    n, k, m, d, b = 12, 4, 1001, 300, 2
    code = cm.Code(n, k, m, d, "repetition")
    A = padded(m, d, 300, 12)
    X_cpu = synth.gaussian((d, b), 13)
    X = X_cpu.to(DEV)
    par = cm.encode(code, A)
    want = orc.matmul(A.cpu().numpy(), X_cpu.numpy())
    rng = np.random.default_rng(14)
    tried = 0
    while tried < 6:                          # decodable masks: a replica of every block
        mask = int(rng.integers(1, 1 << n))
        try:
            orc.repetition_select(n, k, mask)
        except orc.OracleError:
            with pytest.raises(cm.CodedError) as e:
                cm.matvec_decode(code, A, par, X, mask)
            assert e.value.status == cm.CM_ENOTDECODABLE
            continue
        for only in (False, True):
            Y = cm.matvec_decode(code, A, par, X, mask, only_survivors=only)
            torch.cuda.synchronize()
            assert rel_l2_cols(Y.cpu().numpy(), want).max() <= 1e-4
        tried += 1


@pytest.mark.parametrize("only", [False, True], ids=["all-workers", "survivors-only"])
def test_fused_matvec_config_100_repeats(cm, orc, only):
    w = synth.MATVEC
    P = synth.parity_coefficients(w.n, w.k)
    code = cm.Code(w.n, w.k, w.m, w.d, P)
    A, X = synth.matvec_inputs(w, device="cpu")
    Ad, Xd = A.to(DEV), X.to(DEV)
    par = cm.encode(code, Ad)
    want = orc.matmul(A.numpy(), X.numpy())
    ws = torch.empty(cm.matvec_decode_workspace_bytes(code, w.b), dtype=torch.uint8, device=DEV)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    errs = []
    for rep in range(w.repeats):
        mask, _ = cm.draw_erasures(synth.ERASURE_SEED, rep, w.n, w.k)
        Y = cm.matvec_decode(code, Ad, par, Xd, mask, only_survivors=only, ws=ws, status=status)
        errs.append(rel_l2_cols(Y.cpu().numpy(), want).max())
    assert status.item() == 0
    assert max(errs) <= 1e-4, max(errs)


@pytest.mark.parametrize("only", [False, True], ids=["all-workers", "survivors-only"])
def test_fused_bandwidth_config(cm, only):
    """(32,24), A 65536 x 65536 fp32 (16 GiB), b = 8: the fused Y equals the
    separate products and decode bit for bit (the latter is checked element
    by element against the oracle in test_gpu_matvec)."""
    w = synth.BANDWIDTH
    P = synth.parity_coefficients(w.n, w.k)
    code = cm.Code(w.n, w.k, w.m, w.d, P)
    A, X = synth.matvec_inputs(w, device=DEV)
    par = cm.encode(code, A)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    for counter in (0, 1):
        mask, _ = cm.draw_erasures(synth.ERASURE_SEED, counter, w.n, w.k)
        Y = cm.matvec_decode(code, A, par, X, mask, only_survivors=only, status=status)
        Y_sep = separate(cm, code, A, par, X, mask, only)
        torch.cuda.synchronize()
        assert status.item() == 0
        assert torch.equal(Y, Y_sep), counter
    del A, par
    torch.cuda.empty_cache()
