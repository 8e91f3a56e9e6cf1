"""GPU parity of the bf16 coded GEMM path (tcgen05) against the oracle.

The oracle runs the method on the same bf16 blocks: the GPU's bf16 parity
(itself checked against the oracle's fp64 encode to within one bf16 rounding),
worker products C~_j = A~_j B in fp64, fp64 Gaussian-elimination decode.
Tolerances:
  * bf16 encode: |gpu - exact| <= 1 bf16 ulp of the exact value + 2 k u32 sum|P||A|;
  * worker products (exact bf16 products, fp32 accumulation over d terms in
    the tensor core): relative l2 error <= 10 sqrt(d) u32 per worker block per
    column (5.4e-5 at d = 8192), at least 1e-5;
  * decoded A B: relative l2 error <= 1e-2 per column (as the method fixes it
    for the bf16 variant); measured errors are far lower.
"""
import numpy as np
import pytest
import torch

import synth

pytestmark = pytest.mark.gpu
DEV = "cuda:0"
U32 = 2.0 ** -24


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


def bits(t):
    return t.contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


def bf16_ulp(x):
    """Spacing of bf16 numbers at |x| (8 significant bits)."""
    e = np.floor(np.log2(np.maximum(np.abs(x), 2.0 ** -126)))
    return 2.0 ** (e - 7)


def worker_tol(d):
    return max(1e-5, 10 * np.sqrt(d) * U32)


def rel_cols(got, want):
    num = np.linalg.norm(got - want, axis=0)
    den = np.linalg.norm(want, axis=0)
    return num / np.where(den > 0, den, 1.0)


def run(cm, n, k, m, d, N, seed=3, counter=0, inplace=False):
    P = synth.parity_coefficients(n, k)
    code = cm.Code(n, k, m, d, P, dtype="bf16")
    A = synth.gaussian((m, d), seed, dtype=torch.bfloat16).to(DEV)
    B = synth.gaussian((d, N), seed + 1, dtype=torch.bfloat16)
    Bt = B.t().contiguous().to(DEV)
    par = cm.encode(code, A)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    Ct = cm.coded_gemm(code, A, par, Bt, status=status)
    mask, _ = cm.draw_erasures(synth.ERASURE_SEED, counter, n, k)
    C = cm.decode_mat(code, Ct.clone() if inplace else Ct, mask, status=status)
    if inplace:
        Cin = Ct.clone()
        cm.decode_mat(code, Cin, mask, C=Cin, status=status)
    torch.cuda.synchronize()
    assert status.item() == 0
    out = dict(P=P, code=code, A=A, B=B, par=par, Ct=Ct, mask=mask, C=C)
    if inplace:
        out["Cin"] = Cin
    return out


def check_encode_bf16(orc, n, k, A, P, par):
    want, bound = orc.encode_bf16(n, k, bits(A), P.astype(np.float64), with_bound=True)
    got = par.float().double().cpu().numpy()
    tol = bf16_ulp(want) + 2 * k * U32 * bound
    assert np.all(np.abs(got - want) <= tol), np.max(np.abs(got - want) - tol)


@pytest.mark.parametrize("n,k,m,d,ld", [
    (6, 3, 301, 203, 208),       # elementwise form (k <= 8): ragged columns and rows
    (20, 10, 613, 257, 264),     # elementwise form with up to 16 data blocks
    (16, 12, 500, 203, 208),     # tiled form (12 data blocks, 4 parity blocks)
])
def test_encode_bf16_ragged_columns(cm, orc, n, k, m, d, ld):
    """bf16 encode on a padded row pitch with d not a multiple of 4: each
    encode form, its 4-column chunks and its scalar tail, against the
    oracle's bound (RNE output within one bf16 unit)."""
    P = synth.parity_coefficients(n, k)
    code = cm.Code(n, k, m, d, P, dtype="bf16")
    A = synth.gaussian((m, ld), 5, dtype=torch.bfloat16).to(DEV)[:, :d]
    par = cm.encode(code, A)
    torch.cuda.synchronize()
    check_encode_bf16(orc, n, k, A, P, par)


@pytest.mark.parametrize("n,k,m,d,N", [
    (6, 3, 300, 128, 64),        # one partial column tile
    (5, 4, 517, 200, 80),        # d not a multiple of 64, N not of 256, L not of 128
    (16, 12, 1537, 512, 512),    # several row and column tiles
    (4, 3, 40, 64, 16),          # tiny
    (6, 3, 900, 128, 300),       # 3 row tiles per block, ragged last tile and columns
])
def test_coded_gemm_matches_oracle(cm, orc, n, k, m, d, N):
    r = run(cm, n, k, m, d, N)
    check_encode_bf16(orc, n, k, r["A"], r["P"], r["par"])
    want = orc.worker_outputs_bf16(n, k, bits(r["A"]), bits(r["par"]), bits(r["B"]))
    got = r["Ct"].double().cpu().numpy()
    L = r["code"].L
    for j in range(n):
        err = rel_cols(got[j * L:(j + 1) * L], want[j * L:(j + 1) * L])
        assert err.max() <= worker_tol(d), (j, err.max())
    # method-form decode of the oracle's products
    P64 = r["P"].astype(np.float64)
    C_or = orc.decode(n, k, m, P64, r["mask"], want)
    err = rel_cols(r["C"].double().cpu().numpy(), C_or)
    assert err.max() <= 1e-2, err.max()
    assert err.max() <= 1e-4, err.max()      # what the kernels actually reach


def test_decode_mat_in_place_matches(cm, orc):
    r = run(cm, 16, 12, 1000, 256, 256, inplace=True)
    m = r["code"].m
    assert torch.equal(r["Cin"][:m], r["C"])


def test_decode_mat_every_erasure_count(cm, orc):
    n, k, m, d, N = 10, 5, 600, 128, 96
    r = run(cm, n, k, m, d, N)
    want = orc.worker_outputs_bf16(n, k, bits(r["A"]), bits(r["par"]), bits(r["B"]))
    P64 = r["P"].astype(np.float64)
    for e in range(0, n - k + 1):           # e missing systematic blocks
        mask = ((1 << (k - e)) - 1) | (((1 << e) - 1) << k)
        C = cm.decode_mat(r["code"], r["Ct"], mask)
        C_or = orc.decode(n, k, m, P64, mask, want)
        assert rel_cols(C.double().cpu().numpy(), C_or).max() <= 1e-4, e


def test_gemm_config_sampled(cm, orc):
    """(16,12), A 32768 x 8192 bf16, B 8192 x 4096 bf16: sampled block rows
    of every worker against the oracle on the same bf16 blocks, and, over all
    4096 columns, one random row inside every 256-row tile pair of the
    kernel's tiling plus the first and last row of every pair."""
    w = synth.GEMM
    P = synth.parity_coefficients(w.n, w.k)
    code = cm.Code(w.n, w.k, w.m, w.d, P, dtype="bf16")
    L = code.L
    A, B = synth.gemm_inputs(w, device=DEV)
    Bt = B.t().contiguous()
    par = cm.encode(code, A)
    Ct = cm.coded_gemm(code, A, par, Bt)
    mask, _ = cm.draw_erasures(synth.ERASURE_SEED, 0, w.n, w.k)
    C = cm.decode_mat(code, Ct, mask)
    torch.cuda.synchronize()
    rng = np.random.default_rng(5)
    rs = sorted(set([0, L - 1] + rng.integers(0, L, 6).tolist()))
    s = len(rs)
    idx = torch.tensor([i * L + r for i in range(w.k) for r in rs])
    valid = idx < w.m
    A_sub = torch.zeros((w.k * s, w.d), dtype=torch.bfloat16)
    A_sub[valid] = A[idx[valid].to(DEV)].cpu()
    par_rows = torch.tensor([p * L + r for p in range(w.n - w.k) for r in rs])
    par_s = par[par_rows.to(DEV)].cpu()
    check_encode_bf16(orc, w.n, w.k, A_sub, P, par_s)
    Bb = bits(B)
    want = orc.worker_outputs_bf16(w.n, w.k, bits(A_sub), bits(par_s), Bb)
    got = torch.stack([Ct[j * L + r] for j in range(w.n) for r in rs]).double().cpu().numpy()
    for j in range(w.n):
        err = rel_cols(got[j * s:(j + 1) * s], want[j * s:(j + 1) * s])
        # per-column errors over only s sampled rows scatter: allow 2x
        assert err.max() <= 2 * worker_tol(w.d), (j, err.max())
    C_or = orc.decode(w.n, w.k, w.k * s, P.astype(np.float64), mask, want)
    got_c = C[idx[valid].to(DEV)].double().cpu().numpy()
    err = rel_cols(got_c, C_or[valid.numpy()])
    assert err.max() <= 1e-2, err.max()
    # every tile pair: the kernel cuts the m real rows of A and the (n-k) L
    # parity rows into 256-row pairs of their own; the pad rows [m, kL) are
    # stored as zeros
    assert bool((Ct[w.m:w.k * L] == 0).all())
    rng2 = np.random.default_rng(6)
    rows = []
    for lo, hi in ((0, w.m), (w.k * L, w.n * L)):
        for t0 in range(lo, hi, 256):
            t1 = min(hi, t0 + 256)
            rows += [t0, t1 - 1, int(rng2.integers(t0, t1))]
    rows = sorted(set(rows))
    ridx = torch.tensor(rows)
    is_a = ridx < w.m
    coded = torch.empty((len(rows), w.d), dtype=torch.bfloat16)
    coded[is_a] = A[ridx[is_a].to(DEV)].cpu()
    coded[~is_a] = par[(ridx[~is_a] - w.k * L).to(DEV)].cpu()
    # the exact products of the bf16 values, accumulated in fp64
    want_rows = orc.matmul(coded.float().numpy(), B.float().cpu().numpy())
    got_rows = Ct[ridx.to(DEV)].double().cpu().numpy()
    num = np.linalg.norm(got_rows - want_rows, axis=1)
    den = np.linalg.norm(want_rows, axis=1)
    assert (num / den).max() <= 2 * worker_tol(w.d), (num / den).max()
    # survivors only at full size (the bench's launch): the k blocks the
    # decode reads equal the full GEMM's bit for bit, the others untouched
    del C
    Cs = torch.full_like(Ct, float("nan"))
    cm.coded_gemm_survivors(code, A, par, Bt, mask, Ct=Cs)
    torch.cuda.synchronize()
    sel = code.select_decodable(mask)
    for j in range(w.n):
        blk = slice(j * L, (j + 1) * L)
        if (sel >> j) & 1:
            assert torch.equal(Cs[blk], Ct[blk]), j
        else:
            assert bool(torch.isnan(Cs[blk]).all()), j
    del A, B, Bt, par, Ct, Cs
    torch.cuda.empty_cache()


@pytest.mark.parametrize("n,k,m,d,N", [
    (4, 3, 512, 128, 64),        # kL = 513: the pad row lies past the last A tile pair
    (4, 3, 1000, 64, 96),        # kL = 1002 < 1024: the last A pair overhangs the parity rows
    (24, 20, 762, 64, 300),      # 12 pad rows past the last A pair, ragged column tile
])
def test_coded_gemm_writes_every_row_and_nothing_else(cm, orc, n, k, m, d, N):
    P = synth.parity_coefficients(n, k)
    code = cm.Code(n, k, m, d, P, dtype="bf16")
    L = code.L
    A = synth.gaussian((m, d), 11, dtype=torch.bfloat16).to(DEV)
    B = synth.gaussian((d, N), 12, dtype=torch.bfloat16)
    par = cm.encode(code, A)
    guard = 7
    buf = torch.full((n * L + guard, N), float("nan"), dtype=torch.float32, device=DEV)
    Ct = cm.coded_gemm(code, A, par, B.t().contiguous().to(DEV), Ct=buf[:n * L])
    torch.cuda.synchronize()
    got = buf.double().cpu().numpy()
    assert np.isnan(got[n * L:]).all()                       # rows past Ct untouched
    assert not np.isnan(got[:n * L]).any()                   # every Ct row written
    assert (got[m:k * L] == 0).all()                         # pad rows of the last block
    want = orc.worker_outputs_bf16(n, k, bits(A), bits(par), bits(B))
    for j in range(n):
        err = rel_cols(got[j * L:(j + 1) * L], want[j * L:(j + 1) * L])
        assert err.max() <= worker_tol(d), (j, err.max())


@pytest.mark.parametrize("n,k,m,d,N,kind", [
    (16, 12, 3000, 192, 200, "mds"),     # L = 250: one row pair per block, rank 1 short
    (10, 5, 1300, 64, 96, "mds"),        # L = 260: the second pair holds 4 rows
    (24, 20, 762, 64, 300, "mds"),       # pad rows in the last systematic block
    (6, 3, 900, 128, 64, "repetition"),
    (5, 3, 100, 64, 40, "mds"),          # L = 34: a run of one block is shorter than a CTA's rows
])
def test_coded_gemm_survivors_only(cm, orc, n, k, m, d, N, kind):
    """Survivors-only GEMM: the k blocks that the decode reads equal the full
    GEMM's bit for bit, no other row of Ct is written, and the decode of them
    equals the decode after the full GEMM."""
    P = synth.parity_coefficients(n, k) if kind == "mds" else "repetition"
    code = cm.Code(n, k, m, d, P, dtype="bf16")
    L = code.L
    A = synth.gaussian((m, d), 21, dtype=torch.bfloat16).to(DEV)
    Bt = synth.gaussian((N, d), 22, dtype=torch.bfloat16).to(DEV)
    par = cm.encode(code, A)
    full = cm.coded_gemm(code, A, par, Bt)
    if kind == "mds":
        masks = [cm.draw_erasures(synth.ERASURE_SEED, c, n, k)[0] for c in range(3)]
        # one run of all systematic blocks (pad rows at its end); the last k
        # workers (a systematic run ending at block k - 1, then the parity)
        masks += [(1 << k) - 1, ((1 << n) - 1) ^ ((1 << (n - k)) - 1)]
    else:   # block j of worker j mod k: every block among the survivors
        masks = [0b111000, 0b100011, 0b111111]
    for mask in masks:
        sel = code.select_decodable(mask)
        buf = torch.full((n * L + 5, N), float("nan"), dtype=torch.float32, device=DEV)
        status = torch.zeros(1, dtype=torch.int32, device=DEV)
        Ct = cm.coded_gemm_survivors(code, A, par, Bt, mask, Ct=buf[:n * L], status=status)
        C = cm.decode_mat(code, Ct, mask, status=status)
        C_full = cm.decode_mat(code, full, mask)
        torch.cuda.synchronize()
        assert status.item() == 0
        got = buf.cpu()
        for j in range(n):
            blk = got[j * L:(j + 1) * L]
            if (sel >> j) & 1:
                assert torch.equal(blk, full[j * L:(j + 1) * L].cpu()), j
            else:
                assert torch.isnan(blk).all(), j
        assert torch.isnan(got[n * L:]).all()
        assert torch.equal(C, C_full)
    # not decodable: rejected before any launch
    with pytest.raises(cm.CodedError):
        cm.coded_gemm_survivors(code, A, par, Bt, (1 << (k - 1)) - 1)


@pytest.mark.parametrize("n,k,e", [(32, 16, 16), (20, 10, 9)])
def test_decode_mat_many_missing_blocks(cm, orc, n, k, e):
    """Matrix decode with up to 16 missing blocks against the oracle's fp64
    decode of the same fp32 results.  The coefficients are applied in fp32:
    the tolerance grows with the condition number of the e x e block."""
    m, N = 23 * k + 3, 40
    P = synth.parity_coefficients(n, k)
    code = cm.Code(n, k, m, 64, P, dtype="bf16")
    L = code.L
    Ct = synth.gaussian((n * L, N), 31).to(DEV)
    mask = ((1 << (k - e)) - 1) | (((1 << e) - 1) << k)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    C = cm.decode_mat(code, Ct, mask, status=status)
    torch.cuda.synchronize()
    assert status.item() == 0
    want = orc.decode(n, k, m, P.astype(np.float64), mask, Ct.double().cpu().numpy())
    Q = P.astype(np.float64)[:e, k - e:]      # parity rows 0..e-1, missing columns k-e..k-1
    tol = max(1e-5, 100 * np.linalg.cond(Q) * U32)
    assert rel_cols(C.double().cpu().numpy(), want).max() <= tol
