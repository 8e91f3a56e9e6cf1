"""GPU parity of the coded mat-(multi-)vec path against the CPU oracle.

Every test calls the CUDA library through its C ABI (via the ctypes binding)
and compares with the oracle on the same seeded inputs.  Tolerances:
  * encode (fp32 accumulation of k terms): |gpu - exact| <= 2 k u32 sum_i |P||A|
    elementwise (u32 = 2^-24), the standard bound for a k-term dot product;
  * worker products (fp32 partials of <= 16 terms combined in fp64): relative
    l2 error <= 1e-6 per worker block per vector against the oracle's fp64
    products of the same (GPU) coded blocks;
  * decoded A X: relative l2 error <= 1e-4 per output vector against the
    oracle's fp64 A X (the plain definition), as the method fixes it;
  * survivor masks and every index decision: bit-exact;
  * integer single-parity codes: bit-exact.
"""
import itertools
import math

import numpy as np
import pytest
import torch

import synth

pytestmark = pytest.mark.gpu

U32 = 2.0 ** -24
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


def rel_l2_cols(got, want):
    """Relative l2 error of every column (output vector)."""
    got = np.asarray(got, np.float64)
    want = np.asarray(want, np.float64)
    num = np.linalg.norm(got - want, axis=0)
    den = np.linalg.norm(want, axis=0)
    return num / np.where(den > 0, den, 1.0)


def padded(rows, cols, ld, seed, device=DEV):
    """rows x cols N(0,1) fp32 view with leading dimension ld (a strided view)."""
    base = synth.gaussian((rows, ld), seed, "cpu")
    return base.to(device)[:, :cols]


def check_encode(orc, n, k, A_cpu, P, par_gpu):
    want, bound = orc.encode(n, k, A_cpu.numpy(), P.astype(np.float64), with_bound=True)
    got = par_gpu.double().cpu().numpy()
    tol = 2 * k * U32 * bound + 1e-30
    bad = np.abs(got - want) > tol
    assert not bad.any(), "encode: %d elements out of bound, worst excess %g" % (
        bad.sum(), (np.abs(got - want) - tol).max())


def check_workers(orc, n, k, A_cpu, par_gpu, X_cpu, Yt_gpu, L):
    want = orc.worker_outputs(n, k, A_cpu.numpy(), par_gpu.float().cpu().numpy(), X_cpu.numpy())
    got = Yt_gpu.cpu().numpy()
    for j in range(n):
        blk = slice(j * L, (j + 1) * L)
        w = want[blk]
        if np.linalg.norm(w) == 0:
            assert np.all(got[blk] == 0)
            continue
        err = rel_l2_cols(got[blk], w)
        assert err.max() <= 1e-6, (j, err)


def run_path(cm, orc, n, k, m, d, b, seed=7, lda=None, misalign_x=False, counter=0):
    P = synth.parity_coefficients(n, k)
    code = cm.Code(n, k, m, d, P)
    lda = lda or d
    A = padded(m, d, lda, seed)
    A_cpu = A.cpu().contiguous()
    X_cpu = synth.gaussian((d, b), seed + 1)
    if misalign_x:
        buf = torch.zeros(d * b + 1, device=DEV)
        X = buf[1:].view(d, b)
        X.copy_(X_cpu)
    else:
        X = X_cpu.to(DEV)
    par = cm.encode(code, A)
    Yt = cm.matvec(code, A, par, X)
    mask, _ = cm.draw_erasures(synth.ERASURE_SEED, counter, n, k)
    omask, _ = orc.draw_erasures(synth.ERASURE_SEED, counter, n, k)
    assert mask == omask
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    Y = cm.decode(code, Yt, mask, status=status)
    torch.cuda.synchronize()
    assert status.item() == 0
    return dict(P=P, code=code, A=A, A_cpu=A_cpu, X=X, X_cpu=X_cpu, par=par, Yt=Yt, mask=mask,
                Y=Y)


# ---- config 1 and small shapes spanning several tiles with ragged tails ------------

def test_tiny_config_end_to_end(cm, orc):
    w = synth.TINY
    r = run_path(cm, orc, w.n, w.k, w.m, w.d, w.b, seed=synth.DATA_SEED)
    check_encode(orc, w.n, w.k, r["A_cpu"], r["P"], r["par"])
    check_workers(orc, w.n, w.k, r["A_cpu"], r["par"], r["X_cpu"], r["Yt"], r["code"].L)
    want = orc.matmul(r["A_cpu"].numpy(), r["X_cpu"].numpy())
    assert rel_l2_cols(r["Y"].cpu().numpy(), want).max() <= 1e-4
    # stage check: the oracle's own decode (Gaussian elimination) of the GPU's results
    Yo = orc.decode(w.n, w.k, w.m, r["P"].astype(np.float64), r["mask"], r["Yt"].cpu().numpy())
    assert rel_l2_cols(r["Y"].cpu().numpy(), Yo).max() <= 1e-6


SHAPES = [
    # n, k, m, d, b, lda
    (6, 3, 1200, 500, 1, None),
    (5, 4, 37, 130, 1, 132),      # m % k != 0, ragged d, padded leading dimension
    (10, 5, 2003, 1029, 3, 1032),
    (20, 10, 613, 257, 8, 260),
    (32, 24, 1000, 640, 8, None),  # n - k = 8
    (32, 8, 190, 84, 2, None),     # n - k = 24: two encode passes
    (3, 2, 5, 7, 5, 8),            # fewer rows than one warp's group
    (16, 12, 3001, 4096, 4, None),
    (7, 3, 300, 9000, 6, 9004),    # several X chunks (b = 6 pads to 8)
    (12, 5, 700, 17000, 1, None),  # several X chunks at b = 1
    # the (25,23) code on the square, fat and tall matrices of Sec. III-F
    # (rows of 5750 floats padded to a 16-byte pitch)
    (25, 23, 5750, 5750, 1, 5752),
    (25, 23, 5750, 11500, 1, None),
    (25, 23, 11500, 5750, 1, 5752),
]


@pytest.mark.parametrize("n,k,m,d,b,lda", SHAPES)
def test_path_matches_oracle(cm, orc, n, k, m, d, b, lda):
    r = run_path(cm, orc, n, k, m, d, b, lda=lda, seed=n * 1000 + d)
    check_encode(orc, n, k, r["A_cpu"], r["P"], r["par"])
    check_workers(orc, n, k, r["A_cpu"], r["par"], r["X_cpu"], r["Yt"], r["code"].L)
    want = orc.matmul(r["A_cpu"].numpy(), r["X_cpu"].numpy())
    assert rel_l2_cols(r["Y"].cpu().numpy(), want).max() <= 1e-4


def _rows_per_unit(L, nw, warps):
    """The unit height rule of the b = 1 launch, restated: 4-row units when
    they fill the grid's rounds at least 2 points better than 8-row ones."""
    def fill(R):
        units = -(-L // R) * nw
        rounds = -(-units // warps)
        return units / (rounds * warps)
    return 4 if fill(4) >= fill(8) + 0.02 else 8


@pytest.mark.parametrize("n,k,m,d,want_R", [(32, 24, 65536, 64, 8), (10, 5, 12000, 256, 4),
                                            (20, 10, 8000, 128, 8), (6, 3, 1201, 300, 4)])
def test_unit_heights_at_b1(cm, orc, n, k, m, d, want_R):
    # b = 1 products run 8- or 4-row units depending on how the units fill the
    # persistent grid; both heights must give the same results
    warps = torch.cuda.get_device_properties(0).multi_processor_count * 8
    L = -(-m // k)
    if _rows_per_unit(L, n, warps) != want_R:
        pytest.skip("this GPU's SM count selects another height for the shape")
    r = run_path(cm, orc, n, k, m, d, 1, seed=31)
    check_workers(orc, n, k, r["A_cpu"], r["par"], r["X_cpu"], r["Yt"], r["code"].L)
    want = orc.matmul(r["A_cpu"].numpy(), r["X_cpu"].numpy())
    assert rel_l2_cols(r["Y"].cpu().numpy(), want).max() <= 1e-4
    # survivors only: the rule over nw = k workers may pick another height;
    # the blocks agree to the fp32 partial rounding
    Yt2 = cm.matvec_survivors(r["code"], r["A"], r["par"], r["X"], r["mask"])
    torch.cuda.synchronize()
    sel = r["code"].select_decodable(r["mask"])
    got, ref = Yt2.cpu().numpy(), r["Yt"].cpu().numpy()
    for j in range(n):
        if (sel >> j) & 1:
            blk = slice(j * L, (j + 1) * L)
            assert rel_l2_cols(got[blk], ref[blk]).max() <= 1e-6


@pytest.mark.parametrize("b", [1, 4, 8, 3])
def test_misaligned_x_uses_general_staging(cm, orc, b):
    n, k, m, d = 6, 3, 500, 301
    r = run_path(cm, orc, n, k, m, d, b, lda=304, misalign_x=True)
    check_workers(orc, n, k, r["A_cpu"], r["par"], r["X_cpu"], r["Yt"], r["code"].L)


def test_decode_from_every_k_subset(cm, orc):
    for n, k in [(6, 3), (10, 5)]:
        m, d, b = 301, 203, 2
        r = run_path(cm, orc, n, k, m, d, b, lda=204)
        want = orc.matmul(r["A_cpu"].numpy(), r["X_cpu"].numpy())
        for S in itertools.combinations(range(n), k):
            mask = sum(1 << j for j in S)
            Y = cm.decode(r["code"], r["Yt"], mask)
            err = rel_l2_cols(Y.cpu().numpy(), want)
            assert err.max() <= 1e-4, (S, err)


def _masks_with_e_missing(n, k, e, seed):
    """Two survivor masks with exactly e missing systematic blocks: the last
    e systematic and the first e parity workers, and a seeded scatter."""
    masks = [((1 << (k - e)) - 1) | (((1 << e) - 1) << k)]
    rng = np.random.default_rng(seed)
    miss = rng.choice(k, e, replace=False)
    keep = rng.choice(np.arange(k, n), e, replace=False)
    masks.append(sum(1 << j for j in range(k) if j not in miss) + sum(1 << int(j) for j in keep))
    return masks


@pytest.mark.parametrize("n,k,e", [(32, 24, 8), (32, 16, 9), (20, 10, 10), (26, 13, 12),
                                   (32, 16, 16)])
def test_decode_many_missing_blocks(cm, orc, n, k, e):
    """Large erasure counts (up to 16 rows of the inverse per column
    segment): the GPU decode of the GPU's worker results against the
    oracle's fp64 decode of the same results.  Both solve G_S exactly up to
    rounding, so they agree to the fp32 output rounding."""
    m, d, b = 37 * k + 5, 96, 3
    P = synth.parity_coefficients(n, k)
    code = cm.Code(n, k, m, d, P)
    A = synth.gaussian((m, d), 21).to(DEV)
    X = synth.gaussian((d, b), 22).to(DEV)
    par = cm.encode(code, A)
    Yt = cm.matvec(code, A, par, X)
    for mask in _masks_with_e_missing(n, k, e, seed=n * 100 + e):
        assert bin(mask).count("1") == k
        status = torch.zeros(1, dtype=torch.int32, device=DEV)
        Y = cm.decode(code, Yt, mask, status=status)
        torch.cuda.synchronize()
        assert status.item() == 0
        want = orc.decode(n, k, m, P.astype(np.float64), mask, Yt.cpu().numpy())
        err = rel_l2_cols(Y.cpu().numpy(), want)
        assert err.max() <= 1e-6, (hex(mask), err)


@pytest.mark.parametrize("n,k,e,b,m", [(6, 3, 2, 1, 3 * 60000 - 1), (32, 24, 8, 8, 24 * 5200),
                                       (20, 10, 10, 2, 10 * 40000 - 7)])
def test_decode_several_tiles_per_cta(cm, orc, n, k, e, b, m):
    """Problems with more than 152 x 256 row positions (L b) give every CTA of
    the decode several tiles: the first stages while the elimination runs,
    the later ones stage with every thread.  Own decode call and products +
    decode in one call, against the oracle's fp64 decode of the same
    results."""
    d = 16
    P = synth.parity_coefficients(n, k)
    code = cm.Code(n, k, m, d, P)
    assert code.L * b > 152 * 256
    A = synth.gaussian((m, d), 31).to(DEV)
    X = synth.gaussian((d, b), 32).to(DEV)
    par = cm.encode(code, A)
    Yt = cm.matvec(code, A, par, X)
    Yt_cpu = Yt.cpu().numpy()
    drawn = cm.draw_erasures(synth.ERASURE_SEED, 77, n, k)[0]
    for mask in _masks_with_e_missing(n, k, e, seed=n * 1000 + e) + [drawn]:
        status = torch.zeros(1, dtype=torch.int32, device=DEV)
        Y = cm.decode(code, Yt, mask, status=status)
        Yf = cm.matvec_decode(code, A, par, X, mask, status=status)
        torch.cuda.synchronize()
        assert status.item() == 0
        want = orc.decode(n, k, m, P.astype(np.float64), mask, Yt_cpu)
        assert rel_l2_cols(Y.cpu().numpy(), want).max() <= 1e-6, hex(mask)
        assert rel_l2_cols(Yf.cpu().numpy(), want).max() <= 1e-6, hex(mask)


def test_pass_through_is_rounded_to_nearest(cm):
    """Surviving systematic blocks are the fp64 results rounded to fp32 (to
    nearest, ties to even; the kernels convert by integer arithmetic): bit
    for bit equal to the device's own conversion, on values that include
    ties, fp32 subnormals, underflow to zero, overflow and signed zeros."""
    n, k, m = 6, 3, 3000
    code = cm.Code(n, k, m, 16, synth.parity_coefficients(n, k))
    L = code.L
    rng = np.random.default_rng(4)
    y = rng.standard_normal(n * L) * np.exp2(rng.integers(-160, 140, n * L))
    # exact ties: the 29 bits below the fp32 mantissa are 1000...0
    bits = y[:400].view(np.uint64)
    bits &= ~np.uint64((1 << 29) - 1)
    bits |= np.uint64(1 << 28)
    special = np.array([0.0, -0.0, 1e-40, -1e-40, 1e-46, 3e-45, 7e-46, 1.4e-45, 1e39, -1e39,
                        3.4028235677973366e38, 3.4028234663852886e38, np.inf, -np.inf,
                        1.1754942e-38, 5.877471754111438e-39, 1.0 + 2.0 ** -24, 1.0 + 3 * 2.0 ** -24])
    y[400:400 + len(special)] = special
    Yt = torch.from_numpy(y.reshape(n * L, 1)).to(DEV)
    Y = cm.decode(code, Yt, (1 << k) - 1)          # every systematic block survives
    torch.cuda.synchronize()
    want = Yt[:m].float()
    assert torch.equal(Y.view(torch.int32), want.view(torch.int32))
    # with a block to decode the survivors are staged for the decode as well;
    # the surviving systematic blocks 0 and 1 still pass through exactly
    Y = cm.decode(code, Yt, 0b001011)
    torch.cuda.synchronize()
    assert torch.equal(Y[:2 * L].view(torch.int32), want[:2 * L].view(torch.int32))


def test_extra_survivors_use_the_lowest_k(cm, orc):
    n, k, m, d = 10, 5, 400, 128
    r = run_path(cm, orc, n, k, m, d, 1)
    for mask in [0b1111111111, 0b1110111011, 0b1111100000 | 0b1]:
        lowest = 0
        for j in range(n):
            if mask >> j & 1 and bin(lowest).count("1") < k:
                lowest |= 1 << j
        a = cm.decode(r["code"], r["Yt"], mask).cpu()
        bb = cm.decode(r["code"], r["Yt"], lowest).cpu()
        assert torch.equal(a, bb)


@pytest.mark.parametrize("n", [4, 6])
def test_single_parity_integer_code_is_bit_exact(cm, orc, n):
    k = n - 1
    m, d = 1200, 500
    A = synth.small_integers((m, d), -4, 4, seed=11)
    X = synth.small_integers((d, 3), -4, 4, seed=12)
    code = cm.Code(n, k, m, d, np.ones((1, k), np.float32))
    Ad, Xd = A.to(DEV), X.to(DEV)
    par = cm.encode(code, Ad)
    Yt = cm.matvec(code, Ad, par, Xd)
    want = (A.long() @ X.long()).numpy()
    for erased in range(n):
        mask = ((1 << n) - 1) & ~(1 << erased)
        Y = cm.decode(code, Yt, mask)
        assert np.array_equal(Y.cpu().numpy().astype(np.int64), want), erased
        Yo = orc.decode(n, k, m, np.ones((1, k)), mask, Yt.cpu().numpy())
        assert np.array_equal(Yo, want.astype(np.float64))


def test_singular_generator_sets_status(cm):
    n, k, m, d = 6, 3, 90, 40
    P = synth.parity_coefficients(n, k)
    P[1] = P[0]                               # duplicated parity rows
    code = cm.Code(n, k, m, d, P)
    A = synth.gaussian((m, d), 3).to(DEV)
    X = synth.gaussian((d, 1), 4).to(DEV)
    par = cm.encode(code, A)
    Yt = cm.matvec(code, A, par, X)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    Y = torch.full((m, 1), 7.0, device=DEV)
    L = code.L
    cm.decode(code, Yt, 0b011001, Y=Y, status=status)     # survivors {0, 3, 4}
    torch.cuda.synchronize()
    assert status.item() == cm.CM_ESINGULAR
    assert torch.all(Y[L:] == 7.0)            # missing blocks 1, 2: not written
    assert torch.equal(Y[:L], Yt[:L].float()) # surviving block 0 passes through
    P2 = synth.parity_coefficients(n, k)
    P2[2] = 0.0                               # a zero parity row
    code2 = cm.Code(n, k, m, d, P2)
    status.zero_()
    cm.decode(code2, Yt, 0b100011, status=status)
    torch.cuda.synchronize()
    assert status.item() == cm.CM_ESINGULAR
    with pytest.raises(cm.CodedError) as e:
        cm.decode(code, Yt, 0b000011)
    assert e.value.status == cm.CM_ENOTDECODABLE


def test_singular_proportional_rows_and_well_posed_neighbours(cm, orc):
    """Two missing blocks take the closed-form inverse: with parity rows
    proportional by a power of two, q00 q11 - q01 q10 is zero exactly (fp32
    products are exact in fp64), so the set is flagged singular; the sets of
    the same code that avoid the pair decode to the oracle's Y = A X."""
    n, k, m, d = 6, 3, 90, 40
    P = synth.parity_coefficients(n, k)
    P[1] = 2.0 * P[0]                         # rows 3 and 4 of G proportional
    code = cm.Code(n, k, m, d, P)
    A = synth.gaussian((m, d), 5).to(DEV)
    X = synth.gaussian((d, 1), 6).to(DEV)
    par = cm.encode(code, A)
    Yt = cm.matvec(code, A, par, X)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    L = code.L
    Y = torch.full((m, 1), 7.0, device=DEV)
    cm.decode(code, Yt, 0b011001, Y=Y, status=status)     # survivors {0, 3, 4}: e = 2
    torch.cuda.synchronize()
    assert status.item() == cm.CM_ESINGULAR
    assert torch.all(Y[L:] == 7.0)
    want = orc.matmul(A.cpu().numpy().astype(np.float64), X.cpu().numpy().astype(np.float64))
    for mask in (0b101001, 0b110001, 0b101010, 0b100110, 0b001011):   # not both of rows 3, 4
        status.zero_()
        Y = cm.decode(code, Yt, mask, status=status)
        torch.cuda.synchronize()
        assert status.item() == cm.CM_OK, bin(mask)
        assert rel_l2_cols(Y.cpu().numpy(), want).max() <= 1e-4, bin(mask)


def test_concurrent_decodes_on_two_streams(cm, orc):
    """The decode keeps nothing between calls: hundreds of decodes queued on
    two streams at once (behind a device sleep, so they pile up and then run
    concurrently) each give the result of the same decode run alone."""
    n, k, m, d, b = 32, 24, 2000, 256, 2
    r = run_path(cm, orc, n, k, m, d, b)
    code, Yt = r["code"], r["Yt"]
    masks = [cm.draw_erasures(synth.ERASURE_SEED, 500 + i, n, k)[0] for i in range(300)]
    streams = [torch.cuda.Stream(), torch.cuda.Stream()]
    outs = [[torch.empty((m, b), device=DEV) for _ in masks] for _ in streams]
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    torch.cuda.synchronize()
    for si, st in enumerate(streams):
        with torch.cuda.stream(st):
            torch.cuda._sleep(20_000_000)
            order = masks if si == 0 else masks[::-1]
            for i, mask in enumerate(order):
                j = i if si == 0 else len(masks) - 1 - i
                cm.decode(code, Yt, mask, Y=outs[si][j], status=status)
    torch.cuda.synchronize()
    assert status.item() == 0
    want = orc.matmul(r["A_cpu"].numpy(), r["X_cpu"].numpy())
    for j, mask in enumerate(masks):
        alone = cm.decode(code, Yt, mask)
        torch.cuda.synchronize()
        assert torch.equal(outs[0][j], alone), j
        assert torch.equal(outs[1][j], alone), j
        if j % 50 == 0:
            assert rel_l2_cols(alone.cpu().numpy(), want).max() <= 1e-4


def test_outputs_stay_inside_their_buffers(cm):
    """Guard canaries after Yt, Y and the parity buffer stay untouched."""
    n, k, m, d, b = 10, 5, 1003, 515, 3
    P = synth.parity_coefficients(n, k)
    code = cm.Code(n, k, m, d, P)
    L = code.L
    A = padded(m, d, 516, 5)
    X = synth.gaussian((d, b), 6).to(DEV)
    G = 4096
    par_buf = torch.full(((n - k) * L * 516 + G,), 123.0, device=DEV)
    par = par_buf[:(n - k) * L * 516].view((n - k) * L, 516)[:, :d]
    yt_buf = torch.full((n * L * b + G,), 321.0, dtype=torch.float64, device=DEV)
    y_buf = torch.full((m * b + G,), 555.0, device=DEV)
    cm.encode(code, A, par)
    Yt = cm.matvec(code, A, par, X, Yt=yt_buf[:n * L * b].view(n * L, b))
    mask, _ = cm.draw_erasures(1, 1, n, k)
    cm.decode(code, Yt, mask, Y=y_buf[:m * b].view(m, b))
    torch.cuda.synchronize()
    assert torch.all(par_buf[(n - k) * L * 516:] == 123.0)
    assert torch.all(par_buf[:(n - k) * L * 516].view(-1, 516)[:, d:] == 123.0)
    assert torch.all(yt_buf[n * L * b:] == 321.0)
    assert torch.all(y_buf[m * b:] == 555.0)


def test_results_are_bitwise_repeatable(cm, orc):
    n, k, m, d, b = 16, 12, 3000, 3000, 8
    r = run_path(cm, orc, n, k, m, d, b)
    Yt2 = cm.matvec(r["code"], r["A"], r["par"], r["X"])
    par2 = cm.encode(r["code"], r["A"])
    Y2 = cm.decode(r["code"], Yt2, r["mask"])
    torch.cuda.synchronize()
    assert torch.equal(r["par"], par2)
    assert torch.equal(r["Yt"], Yt2)
    assert torch.equal(r["Y"], Y2)


def test_empty_and_degenerate_shapes(cm, orc):
    # one row, one column, k = 1 (repetition of a single block), n = k + 1
    for (n, k, m, d, b) in [(2, 1, 1, 1, 1), (3, 1, 5, 4, 2), (2, 1, 1, 129, 8), (32, 31, 31, 4, 1)]:
        r = run_path(cm, orc, n, k, m, d, b, lda=((d + 3) // 4) * 4)
        want = orc.matmul(r["A_cpu"].numpy(), r["X_cpu"].numpy())
        assert rel_l2_cols(r["Y"].cpu().numpy(), want).max() <= 1e-4


# ---- full-size workloads ---------------------------------------------------------------

def test_matvec_config_100_repeats(cm, orc):
    w = synth.MATVEC
    P = synth.parity_coefficients(w.n, w.k)
    code = cm.Code(w.n, w.k, w.m, w.d, P)
    A, X = synth.matvec_inputs(w, device="cpu")
    Ad, Xd = A.to(DEV), X.to(DEV)
    par = cm.encode(code, Ad)
    want = orc.matmul(A.numpy(), X.numpy())
    G = np.vstack([np.eye(w.k), P.astype(np.float64)])
    errs, kappas = [], []
    for rep in range(w.repeats):
        # each repeat: the n worker products, a fresh erasure set, a decode
        Yt = cm.matvec(code, Ad, par, Xd)
        mask, _ = cm.draw_erasures(synth.ERASURE_SEED, rep, w.n, w.k)
        assert mask == orc.draw_erasures(synth.ERASURE_SEED, rep, w.n, w.k)[0]
        Y = cm.decode(code, Yt, mask)
        errs.append(rel_l2_cols(Y.cpu().numpy(), want).max())
        kappas.append(np.linalg.cond(G[[j for j in range(w.n) if mask >> j & 1]]))
    worst = int(np.argmax(errs))
    assert max(errs) <= 1e-4, (max(errs), kappas[worst])


def test_decode_right_behind_the_products_reads_complete_results(cm):
    """cm_decode is launched as a programmatic dependent of the kernel before
    it: behind the products (which let dependents start during their last
    round) its staging threads must wait for the products to finish.  A
    decode issued right behind a long products launch equals, bit for bit,
    the same decode issued after a synchronize."""
    n, k, m, d, b = 32, 24, 8192, 16384, 8
    code = cm.Code(n, k, m, d, synth.parity_coefficients(n, k))
    g = torch.Generator().manual_seed(11)
    A = torch.randn((m, d), generator=g).to(DEV)
    X = torch.randn((d, b), generator=g).to(DEV)
    par = cm.encode(code, A)
    Yt = torch.empty((n * code.L, b), dtype=torch.float64, device=DEV)
    for c in range(4):
        mask, _ = cm.draw_erasures(synth.ERASURE_SEED, c, n, k)
        Yt.fill_(float("nan"))
        cm.matvec(code, A, par, X, Yt)
        Y_behind = cm.decode(code, Yt, mask)      # right behind the products
        torch.cuda.synchronize()
        Y_after = cm.decode(code, Yt, mask)       # after they are complete
        torch.cuda.synchronize()
        assert not torch.isnan(Y_behind).any()
        assert torch.equal(Y_behind, Y_after)


def test_bandwidth_config_every_element(cm, orc):
    """(32,24), A 65536 x 65536 fp32 (16 GiB), b = 8: the bench's launch
    configuration, checked element by element against the oracle: every
    parity element against the encode bound, every worker result against the
    oracle's products of the same coded blocks, every entry of the decoded Y
    against the plain A X.  The oracle runs on chunks of block rows (all
    blocks' rows r0 .. r1 at a time) to bound host memory."""
    w = synth.BANDWIDTH
    P = synth.parity_coefficients(w.n, w.k)
    code = cm.Code(w.n, w.k, w.m, w.d, P)
    L = code.L
    A, X = synth.matvec_inputs(w, device=DEV)
    par = cm.encode(code, A)
    Yt = cm.matvec(code, A, par, X)
    mask, _ = cm.draw_erasures(synth.ERASURE_SEED, 0, w.n, w.k)
    assert mask == orc.draw_erasures(synth.ERASURE_SEED, 0, w.n, w.k)[0]
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    Y = cm.decode(code, Yt, mask, status=status)
    torch.cuda.synchronize()
    assert status.item() == 0
    X_cpu = X.cpu()
    Yt_cpu = Yt.cpu().numpy()
    Y_cpu = Y.cpu().numpy()
    err2 = np.zeros(w.b)
    ref2 = np.zeros(w.b)
    chunk = 256
    for r0 in range(0, L, chunk):
        r1 = min(L, r0 + chunk)
        s = r1 - r0
        # sub-problem: block i of A_sub holds rows i L + r0 .. i L + r1 - 1 of the padded A
        idx = torch.tensor([i * L + r for i in range(w.k) for r in range(r0, r1)])
        valid = idx < w.m
        A_sub = torch.zeros((w.k * s, w.d))
        A_sub[valid] = A[idx[valid].to(DEV)].cpu()
        par_rows = torch.tensor([p * L + r for p in range(w.n - w.k) for r in range(r0, r1)])
        par_s = par[par_rows.to(DEV)].cpu()
        check_encode(orc, w.n, w.k, A_sub, P, par_s)
        rows = [j * L + r for j in range(w.n) for r in range(r0, r1)]
        check_workers(orc, w.n, w.k, A_sub, par_s, X_cpu, torch.from_numpy(Yt_cpu[rows]), s)
        want = orc.matmul(A_sub[valid].numpy(), X_cpu.numpy())
        got = Y_cpu[idx[valid].numpy()]
        err2 += ((got - want) ** 2).sum(axis=0)
        ref2 += (want ** 2).sum(axis=0)
        del A_sub, par_s
    # decoded A X, every entry: relative l2 error per output vector
    assert (np.sqrt(err2 / ref2)).max() <= 1e-4, np.sqrt(err2 / ref2)
    # surviving systematic blocks pass through exactly rounded
    for i in range(w.k):
        if mask >> i & 1:
            lo, hi = i * L, min((i + 1) * L, w.m)
            assert torch.equal(Y[lo:hi], Yt[lo:hi].float())
    # survivors only at full size: the k blocks the decode reads agree with
    # the all-worker products, the stragglers' rows are not written
    Ys = torch.full_like(Yt, float("nan"))
    cm.matvec_survivors(code, A, par, X, mask, Yt=Ys)
    torch.cuda.synchronize()
    sel = code.select_decodable(mask)
    for j in range(w.n):
        blk = slice(j * L, (j + 1) * L)
        if (sel >> j) & 1:
            assert rel_l2_cols(Ys[blk].cpu().numpy(), Yt_cpu[blk]).max() <= 1e-6, j
        else:
            assert bool(torch.isnan(Ys[blk]).all()), j
    del A, par, Yt, Ys
    torch.cuda.empty_cache()


def test_bounded_wait_gives_up_and_reports(cm):
    """Failure detection: the mbarrier wait that the TMA pipelines use gives
    up on a barrier nothing completes, writes CM_ETIMEOUT, and the context
    keeps working afterwards."""
    import time
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    t0 = time.perf_counter()
    cm.selftest_bounded_wait(status, 20_000_000)      # 20 ms
    torch.cuda.synchronize()
    dt = time.perf_counter() - t0
    assert status.item() == cm.CM_ETIMEOUT
    assert 0.015 < dt < 5.0, dt
    # the context is still usable: a normal coded product runs and is correct
    n, k, m, d = 6, 3, 90, 64
    code = cm.Code(n, k, m, d, synth.parity_coefficients(n, k))
    A = synth.gaussian((m, d), 8).to(DEV)
    X = synth.gaussian((d, 1), 9).to(DEV)
    status.zero_()
    Yt = cm.matvec(code, A, cm.encode(code, A), X, status=status)
    Y = cm.decode(code, Yt, 0b000111, status=status)
    torch.cuda.synchronize()
    assert status.item() == 0
    want = (A.double() @ X.double()).cpu().numpy()
    assert np.linalg.norm(Y.double().cpu().numpy() - want) <= 1e-5 * np.linalg.norm(want)


@pytest.mark.parametrize("n,k,m,d,b", [(10, 5, 2003, 1029, 1), (32, 24, 1000, 640, 8), (6, 3, 37, 130, 3)])
def test_survivors_only_products(cm, orc, n, k, m, d, b):
    """Survivors-only mode computes exactly the rows decode reads, leaves the
    stragglers' rows untouched, and decodes to the same A X."""
    r = run_path(cm, orc, n, k, m, d, b, lda=(d + 3) // 4 * 4)
    L = r["code"].L
    for counter in range(3):
        mask, _ = cm.draw_erasures(synth.ERASURE_SEED, 50 + counter, n, k)
        Yt = torch.full((n * L, b), 12345.0, dtype=torch.float64, device=DEV)
        cm.matvec_survivors(r["code"], r["A"], r["par"], r["X"], mask, Yt=Yt)
        Y = cm.decode(r["code"], Yt, mask)
        torch.cuda.synchronize()
        for j in range(n):
            blk = slice(j * L, (j + 1) * L)
            if mask >> j & 1:
                assert torch.equal(Yt[blk], r["Yt"][blk]), j   # same kernel, same sums
            else:
                assert torch.all(Yt[blk] == 12345.0), j        # never written
        want = orc.matmul(r["A_cpu"].numpy(), r["X_cpu"].numpy())
        assert rel_l2_cols(Y.cpu().numpy(), want).max() <= 1e-4


@pytest.mark.parametrize("n,k,m,d,b", [(12, 4, 1001, 300, 2), (10, 5, 2000, 512, 8), (6, 3, 77, 33, 1)])
def test_repetition_code_end_to_end(cm, orc, n, k, m, d, b):
    """n/k-repetition code (Example "Repetition codes"): parity blocks are
    exact copies, a decode from one replica per block reproduces the product
    of the systematic blocks exactly, and a set missing a block is refused."""
    code = cm.Code(n, k, m, d, "repetition")
    L = code.L
    A = padded(m, d, (d + 3) // 4 * 4, 31)
    X_cpu = synth.gaussian((d, b), 32)
    X = X_cpu.to(DEV)
    par = cm.encode(code, A)
    for p in range(n - k):                     # worker k + p copies block p mod k
        i = p % k
        rows = min(L, m - i * L)
        assert torch.equal(par[p * L:p * L + rows], A[i * L:i * L + rows])
    Yt = cm.matvec(code, A, par, X)
    Y_sys = cm.decode(code, Yt, (1 << k) - 1)  # all systematic workers
    rng = np.random.default_rng(7)
    tried = 0
    while tried < 12:
        mask = int(rng.integers(1, 1 << n))
        try:
            want_sel = orc.repetition_select(n, k, mask)
        except orc.OracleError:
            with pytest.raises(cm.CodedError) as e:
                cm.decode(code, Yt, mask)
            assert e.value.status == cm.CM_ENOTDECODABLE
            continue
        assert code.select_decodable(mask) == want_sel
        Y = cm.decode(code, Yt, mask)
        assert torch.equal(Y, Y_sys), hex(mask)
        tried += 1
    want = orc.matmul(A.cpu().numpy(), X_cpu.numpy())
    assert rel_l2_cols(Y_sys.cpu().numpy(), want).max() <= 1e-4
