"""Pins for the CPU oracle, checked against things other than the oracle.

Each test ties one oracle function to the paper's worked example, a closed
form, a library routine run on an equivalent problem, brute force, or exact
integer arithmetic, so that a dropped term, a wrong sign or index, or a
transposed operand in the oracle fails here.  No GPU is needed.
"""
import itertools
import math
import os

import numpy as np
import pytest
import torch

import synth
from conftest import ROOT, read_golden

pytestmark = pytest.mark.filterwarnings("ignore::DeprecationWarning")


def padded_blocks(A, k):
    """A (m x d) zero-padded to k L rows and reshaped to k blocks (k, L, d)."""
    m, d = A.shape
    L = -(-m // k)
    Ap = np.zeros((k * L, d), A.dtype)
    Ap[:m] = A
    return Ap.reshape(k, L, d)


# ---- Sec. I-A / Fig. 1: the (3,2) worked example ------------------------------

def test_fig1_toy_example(orc):
    g = read_golden("fig1_toy.txt")
    A1, A2 = np.array(g["A1 (2 x 3)"]), np.array(g["A2 (2 x 3)"])
    x = np.array(g["x (3)"]).reshape(3, 1)
    A = np.vstack([A1, A2]).astype(np.float32)
    P = np.array([[1.0, 1.0]])            # worker 3 stores A1 + A2
    par = orc.encode(3, 2, A, P)
    np.testing.assert_array_equal(par, np.array(g["parity A1+A2 (2 x 3)"]))
    Yt = orc.worker_outputs(3, 2, A, par.astype(np.float32), x.astype(np.float32))
    want = {0: g["W1 = A1 x"][0], 1: g["W2 = A2 x"][0], 2: g["W3 = (A1 + A2) x"][0]}
    for j in range(3):
        np.testing.assert_array_equal(Yt[2 * j:2 * j + 2, 0], want[j])
    full = np.concatenate([want[0], want[1]])
    for surv in ([0, 1], [0, 2], [1, 2]):        # any two products suffice
        mask = sum(1 << j for j in surv)
        Y = orc.decode(3, 2, 4, P, mask, Yt)
        np.testing.assert_array_equal(Y[:, 0], full)


# ---- Sec. I-A / III-A: the plain product Y = A X every decode is checked against

def test_matmul_reproduces_fig1_products(orc):
    # Fig. 1: A x is the concatenation of the two block products A1 x, A2 x,
    # worked by hand in the fixture (an exact integer case).
    g = read_golden("fig1_toy.txt")
    A = np.vstack([np.array(g["A1 (2 x 3)"]), np.array(g["A2 (2 x 3)"])])
    x = np.array(g["x (3)"]).reshape(3, 1)
    Y = orc.matmul(A.astype(np.float32), x.astype(np.float32))
    want = np.concatenate([g["W1 = A1 x"][0], g["W2 = A2 x"][0]])
    np.testing.assert_array_equal(Y[:, 0], want)


def test_matmul_small_integers_are_exact():
    # Integer A, X with |A|,|X| <= 4 and d = 500: every partial sum is an
    # integer below 2^53, so fp64 arithmetic must reproduce the int64 product
    # bit for bit, whatever the summation order.
    import oracle
    rng = np.random.default_rng(17)
    A = rng.integers(-4, 5, size=(1200, 500))
    X = rng.integers(-4, 5, size=(500, 3))
    Y = oracle.matmul(A.astype(np.float32), X.astype(np.float32))
    np.testing.assert_array_equal(Y, (A @ X).astype(np.float64))


@pytest.mark.parametrize("m,d,b", [(37, 101, 8), (5, 3, 7), (64, 33, 1)])
def test_matmul_multi_vector_matches_library(orc, m, d, b):
    # b > 1 and m != d: a transposed X index or a swapped operand shape
    # changes the result; numpy's fp64 product is the independent reference.
    rng = np.random.default_rng(m * 1000 + d)
    A = rng.standard_normal((m, d)).astype(np.float32)
    X = rng.standard_normal((d, b)).astype(np.float32)
    want = A.astype(np.float64) @ X.astype(np.float64)
    np.testing.assert_allclose(orc.matmul(A, X), want, rtol=1e-12, atol=1e-12)


# ---- Sec. III-A: encoding, systematic outputs, any-k decoding -----------------

def test_block_rows_padding(orc):
    assert orc.block_rows(1200, 3) == 400
    assert orc.block_rows(65536, 24) == 2731        # 24 * 2731 = 65544: 8 zero rows
    assert orc.block_rows(32768, 12) == 2731
    assert orc.block_rows(7, 7) == 1 and orc.block_rows(8, 7) == 2


@pytest.mark.parametrize("n,k,m,d", [(6, 3, 50, 17), (10, 5, 23, 9), (5, 4, 13, 6)])
def test_encode_matches_library_contraction(orc, n, k, m, d):
    rng = np.random.default_rng(1)
    A = rng.standard_normal((m, d)).astype(np.float32)
    P = rng.standard_normal((n - k, k))
    par, bound = orc.encode(n, k, A, P, with_bound=True)
    blocks = padded_blocks(A.astype(np.float64), k)
    want = np.einsum("pi,ird->prd", P, blocks).reshape(-1, d)
    np.testing.assert_allclose(par, want, rtol=0, atol=1e-12)
    np.testing.assert_allclose(bound, np.einsum("pi,ird->prd", np.abs(P), np.abs(blocks))
                               .reshape(-1, d), rtol=1e-14)
    # appended zero rows contribute nothing: parity of a block row past m only
    # sees the data blocks whose row exists.
    L = -(-m // k)
    if k * L > m:
        r = L - 1
        alive = [i for i in range(k) if i * L + r < m]
        want_r = sum(P[0, i] * A[i * L + r].astype(np.float64) for i in alive)
        np.testing.assert_allclose(par[r], want_r, atol=1e-12)


def test_systematic_outputs_are_uncoded_products(orc):
    # Sec. III-A: with a systematic code A'_i = A_i for i <= k, so worker i's
    # result is the uncoded block product.
    n, k, m, d, b = 6, 3, 61, 29, 3
    rng = np.random.default_rng(2)
    A = rng.standard_normal((m, d)).astype(np.float32)
    X = rng.standard_normal((d, b)).astype(np.float32)
    P = synth.parity_coefficients(n, k)
    par = orc.encode(n, k, A, P).astype(np.float32)
    Yt = orc.worker_outputs(n, k, A, par, X)
    L = -(-m // k)
    blocks = padded_blocks(A.astype(np.float64), k)
    for i in range(k):
        np.testing.assert_allclose(Yt[i * L:(i + 1) * L], blocks[i] @ X.astype(np.float64),
                                   rtol=1e-12, atol=1e-12)
    # parity workers: the given parity times X
    np.testing.assert_allclose(Yt[k * L:], par.astype(np.float64) @ X.astype(np.float64),
                               rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("n,k,m,d,b", [(6, 3, 31, 11, 2), (10, 5, 47, 13, 1)])
def test_decode_from_every_k_subset(orc, n, k, m, d, b):
    # Example "MDS codes" (Sec. III-B): every set of k indices is decodable.
    rng = np.random.default_rng(3)
    A = rng.standard_normal((m, d)).astype(np.float32)
    X = rng.standard_normal((d, b)).astype(np.float32)
    P = synth.parity_coefficients(n, k).astype(np.float64)
    par = orc.encode(n, k, A, P)
    Yt = orc.worker_outputs_f64(n, k, A, par, X)
    want = A.astype(np.float64) @ X.astype(np.float64)
    count = 0
    for S in itertools.combinations(range(n), k):
        mask = sum(1 << j for j in S)
        Y = orc.decode(n, k, m, P, mask, Yt)
        err = np.linalg.norm(Y - want) / np.linalg.norm(want)
        assert err < 1e-10, (S, err)
        count += 1
    assert count == math.comb(n, k)


@pytest.mark.parametrize("n", [4, 6])
def test_single_parity_integer_code_is_exact(orc, n):
    # Sec. III-A: the (n, n-1) code of the toy example generalised (parity =
    # sum of all blocks).  With small integers every product and sum is an
    # integer below 2^24, so results are exact; compare with int64 numpy.
    k = n - 1
    A = synth.small_integers((1200, 500), -4, 4, seed=11).numpy()
    X = synth.small_integers((500, 3), -4, 4, seed=12).numpy()
    P = np.ones((1, k))
    par = orc.encode(n, k, A, P)
    assert np.array_equal(par, np.round(par))
    Yt = orc.worker_outputs(n, k, A, par.astype(np.float32), X)
    want = A.astype(np.int64) @ X.astype(np.int64)
    for erased in range(n):
        mask = ((1 << n) - 1) & ~(1 << erased)
        Y = orc.decode(n, k, A.shape[0], P, mask, Yt)
        assert np.array_equal(Y, want.astype(np.float64)), erased


def test_decode_rejects_too_few_and_singular(orc):
    n, k = 6, 3
    P = synth.parity_coefficients(n, k).astype(np.float64)
    Yt = np.zeros((n * 4, 1))
    with pytest.raises(orc.OracleError, match="not decodable"):
        orc.decode(n, k, 12, P, 0b000011, Yt)
    Pdup = P.copy()
    Pdup[1] = Pdup[0]                       # two identical parity rows
    with pytest.raises(orc.OracleError, match="singular"):
        orc.decode(n, k, 12, Pdup, 0b011001, Yt)   # survivors {0, 3, 4}
    Pz = P.copy()
    Pz[2] = 0.0                             # a zero parity row
    with pytest.raises(orc.OracleError, match="singular"):
        orc.decode(n, k, 12, Pz, 0b100011, Yt)     # survivors {0, 1, 5}


def test_generator_inverse_matches_library(orc):
    n, k = 10, 5
    P = synth.parity_coefficients(n, k).astype(np.float64)
    G = np.vstack([np.eye(k), P])
    for S in [(0, 1, 2, 3, 4), (5, 6, 7, 8, 9), (0, 2, 5, 7, 9)]:
        mask = sum(1 << j for j in S)
        np.testing.assert_allclose(orc.generator_inverse(n, k, P, mask),
                                   np.linalg.inv(G[list(S)]), rtol=1e-10, atol=1e-12)


def test_bf16_paths_match_library(orc):
    n, k, m, d, N = 5, 3, 20, 16, 7
    A = synth.gaussian((m, d), 5, dtype=torch.bfloat16)
    B = synth.gaussian((d, N), 6, dtype=torch.bfloat16)
    P = synth.parity_coefficients(n, k).astype(np.float64)
    Abits = A.view(torch.int16).numpy().view(np.uint16)
    par = orc.encode_bf16(n, k, Abits, P)
    blocks = padded_blocks(A.float().double().numpy(), k)
    np.testing.assert_allclose(par, np.einsum("pi,ird->prd", P, blocks).reshape(-1, d),
                               atol=1e-12)
    parbits = torch.from_numpy(par).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    Bbits = B.view(torch.int16).numpy().view(np.uint16)
    Ct = orc.worker_outputs_bf16(n, k, Abits, parbits, Bbits)
    L = -(-m // k)
    coded = np.vstack([blocks.reshape(-1, d),
                       torch.from_numpy(parbits.view(np.int16)).view(torch.bfloat16)
                       .double().numpy()])
    np.testing.assert_allclose(Ct, coded @ B.double().numpy(), rtol=1e-12, atol=1e-12)


# ---- Sec. III-C/III-D: the straggler model -----------------------------------

def test_splitmix64_published_outputs(orc):
    with open(os.path.join(ROOT, "tests", "golden", "splitmix64.txt")) as f:
        rows = [l.split() for l in f if l.strip() and not l.startswith("#")]
    for seed, i, out in rows:
        assert orc.splitmix64(int(seed), int(i)) == int(out, 16)


def test_survivors_are_the_k_fastest(orc):
    for n, k in [(6, 3), (10, 5), (20, 10), (32, 24), (16, 12)]:
        for c in range(50):
            mask, t = orc.draw_erasures(synth.ERASURE_SEED, c, n, k)
            assert bin(mask).count("1") == k
            fastest = set(np.argsort(t, kind="stable")[:k].tolist())
            assert fastest == {j for j in range(n) if mask >> j & 1}
            assert np.all(t >= 1.0 / k)       # shift 1, scaled by 1/k


def harmonic(n):
    return sum(1.0 / i for i in range(1, n + 1))


@pytest.mark.parametrize("n,k,mu", [(10, 5, 1.0), (10, 10, 1.0), (20, 10, 2.0)])
def test_kth_arrival_mean_matches_closed_form(orc, n, k, mu):
    # Sec. III-D: E[T_MDS] = (1/k)(1 + (H_n - H_{n-k})/mu) (exact harmonic form;
    # k = n is the uncoded case (1/n)(1 + H_n/mu)).  5-sigma Monte-Carlo band.
    draws = 40000
    tk = np.empty(draws)
    for c in range(draws):
        _, t = orc.draw_erasures(12345, c, n, k, 1.0, mu)
        tk[c] = np.sort(t)[k - 1]
    mean = (1 + (harmonic(n) - harmonic(n - k)) / mu) / k
    var = sum(1.0 / (n - i) ** 2 for i in range(k)) / (k * mu) ** 2
    assert abs(tk.mean() - mean) < 5 * math.sqrt(var / draws), (tk.mean(), mean)


def test_kth_arrival_distribution_matches_F_mds(orc):
    # eq. for F_MDS: the k-th order statistic of n i.i.d. F(k t) times; for the
    # shifted exponential its CDF is the binomial tail sum_{i>=k} C(n,i) p^i (1-p)^(n-i)
    # with p = 1 - exp(-mu (k t - 1)).  Kolmogorov-Smirnov at the 1e-3 level.
    from scipy import stats
    n, k, mu = 10, 5, 1.0
    tk = np.array([np.sort(orc.draw_erasures(777, c, n, k, 1.0, mu)[1])[k - 1]
                   for c in range(20000)])

    def cdf(t):
        p = np.clip(1 - np.exp(-mu * (k * np.asarray(t) - 1)), 0, 1)
        return sum(math.comb(n, i) * p ** i * (1 - p) ** (n - i) for i in range(k, n + 1))
    assert stats.kstest(tk, cdf).pvalue > 1e-3


# ---- Sec. III-E: gradient descent -----------------------------------------------

def test_gd_converges_to_least_squares(orc):
    rng = np.random.default_rng(4)
    m, d = 60, 20
    A = rng.standard_normal((m, d)).astype(np.float32)
    y = rng.standard_normal(m).astype(np.float32)
    A64 = A.astype(np.float64)
    eta = 0.5 / (math.sqrt(m) + math.sqrt(d)) ** 2
    x = orc.gd(A, y, eta, 3000)
    x_ls = np.linalg.lstsq(A64, y.astype(np.float64), rcond=None)[0]
    assert np.linalg.norm(x - x_ls) / np.linalg.norm(x_ls) < 1e-10


def test_gd_matches_spectral_closed_form(orc):
    # x_0 = 0: x_t = sum_i (1 - (1 - eta l_i)^t) v_i v_i^T x_LS over the
    # eigenpairs (l_i, v_i) of A^T A.
    rng = np.random.default_rng(5)
    m, d, t = 80, 30, 50
    A = rng.standard_normal((m, d)).astype(np.float32)
    y = rng.standard_normal(m).astype(np.float32)
    A64 = A.astype(np.float64)
    eta = 0.5 / (math.sqrt(m) + math.sqrt(d)) ** 2
    lam, V = np.linalg.eigh(A64.T @ A64)
    x_ls = np.linalg.lstsq(A64, y.astype(np.float64), rcond=None)[0]
    want = V @ ((1 - (1 - eta * lam) ** t) * (V.T @ x_ls))
    x = orc.gd(A, y, eta, t)
    np.testing.assert_allclose(x, want, rtol=1e-10, atol=1e-12)


# ---- the seeded codes are MDS (reading of "(n,k) MDS code") ----------------------

@pytest.mark.parametrize("n,k", [(6, 3), (10, 5), (20, 10), (16, 12), (32, 24)])
def test_seeded_parity_is_mds(n, k):
    # G = [I; P] is MDS iff every square submatrix of P is nonsingular.
    P = synth.parity_coefficients(n, k).astype(np.float64)
    r = n - k
    worst = np.inf
    for s in range(1, min(r, k) + 1):
        cols = np.array(list(itertools.combinations(range(k), s)))
        for rows in itertools.combinations(range(r), s):
            sub = P[list(rows)]
            for c0 in range(0, len(cols), 200000):
                blk = sub[:, cols[c0:c0 + 200000]].transpose(1, 0, 2)
                worst = min(worst, np.abs(np.linalg.det(blk)).min())
    assert worst > 1e-9, worst


# ---- runtime model and repetition codes (Sec. III-B, III-C, III-D) --------------

@pytest.mark.parametrize("scheme,n,k", [("uncoded", 8, 8), ("repetition", 8, 4), ("mds", 8, 4)])
def test_oracle_runtime_simulator_matches_paper_forms(orc, scheme, n, k):
    # the simulated overall runtime follows the paper's distributions (eqs. for
    # F_uncoded, F_rep and the integral F_MDS, by quadrature) and their means
    from scipy import stats
    import oracle.runtime_model as rm
    T = orc.runtime_simulate(scheme, n, k, 1.0, 1.0, 4242, 0, 20000)
    cdf = {"uncoded": lambda t: rm.cdf_uncoded(t, n),
           "repetition": lambda t: rm.cdf_repetition(t, n, k),
           "mds": lambda t: rm.cdf_mds(t, n, k)}[scheme]
    assert stats.kstest(T[:3000], cdf).pvalue > 1e-3
    upper = 60.0 / (k if scheme != "uncoded" else n)
    mean = rm.mean_from_cdf(cdf, upper)
    assert abs(T.mean() - mean) < 5 * T.std() / math.sqrt(T.size)


def test_repetition_select_brute_force(orc):
    # Example "Repetition codes": a survivor set is decodable iff some k of its
    # members give a nonsingular G_S; the selection must be such a set, and
    # must fail exactly when none exists (brute force over all k-subsets)
    for n, k in [(6, 3), (8, 4), (6, 2)]:
        G = np.vstack([np.eye(k), orc.repetition_parity(n, k)])
        for mask in range(1 << n):
            surv = [j for j in range(n) if mask >> j & 1]
            ok = any(np.linalg.matrix_rank(G[list(S)]) == k
                     for S in itertools.combinations(surv, k)) if len(surv) >= k else False
            if ok:
                sel = orc.repetition_select(n, k, mask)
                S = [j for j in range(n) if sel >> j & 1]
                assert len(S) == k and set(S) <= set(surv)
                assert np.linalg.matrix_rank(G[S]) == k
            else:
                with pytest.raises(orc.OracleError):
                    orc.repetition_select(n, k, mask)
