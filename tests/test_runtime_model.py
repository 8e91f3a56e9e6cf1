"""Runtime model (Sec. III-B, III-C, III-D): the library's closed forms,
simulator and planner against the oracle's forms of the paper's equations
(the F_MDS integral by quadrature, means as integrals of 1 - F, scipy's
Lambert W), the paper's printed value 3.15, and Monte Carlo.  No GPU."""
import math

import numpy as np
import pytest

import synth


@pytest.fixture(scope="module")
def cm():
    import os
    import paper_1512_02673_gb300 as cm
    from paper_1512_02673_gb300 import build
    if not os.path.exists(cm.LIB_PATH):
        build.build()
    return cm


@pytest.fixture(scope="module")
def rm():
    import oracle.runtime_model as rm
    return rm


CASES = [("uncoded", 10, 10), ("repetition", 10, 5), ("mds", 10, 5), ("mds", 20, 10),
         ("mds", 32, 24), ("repetition", 12, 4), ("uncoded", 6, 6), ("mds", 6, 3)]


@pytest.mark.parametrize("scheme,n,k", CASES)
def test_simulator_is_bit_exact_with_oracle(cm, orc, scheme, n, k):
    for shift, rate in [(1.0, 1.0), (0.5, 3.0)]:
        a = cm.runtime_simulate(scheme, n, k, 2000, seed=17, counter0=5, shift=shift, rate=rate)
        b = orc.runtime_simulate(scheme, n, k, shift, rate, 17, 5, 2000)
        np.testing.assert_array_equal(a, b)


def test_simulated_mds_runtime_is_the_kth_arrival_of_the_erasure_draw(cm):
    # the MDS round ends at the k-th arrival: the slowest survivor of the draw
    n, k = 10, 5
    T = cm.runtime_simulate("mds", n, k, 50, seed=synth.ERASURE_SEED, counter0=0)
    for c in range(50):
        mask, times = cm.draw_erasures(synth.ERASURE_SEED, c, n, k)
        assert T[c] == max(times[j] for j in range(n) if mask >> j & 1)


@pytest.mark.parametrize("scheme,n,k", CASES)
def test_cdf_matches_paper_forms(cm, rm, scheme, n, k):
    t = np.linspace(0.0, 4.0 / k if scheme != "uncoded" else 4.0 / n, 41)
    F = cm.runtime_cdf(scheme, n, k, t)
    if scheme == "uncoded":
        want = rm.cdf_uncoded(t, n)
    elif scheme == "repetition":
        want = rm.cdf_repetition(t, n, k)
    else:
        want = rm.cdf_mds(t, n, k)          # the paper's integral, by quadrature
    np.testing.assert_allclose(F, want, atol=1e-10)


@pytest.mark.parametrize("scheme,n,k", CASES)
def test_means_are_integrals_of_the_tail(cm, rm, scheme, n, k):
    # E[T] = integral of 1 - F(t) over t >= 0, the library's harmonic forms
    # against quadrature of the library's own CDF and of the paper's forms
    for shift, rate in [(1.0, 1.0), (1.0, 0.25)]:
        mean = cm.runtime_mean(scheme, n, k, shift, rate)
        upper = (shift + 60.0 / rate) / (k if scheme != "uncoded" else n)
        if scheme == "uncoded":
            f = lambda t: rm.cdf_uncoded(t, n, shift, rate)
        elif scheme == "repetition":
            f = lambda t: rm.cdf_repetition(t, n, k, shift, rate)
        else:
            f = lambda t: rm.cdf_mds(t, n, k, shift, rate)
        assert abs(mean - rm.mean_from_cdf(f, upper)) < 1e-7 * mean


@pytest.mark.parametrize("scheme,n,k", [("uncoded", 10, 10), ("repetition", 10, 5), ("mds", 10, 5)])
def test_monte_carlo_agrees_with_closed_forms(cm, scheme, n, k):
    from scipy import stats
    T = cm.runtime_simulate(scheme, n, k, 200000, seed=99)
    mean = cm.runtime_mean(scheme, n, k)
    assert abs(T.mean() - mean) < 5 * T.std() / math.sqrt(T.size)
    assert stats.kstest(T, lambda t: cm.runtime_cdf(scheme, n, k, t)).pvalue > 1e-3


def test_mds_beats_repetition_beats_uncoded_at_paper_sizes(cm):
    # Fig. "runtime distributions": n = 10, k = 5, shifted exponential; the
    # MDS-coded runtime has the lightest tail (remark on dominance)
    t = np.linspace(0.1, 1.0, 50)
    fu = cm.runtime_cdf("uncoded", 10, 10, t)
    fr = cm.runtime_cdf("repetition", 10, 5, t)
    fm = cm.runtime_cdf("mds", 10, 5, t)
    assert np.all(fm >= fr - 1e-15)
    assert cm.runtime_mean("mds", 10, 5) < cm.runtime_mean("repetition", 10, 5)


def test_optimal_mds_rate_lambert(cm, rm):
    # Lemma on optimal MDS-coded algorithms; "3.15 away from the lower bound"
    # (gamma*(1), printed in Sec. III-D)
    k1, g1 = cm.optimal_mds_k(100, 1.0)
    assert abs(g1 - 3.15) < 0.005
    for mu in [0.1, 0.5, 1.0, 2.0, 10.0]:
        ks, g = cm.optimal_mds_k(100, mu)
        ks_or, g_or = rm.lambert_optimal_k(100, mu)
        assert abs(ks - ks_or) < 1e-9 * 100 and abs(g - g_or) < 1e-10 * g_or
        # k* minimises the log-form expected runtime: brute force on a fine grid
        grid = np.linspace(1.0, 99.999, 200001)
        vals = [(1.0 + math.log(100.0 / (100.0 - x)) / mu) / x for x in grid[::100]]
        x_best = grid[::100][int(np.argmin(vals))]
        assert abs(x_best - ks) < 0.1
        # gamma* = n T*: the minimum of n E[T] in the log form
        assert abs(100 * rm.mds_mean_log_form(100, ks, mu) - g) < 1e-9 * g


def test_repetition_code_decodable_sets(cm, orc):
    n, k = 12, 4                               # 3 replicas per block
    code = cm.Code(n, k, 400, 64, "repetition")
    rng = np.random.default_rng(0)
    for _ in range(300):
        mask = int(rng.integers(0, 1 << n))
        try:
            want = orc.repetition_select(n, k, mask)
        except orc.OracleError:
            with pytest.raises(cm.CodedError) as e:
                code.select_decodable(mask)
            assert e.value.status == cm.CM_ENOTDECODABLE
            continue
        assert code.select_decodable(mask) == want
    # a general code takes the first k survivors
    g = cm.Code(10, 5, 100, 64, synth.parity_coefficients(10, 5))
    assert g.select_decodable(0b1111111111) == 0b11111
    assert g.select_decodable(0b1101101101) == 0b0001101101
