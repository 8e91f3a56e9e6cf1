"""Runtime model of uncoded / repetition-coded / MDS-coded algorithms
(Sec. III-B, III-C, III-D), written from the paper's formulas with numpy and
scipy as plain steps.

TEST INFRASTRUCTURE: only tests/ and bench.py's CPU-baseline leg use this.

Mother distribution: the shifted exponential F(t) = 1 - exp(-mu (t - shift))
(eq. for the shifted-exponential model, shift 1 there); a job split l ways
runs each task with P(T <= t) = F(l t).
"""
from __future__ import annotations

import math

import numpy as np
from scipy import integrate, special


def mother_cdf(t, shift, mu):
    t = np.asarray(t, dtype=np.float64)
    return np.where(t >= shift, 1.0 - np.exp(-mu * (t - shift)), 0.0)


def mother_pdf(t, shift, mu):
    t = np.asarray(t, dtype=np.float64)
    return np.where(t >= shift, mu * np.exp(-mu * (t - shift)), 0.0)


def cdf_uncoded(t, n, shift=1.0, mu=1.0):
    """[F(n t)]^n: the last of n tasks of a 1/n split."""
    return mother_cdf(n * np.asarray(t, dtype=np.float64), shift, mu) ** n


def cdf_repetition(t, n, k, shift=1.0, mu=1.0):
    """Eq. for F_rep: [1 - [1 - F(k t)]^(n/k)]^k."""
    return (1.0 - (1.0 - mother_cdf(k * np.asarray(t, dtype=np.float64), shift, mu)) ** (n / k)) ** k


def cdf_mds(t, n, k, shift=1.0, mu=1.0):
    """Eq. for F_MDS as printed: the integral over [0, t] of
    n k f(k tau) C(n-1, k-1) F(k tau)^(k-1) [1 - F(k tau)]^(n-k), by quadrature."""
    c = n * k * math.comb(n - 1, k - 1)

    def dens(tau):
        F = float(mother_cdf(k * tau, shift, mu))
        return c * float(mother_pdf(k * tau, shift, mu)) * F ** (k - 1) * (1.0 - F) ** (n - k)

    out = []
    lo = shift / k          # the density vanishes below shift / k
    for ti in np.atleast_1d(t):
        if ti <= lo:
            out.append(0.0)
        else:
            out.append(integrate.quad(dens, lo, float(ti), limit=200, epsabs=1e-14,
                                      epsrel=1e-12)[0])
    return np.array(out)


def mean_from_cdf(cdf, upper):
    """E[T] = integral of (1 - F(t)) dt over [0, inf) for T >= 0, by quadrature."""
    return integrate.quad(lambda t: 1.0 - float(np.atleast_1d(cdf(t))[0]), 0.0, upper,
                          limit=400, epsabs=1e-13, epsrel=1e-11)[0]


def lambert_optimal_k(n, mu):
    """Lemma on optimal MDS-coded algorithms: k* = [1 + 1/W_{-1}(-e^{-mu-1})] n and
    gamma* = n T* = -W_{-1}(-e^{-mu-1}) / mu, with scipy's W_{-1}."""
    w = float(np.real(special.lambertw(-math.exp(-mu - 1.0), -1)))
    return (1.0 + 1.0 / w) * n, -w / mu


def mds_mean_log_form(n, k, mu, shift=1.0):
    """The expected MDS runtime with H_n - H_{n-k} ~ log(n / (n - k)) (Sec. III-D)."""
    return (shift + math.log(n / (n - k)) / mu) / k
