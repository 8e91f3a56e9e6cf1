// Runtime model of uncoded, repetition-coded and MDS-coded distributed
// algorithms (Sec. III-B, III-C, III-D): closed-form means and distributions
// under the shifted-exponential mother distribution, a Monte-Carlo simulator
// that uses the same straggler draws as cm_draw_erasures, and the optimal
// MDS code rate of the lemma on optimal MDS-coded algorithms (Lambert W).
// Host-only.
#include <algorithm>
#include <cmath>
#include <cstdint>

#include "../../include/cm.h"

namespace {

inline uint64_t mix64(uint64_t seed, uint64_t index)
{
    uint64_t z = seed + index * 0x9E3779B97F4A7C15ull;
    z ^= z >> 30;
    z *= 0xBF58476D1CE4E5B9ull;
    z ^= z >> 27;
    z *= 0x94D049BB133111EBull;
    z ^= z >> 31;
    return z;
}

double harmonic(int n)
{
    double h = 0.0;
    for (int i = n; i >= 1; --i) h += 1.0 / i;   // small terms first
    return h;
}

bool valid(cm_scheme s, int32_t n, int32_t k, double rate)
{
    if (n < 1 || n > 1024 || !(rate > 0.0)) return false;
    if (s == CM_SCHEME_UNCODED) return true;
    if (k < 1 || k > n) return false;
    if (s == CM_SCHEME_REPETITION) return n % k == 0;
    return s == CM_SCHEME_MDS;
}

// Mother distribution F(t) = 1 - exp(-rate (t - shift)) for t >= shift.
double mother(double t, double shift, double rate)
{
    return t <= shift ? 0.0 : -std::expm1(-rate * (t - shift));
}

// log C(n, i)
double log_choose(int n, int i)
{
    return std::lgamma(n + 1.0) - std::lgamma(i + 1.0) - std::lgamma(n - i + 1.0);
}

// Lower branch W_{-1}(x) of the Lambert W function, x in [-1/e, 0): the
// solution w <= -1 of w e^w = x, by Halley's iteration from the branch-point
// series near -1/e or the asymptotic log form near 0.
double lambert_wm1(double x)
{
    const double e = std::exp(1.0);
    if (!(x >= -1.0 / e) || !(x < 0.0)) return NAN;
    double w;
    const double p = std::sqrt(std::max(0.0, 2.0 * (e * x + 1.0)));
    if (x < -0.25) {
        w = -1.0 - p - p * p / 3.0;
    } else {
        const double l1 = std::log(-x), l2 = std::log(-l1);
        w = l1 - l2 + l2 / l1;
    }
    for (int it = 0; it < 60; ++it) {
        const double ew = std::exp(w);
        const double f = w * ew - x;
        const double den = ew * (w + 1.0) - (w + 2.0) * f / (2.0 * w + 2.0);
        if (den == 0.0) break;
        const double step = f / den;
        w -= step;
        if (std::fabs(step) <= 1e-15 * std::fabs(w)) break;
    }
    return w;
}

}  // namespace

extern "C" {

cm_status cm_runtime_mean(cm_scheme scheme, int32_t n, int32_t k, double shift, double rate,
                          double *mean)
{
    if (!mean || !valid(scheme, n, k, rate)) return CM_EINVAL;
    switch (scheme) {
    case CM_SCHEME_UNCODED:   // max of n tasks of a 1/n split: H_n / rate in the exponential part
        *mean = (shift + harmonic(n) / rate) / n;
        break;
    case CM_SCHEME_REPETITION:   // max over k groups of the min of n/k replicas
        *mean = (shift + (double)k / n * harmonic(k) / rate) / k;
        break;
    default:   // MDS: k-th of n arrivals of a 1/k split
        *mean = (shift + (harmonic(n) - harmonic(n - k)) / rate) / k;
        break;
    }
    return CM_OK;
}

cm_status cm_runtime_cdf(cm_scheme scheme, int32_t n, int32_t k, double shift, double rate,
                         const double *t, int64_t count, double *F)
{
    if (!t || !F || count < 0 || !valid(scheme, n, k, rate)) return CM_EINVAL;
    for (int64_t i = 0; i < count; ++i) {
        double v;
        if (scheme == CM_SCHEME_UNCODED) {
            v = std::pow(mother(n * t[i], shift, rate), n);                 // [F(n t)]^n
        } else if (scheme == CM_SCHEME_REPETITION) {
            const double q = 1.0 - mother(k * t[i], shift, rate);
            v = std::pow(1.0 - std::pow(q, (double)n / k), k);               // eq. for F_rep
        } else {
            // k-th order statistic of n tasks with P(T <= t) = F(k t): the
            // binomial tail, equal to the integral form of the paper
            const double p = mother(k * t[i], shift, rate);
            if (p <= 0.0) {
                v = 0.0;
            } else if (p >= 1.0) {
                v = 1.0;
            } else {
                v = 0.0;
                for (int j = k; j <= n; ++j)
                    v += std::exp(log_choose(n, j) + j * std::log(p) + (n - j) * std::log1p(-p));
                v = std::min(1.0, v);
            }
        }
        F[i] = v;
    }
    return CM_OK;
}

cm_status cm_runtime_simulate(cm_scheme scheme, int32_t n, int32_t k, double shift, double rate,
                              uint64_t seed, uint64_t counter0, int64_t count, double *T)
{
    if (!T || count < 0 || n > 32 || !valid(scheme, n, k, rate)) return CM_EINVAL;
    const int kk = scheme == CM_SCHEME_UNCODED ? n : k;   // ways the job is split
    double times[32];
    for (int64_t c = 0; c < count; ++c) {
        const uint64_t counter = counter0 + (uint64_t)c;
        for (int j = 0; j < n; ++j) {
            const uint64_t z = mix64(seed, counter * (uint64_t)n + (uint64_t)j + 1u);
            const double u = std::ldexp((double)(z >> 11), -53);
            times[j] = (shift - std::log1p(-u) / rate) / kk;
        }
        double r;
        if (scheme == CM_SCHEME_UNCODED) {
            r = *std::max_element(times, times + n);
        } else if (scheme == CM_SCHEME_REPETITION) {
            // block i is held by workers i, i + k, i + 2k, ... (n/k replicas)
            r = 0.0;
            for (int i = 0; i < k; ++i) {
                double g = times[i];
                for (int j = i + k; j < n; j += k) g = std::min(g, times[j]);
                r = std::max(r, g);
            }
        } else {
            std::nth_element(times, times + (k - 1), times + n);
            r = times[k - 1];
        }
        T[c] = r;
    }
    return CM_OK;
}

cm_status cm_optimal_mds_k(int32_t n, double rate, double *k_star, double *gamma_star)
{
    if (n < 1 || !(rate > 0.0) || !k_star || !gamma_star) return CM_EINVAL;
    const double w = lambert_wm1(-std::exp(-rate - 1.0));
    if (!std::isfinite(w)) return CM_EINVAL;
    *k_star = (1.0 + 1.0 / w) * n;
    *gamma_star = -w / rate;
    return CM_OK;
}

}  // extern "C"
