// Straggler draw of the shifted-exponential runtime model (Sec. III-C, III-D)
// and survivor selection of an MDS-coded run (eq. for the MDS runtime: the
// run ends at the k-th arrival).  Host-only integer work.
#include <algorithm>
#include <cmath>
#include <cstdint>

#include "../../include/cm.h"

namespace {

// SplitMix64 (Steele, Lea, Flood 2014): Weyl state advanced by the golden
// gamma, then the variant-13 style finaliser with the published constants.
inline uint64_t splitmix64_at(uint64_t seed, uint64_t index)
{
    uint64_t z = seed + index * 0x9E3779B97F4A7C15ull;
    z ^= z >> 30;
    z *= 0xBF58476D1CE4E5B9ull;
    z ^= z >> 27;
    z *= 0x94D049BB133111EBull;
    z ^= z >> 31;
    return z;
}

}  // namespace

extern "C" cm_status cm_draw_erasures(uint64_t seed, uint64_t counter, int32_t n,
                                      int32_t k, double shift, double rate,
                                      uint32_t *survivors, double *times)
{
    if (n < 1 || n > 32 || k < 1 || k > n || !(rate > 0.0) || !survivors) return CM_EINVAL;
    // Key of worker j: its 53-bit uniform (the time increases with it), then
    // its index, so that equal draws rank the lower index first.
    struct Key {
        uint64_t u53;
        int32_t j;
    } keys[32];
    for (int32_t j = 0; j < n; ++j) {
        uint64_t z = splitmix64_at(seed, counter * (uint64_t)n + (uint64_t)j + 1u);
        keys[j].u53 = z >> 11;
        keys[j].j = j;
        if (times) {
            double u = std::ldexp((double)keys[j].u53, -53);
            double e = -std::log1p(-u);                 // Exp(1) by inversion
            times[j] = (shift + e / rate) / (double)k;  // F(k t), shifted exp
        }
    }
    std::sort(keys, keys + n, [](const Key &a, const Key &b) {
        return a.u53 != b.u53 ? a.u53 < b.u53 : a.j < b.j;
    });
    uint32_t mask = 0;
    for (int32_t r = 0; r < k; ++r) mask |= 1u << keys[r].j;
    *survivors = mask;
    return CM_OK;
}
