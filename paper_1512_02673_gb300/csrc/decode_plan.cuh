// The decode plan of one survivor mask (Sec. III-A, last paragraph; Example
// "MDS codes"), formed inside the CTA that applies it.
//
// With S the k survivors used (ascending), the surviving results satisfy
// Yt_S = G_S Z, Z the k uncoded block products.  G_S has a unit row for every
// surviving systematic worker (S[0, ks)) and a parity row P[p] for every
// surviving parity worker (Ps, |Ps| = e, the number of missing systematic
// blocks M).  Gauss-Jordan on G_S that takes the unit rows as the first
// ks = k - e pivots (exact: they are unit vectors) leaves the e x e block
// Q = P[Ps][M]; with Q^-1 the rows of G_S^-1 for the missing blocks are
//   D[c][ks + a] =  Q^-1[c][a]                            (parity survivor Ps[a])
//   D[c][p]      = -sum_a Q^-1[c][a] P[Ps[a]][S[p]]        (systematic survivor S[p])
// and missing block M[c] = sum_p D[c][p] Yt_S[p].
//
// Every CTA that applies a decode forms the plan itself in shared memory, so
// a decode is one launch and keeps no state between calls:
//  * plan_setup (all threads): P into shared memory (16-byte loads of the
//    parameter space), the survivor lists by ballots in warp 0.
//  * plan_eliminate (one warp for e <= 4, else four warps, one per
//    scheduler; e <= 2 in closed form, adj(Q) / det Q, by one warp):
//    Q^-1 in fp64 with [Q | I] held in registers, its 2e^2
//    entries spread over the threads.  The pivot search is one warp
//    reduction over the threads holding the pivot column; that warp hands
//    the pivot key and the column to the others through shared memory (one
//    named barrier per column), and the pivot row travels by shuffles.  The
//    elimination is fraction-free and exchanges no rows: at column c with
//    pivot row b (the largest |W[r][c]| among rows not yet used, compared on
//    the leading 28 bits of the magnitude, lowest row on near-ties) every
//    other row r becomes 2^-s (piv W[r] - W[r][c] W[b]), 2^s the pivot's
//    binade (an exact scale that keeps the rows from growing by a product of
//    pivots).  Afterwards row prow[c] holds column c's pivot d_c and
//    Q^-1[c][a] = W[prow[c]][e + a] / d_c, kept as (high, low) fp32 pairs.
//  * G_S counts as singular when a pivot (det Q for e <= 2) is zero,
//    subnormal or not finite, or when ||Q||_inf ||Q^-1||_inf, bounded by
//    (e max|Q|)(e max|Q^-1|), exceeds 1 / (64 eps) (evaluated in fp32: it is
//    a threshold).
//  * plan_rows (all threads; the matrix decode): the rows D[c][p] above, from
//    the (high, low) pairs of Q^-1 and the exact fp32 values of P in
//    double-float arithmetic.  The vector decode applies the same rows in two
//    factors instead, Q^-1 (Yt_Ps - P[Ps][S_sys] Yt_S_sys).
//
// fp64 runs at a small fraction of the fp32 rate on this part: each warp
// gets about one fp64 instruction per 64 cycles, whatever the independence
// of its instructions, and a division takes about 430 cycles.  So
// conversions and magnitude compares go through integer bit manipulation,
// each column of the elimination costs one fp64 multiply and one fp64 fma per
// entry a thread holds (1 for e <= 8, 4 for e <= 16), spread over warps on
// different schedulers, and the only divisions are the e reciprocals of the
// pivots (the e^2 entries of adj(Q) / det Q for e <= 2), taken in parallel.
#pragma once

#include <cfloat>

#include "cm_internal.cuh"

namespace cm_plan {

constexpr int kMaxE = 16;   // e <= min(k, n - k) <= 16 for n <= 32

struct Plan {
    int32_t e;                    // missing systematic blocks
    int32_t singular;             // G_S judged singular: decode nothing
    int32_t S[CM_MAX_N];          // survivors used, ascending (k of them)
    int32_t Ps[kMaxE];            // surviving parity workers, ascending
    int32_t M[kMaxE];             // missing systematic blocks, ascending
    int32_t prow[kMaxE];          // pivot row of each column
    __align__(16) float P[CM_MAX_P];   // the parity coefficients ((n - k) x k)
    double W[kMaxE][2 * kMaxE];   // the eliminated [Q | I], rows x columns
    double rcp[kMaxE];            // 1 / d_c
    float Qh[kMaxE][kMaxE];       // Q^-1[c][a], high part
    float Ql[kMaxE][kMaxE];       // Q^-1 - Qh
    double fbuf[2][kMaxE];        // the pivot column's entries, per column (double buffered)
    uint32_t kbuf[2];             // the pivot key, per column
};

// x 2^-s for a power-of-two scale, exact, by bit manipulation of the
// exponent (no branch); zero, subnormal and underflowing values give a zero of
// the same sign (they are below 2^-1022 and only ever meet entries of order
// one).
__device__ __forceinline__ double scale_pow2(double x, int s)
{
    const long long b = __double_as_longlong(x);
    const int ex = (int)((b >> 52) & 0x7FF);
    const long long sign = b & (long long)0x8000000000000000ull;
    const long long scaled = (b & ~(0x7FFll << 52)) | ((long long)(ex - s) << 52);
    return __longlong_as_double(ex == 0 || ex - s <= 0 ? sign : scaled);
}

// fp64 -> fp32 rounded to nearest, ties to even (IEEE 754), by integer
// arithmetic: the 52-bit significand keeps its leading 24 bits (with the
// implicit one) and the 29 (or, for fp32 subnormal results, more) bits below
// decide the rounding; a carry out of the significand moves into the exponent
// field, which also turns the largest values into infinity.  Not-a-number
// stays not-a-number (quiet).
__device__ __forceinline__ float rne_float(double x)
{
    const unsigned long long b = (unsigned long long)__double_as_longlong(x);
    const uint32_t sign = (uint32_t)(b >> 32) & 0x80000000u;
    const int ex = (int)((b >> 52) & 0x7FF);
    const unsigned long long man = b & 0xFFFFFFFFFFFFFull;
    if (ex == 0x7FF)
        return __uint_as_float(sign | 0x7F800000u | (man ? 0x400000u : 0u));
    const int e32 = ex - 1023 + 127;
    if (e32 >= 255) return __uint_as_float(sign | 0x7F800000u);
    // significand with the implicit one (none for fp64 zeros and subnormals,
    // which are far below the fp32 range and round to zero below)
    const unsigned long long sig = ex ? (man | (1ull << 52)) : man;
    // bits dropped: 29 for a normal fp32 result, more below its range
    const int shift = e32 >= 1 ? 29 : 29 + 1 - e32;
    if (shift > 54) return __uint_as_float(sign);
    const unsigned long long q = sig >> shift;
    const unsigned long long rem = sig & ((1ull << shift) - 1ull);
    const unsigned long long half = 1ull << (shift - 1);
    const uint32_t up = (rem > half || (rem == half && (q & 1ull))) ? 1u : 0u;
    // normal: exponent field e32 - 1 plus the significand with its implicit
    // one (which adds the last 1); subnormal: the shifted significand alone
    const uint32_t bits = e32 >= 1 ? ((uint32_t)(e32 - 1) << 23) + (uint32_t)q + up
                                   : (uint32_t)q + up;
    return __uint_as_float(sign | bits);
}

// fp64 value of an fp32 value by bit manipulation (exact).
__device__ __forceinline__ double exact_double(float f)
{
    const uint32_t u = __float_as_uint(f);
    const uint32_t ex = (u >> 23) & 0xFFu, man = u & 0x7FFFFFu;
    const unsigned long long sign = (unsigned long long)(u >> 31) << 63;
    if (ex == 0xFFu)   // infinite or not a number
        return __longlong_as_double((long long)(sign | 0x7FF0000000000000ull |
                                                ((unsigned long long)man << 29)));
    if (ex == 0) {     // zero or subnormal: normalise the mantissa
        if (man == 0) return __longlong_as_double((long long)sign);
        const int sh = __clz((int)man) - 8;   // shifts that bring the top bit to bit 23
        const uint32_t m = (man << sh) & 0x7FFFFFu;
        return __longlong_as_double((long long)(sign | ((unsigned long long)(897 - sh) << 52) |
                                                ((unsigned long long)m << 29)));
    }
    return __longlong_as_double((long long)(sign | ((unsigned long long)(ex + 896) << 52) |
                                            ((unsigned long long)man << 29)));
}

// (high, low) fp32 pair of an fp64 value by bit manipulation: high carries the
// leading 24 significant bits (truncated), low the next 29 rounded to 24;
// together about 47 bits.  Values outside the fp32 normal range fall back to a
// rounded conversion (they do not occur for worker results of finite data).
__device__ __forceinline__ void split_double(double y, float &h, float &l)
{
    const unsigned long long b = (unsigned long long)__double_as_longlong(y);
    const uint32_t hi = (uint32_t)(b >> 32), lo = (uint32_t)b;
    const int ex = (int)((hi >> 20) & 0x7FF);
    if (ex < 1023 - 100 || ex > 1023 + 127) {
        h = __double2float_rn(y);
        l = 0.f;
        return;
    }
    const uint32_t sign = hi & 0x80000000u;
    const uint32_t m23 = ((hi & 0xFFFFFu) << 3) | (lo >> 29);
    h = __int_as_float((int)(sign | ((uint32_t)(ex - 1023 + 127) << 23) | m23));
    const uint32_t r29 = lo & 0x1FFFFFFFu;
    // low = r29 * 2^(ex - 1075); below the fp32 normal range it is dropped
    // (it is then under 2^-100 relative to fp32 precision of |y| >= 2^-75)
    const int se = ex - 1075 + 127;
    const float scale = se > 0 ? __int_as_float(se << 23) : 0.f;
    l = __uint_as_float(sign | __float_as_uint(__uint2float_rn(r29) * scale));
}

// split_double and rne_float of the same value, sharing the bit extraction:
// in split_double's own range the rounded value is the truncated high part
// plus one unit in its last place when the 29 dropped bits are above half,
// or exactly half with an odd last bit (a carry moves into the exponent, up
// to infinity, as rounding does); elsewhere rne_float itself.
__device__ __forceinline__ void split_round(double y, float &h, float &l, float &r)
{
    const unsigned long long b = (unsigned long long)__double_as_longlong(y);
    const uint32_t hi = (uint32_t)(b >> 32), lo = (uint32_t)b;
    const int ex = (int)((hi >> 20) & 0x7FF);
    if (ex < 1023 - 100 || ex > 1023 + 127) {
        h = __double2float_rn(y);
        l = 0.f;
        r = rne_float(y);
        return;
    }
    const uint32_t sign = hi & 0x80000000u;
    const uint32_t m23 = ((hi & 0xFFFFFu) << 3) | (lo >> 29);
    const uint32_t hb = sign | ((uint32_t)(ex - 1023 + 127) << 23) | m23;
    h = __uint_as_float(hb);
    const uint32_t r29 = lo & 0x1FFFFFFFu;
    const int se = ex - 1075 + 127;
    const float scale = se > 0 ? __int_as_float(se << 23) : 0.f;
    l = __uint_as_float(sign | __float_as_uint(__uint2float_rn(r29) * scale));
    const uint32_t up = (r29 > 0x10000000u || (r29 == 0x10000000u && (m23 & 1u))) ? 1u : 0u;
    r = __uint_as_float(hb + up);
}

// (sh, sl) += (dh + dl) * (yh + yl), to about 2^-44 relative per term.  The
// rounded operations are explicit intrinsics, which the compiler never
// contracts into fused multiply-adds (that would break the error terms).
__device__ __forceinline__ void df_fma(float dh, float dl, float yh, float yl, float &sh, float &sl)
{
    const float p = __fmul_rn(dh, yh);
    const float pe = __fmaf_rn(dh, yh, -p);                  // exact error of p
    const float t = __fmaf_rn(dh, yl, __fmul_rn(dl, yh));    // cross terms
    const float s1 = __fadd_rn(sh, p);                       // TwoSum(sh, p)
    const float bb = __fsub_rn(s1, sh);
    const float err = __fadd_rn(__fsub_rn(sh, __fsub_rn(s1, bb)), __fsub_rn(p, bb));
    sl = __fadd_rn(sl, __fadd_rn(err, __fadd_rn(pe, t)));
    sh = s1;
}

// (sh, sl) += d (yh + yl) for an fp32 coefficient d (df_fma with a zero low
// part, one rounded product fewer).
__device__ __forceinline__ void df_fma1(float d, float yh, float yl, float &sh, float &sl)
{
    const float p = __fmul_rn(d, yh);
    const float pe = __fmaf_rn(d, yh, -p);                   // exact error of p
    const float t = __fmul_rn(d, yl);
    const float s1 = __fadd_rn(sh, p);                       // TwoSum(sh, p)
    const float bb = __fsub_rn(s1, sh);
    const float err = __fadd_rn(__fsub_rn(sh, __fsub_rn(s1, bb)), __fsub_rn(p, bb));
    sl = __fadd_rn(sl, __fadd_rn(err, __fadd_rn(pe, t)));
    sh = s1;
}

__device__ __forceinline__ double shfl_double(double v, int src)
{
    const long long b = __double_as_longlong(v);
    const int lo = __shfl_sync(0xffffffffu, (int)(b & 0xffffffffll), src);
    const int hi = __shfl_sync(0xffffffffu, (int)(b >> 32), src);
    return __longlong_as_double(((long long)hi << 32) | (unsigned int)lo);
}

// Missing systematic blocks of a survivor mask whose set bits are the k
// survivors used.
__host__ __device__ __forceinline__ int missing_blocks(int k, uint32_t survivors)
{
    const uint32_t sys = k < 32 ? survivors & ((1u << k) - 1u) : survivors;
#ifdef __CUDA_ARCH__
    return k - __popc(sys);
#else
    return k - __builtin_popcount(sys);
#endif
}

// P into shared memory and the survivor lists (warp 0, ballots).  Every
// thread of the CTA calls it; it ends with a CTA barrier.  `survivors` has
// exactly k set bits.
__device__ __forceinline__ void plan_setup(const CodeParams &cp, uint32_t survivors, Plan &pl)
{
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int nwarps = blockDim.x >> 5;
    const int n = cp.n, k = cp.k;
    // 16-byte loads of the parameter space, lane l of warp w taking float4
    // number w + nwarps l (at most one per thread for CTAs of 64 threads or
    // more: (n - k) k <= 256 floats); the first is loaded before the ballots
    // and stored after them, so that its latency covers them
    const int n4 = ((n - k) * k + 3) / 4;
    const float4 *P4 = reinterpret_cast<const float4 *>(cp.P);
    float4 *S4 = reinterpret_cast<float4 *>(pl.P);
    const int i0 = warp + nwarps * lane;
    float4 v0 = make_float4(0.f, 0.f, 0.f, 0.f);
    if (i0 < n4) v0 = P4[i0];
    if (warp == 0) {
        const uint32_t below = (1u << lane) - 1u;
        const bool sel = lane < n && ((survivors >> lane) & 1u);
        const bool miss = lane < k && !sel;
        const uint32_t missm = __ballot_sync(0xffffffffu, miss);
        const bool par = sel && lane >= k;
        const uint32_t parm = __ballot_sync(0xffffffffu, par);
        if (sel) pl.S[__popc(survivors & below)] = lane;
        if (par) pl.Ps[__popc(parm & below)] = lane;
        if (miss) pl.M[__popc(missm & below)] = lane;
        if (lane == 0) {
            pl.e = __popc(missm);
            pl.singular = 0;
        }
    }
    if (i0 < n4) S4[i0] = v0;
    for (int i = i0 + nwarps * 32; i < n4; i += nwarps * 32) S4[i] = P4[i];
    __syncthreads();
}

// Named barrier among the NW eliminating warps (barrier 1; 0 is
// __syncthreads).
template <int NW>
__device__ __forceinline__ void elim_sync()
{
    if (NW == 1) __syncwarp();
    else asm volatile("bar.sync 1, %0;\n" ::"r"(NW * 32) : "memory");
}

// Q^-1 for e <= 2 in closed form, by warp 0 alone (no barrier: the other
// eliminating warps return at once).  Q's entries are fp32 values, so their
// products are exact in fp64: det Q = q00 q11 - q01 q10 carries one rounding
// and Q^-1 = adj(Q) / det Q one more per entry, against a pivot, a scaling
// and a reciprocal per column of the elimination.  G_S counts as singular when
// det Q (Q itself for e = 1) is zero, subnormal or not finite (exactly when Q
// is singular, short of overflow and underflow), or by the elimination's
// condition bound.
__device__ __forceinline__ void plan_inverse_small(Plan &pl, int k)
{
    const int t = threadIdx.x;
    if (t >= 32) return;
    const int e = pl.e;
    // Q[r][j] = P[Ps[r]][M[j]]: row r a surviving parity worker, column j a
    // missing block
    const float f00 = pl.P[(pl.Ps[0] - k) * k + pl.M[0]];
    const float f01 = e == 2 ? pl.P[(pl.Ps[0] - k) * k + pl.M[1]] : 0.f;
    const float f10 = e == 2 ? pl.P[(pl.Ps[1] - k) * k + pl.M[0]] : 0.f;
    const float f11 = e == 2 ? pl.P[(pl.Ps[1] - k) * k + pl.M[1]] : 0.f;
    const float qmax = fmaxf(fmaxf(fabsf(f00), fabsf(f01)), fmaxf(fabsf(f10), fabsf(f11)));
    const double q00 = exact_double(f00), q01 = exact_double(f01);
    const double q10 = exact_double(f10), q11 = exact_double(f11);
    const double det = e == 1 ? q00 : __dsub_rn(__dmul_rn(q00, q11), __dmul_rn(q01, q10));
    const uint32_t ef =
        (uint32_t)((unsigned long long)__double_as_longlong(det) >> 52) & 0x7FFu;
    bool sing = ef == 0u || ef == 0x7FFu;
    float qi = 0.f;
    if (!sing && t < e * e) {
        const int c = t / e, a = t - c * e;      // Q^-1[c][a] = adj(Q)[c][a] / det Q
        double adj = 1.0;                        // e = 1
        if (e == 2) {
            if (c == a) adj = c == 0 ? q11 : q00;
            else adj = c == 0 ? -q01 : -q10;
        }
        float h, l;
        split_double(adj / det, h, l);
        pl.Qh[c][a] = h;
        pl.Ql[c][a] = l;
        qi = fabsf(h);
    }
    qi = __uint_as_float(__reduce_max_sync(0xffffffffu, __float_as_uint(qi)));
    // not-a-number fails the comparison and counts as singular
    if (!sing && !((float)e * qmax * ((float)e * qi) < (float)(1.0 / (64.0 * DBL_EPSILON))))
        sing = true;
    if (t == 0 && sing) pl.singular = 1;
}

// Q^-1 by the first NW warps of the CTA (1, or 4: one per scheduler, since
// each warp gets about one fp64 instruction per 64 cycles); EMAX >= e is a
// power of two (4, 8 or 16) with 2 EMAX^2 >= 32 NW.  The 2 EMAX x EMAX
// entries of [Q | I] are spread over the T = 32 NW threads: thread t holds
// row r = t % EMAX of the columns j = t / EMAX + (T / EMAX) i, i < EPL =
// 2 EMAX^2 / T (1 with EMAX = 4, NW = 1 or EMAX = 8, NW = 4; 4 with EMAX = 16,
// NW = 4).  Column c thus lives in entry c / (T / EMAX) of the EMAX
// consecutive threads from (c % (T / EMAX)) EMAX, one row each, inside one
// warp: the pivot search is one reduction in that warp, which hands the
// pivot key and its rows' multipliers to the other warps through shared
// memory (double buffered, one barrier per column); every thread takes its
// columns' pivot-row entries from its own EMAX threads by shuffles.  Writes
// W, rcp, prow, the (high, low) pairs of Q^-1 and, for a singular G_S, the
// flag.  Pivot keys:
// the upper 32 bits of |W[r][c]| with their lowest 4 bits replaced by
// 15 - r, so the maximum is the largest magnitude to 2^-16 relative, the
// lowest row among those; exponent field 0 (zero, subnormal) or all ones
// (infinite, not a number) marks G_S singular.
template <int EMAX, int NW>
__device__ __forceinline__ void plan_eliminate(Plan &pl, int k)
{
    constexpr int T = 32 * NW;
    constexpr int SL = T / EMAX;                 // column slots
    constexpr int EPL = 2 * EMAX * EMAX / T;     // entries per thread
    static_assert(EPL >= 1 && SL * EPL == 2 * EMAX, "layout");
    if (pl.e <= 2) {
        plan_inverse_small(pl, k);
        return;
    }
    const int t = threadIdx.x;
    const int lane = t & 31;
    const int e = pl.e;
    const int r = t & (EMAX - 1);                // this thread's row
    const int slot = t / EMAX;                   // this thread's column slot
    const int seg0 = lane & ~(EMAX - 1);         // lane of row 0 of this slot
    double w[EPL];
    float qmax = 0.f;
#pragma unroll
    for (int i = 0; i < EPL; ++i) {
        const int j = slot + SL * i;
        double v = 0.0;
        if (r < e) {
            if (j < e) {
                const float q = pl.P[(pl.Ps[r] - k) * k + pl.M[j]];
                qmax = fmaxf(qmax, fabsf(q));
                v = exact_double(q);
            } else if (j - e == r) {
                v = 1.0;
            }
        }
        w[i] = v;
    }
    uint32_t used = 0;
    bool sing = false;
#pragma unroll 1
    for (int col = 0; col < e; ++col) {
        const int ci = col / SL;                 // entry index of column col
        const int cs = col % SL;                 // its slot
        double wc = 0.0;                         // this thread's entry ci
#pragma unroll
        for (int i = 0; i < EPL; ++i)
            if (i == ci) wc = w[i];
        const bool mine = slot == cs;            // this thread holds row r of column col
        uint32_t kc;
        double f, pv;
        if (NW == 1) {
            const uint32_t hi =
                (uint32_t)((unsigned long long)__double_as_longlong(wc) >> 32) & 0x7fffffffu;
            const bool cand = mine && r < e && !((used >> r) & 1u);
            kc = __reduce_max_sync(0xffffffffu, cand ? ((hi & ~15u) | (uint32_t)(15 - r)) : 0u);
            const int bi = 15 - (int)(kc & 15u);
            f = shfl_double(wc, cs * EMAX + r);
            pv = shfl_double(wc, cs * EMAX + bi);
        } else {
            const int buf = col & 1;
            if (t / 32 == cs * EMAX / 32) {      // the pivot column's warp
                const uint32_t hi =
                    (uint32_t)((unsigned long long)__double_as_longlong(wc) >> 32) & 0x7fffffffu;
                const bool cand = mine && r < e && !((used >> r) & 1u);
                const uint32_t kw =
                    __reduce_max_sync(0xffffffffu, cand ? ((hi & ~15u) | (uint32_t)(15 - r)) : 0u);
                if (mine) pl.fbuf[buf][r] = wc;
                if (lane == 0) pl.kbuf[buf] = kw;
            }
            elim_sync<NW>();
            kc = pl.kbuf[buf];
            f = pl.fbuf[buf][r];
            pv = pl.fbuf[buf][15 - (int)(kc & 15u)];
        }
        const uint32_t ef = kc >> 20;            // the pivot's exponent field
        if (ef == 0u || ef >= 0x7FFu) {          // zero, subnormal, infinite or not a number
            sing = true;
            break;
        }
        const int bi = 15 - (int)(kc & 15u);
        used |= 1u << bi;
        if (t == 0) pl.prow[col] = bi;
        const int sc = (int)ef - 1023;
        const double ps = scale_pow2(pv, sc);    // the pivot, scaled into [1, 2)
        const double fs = scale_pow2(f, sc);     // this row's multiplier, scaled alike
        double wb[EPL];                          // pivot-row entries of this thread's columns
#pragma unroll
        for (int i = 0; i < EPL; ++i) wb[i] = shfl_double(w[i], seg0 + bi);
        if (r != bi) {
#pragma unroll
            for (int i = 0; i < EPL; ++i) w[i] = fma(-fs, wb[i], __dmul_rn(ps, w[i]));
        }
    }
    if (!sing) {
        // the eliminated [Q | I] into shared memory
        if (r < e) {
#pragma unroll
            for (int i = 0; i < EPL; ++i) {
                const int j = slot + SL * i;
                if (j < 2 * e) pl.W[r][j] = w[i];
            }
        }
        elim_sync<NW>();
        if (t < e) pl.rcp[t] = 1.0 / pl.W[pl.prow[t]][t];
        elim_sync<NW>();
        // Q^-1 as (high, low) pairs, and the condition bound from the high
        // parts: max |Q^-1| over the e x e entries
        float qi = 0.f;
        for (int u = t; u < e * e; u += T) {
            const int c = u / e, a = u - c * e;
            float h, l;
            split_double(__dmul_rn(pl.W[pl.prow[c]][e + a], pl.rcp[c]), h, l);
            pl.Qh[c][a] = h;
            pl.Ql[c][a] = l;
            qi = fmaxf(qi, fabsf(h));
        }
        // maxima of non-negative floats as their bit patterns
        const uint32_t qiw = __reduce_max_sync(0xffffffffu, __float_as_uint(qi));
        const uint32_t qmw = __reduce_max_sync(0xffffffffu, __float_as_uint(qmax));
        if (NW == 1) {
            qi = __uint_as_float(qiw);
            qmax = __uint_as_float(qmw);
        } else {
            if (t == 0) pl.kbuf[0] = pl.kbuf[1] = 0u;
            elim_sync<NW>();
            if (lane == 0) {
                atomicMax(&pl.kbuf[0], qiw);
                atomicMax(&pl.kbuf[1], qmw);
            }
            elim_sync<NW>();
            qi = __uint_as_float(pl.kbuf[0]);
            qmax = __uint_as_float(pl.kbuf[1]);
        }
        // not-a-number fails the comparison and counts as singular
        if (!((float)e * qmax * ((float)e * qi) < (float)(1.0 / (64.0 * DBL_EPSILON)))) sing = true;
    }
    if (t == 0 && sing) pl.singular = 1;
}

// The rows of the decode, D[c][p] for the e missing blocks c and the k
// survivors p (S order: the surviving systematic workers, then the surviving
// parity workers):
//   D[c][p]      = -sum_q Q^-1[c][q] P[Ps[q]][S[p]]    for p < k - e
//   D[c][k-e+q]  =  Q^-1[c][q]
// formed from the (high, low) pairs of Q^-1 and the exact fp32 values of P
// in double-float arithmetic (about 2^-44 relative), one entry per thread;
// call after the barrier that follows plan_eliminate, then barrier.
__device__ __forceinline__ void plan_rows(const Plan &pl, int k, float (*Dh)[CM_MAX_N],
                                          float (*Dl)[CM_MAX_N])
{
    const int e = pl.e, ks = k - e;
    for (int u = threadIdx.x; u < e * k; u += blockDim.x) {
        const int c = u / k, p = u - c * k;
        if (p < ks) {
            float sh = 0.f, sl = 0.f;
            for (int q = 0; q < e; ++q)
                df_fma(pl.Qh[c][q], pl.Ql[c][q], -pl.P[(pl.Ps[q] - k) * k + pl.S[p]], 0.f, sh,
                       sl);
            Dh[c][p] = sh;
            Dl[c][p] = sl;
        } else {
            Dh[c][p] = pl.Qh[c][p - ks];
            Dl[c][p] = pl.Ql[c][p - ks];
        }
    }
}

}  // namespace cm_plan
