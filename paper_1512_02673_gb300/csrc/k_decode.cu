// K3 / K6: decoding from any k surviving worker results (Sec. III-A, last
// paragraph; Example "MDS codes").
//
// With S the first k survivors (ascending), the surviving results satisfy
// Yt_S = G_S Z, Z = the k uncoded block products.  G_S has a unit row for
// every surviving systematic worker (set Ks) and a parity row P[p] for every
// surviving parity worker (set Ps, |Ps| = e = number of missing systematic
// blocks, set M).  Gauss-Jordan on G_S that takes the unit rows as the first
// k-e pivots (exact: they are unit vectors) leaves the e x e block
// Q = P[Ps][M]; eliminating that block with partial pivoting gives Q^-1, and
// the rows of G_S^-1 for the missing blocks are
//   coefficient of Yt_s, s in Ps  :  Q^-1[c][pos of s in Ps]
//   coefficient of Yt_s, s in Ks  : -sum_a Q^-1[c][a] P[Ps[a]][s]
//
// Two kernels per decode.  A small plan kernel (one CTA) inverts Q in fp64
// on the device and writes the rows of G_S^-1 for the missing blocks to a
// plan slot; the apply kernel is launched right behind it as a programmatic
// dependent launch, so its launch overlaps the inversion: its pass-through
// CTAs (surviving systematic blocks, which need no inverse) run at once, and
// its decode CTAs issue the loads of their k surviving values, then wait for
// the plan (griddepcontrol.wait) and apply it: missing block M[c] row r is
// the combination of the k surviving rows r.  A zero (or relatively
// negligible) pivot marks G_S singular: the kernel writes CM_ESINGULAR to
// the status word and writes no decoded block.  With no missing block there
// is no plan kernel.
//
// fp64 arithmetic runs at about 1/58 of the fp32 rate on this part, so the
// vector decode applies the fp64 coefficients in double-float arithmetic on
// the fp32 pipe: each fp64 coefficient and each fp64 worker result is split
// into a (high, low) fp32 pair (results by integer bit manipulation, no fp64
// instruction), products are formed exactly with an FMA and the sums are kept
// as (sum, compensation) pairs (Knuth's TwoSum), about 2^-44 relative per
// term, far below the rounding of the fp32 output.
#include <algorithm>
#include <atomic>
#include <cfloat>
#include <cmath>

#include "cm_internal.cuh"

namespace {

constexpr int kThreads = 256;       // apply kernels
constexpr int kPlanThreads = 512;   // plan kernel: one entry of [Q | I] per thread
constexpr int kMaxE = 16;   // e <= min(k, n - k) <= 16 for n <= 32

// The decode of one survivor mask, formed in shared memory by every CTA that
// needs it (decode_plan below): the survivors used, the missing systematic
// blocks, the elimination's working matrix and the rows of G_S^-1 for the
// missing blocks as (high, low) fp32 pairs.
struct DecodePlan {
    int32_t e;               // missing systematic blocks
    int32_t singular;        // G_S judged singular: decode nothing
    int32_t S[CM_MAX_N];     // survivors in ascending order (k of them)
    int32_t Ps[kMaxE];       // surviving parity workers, ascending
    int32_t M[kMaxE];        // missing systematic blocks, ascending
    int32_t bi[kMaxE];       // pivot row (in the current row order) of each column
    double piv[kMaxE];       // that pivot's value
    float qmax;              // max |Q| (bounds ||Q||_inf by e max|Q|)
    unsigned long long qimax;   // max |Q^-1| as a magnitude key
    float P[CM_MAX_P];               // the parity coefficients ((n - k) x k)
    double W[2][2 * kMaxE][kMaxE];   // [Q | I] column-major, W[buf][column][row], ping-pong
    double Pd[kMaxE][CM_MAX_N];      // P[Ps[a]][S[p]] for the surviving systematic S[p]
    double rcp[kMaxE];               // 1 / final pivot of each row
    float Dh[kMaxE][CM_MAX_N];       // D[c][p] (p = position in S), high part
    float Dl[kMaxE][CM_MAX_N];       // D - Dh
};

// What the apply kernels need of a plan: written by the plan kernel into a
// slot of a ring in static device memory (no allocation per call).
struct DecodeRows {
    int32_t e;
    int32_t singular;
    int32_t M[kMaxE];
    float Dh[kMaxE][CM_MAX_N];
    float Dl[kMaxE][CM_MAX_N];
};

// Slots in flight at once: a call takes the next slot, so up to this many
// decodes may be pending at a time across streams.
constexpr int kPlanSlots = 256;
__device__ DecodeRows g_decode_rows[kPlanSlots];
std::atomic<uint32_t> g_next_rows{0};

__device__ __forceinline__ void griddep_wait()
{
    asm volatile("griddepcontrol.wait;\n" ::: "memory");
}

__device__ __forceinline__ void griddep_launch_dependents()
{
    asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory");
}

// ---- double-float helpers (fp32 pipe only) -------------------------------------------

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

// (sh, sl) += (dh + dl) * (yh + yl), to about 2^-44 relative per term.
__device__ __forceinline__ void df_fma(float dh, float dl, float yh, float yl, float &sh, float &sl)
{
    const float p = dh * yh;
    const float pe = fmaf(dh, yh, -p);                 // exact error of p
    const float t = fmaf(dh, yl, dl * yh);             // cross terms
    const float s1 = sh + p;                           // TwoSum(sh, p)
    const float bb = s1 - sh;
    const float err = (sh - (s1 - bb)) + (p - bb);
    sl += err + (pe + t);
    sh = s1;
}

// Magnitude key of an fp64 value for pivot search: the bits of |v|, which
// order like the values for every finite |v| (integer compares, no fp64
// instruction); not-a-number counts as the largest, so it is chosen and
// flagged.
__device__ __forceinline__ long long mag_key(double v)
{
    return __double_as_longlong(v) & 0x7fffffffffffffffll;
}

constexpr long long kInfKey = 0x7ff0000000000000ll;

// Largest key over an aligned segment of `seg` lanes (a power of two up to
// 16), lowest row on ties; every lane of the segment ends with the winner's
// row.  All 32 lanes of the warp take part.
__device__ __forceinline__ int seg_argmax(long long key, int row, int seg)
{
#pragma unroll
    for (int off = 8; off; off >>= 1) {
        if (off < seg) {
            const long long ok = __shfl_xor_sync(0xffffffffu, key, off);
            const int orow = __shfl_xor_sync(0xffffffffu, row, off);
            if (ok > key || (ok == key && orow < row)) {
                key = ok;
                row = orow;
            }
        }
    }
    return row;
}

// Largest non-negative float of the CTA into *dst (zero beforehand), by a
// warp maximum and one atomic per warp (an exact, order-free maximum).
__device__ __forceinline__ void cta_max(float v, float *dst)
{
#pragma unroll
    for (int off = 16; off; off >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, off));
    if ((threadIdx.x & 31) == 0 && v > 0.f) atomicMax(reinterpret_cast<int *>(dst), __float_as_int(v));
}

// The same for magnitude keys.
__device__ __forceinline__ void cta_max_key(long long v, unsigned long long *dst)
{
#pragma unroll
    for (int off = 16; off; off >>= 1) {
        const long long o = __shfl_xor_sync(0xffffffffu, v, off);
        v = o > v ? o : v;
    }
    if ((threadIdx.x & 31) == 0 && v > 0) atomicMax(dst, (unsigned long long)v);
}

// x 2^-s for a power-of-two scale, exact, by bit manipulation of the
// exponent (no fp64 instruction); zero, subnormal and underflowing values
// give a zero of the same sign (they are below 2^-1022 and only ever meet
// entries of order one).
__device__ __forceinline__ double scale_pow2(double x, int s)
{
    const long long b = __double_as_longlong(x);
    const int ex = (int)((b >> 52) & 0x7FF);
    const long long sign = b & (long long)0x8000000000000000ull;
    if (ex == 0 || ex - s <= 0) return __longlong_as_double(sign);
    return __longlong_as_double((b & ~(0x7FFll << 52)) | ((long long)(ex - s) << 52));
}

// fp64 value of an fp32 value by bit manipulation (exact; no fp64
// instruction: single fp64 operations have a long latency on this part).
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

// The decode of `survivors` in shared memory, by all kPlanThreads threads of
// the CTA (call it from every thread; it ends with a CTA barrier).
//  * Survivor lists by ballots in warp 0: S (the first k set bits), Ps (the
//    surviving parity workers among them), M (the missing systematic blocks);
//    the ks = k - e surviving systematic workers are S[0, ks).
//  * Gauss-Jordan in fp64 on W = [Q | I], Q = P[Ps][M] (e x e).  Thread t
//    holds entry (row t % E, column t / E), E the power of two at or above
//    e: the rows of a column are an aligned lane segment and the warps are
//    dense (the fp64 pipe of this part takes about 19 cycles per warp
//    instruction, whatever the number of active lanes, and 65 cycles of
//    latency).  The elimination is fraction-free: at column col with pivot
//    row bi, the pivot row moves to position col unchanged and every other
//    row r becomes 2^-s (piv W[r] - W[r][col] W[bi]), 2^s the binade of piv
//    (two separately rounded products, so duplicated rows cancel to exactly
//    zero; the exact power-of-two scale keeps the rows from growing by a
//    product of pivots, which overflows fp64 past about ten columns); each
//    row is scaled by its pivot once at the end:
//    Q^-1[c][a] = W[c][e + a] / W[c][c].
//    The row swap is part of the update, which reads one buffer and writes
//    the other: one CTA barrier per column.  The segment of column col + 1
//    picks that column's pivot right after computing it: the largest
//    |W[a][col + 1]|, a > col (exact magnitudes compared as integers), lowest
//    row on ties.
//  * G_S counts as singular when a pivot is zero, subnormal or not finite,
//    or when ||Q||_inf ||Q^-1||_inf, bounded by (e max|Q|) (e max|Q^-1|),
//    exceeds 1 / (64 eps) (evaluated in fp32: it is a threshold).
//  * D[c][p], the coefficient of the p-th survivor in missing block M[c]:
//    Q^-1[c][a] for the surviving parity worker Ps[a] = S[ks + a], and
//    -sum_a Q^-1[c][a] P[Ps[a]][S[p]] for the surviving systematic worker
//    S[p], p < ks; kept as a (high, low) fp32 pair.
__device__ void decode_plan(const CodeParams &cp, uint32_t survivors, DecodePlan &pl)
{
    const int tid = threadIdx.x, lane = tid & 31;
    const int n = cp.n, k = cp.k;
    {
        // P into shared memory by warp-uniform reads of the parameter space
        // (lanes reading different addresses there are served one address at
        // a time): warp w takes entries [16 w, 16 w + 16)
        const int w = tid >> 5;
        float v = 0.f;
#pragma unroll
        for (int i = 0; i < 16; ++i) {
            const float x = cp.P[(w * 16 + i) & (CM_MAX_P - 1)];
            if (lane == i) v = x;
        }
        if (lane < 16 && w * 16 + lane < CM_MAX_P) pl.P[w * 16 + lane] = v;
    }
    if (tid < 32) {
        const uint32_t below = (1u << lane) - 1u;
        const bool set = lane < n && ((survivors >> lane) & 1u);
        const bool sel = set && __popc(survivors & below) < k;
        const uint32_t selm = __ballot_sync(0xffffffffu, sel);
        const bool miss = lane < k && !sel;
        const uint32_t missm = __ballot_sync(0xffffffffu, miss);
        const bool par = sel && lane >= k;
        const uint32_t parm = __ballot_sync(0xffffffffu, par);
        if (sel) pl.S[__popc(selm & below)] = lane;
        if (par) pl.Ps[__popc(parm & below)] = lane;
        if (miss) pl.M[__popc(missm & below)] = lane;
        if (lane == 0) {
            pl.e = __popc(missm);
            pl.singular = 0;
            pl.qmax = 0.f;
            pl.qimax = 0ull;
        }
    }
    __syncthreads();
    const int e = pl.e, ks = k - e;
    if (e == 0) return;
    const float *P = pl.P;
    const int lg = 32 - __clz(e - 1);   // E = 1 << lg rows per column
    const int E = 1 << lg;
    const int j = tid >> lg, a = tid & (E - 1);
    const bool live = j < 2 * e && a < e;
    {
        // [Q | I] into buffer 0, max |Q|, the pivot of column 0 (exact: the
        // fp64 entries are the fp32 values of P), P at the surviving
        // systematic columns
        float q = 0.f;
        if (live) {
            if (j < e) q = P[(pl.Ps[a] - k) * k + pl.M[j]];
            pl.W[0][j][a] = j < e ? exact_double(q) : (j - e == a ? 1.0 : 0.0);
        }
        const int b0 = seg_argmax(j == 0 && a < e ? (long long)__float_as_int(fabsf(q)) : -1ll, a, E);
        if (tid == b0 && j == 0) {
            pl.bi[0] = b0;
            pl.piv[0] = exact_double(q);
        }
        if (tid < e * ks) {
            const int pa = tid / ks, pp = tid - pa * ks;
            pl.Pd[pa][pp] = exact_double(P[(pl.Ps[pa] - k) * k + pl.S[pp]]);
        }
        cta_max(live && j < e ? fabsf(q) : 0.f, &pl.qmax);
    }
    __syncthreads();
    for (int col = 0; col < e; ++col) {
        const int cur = col & 1, nxt = cur ^ 1;
        const int bi = pl.bi[col];
        const long long pk = mag_key(pl.piv[col]);
        if (pk < (1ll << 52) || pk >= kInfKey) {   // zero, subnormal, infinite or not a number
            __syncthreads();
            if (tid == 0) pl.singular = 1;
            __syncthreads();
            return;
        }
        // the update is scaled by 2^-s, 2^s the pivot's binade: the pivot
        // factor becomes piv 2^-s in [1, 2) and W[r][col] is scaled alike
        // (exact), so rows grow as in Gauss-Jordan with division rather
        // than by a product of pivots per column
        const int sc = (int)(pk >> 52) - 1023;
        const double piv = scale_pow2(pl.piv[col], sc);
        double nv = 0.0;
        if (live) {
            if (a == col) {
                nv = pl.W[cur][j][bi];
            } else if (j != col) {
                const int r = a == bi ? col : a;
                nv = __dsub_rn(__dmul_rn(piv, pl.W[cur][j][r]),
                               __dmul_rn(scale_pow2(pl.W[cur][col][r], sc), pl.W[cur][j][bi]));
            }
            pl.W[nxt][j][a] = nv;
        }
        if (col + 1 < e) {   // the segment of column col + 1 picks its pivot
            const bool cand = j == col + 1 && a > col && a < e;
            const int nb = seg_argmax(cand ? mag_key(nv) : -1ll, a, E);
            if (j == col + 1 && a == nb) {
                pl.bi[col + 1] = nb;
                pl.piv[col + 1] = nv;
            }
        }
        __syncthreads();
    }
    const int fin = e & 1;
    if (tid < e) pl.rcp[tid] = 1.0 / pl.W[fin][tid][tid];
    __syncthreads();
    // D rows, one entry per thread; the dot products run as two chains
    long long qk = 0;
    if (tid < e * k) {
        const int c = tid / k, p = tid - c * k;
        double v;
        if (p >= ks) {
            v = __dmul_rn(pl.W[fin][e + (p - ks)][c], pl.rcp[c]);
            qk = mag_key(v);
        } else {
            double s0 = 0.0, s1 = 0.0;
            for (int aa = 0; aa + 1 < e; aa += 2) {
                s0 = fma(pl.W[fin][e + aa][c], pl.Pd[aa][p], s0);
                s1 = fma(pl.W[fin][e + aa + 1][c], pl.Pd[aa + 1][p], s1);
            }
            if (e & 1) s0 = fma(pl.W[fin][2 * e - 1][c], pl.Pd[e - 1][p], s0);
            v = -__dmul_rn(__dadd_rn(s0, s1), pl.rcp[c]);
        }
        float h, l;
        split_double(v, h, l);
        pl.Dh[c][p] = h;
        pl.Dl[c][p] = l;
    }
    cta_max_key(qk, &pl.qimax);
    __syncthreads();
    const float qi = __double2float_ru(__longlong_as_double((long long)pl.qimax));
    if (!((float)e * pl.qmax * ((float)e * qi) < (float)(1.0 / (64.0 * DBL_EPSILON)))) {
        __syncthreads();   // every thread has read the maxima before the flag is set
        if (tid == 0) pl.singular = 1;
        __syncthreads();
    }
}

// The plan kernel: one CTA inverts Q and writes the decode rows.  It lets
// the apply kernel launch at once; that kernel's griddepcontrol.wait still
// waits for this grid to complete and its writes to be visible.
__global__ void __launch_bounds__(kPlanThreads, 1)
plan_kernel(const CodeParams cp, uint32_t survivors, DecodeRows *out)
{
    griddep_launch_dependents();
    __shared__ DecodePlan pl;
    decode_plan(cp, survivors, pl);
    const int e = pl.e, k = cp.k;
    if (threadIdx.x == 0) {
        out->e = e;
        out->singular = pl.singular;
    }
    if (threadIdx.x < kMaxE) out->M[threadIdx.x] = threadIdx.x < e ? pl.M[threadIdx.x] : 0;
    if (pl.singular) return;
    for (int t = threadIdx.x; t < e * k; t += kPlanThreads) {
        const int c = t / k, p = t - c * k;
        out->Dh[c][p] = pl.Dh[c][p];
        out->Dl[c][p] = pl.Dl[c][p];
    }
}

struct DecodeArgs {
    int64_t L, m;
    int32_t k;
    int32_t b;
    uint32_t survivors;       // the first k set bits are the survivors used
    const DecodeRows *rows;   // the plan kernel's output (when blocks are missing)
    const double *Yt;
    float *Y;
    int32_t *status;
    int mode;
    const float *lab;
    float eta;
    int32_t dec_ctas;         // CTAs of the decode role: the first ones in the grid
    int32_t dec_per_group;    // of those, per group of CG missing blocks
    int32_t pass_per_block;   // pass-through CTAs per surviving systematic block
};

constexpr int CG = 2;   // missing blocks decoded per thread

__device__ __forceinline__ void store_out(const DecodeArgs &a, int64_t out, float y_hi, float y_lo)
{
    if (a.mode == DEC_PLAIN) {
        a.Y[out] = y_hi + y_lo;
    } else if (a.mode == DEC_RESIDUAL) {
        a.Y[out] = (y_hi - a.lab[out]) + y_lo;          // z = A x - y
    } else {
        a.Y[out] = fmaf(-a.eta, y_hi + y_lo, a.Y[out]);  // x -= eta g
    }
}

// Index of the t-th set bit of x (t from 0; x has more than t set bits).
__device__ __forceinline__ int nth_set_bit(uint32_t x, int t)
{
    for (int i = 0; i < t; ++i) x &= x - 1u;
    return __ffs((int)x) - 1;
}

// Loads of the k surviving values at position rv (the survivors are the
// first k set bits of the mask).
__device__ __forceinline__ void load_survivors(const DecodeArgs &a, int64_t per_block, int64_t rv,
                                               double (&yv)[CM_MAX_N])
{
    uint32_t rest = a.survivors;
#pragma unroll
    for (int p = 0; p < CM_MAX_N; ++p) {
        if (p < a.k) {
            const int s = __ffs((int)rest) - 1;
            rest &= rest - 1u;
            yv[p] = a.Yt[(int64_t)s * per_block + rv];
        }
    }
}

// K3, the apply kernel.  Every CTA has one role, fixed by its index with one
// division per CTA: the first dec_ctas CTAs form the missing blocks (group
// g = CTA / dec_per_group of CG blocks, one row position per thread and
// pass), the others pass one surviving systematic block through (kPassItems
// positions per thread, loads issued together).  Decode CTAs come first;
// they issue their first loads, then wait for the plan and copy their CG
// rows of it to shared memory (read there with warp-uniform addresses).
constexpr int kPassItems = 4;

__global__ void __launch_bounds__(kThreads) decode_kernel(const __grid_constant__ DecodeArgs a)
{
    const int k = a.k;
    const int64_t per_block = a.L * a.b;
    const int64_t mb = a.m * a.b;
    int bx = (int)blockIdx.x;
    if (bx < a.dec_ctas) {
        __shared__ float Dh[CG][CM_MAX_N], Dl[CG][CM_MAX_N];
        __shared__ int32_t Mo[CG], ctl[2];
        const int g = bx / a.dec_per_group;
        const int c0 = g * CG;
        const int64_t step = (int64_t)a.dec_per_group * kThreads;
        int64_t rv = (int64_t)(bx - g * a.dec_per_group) * kThreads + threadIdx.x;
        double yv[CM_MAX_N];
        if (rv < per_block) load_survivors(a, per_block, rv, yv);
        griddep_wait();   // the plan kernel has completed
        const DecodeRows *rows = a.rows;
        if (threadIdx.x < 2) ctl[threadIdx.x] = threadIdx.x == 0 ? rows->e : rows->singular;
        if (threadIdx.x < CG) Mo[threadIdx.x] = rows->M[(c0 + threadIdx.x) & (kMaxE - 1)];
        for (int t = threadIdx.x; t < CG * CM_MAX_N; t += kThreads) {
            const int c = t / CM_MAX_N, p = t - c * CM_MAX_N;
            const int cc = (c0 + c) & (kMaxE - 1);
            Dh[c][p] = rows->Dh[cc][p];
            Dl[c][p] = rows->Dl[cc][p];
        }
        __syncthreads();
        if (ctl[1]) {
            if (bx == 0 && threadIdx.x == 0 && a.status) *a.status = CM_ESINGULAR;
            return;
        }
        const int e = ctl[0];
        while (rv < per_block) {
            float sh_[CG], sl_[CG];
#pragma unroll
            for (int c = 0; c < CG; ++c) sh_[c] = sl_[c] = 0.f;
#pragma unroll
            for (int p = 0; p < CM_MAX_N; ++p) {
                if (p < k) {
                    float yh, yl;
                    split_double(yv[p], yh, yl);
#pragma unroll
                    for (int c = 0; c < CG; ++c)
                        if (c0 + c < e) df_fma(Dh[c][p], Dl[c][p], yh, yl, sh_[c], sl_[c]);
                }
            }
#pragma unroll
            for (int c = 0; c < CG; ++c) {
                if (c0 + c < e) {
                    const int64_t out = (int64_t)Mo[c] * per_block + rv;
                    if (out < mb) store_out(a, out, sh_[c], sl_[c]);
                }
            }
            rv += step;
            if (rv >= per_block) break;
            load_survivors(a, per_block, rv, yv);
        }
        return;
    }
    // a surviving systematic block passes through (exactly rounded to fp32);
    // block t is the t-th set bit of the mask below k
    bx -= a.dec_ctas;
    const int t = bx / a.pass_per_block;
    const int64_t base =
        (int64_t)nth_set_bit(a.survivors & (k < 32 ? (1u << k) - 1u : 0xffffffffu), t) * per_block;
    const int64_t lim = (mb - base < per_block ? mb - base : per_block);
    const int64_t step = (int64_t)a.pass_per_block * kThreads * kPassItems;
    for (int64_t i0 = (int64_t)(bx - t * a.pass_per_block) * kThreads * kPassItems + threadIdx.x;
         i0 < lim; i0 += step) {
        double y[kPassItems];
#pragma unroll
        for (int u = 0; u < kPassItems; ++u)
            if (i0 + u * kThreads < lim) y[u] = a.Yt[base + i0 + u * kThreads];
#pragma unroll
        for (int u = 0; u < kPassItems; ++u) {
            if (i0 + u * kThreads >= lim) break;
            const int64_t out = base + i0 + u * kThreads;
            if (a.mode == DEC_PLAIN) {
                a.Y[out] = __double2float_rn(y[u]);
            } else {
                float yh, yl;
                split_double(y[u], yh, yl);
                store_out(a, out, yh, yl);
            }
        }
    }
}

// K6: fp32 results, all e missing blocks of one row position per thread, so
// every surviving element is read once.  Launched behind the plan kernel
// like K3; every CTA waits for the plan and copies its fp32 coefficients
// (the high parts) to shared memory.
template <int EMAX>
__global__ void __launch_bounds__(kThreads)
decode_mat_kernel(int32_t k, int64_t L, int64_t m, uint32_t survivors, const DecodeRows *rows,
                  const float *Ct, int64_t ldc, int N, float *C, int64_t ldcc, int32_t *status)
{
    __shared__ float Dh[EMAX][CM_MAX_N];
    __shared__ int32_t S[CM_MAX_N], Mo[EMAX], ctl[2];
    if (threadIdx.x < CM_MAX_N) {
        // survivors: the first k set bits of the mask
        const uint32_t below = (1u << threadIdx.x) - 1u;
        if (((survivors >> threadIdx.x) & 1u) && __popc(survivors & below) < k)
            S[__popc(survivors & below)] = threadIdx.x;
    }
    griddep_wait();   // the plan kernel has completed
    if (threadIdx.x < 2) ctl[threadIdx.x] = threadIdx.x == 0 ? rows->e : rows->singular;
    if (threadIdx.x < EMAX) Mo[threadIdx.x] = rows->M[threadIdx.x];
    for (int t = threadIdx.x; t < EMAX * CM_MAX_N; t += kThreads)
        Dh[t / CM_MAX_N][t % CM_MAX_N] = rows->Dh[t / CM_MAX_N][t % CM_MAX_N];
    __syncthreads();
    if (ctl[1]) {
        if (blockIdx.x == 0 && threadIdx.x == 0 && status) *status = CM_ESINGULAR;
        return;
    }
    const int e = ctl[0];
    const bool inplace = C == Ct;
    const bool vec = (N % 4 == 0) && (ldc % 4 == 0) && (ldcc % 4 == 0) &&
                     (((uintptr_t)Ct | (uintptr_t)C) & 15u) == 0;
    const int W = vec ? 4 : 1;
    const int64_t nw = N / W;
    const int64_t total = L * nw;
    // survivors whose loads are issued together (fewer with more accumulators)
    constexpr int kBatch = EMAX <= 8 ? 4 : 2;
    int M[EMAX];
#pragma unroll
    for (int c = 0; c < EMAX; ++c) M[c] = c < e ? Mo[c] : 0;
    for (int64_t it = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; it < total;
         it += (int64_t)gridDim.x * blockDim.x) {
        const int64_t r = it / nw;
        const int64_t col = (it - r * nw) * W;
        float4 acc[EMAX];
#pragma unroll
        for (int c = 0; c < EMAX; ++c) acc[c] = make_float4(0.f, 0.f, 0.f, 0.f);
        // survivors in batches of kBatch: their loads are issued together
        for (int p0 = 0; p0 < k; p0 += kBatch) {
            float4 v[kBatch];
#pragma unroll
            for (int u = 0; u < kBatch; ++u) {
                if (p0 + u < k) {
                    const float *src = Ct + ((int64_t)S[p0 + u] * L + r) * ldc + col;
                    v[u] = vec ? __ldg(reinterpret_cast<const float4 *>(src))
                               : make_float4(__ldg(src), 0.f, 0.f, 0.f);
                }
            }
#pragma unroll
            for (int u = 0; u < kBatch; ++u) {
                const int p = p0 + u;
                if (p >= k) break;
                const int s = S[p];
                if (!inplace && s < k) {   // surviving systematic block passes through
                    const int64_t g = (int64_t)s * L + r;
                    if (g < m) {
                        float *dst = C + g * ldcc + col;
                        if (vec) *reinterpret_cast<float4 *>(dst) = v[u];
                        else *dst = v[u].x;
                    }
                }
#pragma unroll
                for (int c = 0; c < EMAX; ++c) {
                    if (c < e) {
                        const float w = Dh[c][p];
                        acc[c].x = fmaf(w, v[u].x, acc[c].x);
                        acc[c].y = fmaf(w, v[u].y, acc[c].y);
                        acc[c].z = fmaf(w, v[u].z, acc[c].z);
                        acc[c].w = fmaf(w, v[u].w, acc[c].w);
                    }
                }
            }
        }
#pragma unroll
        for (int c = 0; c < EMAX; ++c) {
            if (c < e) {
                const int64_t g = (int64_t)M[c] * L + r;
                if (g < m) {
                    float *dst = C + g * ldcc + col;
                    if (vec) *reinterpret_cast<float4 *>(dst) = acc[c];
                    else *dst = acc[c].x;
                }
            }
        }
    }
}

// CTAs for `items` independent items, at most `per_sm` per SM.
int grid_for(int64_t items, int per_sm)
{
    int64_t g = (items + kThreads - 1) / kThreads;
    const int64_t cap = (int64_t)(cm_sm_count() > 0 ? cm_sm_count() : 1) * per_sm;
    if (g > cap) g = cap;
    if (g < 1) g = 1;
    return (int)g;
}

// Missing systematic blocks of a survivor mask (its first k set bits).
int missing_blocks(int k, uint32_t survivors)
{
    const uint32_t sys = k < 32 ? survivors & ((1u << k) - 1u) : survivors;
    return k - __builtin_popcount(sys);
}

// Launches the plan kernel into the next slot of the ring.
cudaError_t launch_plan(const CodeParams &cp, uint32_t survivors, cudaStream_t s,
                        DecodeRows **rows)
{
    void *base = nullptr;
    cudaError_t e = cudaGetSymbolAddress(&base, g_decode_rows);
    if (e != cudaSuccess) return e;
    *rows = static_cast<DecodeRows *>(base) +
            g_next_rows.fetch_add(1, std::memory_order_relaxed) % kPlanSlots;
    plan_kernel<<<1, kPlanThreads, 0, s>>>(cp, survivors, *rows);
    return cudaGetLastError();
}

// Launch behind the plan kernel as a programmatic dependent launch.
template <typename... KArgs, typename... Args>
cudaError_t launch_behind_plan(void (*kern)(KArgs...), unsigned grid, cudaStream_t s,
                               Args... args)
{
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = 0;
    cfg.stream = s;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kern, args...);
}

}  // namespace

cudaError_t launch_decode(const CodeParams &cp, const double *Yt, uint32_t survivors, int b,
                          float *Y, int32_t *status, int mode, const float *lab, float eta,
                          cudaStream_t s)
{
    DecodeArgs a;
    a.L = cp.L;
    a.m = cp.m;
    a.k = cp.k;
    a.b = b;
    a.survivors = survivors;
    a.rows = nullptr;
    a.Yt = Yt;
    a.Y = Y;
    a.status = status;
    a.mode = mode;
    a.lab = lab;
    a.eta = eta;
    // CTAs per role, capped (threads then loop) so the grid stays well inside
    // the launch limit for any block size
    const int e = missing_blocks(cp.k, survivors), ngroups = (e + CG - 1) / CG;
    const int64_t per_block = cp.L * (int64_t)b;
    const int64_t cap = 1 << 20;
    a.dec_per_group = (int32_t)std::min(cap, (per_block + kThreads - 1) / kThreads);
    a.dec_ctas = ngroups * a.dec_per_group;
    a.pass_per_block = (int32_t)std::min(
        cap, (per_block + kThreads * kPassItems - 1) / (kThreads * kPassItems));
    const int64_t grid = a.dec_ctas + (int64_t)(cp.k - e) * a.pass_per_block;
    if (grid < 1) return cudaSuccess;
    if (e == 0) {   // nothing to invert: the pass-through alone
        decode_kernel<<<(unsigned)grid, kThreads, 0, s>>>(a);
        return cudaGetLastError();
    }
    DecodeRows *rows = nullptr;
    cudaError_t err = launch_plan(cp, survivors, s, &rows);
    if (err != cudaSuccess) return err;
    a.rows = rows;
    return launch_behind_plan(decode_kernel, (unsigned)grid, s, a);
}

cudaError_t launch_decode_mat(const CodeParams &cp, const float *Ct, int64_t ldc,
                              uint32_t survivors, int N, float *C, int64_t ldcc, int32_t *status,
                              cudaStream_t s)
{
    const int e = missing_blocks(cp.k, survivors);
    DecodeRows *rows = nullptr;
    cudaError_t err = launch_plan(cp, survivors, s, &rows);
    if (err != cudaSuccess) return err;
    const int64_t items = cp.L * (int64_t)N / 4 + 1;
    const unsigned g = (unsigned)grid_for(items, 8);
    const int32_t k = cp.k;
    const int64_t L = cp.L, m = cp.m;
    if (e <= 4)
        return launch_behind_plan(decode_mat_kernel<4>, g, s, k, L, m, survivors,
                                  (const DecodeRows *)rows, Ct, ldc, N, C, ldcc, status);
    if (e <= 8)
        return launch_behind_plan(decode_mat_kernel<8>, g, s, k, L, m, survivors,
                                  (const DecodeRows *)rows, Ct, ldc, N, C, ldcc, status);
    return launch_behind_plan(decode_mat_kernel<16>, g, s, k, L, m, survivors,
                              (const DecodeRows *)rows, Ct, ldc, N, C, ldcc, status);
}
