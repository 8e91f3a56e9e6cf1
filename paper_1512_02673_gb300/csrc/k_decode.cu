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
// The master knows the survivors when it decodes, so the library's host code
// forms these coefficients once per call (plan_decode, fp64, a few
// microseconds; formed on the device they cost every CTA ~10 us of
// latency-bound fp64 work) and passes them to the kernel by value; the
// kernel's threads apply them: missing block M[c] row r is the combination of
// the k surviving rows r, surviving systematic blocks pass through.  A zero
// (or relatively negligible) pivot marks G_S singular: the kernel writes
// CM_ESINGULAR to the status word and writes no decoded block.
//
// fp64 arithmetic runs at about 1/58 of the fp32 rate on this part, so the
// vector decode applies the fp64 coefficients in double-float arithmetic on
// the fp32 pipe: each fp64 coefficient and each fp64 worker result is split
// into a (high, low) fp32 pair (results by integer bit manipulation, no fp64
// instruction), products are formed exactly with an FMA and the sums are kept
// as (sum, compensation) pairs (Knuth's TwoSum), about 2^-44 relative per
// term, far below the rounding of the fp32 output.
#include <algorithm>
#include <cfloat>
#include <cmath>
#include <cstring>

#include "cm_internal.cuh"

namespace {

constexpr int kThreads = 256;
constexpr int kMaxE = 16;   // e <= min(k, n - k) <= 16 for n <= 32

// The decode of one survivor mask, formed on the host (plan_decode below) and
// passed to the kernels by value: the survivors used, the missing systematic
// blocks, and the rows of G_S^-1 for those blocks as (high, low) fp32 pairs.
struct DecodePlan {
    int32_t e;               // missing systematic blocks
    int32_t singular;        // G_S judged singular: decode nothing
    int32_t S[CM_MAX_N];     // survivors in ascending order (k of them)
    int32_t M[kMaxE];        // missing systematic blocks, ascending
    float Dh[kMaxE][CM_MAX_N];   // D[c][p] (p = position in S), rounded to fp32
    float Dl[kMaxE][CM_MAX_N];   // D - Dh, rounded to fp32
};

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

struct DecodeArgs {
    int64_t L, m;
    int32_t k;
    int32_t b;
    DecodePlan plan;
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

// The plan stays in the parameter space: every access below is uniform
// across a warp (one (c, p) at a time; S and M indexed by a block number that
// is fixed per CTA), which the constant cache serves by broadcast; copying it
// to shared memory would read it divergently.
//
// Every CTA has one role, fixed by its index with one division per CTA: the
// first dec_ctas CTAs form the missing blocks (group g = CTA / dec_per_group
// of CG blocks, one row position per thread and pass), the others pass one
// surviving systematic block through (kPassItems positions per thread, loads
// issued together).  Decode CTAs come first so that their longer chains
// (k loads, then k CG double-float FMAs) start first.
constexpr int kPassItems = 4;

__global__ void __launch_bounds__(kThreads) decode_kernel(const __grid_constant__ DecodeArgs a)
{
    const DecodePlan &sh = a.plan;
    const int k = a.k, e = sh.e;
    const int64_t per_block = a.L * a.b;
    const int64_t mb = a.m * a.b;
    int bx = (int)blockIdx.x;
    if (bx < a.dec_ctas) {
        if (sh.singular) {
            if (bx == 0 && threadIdx.x == 0 && a.status) *a.status = CM_ESINGULAR;
            return;
        }
        const int g = bx / a.dec_per_group;
        const int c0 = g * CG;
        const int64_t step = (int64_t)a.dec_per_group * kThreads;
        for (int64_t rv = (int64_t)(bx - g * a.dec_per_group) * kThreads + threadIdx.x;
             rv < per_block; rv += step) {
            double yv[CM_MAX_N];
#pragma unroll
            for (int p = 0; p < CM_MAX_N; ++p)
                if (p < k) yv[p] = a.Yt[(int64_t)sh.S[p] * per_block + rv];
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
                        if (c0 + c < e)
                            df_fma(sh.Dh[c0 + c][p], sh.Dl[c0 + c][p], yh, yl, sh_[c], sl_[c]);
                }
            }
#pragma unroll
            for (int c = 0; c < CG; ++c) {
                if (c0 + c < e) {
                    const int64_t out = (int64_t)sh.M[c0 + c] * per_block + rv;
                    if (out < mb) store_out(a, out, sh_[c], sl_[c]);
                }
            }
        }
        return;
    }
    // a surviving systematic block passes through (exactly rounded to fp32)
    bx -= a.dec_ctas;
    const int t = bx / a.pass_per_block;
    const int64_t base = (int64_t)sh.S[t] * per_block;
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
// every surviving element is read once.
template <int EMAX>
__global__ void __launch_bounds__(kThreads)
decode_mat_kernel(const CodeParams cp, const __grid_constant__ DecodePlan plan, const float *Ct,
                  int64_t ldc, int N, float *C, int64_t ldcc, int32_t *status)
{
    const DecodePlan &sh = plan;   // read in place (uniform accesses)
    if (sh.singular) {
        if (blockIdx.x == 0 && threadIdx.x == 0 && status) *status = CM_ESINGULAR;
        return;
    }
    const int k = cp.k, e = sh.e;
    const int64_t L = cp.L, m = cp.m;
    const bool inplace = C == Ct;
    const bool vec = (N % 4 == 0) && (ldc % 4 == 0) && (ldcc % 4 == 0) &&
                     (((uintptr_t)Ct | (uintptr_t)C) & 15u) == 0;
    const int W = vec ? 4 : 1;
    const int64_t nw = N / W;
    const int64_t total = L * nw;
    int M[EMAX];
#pragma unroll
    for (int c = 0; c < EMAX; ++c) M[c] = c < e ? sh.M[c] : 0;
    for (int64_t it = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; it < total;
         it += (int64_t)gridDim.x * blockDim.x) {
        const int64_t r = it / nw;
        const int64_t col = (it - r * nw) * W;
        float4 acc[EMAX];
#pragma unroll
        for (int c = 0; c < EMAX; ++c) acc[c] = make_float4(0.f, 0.f, 0.f, 0.f);
        for (int p = 0; p < k; ++p) {
            const int s = sh.S[p];
            const float *src = Ct + ((int64_t)s * L + r) * ldc + col;
            float4 v;
            if (vec) {
                v = __ldg(reinterpret_cast<const float4 *>(src));
            } else {
                v = make_float4(__ldg(src), 0.f, 0.f, 0.f);
            }
            if (!inplace && s < k) {   // surviving systematic block passes through
                const int64_t g = (int64_t)s * L + r;
                if (g < m) {
                    float *dst = C + g * ldcc + col;
                    if (vec) *reinterpret_cast<float4 *>(dst) = v;
                    else *dst = v.x;
                }
            }
#pragma unroll
            for (int c = 0; c < EMAX; ++c) {
                if (c < e) {
                    const float w = sh.Dh[c][p];
                    acc[c].x = fmaf(w, v.x, acc[c].x);
                    acc[c].y = fmaf(w, v.y, acc[c].y);
                    acc[c].z = fmaf(w, v.z, acc[c].z);
                    acc[c].w = fmaf(w, v.w, acc[c].w);
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

// The decode of `survivors` (host, fp64): the survivor lists, then
// Gauss-Jordan on [Q | I], Q = P[Ps][M] (e x e), fraction-free (a non-pivot
// row becomes piv W[a] - W[a][col] W[col], two separately rounded products),
// with partial pivoting on the fp32 image of |W[a][col]| (lowest index on
// ties) and one division per row at the end: Q^-1[c][a] = W[c][e+a] / W[c][c].
// G_S counts as singular when a pivot is zero or not finite, or when
// ||Q||_inf ||Q^-1||_inf, bounded by ||Q||_inf e max|Q^-1|, exceeds
// 1 / (64 eps).  Host code is compiled without floating-point contraction, so
// the plan is the same on every host.
void plan_decode(const CodeParams &cp, uint32_t survivors, DecodePlan &pl)
{
    const int n = cp.n, k = cp.k;
    int Ps[kMaxE];
    int ns = 0, e = 0, np = 0;
    for (int j = 0; j < n && ns < k; ++j)
        if ((survivors >> j) & 1u) {
            pl.S[ns++] = j;
            if (j >= k) Ps[np++] = j;
        }
    for (int i = 0; i < k; ++i) {
        bool in = false;
        for (int p = 0; p < ns; ++p) in = in || pl.S[p] == i;
        if (!in) pl.M[e++] = i;
    }
    pl.e = e;
    pl.singular = 0;
    if (e == 0) return;
    double W[kMaxE][2 * kMaxE];
    double qnorm = 0.0;
    for (int a = 0; a < e; ++a) {
        double row = 0.0;
        for (int c = 0; c < e; ++c) {
            W[a][c] = (double)cp.P[(Ps[a] - k) * k + pl.M[c]];
            row += std::fabs(W[a][c]);
        }
        for (int c = 0; c < e; ++c) W[a][e + c] = a == c ? 1.0 : 0.0;
        qnorm = std::max(qnorm, row);
    }
    for (int col = 0; col < e; ++col) {
        int bi = col;
        float best = -1.f;
        for (int a = col; a < e; ++a) {
            const float f = (float)std::fabs(W[a][col]);
            if (f > best) {
                best = f;
                bi = a;
            }
        }
        const double piv = W[bi][col];
        if (!(std::fabs(piv) > 0.0) || !std::isfinite(piv)) {
            pl.singular = 1;
            return;
        }
        if (bi != col)
            for (int j = 0; j < 2 * e; ++j) std::swap(W[col][j], W[bi][j]);
        for (int a = 0; a < e; ++a) {
            if (a == col) continue;
            const double fa = W[a][col];
            for (int j = 0; j < 2 * e; ++j) {
                const double p1 = piv * W[a][j], p2 = fa * W[col][j];
                W[a][j] = j == col ? 0.0 : p1 - p2;
            }
        }
    }
    double Qi[kMaxE][kMaxE], qimax = 0.0;
    for (int c = 0; c < e; ++c) {
        const double dinv = 1.0 / W[c][c];
        for (int a = 0; a < e; ++a) {
            Qi[c][a] = W[c][e + a] * dinv;
            qimax = std::max(qimax, std::fabs(Qi[c][a]));
        }
    }
    if (!(qnorm * qimax * e < 1.0 / (64.0 * DBL_EPSILON))) {
        pl.singular = 1;
        return;
    }
    for (int c = 0; c < e; ++c)
        for (int p = 0; p < k; ++p) {
            const int sp = pl.S[p];
            double v = 0.0;
            if (sp >= k) {
                for (int a = 0; a < e; ++a)
                    if (Ps[a] == sp) v = Qi[c][a];
            } else {
                for (int a = 0; a < e; ++a)
                    v = std::fma(-Qi[c][a], (double)cp.P[(Ps[a] - k) * k + sp], v);
            }
            const float h = (float)v;
            pl.Dh[c][p] = h;
            pl.Dl[c][p] = (float)(v - (double)h);
        }
}

}  // namespace

cudaError_t launch_decode(const CodeParams &cp, const double *Yt, uint32_t survivors, int b,
                          float *Y, int32_t *status, int mode, const float *lab, float eta,
                          cudaStream_t s)
{
    DecodeArgs a;
    std::memset(&a.plan, 0, sizeof(a.plan));
    plan_decode(cp, survivors, a.plan);
    a.L = cp.L;
    a.m = cp.m;
    a.k = cp.k;
    a.b = b;
    a.Yt = Yt;
    a.Y = Y;
    a.status = status;
    a.mode = mode;
    a.lab = lab;
    a.eta = eta;
    // CTAs per role, capped (threads then loop) so the grid stays well inside
    // the launch limit for any block size
    const int64_t per_block = cp.L * (int64_t)b;
    const int64_t cap = 1 << 20;
    const int e = a.plan.e, ngroups = (e + CG - 1) / CG;
    a.dec_per_group = (int32_t)std::min(cap, (per_block + kThreads - 1) / kThreads);
    a.dec_ctas = a.plan.singular ? 1 : ngroups * a.dec_per_group;
    a.pass_per_block = (int32_t)std::min(
        cap, (per_block + kThreads * kPassItems - 1) / (kThreads * kPassItems));
    const int64_t grid = a.dec_ctas + (int64_t)(cp.k - e) * a.pass_per_block;
    if (grid < 1) return cudaSuccess;
    decode_kernel<<<(unsigned)grid, kThreads, 0, s>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_decode_mat(const CodeParams &cp, const float *Ct, int64_t ldc,
                              uint32_t survivors, int N, float *C, int64_t ldcc, int32_t *status,
                              cudaStream_t s)
{
    DecodePlan plan;
    std::memset(&plan, 0, sizeof(plan));
    plan_decode(cp, survivors, plan);
    const int64_t items = cp.L * (int64_t)N / 4 + 1;
    const int g = grid_for(items, 8);
    if (plan.e <= 4)
        decode_mat_kernel<4><<<g, kThreads, 0, s>>>(cp, plan, Ct, ldc, N, C, ldcc, status);
    else if (plan.e <= 8)
        decode_mat_kernel<8><<<g, kThreads, 0, s>>>(cp, plan, Ct, ldc, N, C, ldcc, status);
    else
        decode_mat_kernel<16><<<g, kThreads, 0, s>>>(cp, plan, Ct, ldc, N, C, ldcc, status);
    return cudaGetLastError();
}
