// K3 / K6: decoding from any k surviving worker results (Sec. III-A, last
// paragraph; Example "MDS codes").
//
// One launch per decode and no state kept between calls: every CTA forms the
// decode in its own shared memory (decode_plan.cuh: the e x e block Q of G_S
// inverted in fp64 in registers by one or four warps) and applies it.  The
// vector decode applies the rows of G_S^-1 for the missing systematic blocks
// in two factors, Z_M = Q^-1 (Y_par - P[Ps][S_sys] Y_sys), the second formed
// while the elimination runs; the matrix decode forms the rows D of G_S^-1
// and sums M[c] = sum_p D[c][p] Yt_S[p] over the k surviving results.
// Surviving systematic blocks pass through.  Each surviving value is loaded
// once per CTA.  A zero (or relatively negligible) pivot marks G_S singular:
// CM_ESINGULAR goes to the status word and no missing block is written
// (surviving systematic blocks are still copied).
//
// fp64 arithmetic runs at a small fraction of the fp32 rate on this part, so
// the vector decode works in double-float arithmetic on the fp32 pipe: each
// fp64 worker result and each entry of Q^-1 is a (high, low) fp32 pair split by
// integer bit manipulation, products are formed exactly with an FMA and the
// sums are kept as (sum, compensation) pairs (Knuth's TwoSum), about 2^-44
// relative per term, far below the rounding of the fp32 output; fp32 outputs
// of fp64 values are rounded to nearest even by integer arithmetic.  The
// matrix decode (fp32 results of the tensor-core products) applies the rows'
// high parts in fp32.
#include <algorithm>

#include "cm_internal.cuh"
#include "decode_plan.cuh"

using namespace cm_plan;

namespace {

constexpr int kThreads = 1024;     // vector decode: one CTA per SM
constexpr int kTile = 256;         // row positions staged at a time
constexpr int kMatThreads = 256;   // matrix decode

struct DecodeArgs {
    CodeParams cp;
    int32_t b;
    uint32_t survivors;       // exactly k set bits: the survivors used
    const double *Yt;
    float *Y;
    int32_t *status;
    int mode;
    const float *lab;
    float eta;
    int64_t chunk;            // row positions per CTA
    int32_t dependent;        // launched as a programmatic dependent of the products
    int32_t nparts;           // Yt holds this many partial results of the products ...
    int64_t part_stride;      // ... this many doubles apart; their sum is the result
};

__device__ __forceinline__ void griddep_wait()
{
    asm volatile("griddepcontrol.wait;\n" ::: "memory");
}

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

// Named barrier among the warps that stage while the first NW warps
// eliminate (barrier 2; 0 is __syncthreads, 1 the eliminating warps').
__device__ __forceinline__ void staging_sync(int threads)
{
    asm volatile("bar.sync 2, %0;\n" ::"r"(threads) : "memory");
}

// K3.  A persistent grid, one CTA of 1024 threads per SM; CTA i owns the row
// positions [i chunk, (i + 1) chunk) (row r of every block and vector v,
// position r b + v) of all k output blocks, taken in tiles of kTile.  With
// Y_par the results of the e surviving parity workers and Y_sys those of
// the ks = k - e surviving systematic ones, the missing blocks are
//   Z_M = Q^-1 R,   R = Y_par - P[Ps][S_sys] Y_sys,
// the same rows of G_S^-1 applied in two factors: R needs only P, so it is
// formed while the elimination runs, and what follows the elimination is a
// sum of e terms per output.
//  1. plan_setup.
//  2. For every tile: the k surviving values of its positions are loaded
//     (position fastest, coalesced; a thread's loads issued together) and
//     staged in shared memory as (high, low) fp32 pairs, and those of the
//     surviving systematic blocks are written out at once (the pass-through,
//     fp32 rounding of the fp64 results).  For the first tile of a decode
//     call of its own the first NW warps eliminate meanwhile (when blocks
//     are missing), so the loads overlap the elimination.
//  3. Every (parity survivor a, position) of the tile is one thread's item:
//     R[a] = y_Ps[a] - sum_p P[Ps[a]][S[p]] y_S[p] over the systematic
//     survivors, in double-float arithmetic, written over y_Ps[a]'s slot
//     (the only item that reads it).  The staging warps do this while the
//     first tile's elimination is still running.
//  4. Every (missing block c, position) is one thread's item: sum_a
//     Q^-1[c][a] R[a] in double-float arithmetic.  Many short items keep
//     every scheduler busy (a thread per position with all e blocks left one
//     warp per scheduler waiting on its own dependent operations), and code
//     that runs once per item stays small (fully unrolled loops spent most
//     of their time fetching instructions).
template <int EMAX, int NW>
__global__ void __launch_bounds__(kThreads, 1) decode_kernel(const __grid_constant__ DecodeArgs a)
{
    extern __shared__ float2 ysm[];   // [CM_MAX_N][kTile] (high, low) pairs of the survivors
    __shared__ Plan pl;
    __shared__ float Pn[kMaxE][CM_MAX_N + 1];   // -P[Ps[a]][S[p]], p < ks (padded rows)
    const int k = a.cp.k;
    const int e = missing_blocks(k, a.survivors);
    const int ks = k - e;
    const int tid = threadIdx.x;
    const int64_t per_block = a.cp.L * a.b;
    const int64_t mb = a.cp.m * a.b;
    const int64_t p0 = (int64_t)blockIdx.x * a.chunk;
    const int64_t n = (per_block - p0 < a.chunk ? per_block - p0 : a.chunk);
    plan_setup(a.cp, a.survivors, pl);
    // Every decode is launched as a programmatic dependent of the kernel
    // before it.  In the plan-first form (products and decode in one call)
    // the eliminating warps form Q^-1 from the kernel parameters while the
    // products finish, and every thread waits for the products before it
    // reads a result.  In the overlap form (a decode call of its own) the
    // eliminating warps start at once and the staging threads wait before
    // their loads, so the elimination overlaps the previous kernel's tail
    // (when that kernel lets dependents start, as the products do), the
    // first tile's loads and its R.
    const bool overlap = !a.dependent;
    if (!overlap) {
        if (e > 0 && tid < 32 * NW) plan_eliminate<EMAX, NW>(pl, k);
        griddep_wait();
    }
    bool dec = false;
    for (int64_t t0 = 0; t0 < n; t0 += kTile) {
        const int tn = (int)(n - t0 < kTile ? n - t0 : kTile);
        const bool first = t0 == 0;
        const bool split = overlap && first && e > 0;   // the first NW warps eliminate
        const int lo = split ? 32 * NW : 0;
        if (split && tid < lo) {
            plan_eliminate<EMAX, NW>(pl, k);
            griddep_wait();   // before the later tiles' loads and any store
        } else {
            if (overlap && first) griddep_wait();
            const int tt = tid - lo;
            if (first) {
                for (int u = tt; u < e * ks; u += kThreads - lo) {
                    const int c = u / ks, p = u - c * ks;
                    Pn[c][p] = -pl.P[(pl.Ps[c] - k) * k + pl.S[p]];
                }
            }
            // stage the tile: thread tt takes position q = tt % tn of
            // survivors tt / tn, tt / tn + per, ... (per = threads / tn), SB
            // of them with their loads issued before any store (one division
            // per thread, none per value)
            constexpr int SB = 4;
            const int per = (kThreads - lo) / tn;
            if (tt < per * tn) {
                const int q = tt % tn;
                const int64_t base = p0 + t0 + q;
                for (int pb = tt / tn; pb < k; pb += SB * per) {
                    double y[SB];
#pragma unroll
                    for (int j = 0; j < SB; ++j) {
                        const int p = pb + j * per;
                        if (p < k) y[j] = a.Yt[(int64_t)pl.S[p] * per_block + base];
                    }
                    for (int h = 1; h < a.nparts; ++h) {
#pragma unroll
                        for (int j = 0; j < SB; ++j) {
                            const int p = pb + j * per;
                            if (p < k) y[j] += a.Yt[(int64_t)pl.S[p] * per_block + base + h * a.part_stride];
                        }
                    }
#pragma unroll
                    for (int j = 0; j < SB; ++j) {
                        const int p = pb + j * per;
                        if (p >= k) break;
                        const int s = pl.S[p];
                        float yh, yl, yr;
                        if (a.mode == DEC_PLAIN) split_round(y[j], yh, yl, yr);
                        else split_double(y[j], yh, yl);
                        if (e > 0) ysm[p * kTile + q] = make_float2(yh, yl);
                        const int64_t src = (int64_t)s * per_block + base;
                        if (s < k && src < mb) {   // surviving systematic block: pass through
                            if (a.mode == DEC_PLAIN) a.Y[src] = yr;
                            else store_out(a, src, yh, yl);
                        }
                    }
                }
            }
            if (e > 0) {
                if (split) staging_sync(kThreads - lo);
                else __syncthreads();
                for (int u = tt; u < e * tn; u += kThreads - lo) {
                    const int c = u / tn, q = u - c * tn;
                    float2 *r = &ysm[(ks + c) * kTile + q];
                    float sh = r->x, sl = r->y;
#pragma unroll 4
                    for (int p = 0; p < ks; ++p) {
                        const float2 y = ysm[p * kTile + q];
                        df_fma1(Pn[c][p], y.x, y.y, sh, sl);
                    }
                    *r = make_float2(sh, sl);
                }
            }
        }
        if (e == 0) continue;
        __syncthreads();
        if (first) {
            if (pl.singular && blockIdx.x == 0 && tid == 0 && a.status) *a.status = CM_ESINGULAR;
            dec = !pl.singular;
        }
        if (dec) {
            for (int u = tid; u < e * tn; u += kThreads) {
                const int c = u / tn, q = u - c * tn;
                float sh = 0.f, sl = 0.f;
#pragma unroll 4
                for (int j = 0; j < e; ++j) {
                    const float2 r = ysm[(ks + j) * kTile + q];
                    df_fma(pl.Qh[c][j], pl.Ql[c][j], r.x, r.y, sh, sl);
                }
                const int64_t out = (int64_t)pl.M[c] * per_block + p0 + t0 + q;
                if (out < mb) store_out(a, out, sh, sl);
            }
        }
        __syncthreads();   // before the next tile overwrites the staging
    }
}

struct DecodeMatArgs {
    CodeParams cp;
    uint32_t survivors;
    const float *Ct;
    int64_t ldc;
    int32_t N;
    float *C;
    int64_t ldcc;
    int32_t *status;
};

// K6: fp32 results, all e missing blocks of one row position (4 columns when
// aligned) per thread, so every surviving element is read once.  Every CTA
// forms the plan and the rows D (as K3), then streams: the loads of a batch
// of survivors are issued together before their FMAs, which apply the rows'
// high parts in fp32.
template <int EMAX>
__global__ void __launch_bounds__(kMatThreads) decode_mat_kernel(const __grid_constant__ DecodeMatArgs a)
{
    __shared__ Plan pl;
    __shared__ float Dh[kMaxE][CM_MAX_N], Dl[kMaxE][CM_MAX_N];
    plan_setup(a.cp, a.survivors, pl);
    const int k = a.cp.k, e = pl.e;
    constexpr int NW = EMAX == 4 ? 1 : 4;
    if (e > 0 && (int)(threadIdx.x >> 5) < NW) plan_eliminate<EMAX, NW>(pl, k);
    __syncthreads();
    const bool dec = e > 0 && !pl.singular;
    if (dec) plan_rows(pl, k, Dh, Dl);
    __syncthreads();
    if (e > 0 && pl.singular && blockIdx.x == 0 && threadIdx.x == 0 && a.status)
        *a.status = CM_ESINGULAR;
    const float *Ct = a.Ct;
    float *C = a.C;
    const int64_t L = a.cp.L, m = a.cp.m, ldc = a.ldc, ldcc = a.ldcc;
    const int N = a.N;
    const bool inplace = C == Ct;
    if (inplace && !dec) return;   // survivors already in place, nothing to decode
    const bool vec = (N % 4 == 0) && (ldc % 4 == 0) && (ldcc % 4 == 0) &&
                     (((uintptr_t)Ct | (uintptr_t)C) & 15u) == 0;
    const int W = vec ? 4 : 1;
    const int64_t nw = N / W;
    const int64_t total = L * nw;
    // survivors whose loads are issued together (fewer with more accumulators)
    constexpr int kBatch = EMAX <= 8 ? 4 : 2;
    for (int64_t it = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; it < total;
         it += (int64_t)gridDim.x * blockDim.x) {
        const int64_t r = it / nw;
        const int64_t col = (it - r * nw) * W;
        float4 acc[EMAX];
#pragma unroll
        for (int c = 0; c < EMAX; ++c) acc[c] = make_float4(0.f, 0.f, 0.f, 0.f);
        for (int p0 = 0; p0 < k; p0 += kBatch) {
            float4 v[kBatch];
#pragma unroll
            for (int u = 0; u < kBatch; ++u) {
                if (p0 + u < k) {
                    const float *src = Ct + ((int64_t)pl.S[p0 + u] * L + r) * ldc + col;
                    v[u] = vec ? __ldg(reinterpret_cast<const float4 *>(src))
                               : make_float4(__ldg(src), 0.f, 0.f, 0.f);
                }
            }
#pragma unroll
            for (int u = 0; u < kBatch; ++u) {
                const int p = p0 + u;
                if (p >= k) break;
                const int s = pl.S[p];
                if (!inplace && s < k) {   // surviving systematic block passes through
                    const int64_t g = (int64_t)s * L + r;
                    if (g < m) {
                        float *dst = C + g * ldcc + col;
                        if (vec) *reinterpret_cast<float4 *>(dst) = v[u];
                        else *dst = v[u].x;
                    }
                }
                if (dec) {
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
        }
        if (dec) {
#pragma unroll
            for (int c = 0; c < EMAX; ++c) {
                if (c < e) {
                    const int64_t g = (int64_t)pl.M[c] * L + r;
                    if (g < m) {
                        float *dst = C + g * ldcc + col;
                        if (vec) *reinterpret_cast<float4 *>(dst) = acc[c];
                        else *dst = acc[c].x;
                    }
                }
            }
        }
    }
}

// CTAs for `items` independent items of `threads` threads, at most `per_sm` per SM.
unsigned grid_for(int64_t items, int threads, int per_sm)
{
    int64_t g = (items + threads - 1) / threads;
    const int64_t cap = (int64_t)(cm_sm_count() > 0 ? cm_sm_count() : 1) * per_sm;
    if (g > cap) g = cap;
    if (g < 1) g = 1;
    return (unsigned)g;
}

// The vector decode, launched as a programmatic dependent.  The dynamic
// shared-memory limit is a property of the function in each device's context,
// so it is set on every call (about 0.2 us), as the other launchers do.
template <int EMAX, int NW>
cudaError_t launch_k3(const DecodeArgs &a, unsigned grid, cudaStream_t s)
{
    constexpr int kSmem = CM_MAX_N * kTile * (int)sizeof(float2);
    auto kern = decode_kernel<EMAX, NW>;
    const cudaError_t attr =
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmem);
    if (attr != cudaSuccess) return attr;
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = kSmem;
    cfg.stream = s;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kern, a);
}

}  // namespace

cudaError_t launch_decode(const CodeParams &cp, const double *Yt, uint32_t survivors, int b,
                          float *Y, int32_t *status, int mode, const float *lab, float eta,
                          bool dependent, cudaStream_t s, int nparts, int64_t part_stride)
{
    DecodeArgs a;
    a.dependent = dependent ? 1 : 0;
    a.nparts = nparts;
    a.part_stride = part_stride;
    a.cp = cp;
    a.b = b;
    a.survivors = survivors;
    a.Yt = Yt;
    a.Y = Y;
    a.status = status;
    a.mode = mode;
    a.lab = lab;
    a.eta = eta;
    // one CTA per SM, at least 64 positions each
    const int64_t per_block = cp.L * (int64_t)b;
    int64_t grid = (per_block + 63) / 64;
    const int64_t sms = cm_sm_count() > 0 ? cm_sm_count() : 1;
    if (grid > sms) grid = sms;
    if (grid < 1) grid = 1;
    a.chunk = (per_block + grid - 1) / grid;
    grid = (per_block + a.chunk - 1) / a.chunk;
    const int e = missing_blocks(cp.k, survivors);
    if (e <= 4) return launch_k3<4, 1>(a, (unsigned)grid, s);
    if (e <= 8) return launch_k3<8, 4>(a, (unsigned)grid, s);
    return launch_k3<16, 4>(a, (unsigned)grid, s);
}

cudaError_t launch_decode_mat(const CodeParams &cp, const float *Ct, int64_t ldc,
                              uint32_t survivors, int N, float *C, int64_t ldcc, int32_t *status,
                              cudaStream_t s)
{
    DecodeMatArgs a;
    a.cp = cp;
    a.survivors = survivors;
    a.Ct = Ct;
    a.ldc = ldc;
    a.N = N;
    a.C = C;
    a.ldcc = ldcc;
    a.status = status;
    const int e = missing_blocks(cp.k, survivors);
    const unsigned g = grid_for(cp.L * (int64_t)N / 4 + 1, kMatThreads, 4);
    if (e <= 4) decode_mat_kernel<4><<<g, kMatThreads, 0, s>>>(a);
    else if (e <= 8) decode_mat_kernel<8><<<g, kMatThreads, 0, s>>>(a);
    else decode_mat_kernel<16><<<g, kMatThreads, 0, s>>>(a);
    return cudaGetLastError();
}
