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
// Every CTA forms these coefficients itself in shared memory (one warp, fp64),
// then the CTA's threads apply them: missing block M[c] row r is the
// combination of the k surviving rows r, surviving systematic blocks pass
// through.  A zero (or relatively negligible) pivot marks G_S singular: the
// kernel writes CM_ESINGULAR to the status word and writes no output.
//
// fp64 arithmetic runs at about 1/58 of the fp32 rate on this part, so the
// vector decode applies the fp64 coefficients in double-float arithmetic on
// the fp32 pipe: each fp64 coefficient and each fp64 worker result is split
// into a (high, low) fp32 pair (results by integer bit manipulation, no fp64
// instruction), products are formed exactly with an FMA and the sums are kept
// as (sum, compensation) pairs (Knuth's TwoSum), about 2^-44 relative per
// term, far below the rounding of the fp32 output.
#include <cfloat>

#include "cm_internal.cuh"

namespace {

constexpr int kThreads = 256;
constexpr int kMaxE = 16;   // e <= min(k, n - k) <= 16 for n <= 32

struct DecodeShared {
    int S[CM_MAX_N];       // survivors in ascending order (k of them)
    int role[CM_MAX_N];    // block i < k: -1 passes through, else its row c in M
    int M[kMaxE];          // missing systematic blocks, ascending
    int Ps[kMaxE];         // surviving parity workers, ascending
    int e;
    int singular;
    double W[kMaxE][2 * kMaxE];   // [Q | I] during elimination
    double Qi[kMaxE][kMaxE];      // Q^-1
    double D[kMaxE][CM_MAX_N];    // decode rows: D[c][p], p = position in S
    float Dh[kMaxE][CM_MAX_N];    // D as (high, low) fp32 pairs
    float Dl[kMaxE][CM_MAX_N];
};

// Warp 0: the survivor lists (S, role, M, Ps, e) from the mask, by ballots.
__device__ void decode_select(const CodeParams &cp, uint32_t survivors, DecodeShared &sh)
{
    const int lane = threadIdx.x & 31;
    const int n = cp.n, k = cp.k;
    const uint32_t below = (1u << lane) - 1u;
    // the first k set bits of the mask are the survivors used
    const bool set = lane < n && ((survivors >> lane) & 1u);
    const bool sel = set && __popc(survivors & below) < k;
    const uint32_t selm = __ballot_sync(0xffffffffu, sel);
    const bool miss = lane < k && !sel;
    const uint32_t missm = __ballot_sync(0xffffffffu, miss);
    const bool par = sel && lane >= k;
    const uint32_t parm = __ballot_sync(0xffffffffu, par);
    if (sel) sh.S[__popc(selm & below)] = lane;
    if (par) sh.Ps[__popc(parm & below)] = lane;
    if (miss) sh.M[__popc(missm & below)] = lane;
    if (lane < k) sh.role[lane] = miss ? __popc(missm & below) : -1;
    if (lane == 0) {
        sh.e = __popc(missm);
        sh.singular = 0;
    }
}

// Warp 0: rows of G_S^-1 for the missing blocks (D, and D as fp32 pairs).
// fp64 instructions have long latency on this part (about 64 cycles for a
// multiply or FMA, about 440 for a reciprocal), so the elimination is
// fraction-free: a non-pivot row becomes piv * W[a] - W[a][col] * W[col]
// (separate products, so duplicated rows cancel to exactly zero), with one
// reciprocal per row at the end; partial pivoting is unaffected because all
// non-pivot rows are scaled alike.  G_S counts as singular when a pivot is
// zero or not finite, or when ||Q||_inf ||Q^-1||_inf exceeds 1 / (64 eps).
__device__ void decode_coefficients(const CodeParams &cp, DecodeShared &sh)
{
    const int lane = threadIdx.x & 31;
    const int k = cp.k, e = sh.e;
    if (e == 0) return;
    const int mc = lane < e ? sh.M[lane] : 0;
    // W = [Q | I], Q[a][c] = P[Ps[a] - k][M[c]]; lane owns column `lane`.
    double qnorm = 0.0;   // row sums of |Q| (lane a < e holds row a)
    for (int a = 0; a < e; ++a) {
        const int ps = sh.Ps[a];
        double w = 0.0;
        if (lane < e) w = (double)cp.P[(ps - k) * k + mc];
        else if (lane < 2 * e) w = (lane - e == a) ? 1.0 : 0.0;
        if (lane < 2 * e) sh.W[a][lane] = w;
    }
    __syncwarp();
    if (lane < e)
        for (int c = 0; c < e; ++c) qnorm += fabs(sh.W[lane][c]);
    for (int off = 16; off; off >>= 1) qnorm = fmax(qnorm, __shfl_xor_sync(0xffffffffu, qnorm, off));
    int singular = 0;
    for (int col = 0; col < e; ++col) {
        // partial pivoting on the fp32 image of |W[a][col]| (a >= col), lowest
        // index on ties; any near-largest pivot is as good numerically
        const double wl = lane >= col && lane < e ? sh.W[lane][col] : 0.0;
        float best = lane >= col && lane < e ? (float)fabs(wl) : -1.f;
        int bi = lane;
        for (int off = 16; off; off >>= 1) {
            const float ob = __shfl_xor_sync(0xffffffffu, best, off);
            const int oi = __shfl_xor_sync(0xffffffffu, bi, off);
            if (ob > best || (ob == best && oi < bi)) {
                best = ob;
                bi = oi;
            }
        }
        const double bval = __shfl_sync(0xffffffffu, wl, bi);
        if (!(fabs(bval) > 0.0) || !isfinite(bval)) {
            singular = 1;
            break;
        }
        if (bi != col && lane < 2 * e) {
            const double t = sh.W[col][lane];
            sh.W[col][lane] = sh.W[bi][lane];
            sh.W[bi][lane] = t;
        }
        __syncwarp();
        if (lane < 2 * e) {
            // lane owns column `lane`; column `col` of the non-pivot rows becomes 0
            const double piv = bval;
            const double wc = sh.W[col][lane];
            for (int a = 0; a < e; ++a) {
                if (a == col) continue;
                const double fa = sh.W[a][col];      // read before anyone writes it
                const double wa = sh.W[a][lane];
                __syncwarp(__activemask());
                sh.W[a][lane] = lane == col ? 0.0 : piv * wa - fa * wc;
            }
        }
        __syncwarp();
    }
    if (!singular) {
        // Q^-1[c][a] = W[c][e + a] / W[c][c]
        const double dinv = lane < e ? 1.0 / sh.W[lane][lane] : 0.0;
        double qimax = 0.0;
        for (int t = lane; t < 32 * ((e * e + 31) / 32); t += 32) {
            const int c = t / e, aa = t % e;
            const double dc = __shfl_sync(0xffffffffu, dinv, t < e * e ? c : 0);
            if (t < e * e) {
                const double q = sh.W[c][e + aa] * dc;
                sh.Qi[c][aa] = q;
                qimax = fmax(qimax, fabs(q));
            }
        }
        for (int off = 16; off; off >>= 1)
            qimax = fmax(qimax, __shfl_xor_sync(0xffffffffu, qimax, off));
        // ||Q^-1||_inf <= e max|Q^-1|
        if (!(qnorm * qimax * e < 1.0 / (64.0 * DBL_EPSILON))) singular = 1;
    }
    if (singular) {
        if (lane == 0) sh.singular = 1;
        __syncwarp();
        return;
    }
    __syncwarp();
    // D[c][p] (p = position in S): independent e-term chains, two per lane
    auto d_entry = [&](int t, double &v) {
        const int c = t / k, p = t % k;
        const int s = sh.S[p];
        if (s >= k) {
            int aa = 0;
            while (sh.Ps[aa] != s) ++aa;
            v = sh.Qi[c][aa];
            return;
        }
        v = 0.0;
        for (int aa = 0; aa < e; ++aa)
            v = fma(-sh.Qi[c][aa], (double)cp.P[(sh.Ps[aa] - k) * k + s], v);
    };
    for (int t = lane; t < e * k; t += 64) {
        double v0 = 0.0, v1 = 0.0;
        const int t1 = t + 32;
        d_entry(t, v0);
        if (t1 < e * k) d_entry(t1, v1);
        for (int q = 0; q < 2; ++q) {
            const int tt = q ? t1 : t;
            if (tt >= e * k) break;
            const double v = q ? v1 : v0;
            const int c = tt / k, p = tt % k;
            sh.D[c][p] = v;
            const float h = __double2float_rn(v);
            sh.Dh[c][p] = h;
            sh.Dl[c][p] = __double2float_rn(v - (double)h);
        }
    }
    __syncwarp();
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

struct DecodeArgs {
    CodeParams cp;
    const double *Yt;
    uint32_t survivors;
    int b;
    float *Y;
    int32_t *status;
    int mode;
    const float *lab;
    float eta;
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

__global__ void __launch_bounds__(kThreads) decode_kernel(const DecodeArgs a)
{
    __shared__ DecodeShared sh;
    const int warp = threadIdx.x >> 5;
    if (warp == 0) decode_select(a.cp, a.survivors, sh);
    __syncthreads();
    const int k = a.cp.k, e = sh.e;
    const int64_t L = a.cp.L, m = a.cp.m;
    const int b = a.b;
    const int64_t per_block = L * b;
    if (warp == 0) {
        decode_coefficients(a.cp, sh);
    } else {
        // meanwhile the other warps pass the surviving systematic blocks
        // through (exactly rounded to fp32), four independent loads at a time
        const int64_t npass = (int64_t)(k - e) * per_block;
        const int64_t stride = (int64_t)gridDim.x * (blockDim.x - 32);
        for (int64_t it0 = (int64_t)blockIdx.x * (blockDim.x - 32) + threadIdx.x - 32;
             it0 < npass; it0 += 4 * stride) {
            double y[4];
            int64_t out[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int64_t it = it0 + u * stride;
                out[u] = -1;
                if (it < npass) {
                    const int t = (int)(it / per_block);
                    const int64_t o = (int64_t)sh.S[t] * per_block + (it - (int64_t)t * per_block);
                    if (o < m * b) {
                        out[u] = o;
                        y[u] = a.Yt[o];
                    }
                }
            }
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                if (out[u] < 0) continue;
                if (a.mode == DEC_PLAIN) {
                    a.Y[out[u]] = __double2float_rn(y[u]);
                } else {
                    float yh, yl;
                    split_double(y[u], yh, yl);
                    store_out(a, out[u], yh, yl);
                }
            }
        }
    }
    __syncthreads();
    if (sh.singular) {
        if (threadIdx.x == 0 && a.status) *a.status = CM_ESINGULAR;
        return;
    }
    // missing systematic blocks: up to CG of them per thread, one row position;
    // the k surviving values are loaded before any arithmetic
    const int ngroups = (e + CG - 1) / CG;
    const int64_t ndec = (int64_t)ngroups * per_block;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t it = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; it < ndec; it += stride) {
        const int g = (int)(it / per_block);
        const int64_t rv = it - (int64_t)g * per_block;
        const int c0 = g * CG;
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
                if (out < m * b) store_out(a, out, sh_[c], sl_[c]);
            }
        }
    }
}

// K6: fp32 results, all e missing blocks of one row position per thread, so
// every surviving element is read once.
template <int EMAX>
__global__ void __launch_bounds__(kThreads)
decode_mat_kernel(const CodeParams cp, const float *Ct, int64_t ldc, uint32_t survivors, int N,
                  float *C, int64_t ldcc, int32_t *status)
{
    __shared__ DecodeShared sh;
    __shared__ float Df[kMaxE][CM_MAX_N];
    if (threadIdx.x < 32) {
        decode_select(cp, survivors, sh);
        __syncwarp();
        decode_coefficients(cp, sh);
    }
    __syncthreads();
    if (sh.singular) {
        if (threadIdx.x == 0 && status) *status = CM_ESINGULAR;
        return;
    }
    const int k = cp.k, e = sh.e;
    for (int t = threadIdx.x; t < e * k; t += blockDim.x) Df[t / k][t % k] = (float)sh.D[t / k][t % k];
    __syncthreads();
    const int64_t L = cp.L, m = cp.m;
    const bool inplace = C == Ct;
    const bool vec = (N % 4 == 0) && (ldc % 4 == 0) && (ldcc % 4 == 0) &&
                     (((uintptr_t)Ct | (uintptr_t)C) & 15u) == 0;
    const int W = vec ? 4 : 1;
    const int64_t nw = N / W;
    const int64_t total = L * nw;
    int M[EMAX];
    {
        int cnt = 0;
        for (int i = 0; i < k && cnt < EMAX; ++i)
            if (sh.role[i] >= 0) M[cnt++] = i;
        for (; cnt < EMAX; ++cnt) M[cnt] = 0;
    }
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
                    const float w = Df[c][p];
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

// Every CTA inverts the small block of G_S itself, so the grid is capped at
// `per_sm` CTAs per SM: enough to stream the results, few enough that the
// (slow on this part) fp64 inverse is not repeated needlessly.
int grid_for(int64_t items, int per_sm)
{
    int64_t g = (items + kThreads - 1) / kThreads;
    const int64_t cap = (int64_t)(cm_sm_count() > 0 ? cm_sm_count() : 1) * per_sm;
    if (g > cap) g = cap;
    if (g < 1) g = 1;
    return (int)g;
}

}  // namespace

cudaError_t launch_decode(const CodeParams &cp, const double *Yt, uint32_t survivors, int b,
                          float *Y, int32_t *status, int mode, const float *lab, float eta,
                          cudaStream_t s)
{
    DecodeArgs a;
    a.cp = cp;
    a.Yt = Yt;
    a.survivors = survivors;
    a.b = b;
    a.Y = Y;
    a.status = status;
    a.mode = mode;
    a.lab = lab;
    a.eta = eta;
    decode_kernel<<<grid_for((int64_t)cp.k * cp.L * b / 2 + 1, 2), kThreads, 0, s>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_decode_mat(const CodeParams &cp, const float *Ct, int64_t ldc,
                              uint32_t survivors, int N, float *C, int64_t ldcc, int32_t *status,
                              cudaStream_t s)
{
    // e = number of missing systematic blocks among the first k survivors
    int e = 0, cnt = 0;
    for (int j = 0; j < cp.n && cnt < cp.k; ++j)
        if ((survivors >> j) & 1u) {
            ++cnt;
            if (j >= cp.k) ++e;
        }
    const int64_t items = cp.L * (int64_t)N / 4 + 1;
    const int g = grid_for(items, 4);
    if (e <= 4)
        decode_mat_kernel<4><<<g, kThreads, 0, s>>>(cp, Ct, ldc, survivors, N, C, ldcc, status);
    else if (e <= 8)
        decode_mat_kernel<8><<<g, kThreads, 0, s>>>(cp, Ct, ldc, survivors, N, C, ldcc, status);
    else
        decode_mat_kernel<16><<<g, kThreads, 0, s>>>(cp, Ct, ldc, survivors, N, C, ldcc, status);
    return cudaGetLastError();
}
