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
#include <cfloat>

#include "cm_internal.cuh"

namespace {

constexpr int kThreads = 256;
constexpr int kMaxE = 16;   // e <= min(k, n - k) <= 16 for n <= 32

struct DecodeShared {
    int S[CM_MAX_N];       // survivors in ascending order (k of them)
    int role[CM_MAX_N];    // block i < k: -1 passes through, else its row c in M
    int Ps[kMaxE];         // surviving parity workers, ascending
    int e;
    int singular;
    double W[kMaxE][2 * kMaxE];   // [Q | I] during elimination
    double Qi[kMaxE][kMaxE];      // Q^-1
    double D[kMaxE][CM_MAX_N];    // decode rows: D[c][p], p = position in S
};

// Warp 0 of the CTA fills sh (S, role, e, D, singular).
__device__ void decode_coefficients(const CodeParams &cp, uint32_t survivors, DecodeShared &sh)
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
    const int e = __popc(missm);
    if (sel) sh.S[__popc(selm & below)] = lane;
    if (par) sh.Ps[__popc(parm & below)] = lane;
    if (lane < k) sh.role[lane] = miss ? __popc(missm & below) : -1;
    // per-lane copies of the M and Ps lists (lane-indexed via shuffles)
    int Mi = -1, Pi = -1;
    {
        // position of each missing / parity worker in its list
        int mpos = miss ? __popc(missm & below) : -1;
        int ppos = par ? __popc(parm & below) : -1;
        // gather: list element t is the lane whose pos == t
        for (int src = 0; src < 32; ++src) {
            int pm = __shfl_sync(0xffffffffu, mpos, src);
            int pp = __shfl_sync(0xffffffffu, ppos, src);
            if (pm == lane) Mi = src;
            if (pp == lane) Pi = src;
        }
    }
    if (lane == 0) {
        sh.e = e;
        sh.singular = 0;
    }
    if (e == 0) {
        __syncwarp();
        return;
    }
    // W = [Q | I], Q[a][c] = P[Ps[a] - k][M[c]]; lane owns column `lane`.
    double scale = 0.0;
    const int mc = __shfl_sync(0xffffffffu, Mi, lane < e ? lane : 0);   // M[lane]
    for (int a = 0; a < e; ++a) {
        const int ps = __shfl_sync(0xffffffffu, Pi, a);                   // Ps[a]
        double w = 0.0;
        if (lane < e) {
            w = (double)cp.P[(ps - k) * k + mc];
            scale = fmax(scale, fabs(w));
        } else if (lane < 2 * e) {
            w = (lane - e == a) ? 1.0 : 0.0;
        }
        if (lane < 2 * e) sh.W[a][lane] = w;
    }
    for (int off = 16; off; off >>= 1) scale = fmax(scale, __shfl_xor_sync(0xffffffffu, scale, off));
    const double tol = 64.0 * DBL_EPSILON * scale;
    __syncwarp();
    int singular = 0;
    for (int col = 0; col < e && !singular; ++col) {
        // partial pivoting: largest |W[a][col]| over a >= col, lowest index on ties
        double best = lane >= col && lane < e ? fabs(sh.W[lane][col]) : -1.0;
        int bi = lane;
        for (int off = 16; off; off >>= 1) {
            const double ob = __shfl_xor_sync(0xffffffffu, best, off);
            const int oi = __shfl_xor_sync(0xffffffffu, bi, off);
            if (ob > best || (ob == best && oi < bi)) {
                best = ob;
                bi = oi;
            }
        }
        if (!(best > tol)) {   // also catches NaN
            singular = 1;
            break;
        }
        if (bi != col && lane < 2 * e) {
            const double t = sh.W[col][lane];
            sh.W[col][lane] = sh.W[bi][lane];
            sh.W[bi][lane] = t;
        }
        __syncwarp();
        const double rp = 1.0 / sh.W[col][col];
        double f[kMaxE];
#pragma unroll
        for (int a = 0; a < kMaxE; ++a) f[a] = a < e ? sh.W[a][col] * rp : 0.0;
        __syncwarp();
        if (lane < 2 * e) {
            const double wc = sh.W[col][lane];
#pragma unroll
            for (int a = 0; a < kMaxE; ++a)
                if (a < e && a != col) sh.W[a][lane] -= f[a] * wc;
        }
        __syncwarp();
    }
    if (singular) {
        if (lane == 0) sh.singular = 1;
        __syncwarp();
        return;
    }
    // Q^-1[c][a] = W[c][e + a] / W[c][c]
    for (int t = lane; t < e * e; t += 32) {
        const int c = t / e, aa = t % e;
        sh.Qi[c][aa] = sh.W[c][e + aa] / sh.W[c][c];
    }
    __syncwarp();
    // lane p < k builds column p of D (p = position in S)
    if (lane < k) {
        const int s = sh.S[lane];
        if (s >= k) {
            const int aa = __popc(parm & ((1u << s) - 1u));
            for (int c = 0; c < e; ++c) sh.D[c][lane] = sh.Qi[c][aa];
        } else {
            for (int c = 0; c < e; ++c) {
                double v = 0.0;
                for (int aa = 0; aa < e; ++aa)
                    v = fma(-sh.Qi[c][aa], (double)cp.P[(sh.Ps[aa] - k) * k + s], v);
                sh.D[c][lane] = v;
            }
        }
    }
    __syncwarp();
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

__global__ void __launch_bounds__(kThreads) decode_kernel(const DecodeArgs a)
{
    __shared__ DecodeShared sh;
    if (threadIdx.x < 32) decode_coefficients(a.cp, a.survivors, sh);
    __syncthreads();
    if (sh.singular) {
        if (threadIdx.x == 0 && a.status) *a.status = CM_ESINGULAR;
        return;
    }
    const int k = a.cp.k;
    const int64_t L = a.cp.L, m = a.cp.m;
    const int b = a.b;
    const int64_t per_block = L * b;
    const int64_t total = (int64_t)k * per_block;
    for (int64_t it = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; it < total;
         it += (int64_t)gridDim.x * blockDim.x) {
        const int i = (int)(it / per_block);
        const int64_t rv = it - (int64_t)i * per_block;     // r * b + v within the block
        const int64_t out = (int64_t)i * per_block + rv;     // row-major index into Y
        if (out >= m * b) continue;                          // appended zero rows
        const int c = sh.role[i];
        double y;
        if (c < 0) {
            y = a.Yt[out];                                   // surviving systematic block
        } else {
            y = 0.0;
            for (int p = 0; p < k; ++p) y = fma(sh.D[c][p], a.Yt[(int64_t)sh.S[p] * per_block + rv], y);
        }
        if (a.mode == DEC_PLAIN) {
            a.Y[out] = (float)y;
        } else if (a.mode == DEC_RESIDUAL) {
            a.Y[out] = (float)(y - (double)a.lab[out]);         // z = A x - y
        } else {
            a.Y[out] = (float)((double)a.Y[out] - (double)a.eta * y);   // x -= eta g
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
    if (threadIdx.x < 32) decode_coefficients(cp, survivors, sh);
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
    decode_kernel<<<grid_for((int64_t)cp.k * cp.L * b, 1), kThreads, 0, s>>>(a);
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
