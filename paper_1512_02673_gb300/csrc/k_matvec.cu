// K2: the n worker products of coded mat-(multi-)vec (Sec. III-A protocol).
//
// Yt[j L + r][v] = sum_c A~_j[r][c] X[c][v] for every worker j < n, block row
// r < L and vector v < b <= 8.  Worker j < k reads its block in place from A
// (rows past m are virtual zeros: never read, result 0); worker j >= k reads
// the parity buffer.
//
// Mapping.  A persistent grid (SMs x resident CTAs).  Work unit = a group of
// R consecutive block rows of one worker, owned by one warp; unit u belongs to
// worker u % n, so consecutive warps stream different workers and all n
// workers progress together, as the n workers of the protocol do.  Lane l of
// a warp reads columns [4l, 4l+4) of every 128-column step of its R rows with
// 128-bit streaming loads (L1 no-allocate), so each coded element is read
// exactly once.  The CTA's warps sweep the columns in lockstep through chunks
// of X staged in shared memory by cp.async (double buffered, one barrier per
// chunk); the smem layout gives every lane its 4 columns x BP vectors with
// conflict-free 128-bit loads.
//
// Precision.  Each lane accumulates R x BP fp32 partials over F steps (4F
// terms).  Then a transposing butterfly over the 32 lanes (each level sends
// half of the values, so 32 values cost 31 shuffles) leaves every lane with
// one complete fp32 partial of 128 F columns, which is added to an fp64
// accumulator.  Results are fp64: decoding multiplies worker results by the
// entries of G_S^-1, so an fp32 rounding of them would be amplified.
#include "cm_internal.cuh"

namespace {

constexpr int kWarps = 8;
constexpr int kThreads = kWarps * 32;

template <int BP>
struct XCfg {
    // columns per staged chunk (about 32 KB of X per buffer)
    static constexpr int CX = 8192 / BP;
    // float stride between the smem groups of the BP = 4 / 8 layouts: the
    // padding makes both the 16-byte cp.async stores and the lane loads hit
    // distinct bank groups.
    static constexpr int GS = BP == 1 ? 0 : (BP == 4 ? CX + 8 : CX + 4);
    static constexpr int FLOATS = BP == 1 ? CX : (BP == 4 ? 4 * GS : 8 * GS);
    static constexpr int BYTES = FLOATS * 4;
};

struct MatvecArgs {
    const float *A;
    int64_t lda;
    const float *par;
    int64_t ldp;
    const float *X;
    double *Yt;
    int64_t m, d, L;
    int32_t n, k, b;
    int32_t fast16;        // X chunks may be staged with 16-byte copies
    int64_t groups;        // total work units
    int64_t groups_per_worker;
};

__device__ __forceinline__ uint32_t smem_addr(const void *p)
{
    return (uint32_t)__cvta_generic_to_shared(p);
}

__device__ __forceinline__ void cp_async16(float *dst, const float *src, int bytes)
{
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(smem_addr(dst)),
                 "l"(src), "r"(bytes));
}

__device__ __forceinline__ void cp_async4(float *dst, const float *src, int bytes)
{
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;\n" ::"r"(smem_addr(dst)),
                 "l"(src), "r"(bytes));
}

__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n"); }
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_group 0;\n" ::: "memory"); }

__device__ __forceinline__ float4 ld_stream4(const float *p)
{
    float4 v;
    asm("ld.global.nc.L1::no_allocate.v4.f32 {%0, %1, %2, %3}, [%4];\n"
        : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
        : "l"(p));
    return v;
}

// Stage columns [c0, c0 + CX) of X into smem buffer xs (zero past d / b).
template <int BP>
__device__ __forceinline__ void stage_x(const MatvecArgs &a, float *xs, int64_t c0)
{
    using C = XCfg<BP>;
    const int tid = threadIdx.x;
    const float *X = a.X;
    if (a.fast16) {
        if constexpr (BP == 1) {
            for (int u = tid; u < C::CX / 4; u += kThreads) {
                int64_t col = c0 + 4 * u;
                int64_t left = a.d - col;
                int bytes = left >= 4 ? 16 : (left > 0 ? (int)left * 4 : 0);
                cp_async16(xs + 4 * u, bytes ? X + col : X, bytes);
            }
        } else {
            constexpr int H = BP / 4;
            for (int u = tid; u < C::CX * H; u += kThreads) {
                int col = u / H, h = u % H;
                int g = (col & 3) * H + h;
                int64_t gc = c0 + col;
                bool in = gc < a.d;
                cp_async16(xs + g * C::GS + (col >> 2) * 4,
                           in ? X + gc * BP + 4 * h : X, in ? 16 : 0);
            }
        }
    } else {
        for (int e = tid; e < C::CX * BP; e += kThreads) {
            int col = e / BP, v = e % BP;
            int64_t gc = c0 + col;
            bool in = gc < a.d && v < a.b;
            int dst;
            if constexpr (BP == 1)
                dst = col;
            else
                dst = ((col & 3) * (BP / 4) + (v >> 2)) * C::GS + (col >> 2) * 4 + (v & 3);
            cp_async4(xs + dst, in ? X + gc * a.b + v : X, in ? 4 : 0);
        }
    }
    cp_async_commit();
}

// Transposing butterfly: V fp32 values per lane -> max(1, V/32) complete sums
// per lane (see the header comment), added into acc64.
template <int V>
__device__ __forceinline__ void flush(float (&t)[V], double (&acc64)[V >= 32 ? V / 32 : 1], int lane)
{
    constexpr int LOGV = V == 1 ? 0 : V == 2 ? 1 : V == 4 ? 2 : V == 8 ? 3 : V == 16 ? 4
                       : V == 32 ? 5 : 6;
#pragma unroll
    for (int l = 0; l < 5; ++l) {
        const int mask = 16 >> l;
        if (l < LOGV) {
            const int half = (V >> l) / 2;
            const bool upper = lane & mask;
#pragma unroll
            for (int i = 0; i < half; ++i) {
                float send = upper ? t[i] : t[i + half];
                float keep = upper ? t[i + half] : t[i];
                t[i] = keep + __shfl_xor_sync(0xffffffffu, send, mask);
            }
        } else {
            t[0] += __shfl_xor_sync(0xffffffffu, t[0], mask);
        }
    }
    constexpr int NH = V >= 32 ? V / 32 : 1;
#pragma unroll
    for (int i = 0; i < NH; ++i) acc64[i] += (double)t[i];
#pragma unroll
    for (int i = 0; i < V; ++i) t[i] = 0.f;
}

template <int BP, int R, int F>
__global__ void __launch_bounds__(kThreads)
matvec_kernel(const MatvecArgs a)
{
    using C = XCfg<BP>;
    constexpr int V = R * BP;
    constexpr int NH = V >= 32 ? V / 32 : 1;
    extern __shared__ __align__(16) float smem[];
    const int lane = threadIdx.x & 31;
    const int warp = threadIdx.x >> 5;
    const int64_t total_warps = (int64_t)gridDim.x * kWarps;
    const int64_t gw = (int64_t)blockIdx.x * kWarps + warp;
    const int64_t rounds = (a.groups + total_warps - 1) / total_warps;
    const int64_t nchunks = (a.d + C::CX - 1) / C::CX;
    const int64_t nseq = rounds * nchunks;
    const int64_t steps = (a.d + 127) / 128;

    stage_x<BP>(a, smem, 0);
    int64_t seq = 0;
    for (int64_t round = 0; round < rounds; ++round) {
        const int64_t g = round * total_warps + gw;
        const bool has = g < a.groups;
        // unit g -> worker j = g % n, rows [rr0, rr0 + R) of that worker
        const int j = has ? (int)(g % a.n) : 0;
        const int64_t rr0 = has ? (g / a.n) * R : 0;
        const float *rowp[R];
#pragma unroll
        for (int r = 0; r < R; ++r) {
            const int64_t rr = rr0 + r;
            rowp[r] = nullptr;
            if (has && rr < a.L) {
                if (j < a.k) {
                    const int64_t gr = (int64_t)j * a.L + rr;
                    if (gr < a.m) rowp[r] = a.A + gr * a.lda;
                } else {
                    rowp[r] = a.par + ((int64_t)(j - a.k) * a.L + rr) * a.ldp;
                }
            }
        }
        float acc[V];
        double acc64[NH];
#pragma unroll
        for (int i = 0; i < V; ++i) acc[i] = 0.f;
#pragma unroll
        for (int i = 0; i < NH; ++i) acc64[i] = 0.0;

        // A for step s of this lane: columns [128 s + 4 lane, +4)
        auto load_step = [&](int64_t s, float4 (&v)[R]) {
            const int64_t col = 128 * s + 4 * lane;
            const bool full = 128 * s + 128 <= a.d;
#pragma unroll
            for (int r = 0; r < R; ++r) {
                v[r] = make_float4(0.f, 0.f, 0.f, 0.f);
                if (rowp[r]) {
                    if (full) {
                        v[r] = ld_stream4(rowp[r] + col);
                    } else {
                        const float *p = rowp[r] + col;
                        if (col + 0 < a.d) v[r].x = __ldg(p + 0);
                        if (col + 1 < a.d) v[r].y = __ldg(p + 1);
                        if (col + 2 < a.d) v[r].z = __ldg(p + 2);
                        if (col + 3 < a.d) v[r].w = __ldg(p + 3);
                    }
                }
            }
        };

        float4 cur[R], nxt[R];
        if (has) load_step(0, cur);
        int fl = 0;
        int64_t s = 0;
        for (int64_t ch = 0; ch < nchunks; ++ch, ++seq) {
            cp_async_wait_all();
            __syncthreads();   // chunk `seq` visible; buffer of seq+1 free
            if (seq + 1 < nseq)
                stage_x<BP>(a, smem + ((seq + 1) & 1) * C::FLOATS,
                            ((seq + 1) % nchunks) * C::CX);
            if (!has) continue;
            const float *xb = smem + (seq & 1) * C::FLOATS;
            const int64_t send = min(steps, (ch + 1) * (C::CX / 128));
            for (; s < send; ++s) {
                if (s + 1 < steps) load_step(s + 1, nxt);
                const int c4 = (int)(s - ch * (C::CX / 128)) * 32 + lane;
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    float x[BP];
                    if constexpr (BP == 1) {
                        const float4 xv = *reinterpret_cast<const float4 *>(xb + 4 * c4);
                        x[0] = q == 0 ? xv.x : q == 1 ? xv.y : q == 2 ? xv.z : xv.w;
                    } else {
#pragma unroll
                        for (int h = 0; h < BP / 4; ++h) {
                            const float4 xv = *reinterpret_cast<const float4 *>(
                                xb + (q * (BP / 4) + h) * C::GS + 4 * c4);
                            x[4 * h + 0] = xv.x;
                            x[4 * h + 1] = xv.y;
                            x[4 * h + 2] = xv.z;
                            x[4 * h + 3] = xv.w;
                        }
                    }
#pragma unroll
                    for (int r = 0; r < R; ++r) {
                        const float av = q == 0 ? cur[r].x : q == 1 ? cur[r].y
                                       : q == 2 ? cur[r].z : cur[r].w;
#pragma unroll
                        for (int v = 0; v < BP; ++v)
                            acc[r * BP + v] = fmaf(av, x[v], acc[r * BP + v]);
                    }
                }
#pragma unroll
                for (int r = 0; r < R; ++r) cur[r] = nxt[r];
                if (++fl == F) {
                    flush<V>(acc, acc64, lane);
                    fl = 0;
                }
            }
        }
        if (!has) continue;
        if (fl) flush<V>(acc, acc64, lane);
        // lane holds value index vi = r * BP + v
        const int64_t base = (int64_t)j * a.L + rr0;
        if constexpr (V >= 32) {
#pragma unroll
            for (int i = 0; i < NH; ++i) {
                const int vi = lane * NH + i;
                const int r = vi / BP, v = vi % BP;
                if (v < a.b && rr0 + r < a.L) a.Yt[(base + r) * a.b + v] = acc64[i];
            }
        } else {
            constexpr int SHIFT = V == 1 ? 5 : V == 2 ? 4 : V == 4 ? 3 : V == 8 ? 2 : 1;
            if ((lane & ((1 << SHIFT) - 1)) == 0) {
                const int vi = lane >> SHIFT;
                const int r = vi / BP, v = vi % BP;
                if (v < a.b && rr0 + r < a.L) a.Yt[(base + r) * a.b + v] = acc64[0];
            }
        }
    }
    cp_async_wait_all();
}

template <int BP, int R, int F>
cudaError_t launch_bp(MatvecArgs a, cudaStream_t s)
{
    using C = XCfg<BP>;
    auto kern = matvec_kernel<BP, R, F>;
    const int smem = 2 * C::BYTES;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    int per_sm = 0;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kThreads, smem);
    if (e != cudaSuccess) return e;
    if (per_sm < 1) per_sm = 1;
    a.groups_per_worker = (a.L + R - 1) / R;
    a.groups = a.groups_per_worker * a.n;
    const int64_t need = (a.groups + kWarps - 1) / kWarps;
    int64_t grid = (int64_t)cm_sm_count() * per_sm;
    if (grid < 1) grid = 1;
    if (grid > need) grid = need;
    kern<<<(unsigned)grid, kThreads, smem, s>>>(a);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_matvec(const CodeParams &cp, const float *A, int64_t lda, const float *par,
                          int64_t ldp, const float *X, int b, double *Yt, cudaStream_t s)
{
    MatvecArgs a;
    a.A = A;
    a.lda = lda;
    a.par = par;
    a.ldp = ldp;
    a.X = X;
    a.Yt = Yt;
    a.m = cp.m;
    a.d = cp.d;
    a.L = cp.L;
    a.n = cp.n;
    a.k = cp.k;
    a.b = b;
    a.groups = 0;
    a.groups_per_worker = 0;
    const bool x16 = ((uintptr_t)X & 15u) == 0;
    if (b == 1) {
        a.fast16 = x16;
        return launch_bp<1, 8, 8>(a, s);
    }
    if (b <= 4) {
        a.fast16 = x16 && b == 4;
        return launch_bp<4, 4, 4>(a, s);
    }
    a.fast16 = x16 && b == 8;
    return launch_bp<8, 4, 4>(a, s);
}
