// K1: encoding (Sec. III-A): parity block p = sum_i P[p][i] A_i for every
// parity block p of the (n,k) code, applied elementwise across the k row
// blocks of A (rows past m are the appended zero rows and are skipped).
//
// A short contraction (k <= 31) that streams A once: each thread owns one
// 16-byte vector of columns of one block row r, reads the k vectors
// A_i[r][cols] with 128-bit loads (held in flight in groups of 4) and keeps
// all NPG parity accumulators of that vector in registers, so every element
// of A is read once per pass and every parity element written once
// (n - k <= NPG: one pass).  fp32 accumulation; bf16 outputs are rounded to
// nearest even once, at the end.  The grid is persistent (SMs x resident
// CTAs) over a flattened (row, column vector) space, so accesses are
// coalesced along rows.
#include <cuda_bf16.h>

#include "cm_internal.cuh"

namespace {

constexpr int kThreads = 256;

struct EncodeArgs {
    CodeParams cp;
    const void *A;
    int64_t lda;
    void *par;
    int64_t ldp;
    int p0;   // first parity block of this pass
    int np;   // parity blocks in this pass
};

template <typename T>
struct Vec;
template <>
struct Vec<float> {
    static constexpr int W = 4;
    __device__ static void load(const float *p, float (&v)[4])
    {
        float4 t;
        asm("ld.global.nc.L1::no_allocate.v4.f32 {%0, %1, %2, %3}, [%4];\n"
            : "=f"(t.x), "=f"(t.y), "=f"(t.z), "=f"(t.w)
            : "l"(p));
        v[0] = t.x; v[1] = t.y; v[2] = t.z; v[3] = t.w;
    }
    __device__ static float scalar(const float *p) { return __ldg(p); }
    __device__ static void store(float *p, const float (&v)[4])
    {
        __stcs(reinterpret_cast<float4 *>(p), make_float4(v[0], v[1], v[2], v[3]));
    }
    __device__ static void store_scalar(float *p, float v) { *p = v; }
};
template <>
struct Vec<uint16_t> {   // bf16 bits
    static constexpr int W = 8;
    __device__ static float widen(uint32_t h) { return __uint_as_float(h << 16); }
    __device__ static void load(const uint16_t *p, float (&v)[8])
    {
        uint4 t;
        asm("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];\n"
            : "=r"(t.x), "=r"(t.y), "=r"(t.z), "=r"(t.w)
            : "l"(p));
        const uint32_t w[4] = {t.x, t.y, t.z, t.w};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            v[2 * i] = widen(w[i] & 0xffffu);
            v[2 * i + 1] = widen(w[i] >> 16);
        }
    }
    __device__ static float scalar(const uint16_t *p) { return widen(__ldg(p)); }
    __device__ static uint32_t rne(float f)
    {
        return (uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(f));
    }
    __device__ static void store(uint16_t *p, const float (&v)[8])
    {
        uint4 t;
        t.x = rne(v[0]) | (rne(v[1]) << 16);
        t.y = rne(v[2]) | (rne(v[3]) << 16);
        t.z = rne(v[4]) | (rne(v[5]) << 16);
        t.w = rne(v[6]) | (rne(v[7]) << 16);
        __stcs(reinterpret_cast<uint4 *>(p), t);
    }
    __device__ static void store_scalar(uint16_t *p, float v) { *p = (uint16_t)rne(v); }
};

template <typename T, int NPG>
__global__ void __launch_bounds__(kThreads) encode_kernel(const EncodeArgs a)
{
    constexpr int W = Vec<T>::W;
    constexpr int G = 4;   // data blocks loaded per group
    const int k = a.cp.k, np = a.np, p0 = a.p0;
    const int64_t L = a.cp.L, m = a.cp.m, d = a.cp.d;
    const int64_t nvec = (d + W - 1) / W;
    const int64_t total = L * nvec;
    const T *A = static_cast<const T *>(a.A);
    T *par = static_cast<T *>(a.par);
    for (int64_t it = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; it < total;
         it += (int64_t)gridDim.x * blockDim.x) {
        const int64_t r = it / nvec;
        const int64_t col = (it - r * nvec) * W;
        const bool full = col + W <= d;
        float acc[NPG][W];
#pragma unroll
        for (int j = 0; j < NPG; ++j)
#pragma unroll
            for (int e = 0; e < W; ++e) acc[j][e] = 0.f;
        for (int i0 = 0; i0 < k; i0 += G) {
            float v[G][W];
#pragma unroll
            for (int g = 0; g < G; ++g) {
                const int i = i0 + g;
                const int64_t row = (int64_t)i * L + r;
#pragma unroll
                for (int e = 0; e < W; ++e) v[g][e] = 0.f;
                if (i < k && row < m) {
                    const T *src = A + row * a.lda + col;
                    if (full) {
                        Vec<T>::load(src, v[g]);
                    } else {
#pragma unroll
                        for (int e = 0; e < W; ++e)
                            if (col + e < d) v[g][e] = Vec<T>::scalar(src + e);
                    }
                }
            }
#pragma unroll
            for (int g = 0; g < G; ++g) {
                const int i = i0 + g;
                if (i >= k) break;
#pragma unroll
                for (int j = 0; j < NPG; ++j) {
                    if (j < np) {
                        const float w = a.cp.P[(p0 + j) * k + i];
#pragma unroll
                        for (int e = 0; e < W; ++e) acc[j][e] = fmaf(w, v[g][e], acc[j][e]);
                    }
                }
            }
        }
#pragma unroll
        for (int j = 0; j < NPG; ++j) {
            if (j < np) {
                T *dst = par + ((int64_t)(p0 + j) * L + r) * a.ldp + col;
                if (full) {
                    Vec<T>::store(dst, acc[j]);
                } else {
#pragma unroll
                    for (int e = 0; e < W; ++e)
                        if (col + e < d) Vec<T>::store_scalar(dst + e, acc[j][e]);
                }
            }
        }
    }
}

template <typename T, int NPG>
cudaError_t launch_passes(const CodeParams &cp, const void *A, int64_t lda, void *par,
                          int64_t ldp, cudaStream_t s)
{
    auto kern = encode_kernel<T, NPG>;
    int per_sm = 0;
    cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kThreads, 0);
    if (e != cudaSuccess) return e;
    if (per_sm < 1) per_sm = 1;
    const int64_t W = Vec<T>::W;
    const int64_t items = cp.L * ((cp.d + W - 1) / W);
    int64_t grid = (int64_t)cm_sm_count() * per_sm;
    const int64_t need = (items + kThreads - 1) / kThreads;
    if (grid > need) grid = need;
    if (grid < 1) grid = 1;
    EncodeArgs a;
    a.cp = cp;
    a.A = A;
    a.lda = lda;
    a.par = par;
    a.ldp = ldp;
    for (int p0 = 0; p0 < cp.n - cp.k; p0 += NPG) {
        a.p0 = p0;
        a.np = cp.n - cp.k - p0 < NPG ? cp.n - cp.k - p0 : NPG;
        kern<<<(unsigned)grid, kThreads, 0, s>>>(a);
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
    }
    return cudaSuccess;
}

}  // namespace

cudaError_t launch_encode_f32(const CodeParams &cp, const float *A, int64_t lda, float *par,
                              int64_t ldp, cudaStream_t s)
{
    if (cp.n - cp.k <= 8) return launch_passes<float, 8>(cp, A, lda, par, ldp, s);
    return launch_passes<float, 16>(cp, A, lda, par, ldp, s);
}

cudaError_t launch_encode_bf16(const CodeParams &cp, const uint16_t *A, int64_t lda,
                               uint16_t *par, int64_t ldp, cudaStream_t s)
{
    return launch_passes<uint16_t, 8>(cp, A, lda, par, ldp, s);
}
