// K1: encoding (Sec. III-A): parity block p = sum_i P[p][i] A_i for every
// parity block p of the (n,k) code, applied elementwise across the k row
// blocks of A (rows past m are the appended zero rows).
//
// A short contraction (k <= 31 terms per output) that streams A once and
// writes the parity once.  Two forms, both with fp32 accumulation in the
// order i = 0..k-1 (so they give the same bits) and bf16 outputs rounded to
// nearest even once:
//
// Elementwise (k <= 8, or k <= 16 with at least k/2 parity blocks): thread t
// loads 4 columns of one block row from every data block with plain vector
// loads, forms every parity block's sum with the coefficients as constant
// operands, and stores 4 columns of every parity block.  Many resident warps
// with few instructions per byte: on short codes, whose writes are as large
// as their reads, this keeps more requests in flight than a TMA ring in the
// same shared memory, and runs at the rate of a plain copy of the same bytes.
//
// Tiled (the rest): a work unit = one block row r and a segment of steps of
// 128 columns, owned by one CTA; warp w takes the segment's steps w, w + 8,
// ..., so that the CTA's warps read and write adjacent 512-byte pieces of
// every row at once.  A persistent grid sweeps the units; the launcher takes
// the longest segment whose units fill the rounds of the grid to 90 %.  Each
// step gathers row r of every data block into shared memory with TMA in
// sub-steps of KC blocks: 3-D boxes of KC full blocks (block stride L rows;
// boxes past the last full block read as zero) plus, if m is not a multiple
// of L, one 2-D box of the partial block whose rows past m read as zero;
// blocks wholly past m are skipped.  Sub-steps stream through a per-warp ring
// of ST = 2 slots with one mbarrier each (lane 0 issues, the warp consumes),
// so several KB per warp are in flight with no per-lane copy work, and small
// rings leave room for 2 or 3 CTAs of 8 warps per SM (registers decide: 3
// for up to 4 parity blocks).  A third slot per warp measured up to 5 %
// slower.  Lane l owns columns [4l, 4l+4) of
// the step and keeps the accumulators of all parity blocks of the pass in
// registers (packed fp32x2 FMAs with the coefficient pair (P[p][i], P[p][i])
// read as a shared-memory broadcast), then stores them with coalesced
// streaming stores.  n - k <= 16 is one pass.  Waits are bounded (about 2 s):
// a time-out writes CM_ETIMEOUT to the status word and the warp stops.
#include <cuda_bf16.h>

#include "cm_internal.cuh"
#include "tma.cuh"

namespace {

constexpr int STEP = 128;       // columns per step
constexpr int SEG = 32;         // steps per work unit, at most
constexpr int KC = 8;           // data blocks per sub-step (one TMA box)
constexpr int ST = 2;           // ring slots per warp
constexpr int kWarps = 8;

template <typename T>
struct Elem;

template <>
struct Elem<float> {
    static constexpr CUtensorMapDataType TM = CU_TENSOR_MAP_DATA_TYPE_FLOAT32;
    __device__ static void load4(const float *p, float2 &a, float2 &b)
    {
        const float4 v = *reinterpret_cast<const float4 *>(p);
        a = make_float2(v.x, v.y);
        b = make_float2(v.z, v.w);
    }
    __device__ static void store4(float *p, float2 a, float2 b)
    {
        __stcs(reinterpret_cast<float4 *>(p), make_float4(a.x, a.y, b.x, b.y));
    }
    __device__ static void store1(float *p, float v) { *p = v; }
    __device__ static float load1(const float *p) { return *p; }
};

template <>
struct Elem<uint16_t> {   // bf16 bits
    static constexpr CUtensorMapDataType TM = CU_TENSOR_MAP_DATA_TYPE_BFLOAT16;
    __device__ static float widen(uint32_t h) { return __uint_as_float(h << 16); }
    __device__ static uint32_t rne(float f)
    {
        return (uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(f));
    }
    __device__ static void load4(const uint16_t *p, float2 &a, float2 &b)
    {
        const uint2 v = *reinterpret_cast<const uint2 *>(p);
        a = make_float2(widen(v.x & 0xffffu), widen(v.x >> 16));
        b = make_float2(widen(v.y & 0xffffu), widen(v.y >> 16));
    }
    __device__ static void store4(uint16_t *p, float2 a, float2 b)
    {
        uint2 v;
        v.x = rne(a.x) | (rne(a.y) << 16);
        v.y = rne(b.x) | (rne(b.y) << 16);
        __stcs(reinterpret_cast<uint2 *>(p), v);
    }
    __device__ static void store1(uint16_t *p, float v) { *p = (uint16_t)rne(v); }
    __device__ static float load1(const uint16_t *p) { return widen(*p); }
};

struct EncodeArgs {
    void *par;
    int64_t ldp;
    int32_t *status;
    int64_t d, L;
    int32_t k;
    int32_t kf;          // data blocks with all L rows below m
    int32_t kv;          // data blocks with at least one row below m
    int32_t p0, np;      // parity blocks of this pass
    int32_t steps;       // 128-column steps per row
    int32_t seg;         // steps per segment
    int32_t nseg;        // segments per row
    int32_t nsub;        // sub-steps per step: ceil(kf / KC) + (kv > kf)
    int64_t units;       // L * nseg
};

template <typename T, int NPG>
__device__ __forceinline__ void encode_body(const CUtensorMap &tmF, const CUtensorMap &tmP,
                                            const CodeParams &cp, const EncodeArgs &a)
{
    constexpr uint32_t SLOT = KC * STEP * sizeof(T);
    // dynamic shared memory: [rings, 1024-aligned][coefficient pairs][mbarriers]
    extern __shared__ __align__(16) unsigned char smem_raw[];
    const uint32_t raw0 = cm_smem_u32(smem_raw);
    unsigned char *rings = smem_raw + (((raw0 + 1023) & ~1023u) - raw0);
    float2 *pairs = reinterpret_cast<float2 *>(rings + kWarps * ST * SLOT);   // i * NPG + j
    uint64_t *bars = reinterpret_cast<uint64_t *>(pairs + 32 * NPG);
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    unsigned char *ring = rings + warp * ST * SLOT;
    uint64_t *bar = bars + warp * ST;

    for (int t = threadIdx.x; t < a.kv * NPG; t += blockDim.x) {
        const int i = t / NPG, j = t % NPG;
        const float w = j < a.np ? cp.P[(a.p0 + j) * a.k + i] : 0.f;
        pairs[t] = make_float2(w, w);
    }
    if (threadIdx.x < kWarps * ST) cm_mbar_init(&bars[threadIdx.x], 1);
    cm_fence_mbar_init();
    __syncthreads();

    // a unit (block row r, segment of seg steps) belongs to one CTA; warp w
    // takes the unit's steps w, w + kWarps, ..., so that the CTA's warps read
    // and write adjacent 512-byte pieces of every row at once
    const int64_t cta_units = (int64_t)gridDim.x;
    if ((int64_t)blockIdx.x >= a.units) return;
    const int nfull = (a.kf + KC - 1) / KC;      // sub-steps of full blocks

    auto warp_steps = [&](int64_t u) {           // this warp's steps in unit u
        const int s0 = (int)(u % a.nseg) * a.seg;
        const int ns = (a.steps - s0) < a.seg ? a.steps - s0 : a.seg;
        return ns > warp ? (ns - warp + kWarps - 1) / kWarps : 0;
    };
    auto next_unit = [&](int64_t u) {            // the next unit with steps for this warp
        do u += cta_units; while (u < a.units && warp_steps(u) == 0);
        return u;
    };
    int64_t first = blockIdx.x;
    if (warp_steps(first) == 0) first = next_unit(first);

    // ---- producer (lane 0): sub-step c of step p_s of unit p_unit ----
    int64_t p_unit = first;
    int p_s = 0, p_c = 0, p_slot = 0, in_flight = 0;
    auto produce = [&]() {
        const int64_t r = p_unit / a.nseg;
        const int32_t x = ((int)(p_unit % a.nseg) * a.seg + warp + kWarps * p_s) * STEP;
        unsigned char *dst = ring + p_slot * SLOT;
        if (p_c < nfull) {
            cm_mbar_arrive_expect_tx(&bar[p_slot], SLOT);
            cm_tma_load_3d(dst, &tmF, x, (int32_t)r, p_c * KC, &bar[p_slot]);
        } else {
            cm_mbar_arrive_expect_tx(&bar[p_slot], STEP * sizeof(T));
            cm_tma_load_2d(dst, &tmP, x, (int32_t)r, &bar[p_slot]);
        }
        p_slot = p_slot + 1 == ST ? 0 : p_slot + 1;
        ++in_flight;
        if (++p_c == a.nsub) {
            p_c = 0;
            if (++p_s == warp_steps(p_unit)) {
                p_s = 0;
                p_unit = next_unit(p_unit);
            }
        }
    };
    if (lane == 0)
        while (in_flight < ST && p_unit < a.units) produce();

    // ---- consumer ----
    int slot = 0;
    uint32_t phase = 0;
    T *par = static_cast<T *>(a.par);
    for (int64_t u = first; u < a.units; u = next_unit(u)) {
        const int64_t r = u / a.nseg;
        const int seg = (int)(u % a.nseg);
        const int ns = warp_steps(u);
        for (int s = 0; s < ns; ++s) {
            float2 acc[NPG][2];
#pragma unroll
            for (int j = 0; j < NPG; ++j) acc[j][0] = acc[j][1] = make_float2(0.f, 0.f);
            for (int c = 0; c < a.nsub; ++c) {
                if (!cm_mbar_wait(&bar[slot], phase)) {
                    if (lane == 0) {
                        if (a.status) *a.status = CM_ETIMEOUT;
                        // wait (bounded) for this warp's copies still in flight
                        for (int i = 0; i < in_flight; ++i) {
                            cm_mbar_wait(&bar[slot], phase, 100000000ull);
                            if (++slot == ST) {
                                slot = 0;
                                phase ^= 1u;
                            }
                        }
                    }
                    return;   // no CTA barrier follows: the warp may leave
                }
                // blocks of this sub-step: [i0, i0 + nb)
                const int i0 = c < nfull ? c * KC : a.kf;
                const int nb = c < nfull ? (a.kf - i0 < KC ? a.kf - i0 : KC) : 1;
                const T *src = reinterpret_cast<const T *>(ring + slot * SLOT) + 4 * lane;
                const float2 *pp = pairs + i0 * NPG;
#pragma unroll 2
                for (int i = 0; i < nb; ++i) {
                    float2 a01, a23;
                    Elem<T>::load4(src + i * STEP, a01, a23);
#pragma unroll
                    for (int j = 0; j < NPG; ++j) {
                        if (j < a.np) {
                            const float2 w = pp[i * NPG + j];
                            acc[j][0] = __ffma2_rn(w, a01, acc[j][0]);
                            acc[j][1] = __ffma2_rn(w, a23, acc[j][1]);
                        }
                    }
                }
                if (++slot == ST) {
                    slot = 0;
                    phase ^= 1u;
                }
                __syncwarp();   // every lane is done reading the slot
                if (lane == 0) {
                    --in_flight;
                    if (p_unit < a.units) produce();   // refill it
                }
            }
            const int64_t col = (int64_t)(seg * a.seg + warp + kWarps * s) * STEP + 4 * lane;
            if (col < a.d) {
#pragma unroll
                for (int j = 0; j < NPG; ++j) {
                    if (j < a.np) {
                        T *dst = par + ((int64_t)(a.p0 + j) * a.L + r) * a.ldp + col;
                        if (col + 4 <= a.d) {
                            Elem<T>::store4(dst, acc[j][0], acc[j][1]);
                        } else {
                            const float v[4] = {acc[j][0].x, acc[j][0].y, acc[j][1].x,
                                                acc[j][1].y};
                            for (int e = 0; col + e < a.d; ++e) Elem<T>::store1(dst + e, v[e]);
                        }
                    }
                }
            }
        }
    }
}

// up to 12 parity blocks per pass: the compiler's own register choice (two or
// three CTAs per SM); 16: capped at 128 registers, two CTAs per SM
template <typename T, int NPG>
__global__ void __launch_bounds__(kWarps * 32)
encode_kernel(const __grid_constant__ CUtensorMap tmF, const __grid_constant__ CUtensorMap tmP,
              const CodeParams cp, const EncodeArgs a)
{
    encode_body<T, NPG>(tmF, tmP, cp, a);
}

template <typename T>
__global__ void __launch_bounds__(kWarps * 32, 2)
encode_kernel16(const __grid_constant__ CUtensorMap tmF, const __grid_constant__ CUtensorMap tmP,
                const CodeParams cp, const EncodeArgs a)
{
    encode_body<T, 16>(tmF, tmP, cp, a);
}

// Elementwise form for short codes (at most KE data blocks with rows below m,
// at most 8 parity blocks).  Thread t takes 4 columns of one block row: it
// loads them from every data block (zeros past m), forms the parity blocks'
// sums in the same order i = 0..k-1 as the tiled kernel (so the results are
// the same bits), and stores 4 columns of every parity block.  The
// coefficients sit in the kernel's parameter space as constant operands.
template <int NPG, int KE>
struct EwArgs {
    const void *A;
    void *par;
    int64_t lda, ldp;
    int64_t m, d, L;
    int64_t nc;          // 4-column chunks per row
    int32_t k, np;
    float w[NPG][KE];    // w[j][i] = P[j][i]
};

template <typename T, int NPG, int KE>
__global__ void __launch_bounds__(256)
encode_ew_kernel(const __grid_constant__ EwArgs<NPG, KE> a)
{
    const T *A = static_cast<const T *>(a.A);
    T *par = static_cast<T *>(a.par);
    const int64_t S = (int64_t)gridDim.x * blockDim.x;
    const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    int64_t r = t / a.nc, c = t - r * a.nc;
    const int64_t qS = S / a.nc, rS = S - qS * a.nc;
    while (r < a.L) {
        const int64_t col = 4 * c;
        const bool full = col + 4 <= a.d;
        float2 x[KE][2];
#pragma unroll
        for (int i = 0; i < KE; ++i) {
            x[i][0] = x[i][1] = make_float2(0.f, 0.f);
            const int64_t row = (int64_t)i * a.L + r;
            if (i < a.k && row < a.m) {
                const T *src = A + row * a.lda + col;
                if (full) {
                    Elem<T>::load4(src, x[i][0], x[i][1]);
                } else {
                    float v[4] = {0.f, 0.f, 0.f, 0.f};
                    for (int e = 0; col + e < a.d; ++e) v[e] = Elem<T>::load1(src + e);
                    x[i][0] = make_float2(v[0], v[1]);
                    x[i][1] = make_float2(v[2], v[3]);
                }
            }
        }
        float2 acc[NPG][2];
#pragma unroll
        for (int j = 0; j < NPG; ++j) acc[j][0] = acc[j][1] = make_float2(0.f, 0.f);
#pragma unroll
        for (int i = 0; i < KE; ++i) {
            if (i < a.k) {
#pragma unroll
                for (int j = 0; j < NPG; ++j) {
                    const float2 w = make_float2(a.w[j][i], a.w[j][i]);
                    acc[j][0] = __ffma2_rn(w, x[i][0], acc[j][0]);
                    acc[j][1] = __ffma2_rn(w, x[i][1], acc[j][1]);
                }
            }
        }
#pragma unroll
        for (int j = 0; j < NPG; ++j) {
            if (j < a.np) {
                T *dst = par + ((int64_t)j * a.L + r) * a.ldp + col;
                if (full) {
                    Elem<T>::store4(dst, acc[j][0], acc[j][1]);
                } else {
                    const float v[4] = {acc[j][0].x, acc[j][0].y, acc[j][1].x, acc[j][1].y};
                    for (int e = 0; col + e < a.d; ++e) Elem<T>::store1(dst + e, v[e]);
                }
            }
        }
        c += rS;
        r += qS;
        if (c >= a.nc) {
            c -= a.nc;
            ++r;
        }
    }
}

template <typename T, int NPG, int KE>
cudaError_t launch_ew(const CodeParams &cp, const T *A, int64_t lda, T *par, int64_t ldp,
                      cudaStream_t s)
{
    EwArgs<NPG, KE> a;
    a.A = A;
    a.par = par;
    a.lda = lda;
    a.ldp = ldp;
    a.m = cp.m;
    a.d = cp.d;
    a.L = cp.L;
    a.nc = (cp.d + 3) / 4;
    a.k = cp.k;
    a.np = cp.n - cp.k;
    for (int j = 0; j < NPG; ++j)
        for (int i = 0; i < KE; ++i)
            a.w[j][i] = j < a.np && i < cp.k ? cp.P[j * cp.k + i] : 0.f;
    auto kern = encode_ew_kernel<T, NPG, KE>;
    int per_sm = 0;
    cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, 256, 0);
    if (e != cudaSuccess) return e;
    if (per_sm < 1) per_sm = 1;
    const int64_t items = cp.L * a.nc;
    int64_t grid = (int64_t)(cm_sm_count() > 0 ? cm_sm_count() : 1) * per_sm;
    if (grid > (items + 255) / 256) grid = (items + 255) / 256;
    if (grid < 1) grid = 1;
    kern<<<(unsigned)grid, 256, 0, s>>>(a);
    return cudaGetLastError();
}

template <typename T, int NPG>
cudaError_t launch_passes(const CodeParams &cp, const T *A, int64_t lda, T *par, int64_t ldp,
                          int32_t *status, cudaStream_t s)
{
    const int64_t es = sizeof(T);
    const int kf = (int)(cp.m / cp.L);                 // >= 1 since L <= m
    const int kv = (int)((cp.m + cp.L - 1) / cp.L);
    if constexpr (NPG <= 8) {   // short codes: the elementwise form (see above)
        if (cp.k <= 8) return launch_ew<T, NPG, 8>(cp, A, lda, par, ldp, s);
    }
    if constexpr (NPG <= 12) {
        if (cp.k <= 16 && 2 * (cp.n - cp.k) >= cp.k)
            return launch_ew<T, NPG, 16>(cp, A, lda, par, ldp, s);
    }
    CUtensorMap tmF, tmP;
    if (!cm_make_tmap_3d(&tmF, Elem<T>::TM, A, (uint64_t)cp.d, (uint64_t)cp.L, (uint64_t)kf,
                         (uint64_t)(lda * es), (uint64_t)(cp.L * lda * es), STEP, 1, KC))
        return cudaErrorInvalidValue;
    if (kv > kf) {
        if (!cm_make_tmap_2d(&tmP, Elem<T>::TM, A + (int64_t)kf * cp.L * lda, (uint64_t)cp.d,
                             (uint64_t)(cp.m - (int64_t)kf * cp.L), (uint64_t)(lda * es), STEP, 1,
                             CU_TENSOR_MAP_SWIZZLE_NONE))
            return cudaErrorInvalidValue;
    } else {
        tmP = tmF;   // unused
    }
    EncodeArgs a;
    a.par = par;
    a.ldp = ldp;
    a.status = status;
    a.d = cp.d;
    a.L = cp.L;
    a.k = cp.k;
    a.kf = kf;
    a.kv = kv;
    a.steps = (int)((cp.d + STEP - 1) / STEP);
    a.nsub = (kf + KC - 1) / KC + (kv > kf ? 1 : 0);
    void (*kern)(const CUtensorMap, const CUtensorMap, const CodeParams, const EncodeArgs);
    if constexpr (NPG == 16)
        kern = encode_kernel16<T>;
    else
        kern = encode_kernel<T, NPG>;
    const int smem = 1024 + kWarps * ST * KC * STEP * (int)es + 32 * NPG * 8 + kWarps * ST * 8;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    int per_sm = 0;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kWarps * 32, smem);
    if (e != cudaSuccess) return e;
    if (per_sm < 1) per_sm = 1;
    int64_t grid = (int64_t)cm_sm_count() * per_sm;
    {   // segment length: CTA-level units, warps interleaved over the steps
        double best = -1.0;
        for (int ns = (a.steps + kWarps * SEG - 1) / (kWarps * SEG); ns <= a.steps; ++ns) {
            const int sg = (a.steps + ns - 1) / ns;
            const int nsg = (a.steps + sg - 1) / sg;
            const int64_t units = cp.L * nsg;
            const int64_t rounds = (units + grid - 1) / grid;
            const int wsteps = (sg + kWarps - 1) / kWarps;
            const double fill = (double)cp.L * a.steps / ((double)rounds * wsteps * kWarps * grid);
            if (fill > best + 1e-9) {
                best = fill;
                a.seg = sg;
                a.nseg = nsg;
            }
            if (fill >= 0.9) break;
        }
    }
    a.units = cp.L * a.nseg;
    const int64_t need = a.units;
    if (grid > need) grid = need;
    if (grid < 1) grid = 1;
    for (int p0 = 0; p0 < cp.n - cp.k; p0 += NPG) {
        a.p0 = p0;
        a.np = cp.n - cp.k - p0 < NPG ? cp.n - cp.k - p0 : NPG;
        kern<<<(unsigned)grid, kWarps * 32, smem, s>>>(tmF, tmP, cp, a);
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
    }
    return cudaSuccess;
}

// Parity blocks per pass: the smallest instance at or above n - k, so that
// few accumulators and coefficient slots go to blocks that do not exist
// (n - k > 16 takes several passes of 16).
template <typename T>
cudaError_t launch_np(const CodeParams &cp, const T *A, int64_t lda, T *par, int64_t ldp,
                      int32_t *status, cudaStream_t s)
{
    const int np = cp.n - cp.k;
    if (np <= 2) return launch_passes<T, 2>(cp, A, lda, par, ldp, status, s);
    if (np <= 3) return launch_passes<T, 3>(cp, A, lda, par, ldp, status, s);
    if (np <= 4) return launch_passes<T, 4>(cp, A, lda, par, ldp, status, s);
    if (np <= 5) return launch_passes<T, 5>(cp, A, lda, par, ldp, status, s);
    if (np <= 6) return launch_passes<T, 6>(cp, A, lda, par, ldp, status, s);
    if (np <= 8) return launch_passes<T, 8>(cp, A, lda, par, ldp, status, s);
    if (np <= 10) return launch_passes<T, 10>(cp, A, lda, par, ldp, status, s);
    if (np <= 12) return launch_passes<T, 12>(cp, A, lda, par, ldp, status, s);
    return launch_passes<T, 16>(cp, A, lda, par, ldp, status, s);
}

}  // namespace

cudaError_t launch_encode_f32(const CodeParams &cp, const float *A, int64_t lda, float *par,
                              int64_t ldp, int32_t *status, cudaStream_t s)
{
    return launch_np<float>(cp, A, lda, par, ldp, status, s);
}

cudaError_t launch_encode_bf16(const CodeParams &cp, const uint16_t *A, int64_t lda,
                               uint16_t *par, int64_t ldp, int32_t *status, cudaStream_t s)
{
    return launch_np<uint16_t>(cp, A, lda, par, ldp, status, s);
}
