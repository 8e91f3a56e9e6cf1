// K5: coded matrix-matrix products on tcgen05 tensor cores (the s-column X of
// the Sec. I-A example, bf16 inputs, fp32 accumulation).
//
// Ct[j L + r][c] = sum_t A~_j[r][t] Bt[c][t] for every worker j < n, block row
// r < L and column c < N.  Worker j < k reads rows of A in place, worker
// j >= k rows of the bf16 parity buffer (both K-major, i.e. row-major); B is
// given transposed (N x d, K-major).
//
// Tiles.  128 x 256 output tiles that never straddle a worker block: worker j
// has ceil(L / 128) row tiles; the last one reads past the block (zeros past
// m or the parity buffer, or the next block's rows) and stores only rows < L.
// Tile order: column tile fastest, so the 16 column tiles of one row tile run
// at the same time on different SMs and the 2 MB row slab of A~ comes from
// HBM once and from L2 after that; Bt (64 MB) stays L2-resident.
//
// One persistent CTA per SM, warp-specialised:
//   warp 0 lane 0  TMA producer: 128B-swizzled boxes of A~ (128 x 64) and Bt
//                  (256 x 64) into a 4-stage shared-memory ring (48 KB per stage);
//   warp 1         allocates 512 TMEM columns (two 128 x 256 fp32 accumulators);
//                  lane 0 issues tcgen05.mma.cta_group::1.kind::f16 (M=128,
//                  N=256, K=16, four per stage) and tcgen05.commit to free a
//                  stage / publish an accumulator;
//   warps 2..5     epilogue: tcgen05.ld (32 lanes x 32 columns per load) from
//                  the accumulator of their TMEM lane quarter, fp32 stores to Ct,
//                  then release the accumulator, so the epilogue of one tile
//                  overlaps the MMAs of the next.
// Every wait is bounded (about 2 s); on a time-out the kernel writes
// CM_ETIMEOUT to the status word, every role stops, outstanding work is
// drained with bounded waits and the TMEM is freed before the CTA exits.
#include "cm_internal.cuh"
#include "tma.cuh"

namespace {

constexpr int BM = 128, BN = 256, BK = 64, STAGES = 4, ACCS = 2;
constexpr int TMEM_COLS = ACCS * BN;   // 512
constexpr int kThreads = 192;
constexpr uint32_t A_BYTES = BM * BK * 2;
constexpr uint32_t B_BYTES = BN * BK * 2;
constexpr uint32_t STAGE_BYTES = A_BYTES + B_BYTES;
constexpr int SMEM_BYTES = 1024 + STAGES * STAGE_BYTES + 256;

struct GemmArgs {
    float *Ct;
    int64_t ldc;
    int32_t *status;
    int64_t L;
    int32_t n, k, N;
    int32_t mtiles;    // row tiles per worker block
    int32_t ntiles;    // column tiles
    int32_t kblocks;   // 64-wide K blocks
    int64_t tiles;
};

// ---- tcgen05 helpers (inline PTX) ---------------------------------------------------

// Shared-memory matrix descriptor of a K-major operand tile written by TMA with
// 128-byte swizzling: 8-row groups 1024 bytes apart (stride byte offset), the
// leading byte offset unused for this layout, descriptor version 1, swizzle
// mode "128B" (2).
__device__ __forceinline__ uint64_t smem_desc_sw128(uint32_t saddr)
{
    return (uint64_t)((saddr & 0x3FFFFu) >> 4) | ((uint64_t)1 << 16) |
           ((uint64_t)(1024 >> 4) << 32) | ((uint64_t)1 << 46) | ((uint64_t)2 << 61);
}

// Instruction descriptor for kind::f16: fp32 accumulator, bf16 A and B, both
// K-major, N = BN, M = BM.
constexpr uint32_t kIdesc = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(BN >> 3) << 17) |
                            ((uint32_t)(BM >> 4) << 24);

__device__ __forceinline__ void mma_bf16(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc,
                                         uint32_t accumulate)
{
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}\n" ::"r"(d_tmem),
        "l"(adesc), "l"(bdesc), "r"(kIdesc), "r"(accumulate)
        : "memory");
}

__device__ __forceinline__ void mma_commit(uint64_t *bar)
{
    asm volatile(
        "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];\n" ::"r"(
            cm_smem_u32(bar))
        : "memory");
}

__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;\n" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;\n" ::: "memory"); }

// 32 lanes x 32 consecutive fp32 columns of TMEM into 32 registers per thread.
__device__ __forceinline__ void tmem_load32(uint32_t taddr, float (&v)[32])
{
    uint32_t r[32];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
        "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
        "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, "
        "[%32];\n"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
          "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]),
          "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]),
          "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
          "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]),
          "=r"(r[31])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;\n" ::: "memory");
#pragma unroll
    for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

struct Tile {
    int j;          // worker
    int mt;         // row tile within the worker block
    int n0;         // first output column
    bool parity;    // rows come from the parity buffer
    int32_t y;      // row coordinate in A or in the parity buffer
};

__device__ __forceinline__ Tile tile_of(const GemmArgs &g, int64_t t)
{
    Tile x;
    const int nt = (int)(t % g.ntiles);
    const int64_t rest = t / g.ntiles;
    x.mt = (int)(rest % g.mtiles);
    x.j = (int)(rest / g.mtiles);
    x.n0 = nt * BN;
    x.parity = x.j >= g.k;
    const int64_t r0 = (int64_t)x.mt * BM;
    x.y = (int32_t)(x.parity ? (int64_t)(x.j - g.k) * g.L + r0 : (int64_t)x.j * g.L + r0);
    return x;
}

__global__ void __launch_bounds__(kThreads, 1)
gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmP,
            const __grid_constant__ CUtensorMap tmB, const GemmArgs g)
{
    extern __shared__ __align__(16) unsigned char smem_raw[];
    unsigned char *base = smem_raw + ((1024 - (cm_smem_u32(smem_raw) & 1023)) & 1023);
    uint64_t *full = reinterpret_cast<uint64_t *>(base + STAGES * STAGE_BYTES);
    uint64_t *empty = full + STAGES;
    uint64_t *tfull = empty + STAGES;
    uint64_t *tempty = tfull + ACCS;
    uint64_t *drain = tempty + ACCS;
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(drain + 1);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(tmem_slot + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            cm_mbar_init(&full[s], 1);
            cm_mbar_init(&empty[s], 1);
        }
        for (int a = 0; a < ACCS; ++a) {
            cm_mbar_init(&tfull[a], 1);
            cm_mbar_init(&tempty[a], 128);
        }
        cm_mbar_init(drain, 1);
        *abort_flag = 0;
        cm_fence_mbar_init();
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;\n" ::"r"(
                         cm_smem_u32(tmem_slot)),
                     "r"(TMEM_COLS)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;\n" ::: "memory");
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;

    auto fail = [&]() {
        *abort_flag = 1;
        if (g.status) *g.status = CM_ETIMEOUT;
    };

    if (warp == 0 && lane == 0) {
        // ---- TMA producer ----
        int s = 0;
        uint32_t ph = 0;
        int64_t issued = 0;
        for (int64_t t = blockIdx.x; t < g.tiles && !*abort_flag; t += gridDim.x) {
            const Tile x = tile_of(g, t);
            const CUtensorMap *ma = x.parity ? &tmP : &tmA;
            for (int kb = 0; kb < g.kblocks; ++kb) {
                if (*abort_flag || !cm_mbar_wait(&empty[s], ph ^ 1u)) {
                    fail();
                    break;
                }
                unsigned char *sa = base + s * STAGE_BYTES;
                cm_mbar_arrive_expect_tx(&full[s], STAGE_BYTES);
                cm_tma_load_2d(sa, ma, kb * BK, x.y, &full[s]);
                cm_tma_load_2d(sa + A_BYTES, &tmB, kb * BK, x.n0, &full[s]);
                ++issued;
                if (++s == STAGES) {
                    s = 0;
                    ph ^= 1u;
                }
            }
        }
        if (*abort_flag) {
            // drain: wait (bounded) for the last phase of every stage in flight
            for (int i = 0; i < STAGES && i < issued; ++i) {
                if (--s < 0) {
                    s = STAGES - 1;
                    ph ^= 1u;
                }
                cm_mbar_wait(&full[s], ph, 100000000ull);
            }
        }
    } else if (warp == 1 && lane == 0) {
        // ---- MMA issuer ----
        int s = 0, acc = 0;
        uint32_t ph = 0, aph = 0;
        for (int64_t t = blockIdx.x; t < g.tiles && !*abort_flag; t += gridDim.x) {
            if (!cm_mbar_wait(&tempty[acc], aph ^ 1u)) {
                fail();
                break;
            }
            tc_fence_after();
            const uint32_t d_tmem = tmem_base + (uint32_t)(acc * BN);
            bool ok = true;
            for (int kb = 0; kb < g.kblocks; ++kb) {
                if (*abort_flag || !cm_mbar_wait(&full[s], ph)) {
                    fail();
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t sa = cm_smem_u32(base + s * STAGE_BYTES);
                const uint32_t sb = sa + A_BYTES;
#pragma unroll
                for (int kk = 0; kk < BK / 16; ++kk)
                    mma_bf16(d_tmem, smem_desc_sw128(sa + kk * 32), smem_desc_sw128(sb + kk * 32),
                             (kb | kk) != 0);
                mma_commit(&empty[s]);   // the stage is free once these MMAs finish
                if (++s == STAGES) {
                    s = 0;
                    ph ^= 1u;
                }
            }
            if (!ok) break;
            mma_commit(&tfull[acc]);     // accumulator ready for the epilogue
            if (++acc == ACCS) {
                acc = 0;
                aph ^= 1u;
            }
        }
        // all MMAs issued by this thread have completed once `drain` fires
        mma_commit(drain);
        cm_mbar_wait(drain, 0, 100000000ull);
    } else if (warp >= 2) {
        // ---- epilogue: TMEM -> registers -> Ct ----
        const int q = warp & 3;                  // TMEM lane quarter of this warp
        const int row = q * 32 + lane;           // row of the tile
        int acc = 0;
        uint32_t aph = 0;
        for (int64_t t = blockIdx.x; t < g.tiles; t += gridDim.x) {
            // warp-uniform decisions: tcgen05.ld below is .sync.aligned
            if (__shfl_sync(0xffffffffu, *abort_flag, 0)) break;
            const bool ok = cm_mbar_wait(&tfull[acc], aph);
            if (!__all_sync(0xffffffffu, ok)) {
                if (lane == 0) fail();
                break;
            }
            tc_fence_after();
            const Tile x = tile_of(g, t);
            const int64_t r = (int64_t)x.mt * BM + row;
            const bool valid = r < g.L;
            float *dst = g.Ct + ((int64_t)x.j * g.L + r) * g.ldc + x.n0;
            const uint32_t taddr = tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(acc * BN);
#pragma unroll 1
            for (int c = 0; c < BN / 32; ++c) {
                float v[32];
                tmem_load32(taddr + c * 32, v);
                const int col = x.n0 + c * 32;
                if (valid && col < g.N) {
                    float *p = dst + c * 32;
                    if (col + 32 <= g.N && ((g.ldc & 3) == 0)) {
#pragma unroll
                        for (int i = 0; i < 32; i += 4)
                            *reinterpret_cast<float4 *>(p + i) =
                                make_float4(v[i], v[i + 1], v[i + 2], v[i + 3]);
                    } else {
#pragma unroll
                        for (int i = 0; i < 32; ++i)
                            if (col + i < g.N) p[i] = v[i];
                    }
                }
            }
            tc_fence_before();
            cm_mbar_arrive(&tempty[acc]);
            if (++acc == ACCS) {
                acc = 0;
                aph ^= 1u;
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        __syncwarp();
        tc_fence_after();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;\n" ::"r"(tmem_base),
                     "r"(TMEM_COLS)
                     : "memory");
    }
}

}  // namespace

cudaError_t launch_coded_gemm(const CodeParams &cp, const uint16_t *A, int64_t lda,
                              const uint16_t *par, int64_t ldp, const uint16_t *Bt, int64_t ldb,
                              int N, float *Ct, int64_t ldc, int32_t *status, cudaStream_t s)
{
    CUtensorMap tmA, tmP, tmB;
    const uint64_t d = (uint64_t)cp.d;
    if (!cm_make_tmap_2d(&tmA, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, A, d, (uint64_t)cp.m,
                         (uint64_t)lda * 2, BK, BM, CU_TENSOR_MAP_SWIZZLE_128B) ||
        !cm_make_tmap_2d(&tmP, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, par, d,
                         (uint64_t)(cp.n - cp.k) * cp.L, (uint64_t)ldp * 2, BK, BM,
                         CU_TENSOR_MAP_SWIZZLE_128B) ||
        !cm_make_tmap_2d(&tmB, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, Bt, d, (uint64_t)N,
                         (uint64_t)ldb * 2, BK, BN, CU_TENSOR_MAP_SWIZZLE_128B))
        return cudaErrorInvalidValue;
    GemmArgs g;
    g.Ct = Ct;
    g.ldc = ldc;
    g.status = status;
    g.L = cp.L;
    g.n = cp.n;
    g.k = cp.k;
    g.N = N;
    g.mtiles = (int)((cp.L + BM - 1) / BM);
    g.ntiles = (N + BN - 1) / BN;
    g.kblocks = (int)((cp.d + BK - 1) / BK);
    g.tiles = (int64_t)cp.n * g.mtiles * g.ntiles;
    cudaError_t e = cudaFuncSetAttribute(gemm_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         SMEM_BYTES);
    if (e != cudaSuccess) return e;
    int64_t grid = cm_sm_count();
    if (grid < 1) grid = 1;
    if (grid > g.tiles) grid = g.tiles;
    gemm_kernel<<<(unsigned)grid, kThreads, SMEM_BYTES, s>>>(tmA, tmP, tmB, g);
    return cudaGetLastError();
}
