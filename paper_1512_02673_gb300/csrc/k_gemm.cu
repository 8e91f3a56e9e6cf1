// K5: coded matrix-matrix products on tcgen05 tensor cores (the s-column X of
// the Sec. I-A example, bf16 inputs, fp32 accumulation).
//
// Ct[j L + r][c] = sum_t A~_j[r][t] Bt[c][t] for every worker j < n, block row
// r < L and column c < N.  Worker j < k reads rows of A in place, worker
// j >= k rows of the bf16 parity buffer (both K-major, i.e. row-major); B is
// given transposed (N x d, K-major).
//
// Two-SM tiles.  A cluster of two CTAs on a pair of SMs computes one 256 x 256
// output tile with tcgen05.mma.cta_group::2 (M = 256 over the pair, N = 256,
// K = 16): CTA r stages rows [128 r, 128 r + 128) of the A~ tile and rows
// [128 r, 128 r + 128) of the Bt tile, and accumulates its 128 output rows in
// its own tensor memory.  Per K block of 64 each SM thus stages 32 KB (instead
// of 48 KB for a one-SM 128 x 256 tile), which leaves six stages in shared
// memory and halves the Bt bytes every SM reads per MMA: the one-SM version
// was held near 0.8 of peak by shared-memory traffic (TMA fills plus tensor-
// core operand reads).
//
// Row tiling (all workers).  The coded rows are two contiguous ranges: Ct rows [0, kL) are
// rows of A in place (worker j < k owns [jL, jL + L)), Ct rows [kL, nL) are
// rows of the parity buffer.  Each range is cut into 256-row pairs of its
// own, A's over its m real rows only, so no tile computes the virtual zero
// rows of every block's ragged end or reads a neighbour's rows: at (16,12)
// with m = 32768 this gives 128 + 43 row pairs x 16 column tiles = 2736 work
// items, 36 full waves of 76 pairs (per-worker tiles needed 2816, 38 waves
// with a 4-item tail).  Rows past a range's end load as zeros (TMA
// out-of-bounds fill) and are not stored; the pad rows [m, kL) of the last
// systematic block are stored as zeros, by the last A pair's tiles where they
// cover them and by its rank-1 CTA's epilogue past its end.  Work order: bands
// of 16 column tiles, every row pair of a band before the next band, the
// band's tiles of one pair consecutive (at N = 4096 one band: the 16 column
// tiles of a row pair run together and read its A~ slab from HBM once).
// Bt is loaded with an evict-last L2 policy and Ct is stored with streaming
// stores, so that the A~ slabs and Ct pass through L2 without displacing Bt.
// Narrower bands (8 tiles, 32 MB of Bt at d = 8192) cut the DRAM reads of the
// profiling case from 1.73 to 1.43 GB but ran 0.6 % slower: DRAM runs at about
// 30 % of its peak here and is not what limits the kernel.
//
// Survivors only (cm_coded_gemm_survivors): the listed workers fall into
// runs of consecutive workers (none across the A | parity boundary), each a
// contiguous row range of A or of the parity and of Ct, tiled like the two
// ranges above; the other blocks of Ct are not written.
//
// One persistent CTA per SM, warp-specialised, in both CTAs of a pair:
//   warp 0 lane 0  TMA producer of the CTA's halves (128B-swizzled 128 x 64
//                  boxes) into a 6-stage ring whose stages are guarded in
//                  pairs (one full and one empty barrier per 2 K blocks: half
//                  the barrier round trips, +1 %; three per barrier left two
//                  groups and ran 10 % slower); every load completes on the
//                  leader CTA's barrier, which the leader's producer arms
//                  with the bytes of both CTAs;
//   warp 1         allocates 512 TMEM columns together with the peer
//                  (cta_group::2: two 128 x 256 fp32 accumulators per CTA);
//                  in the leader (rank 0), lane 0 issues the MMAs and
//                  tcgen05.commit, multicast to both CTAs, to free a stage or
//                  publish an accumulator;
//   warps 2..5     epilogue: tcgen05.ld (32 lanes x 32 columns per load) from
//                  the CTA's accumulator, fp32 stores to Ct, then release of
//                  the accumulator on the leader's barrier (the peer's
//                  threads arrive remotely), so the epilogue of one tile
//                  overlaps the MMAs of the next.
// Every wait is bounded (about 2 s); on a time-out the kernel writes
// CM_ETIMEOUT to the status word, every role stops, outstanding work is
// drained with bounded waits, and both CTAs meet at a cluster barrier before
// the TMEM is freed and they exit, so neither touches the other's shared
// memory while it is not live.
#include <atomic>

#include "cm_internal.cuh"
#include "tma.cuh"

namespace {

constexpr int BM = 128;              // rows per CTA (256 per pair)
constexpr int kBand = 16;            // column tiles per band of the work order
constexpr int BN = 256, BK = 64, STAGES = 6, ACCS = 2;
constexpr int KG = 2;                 // K blocks per barrier
constexpr int GROUPS = STAGES / KG;   // barrier groups in the ring
constexpr int BNH = BN / 2;          // Bt rows staged per CTA
constexpr int TMEM_COLS = ACCS * BN;   // 512
constexpr int kThreads = 192;
constexpr uint32_t A_BYTES = BM * BK * 2;
constexpr uint32_t B_BYTES = BNH * BK * 2;
constexpr uint32_t STAGE_BYTES = A_BYTES + B_BYTES;   // 32 KB per CTA
constexpr int SMEM_BYTES = 1024 + STAGES * STAGE_BYTES + 256;

struct GemmArgs {
    float *Ct;
    int64_t ldc;
    int32_t *status;
    int64_t kL;        // Ct rows from A (systematic blocks, pad rows included)
    int64_t pL;        // Ct rows from the parity buffer, (n - k) L
    int32_t N;
    int32_t psys;      // 256-row pairs over A's m rows
    int32_t ppar;      // 256-row pairs over the parity rows
    int32_t ntiles;    // column tiles
    int32_t kblocks;   // 64-wide K blocks
    int64_t pairs;     // (row pair, column tile) work items
    // survivors only: runs of consecutive computed workers (0 runs: all of
    // them, two contiguous ranges)
    int64_t L;
    int32_t k;
    int32_t nruns;
    int32_t run_p0[CM_MAX_N + 1];   // first row pair of each run; run_p0[nruns] = all
    int8_t run_w[CM_MAX_N];         // first worker of each run
    int8_t run_cnt[CM_MAX_N];       // workers in each run
};

// ---- tcgen05 / cluster helpers (inline PTX) ------------------------------------------

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
// K-major, N = BN, M = 256 (the pair).
constexpr uint32_t kIdesc = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(BN >> 3) << 17) |
                            ((uint32_t)((2 * BM) >> 4) << 24);

__device__ __forceinline__ void mma_bf16_pair(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc,
                                              uint32_t accumulate)
{
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}\n" ::"r"(d_tmem),
        "l"(adesc), "l"(bdesc), "r"(kIdesc), "r"(accumulate)
        : "memory");
}

// Arrive on the mbarrier at this offset in both CTAs of the pair once the
// MMAs issued so far have completed.
__device__ __forceinline__ void mma_commit_pair(uint64_t *bar)
{
    asm volatile(
        "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster"
        ".b64 [%0], %1;\n" ::"r"(cm_smem_u32(bar)),
        "h"((uint16_t)0x3)
        : "memory");
}

// Arrive on a local mbarrier once this thread's MMAs have completed.
__device__ __forceinline__ void mma_commit_local(uint64_t *bar)
{
    asm volatile(
        "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.b64 [%0];\n" ::"r"(
            cm_smem_u32(bar))
        : "memory");
}

__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;\n" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;\n" ::: "memory"); }

__device__ __forceinline__ uint32_t cluster_ctarank()
{
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;\n" : "=r"(r));
    return r;
}

__device__ __forceinline__ uint32_t cluster_id()
{
    uint32_t r;
    asm volatile("mov.u32 %0, %%clusterid.x;\n" : "=r"(r));
    return r;
}

__device__ __forceinline__ uint32_t cluster_count()
{
    uint32_t r;
    asm volatile("mov.u32 %0, %%nclusterid.x;\n" : "=r"(r));
    return r;
}

// Shared::cluster address of the same shared-memory location in CTA `rank`.
__device__ __forceinline__ uint32_t map_to_rank(const void *p, uint32_t rank)
{
    uint32_t r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;\n" : "=r"(r) : "r"(cm_smem_u32(p)), "r"(rank));
    return r;
}

// Every thread of both CTAs: release its earlier writes, wait for the others.
__device__ __forceinline__ void cluster_sync()
{
    asm volatile("barrier.cluster.arrive.release;\n\tbarrier.cluster.wait.acquire;\n" ::: "memory");
}

// Arrive (release, cluster scope) on an mbarrier given by its shared::cluster
// address, possibly in the peer CTA.
__device__ __forceinline__ void mbar_arrive_cluster(uint32_t cl_addr)
{
    asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];\n" ::"r"(cl_addr)
                 : "memory");
}

// 2-D TMA load into this CTA's shared memory whose completion is counted on an
// mbarrier of either CTA of the pair (shared::cluster address).
__device__ __forceinline__ void tma_load_2d_pair(void *smem_dst, const CUtensorMap *map, int32_t x,
                                                 int32_t y, uint32_t bar_cl)
{
    asm volatile(
        "cp.async.bulk.tensor.2d.cta_group::2.shared::cluster.global.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3}], [%4];\n" ::"r"(cm_smem_u32(smem_dst)),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar_cl)
        : "memory");
}

// The same with an L2 cache policy (createpolicy): the Bt tiles are read by
// every row pair, so they are loaded with an evict-last policy and stay in L2
// while the A~ slabs and the streaming Ct stores pass through.
__device__ __forceinline__ void tma_load_2d_pair_hint(void *smem_dst, const CUtensorMap *map,
                                                      int32_t x, int32_t y, uint32_t bar_cl,
                                                      uint64_t policy)
{
    asm volatile(
        "cp.async.bulk.tensor.2d.cta_group::2.shared::cluster.global.mbarrier::complete_tx::bytes"
        ".L2::cache_hint [%0], [%1, {%2, %3}], [%4], %5;\n" ::"r"(cm_smem_u32(smem_dst)),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar_cl), "l"(policy)
        : "memory");
}

__device__ __forceinline__ uint64_t l2_evict_last_policy()
{
    uint64_t p;
    asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;\n" : "=l"(p));
    return p;
}

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
    bool parity;    // rows come from the parity buffer
    int32_t y;      // first row in A or in the parity buffer
    int n0;         // first output column
    int64_t crow;   // Ct row of the tile's first row
    int32_t rows;   // rows of the tile that exist in Ct (may be <= 0)
    int32_t pad;    // pad rows [crow + BM, crow + BM + pad) to store as zeros
};

// CTA `rank`'s half of work item p: rows [128 rank, 128 rank + 128) of p's
// row pair.
__device__ __forceinline__ Tile tile_of(const GemmArgs &g, int64_t p, int rank)
{
    Tile x;
    // bands of kBand column tiles, every row pair of a band before the next
    // band, the band's tiles of one pair consecutive
    const int64_t npairs = g.pairs / g.ntiles;
    const int band = (int)(p / (npairs * kBand));
    const int bw = g.ntiles - band * kBand < kBand ? g.ntiles - band * kBand : kBand;
    const int64_t in = p - (int64_t)band * npairs * kBand;
    const int nt = band * kBand + (int)(in % bw);
    const int rp = (int)(in / bw);
    x.n0 = nt * BN;
    if (g.nruns > 0) {
        // survivors only: a pair of one run of consecutive workers; a tile may
        // read past its run (the next block's rows, or zeros past m) but
        // stores only the run's rows, its pad rows (zeros past m) included
        int r = 0;
        while (r + 1 < g.nruns && rp >= g.run_p0[r + 1]) ++r;
        const int j = g.run_w[r];
        const int64_t R = (int64_t)g.run_cnt[r] * g.L;
        const int64_t r0 = (int64_t)(rp - g.run_p0[r]) * (2 * BM) + rank * BM;
        x.parity = j >= g.k;
        x.y = (int32_t)((x.parity ? (int64_t)(j - g.k) : (int64_t)j) * g.L + r0);
        x.crow = (int64_t)j * g.L + r0;
        x.rows = (int32_t)(R - r0 < BM ? R - r0 : BM);
        x.pad = 0;
        return x;
    }
    x.parity = rp >= g.psys;
    const int64_t y = (int64_t)(x.parity ? rp - g.psys : rp) * (2 * BM) + rank * BM;
    x.y = (int32_t)y;
    const int64_t end = x.parity ? g.pL : g.kL;
    x.crow = x.parity ? g.kL + y : y;
    x.rows = (int32_t)(end - y < BM ? end - y : BM);
    x.pad = (!x.parity && rank == 1 && rp == g.psys - 1 && y + BM < g.kL) ? (int32_t)(g.kL - y - BM)
                                                                          : 0;
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
    const int rank = (int)cluster_ctarank();
    const bool leader = rank == 0;
    if (threadIdx.x == 0) {
        for (int s = 0; s < GROUPS; ++s) {
            cm_mbar_init(&full[s], 1);    // leader: its producer's arrive (+ both CTAs' bytes)
            cm_mbar_init(&empty[s], 1);   // the leader's MMA commit
        }
        for (int a = 0; a < ACCS; ++a) {
            cm_mbar_init(&tfull[a], 1);                // the leader's MMA commit
            cm_mbar_init(&tempty[a], 2 * 4 * 32);      // leader: both CTAs' epilogue threads
        }
        cm_mbar_init(drain, 1);
        *abort_flag = 0;
        cm_fence_mbar_init();
    }
    if (warp == 1) {   // with the peer's warp 1: the same columns in both CTAs
        asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;\n" ::"r"(
                         cm_smem_u32(tmem_slot)),
                     "r"(TMEM_COLS)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;\n" ::: "memory");
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;
    const int64_t first = cluster_id(), stride = cluster_count();
    cluster_sync();   // both CTAs' barriers exist before either signals the other

    auto fail = [&]() {
        *abort_flag = 1;
        if (g.status) *g.status = CM_ETIMEOUT;
    };

    if (warp == 0 && lane == 0) {
        // ---- TMA producer (both CTAs) ----
        const uint64_t keep = l2_evict_last_policy();
        int s = 0;
        uint32_t ph = 0;
        int64_t issued = 0;
        for (int64_t p = first; p < g.pairs && !*abort_flag; p += stride) {
            const Tile x = tile_of(g, p, rank);
            const CUtensorMap *ma = x.parity ? &tmP : &tmA;
            for (int kb = 0; kb < g.kblocks; kb += KG) {
                if (*abort_flag || !cm_mbar_wait(&empty[s], ph ^ 1u)) {
                    fail();
                    break;
                }
                const int nb = g.kblocks - kb < KG ? g.kblocks - kb : KG;
                const uint32_t bar = map_to_rank(&full[s], 0);   // the leader's stage barrier
                if (leader) cm_mbar_arrive_expect_tx(&full[s], 2 * STAGE_BYTES * nb);
                for (int u = 0; u < nb; ++u) {
                    unsigned char *sa = base + (s * KG + u) * STAGE_BYTES;
                    tma_load_2d_pair(sa, ma, (kb + u) * BK, x.y, bar);
                    tma_load_2d_pair_hint(sa + A_BYTES, &tmB, (kb + u) * BK, x.n0 + rank * BNH,
                                          bar, keep);
                }
                ++issued;
                if (++s == GROUPS) {
                    s = 0;
                    ph ^= 1u;
                }
            }
        }
        if (*abort_flag && leader) {
            // drain: wait (bounded) for the last phase of every stage in flight
            for (int i = 0; i < GROUPS && i < issued; ++i) {
                if (--s < 0) {
                    s = GROUPS - 1;
                    ph ^= 1u;
                }
                cm_mbar_wait(&full[s], ph, 100000000ull);
            }
        }
    } else if (warp == 1 && lane == 0 && leader) {
        // ---- MMA issuer (leader only) ----
        int s = 0, acc = 0;
        uint32_t ph = 0, aph = 0;
        for (int64_t p = first; p < g.pairs && !*abort_flag; p += stride) {
            if (!cm_mbar_wait(&tempty[acc], aph ^ 1u)) {
                fail();
                break;
            }
            tc_fence_after();
            const uint32_t d_tmem = tmem_base + (uint32_t)(acc * BN);
            bool ok = true;
            for (int kb = 0; kb < g.kblocks; kb += KG) {
                if (*abort_flag || !cm_mbar_wait(&full[s], ph)) {
                    fail();
                    ok = false;
                    break;
                }
                tc_fence_after();
                const int nb = g.kblocks - kb < KG ? g.kblocks - kb : KG;
                for (int u = 0; u < nb; ++u) {
                    const uint32_t sa = cm_smem_u32(base + (s * KG + u) * STAGE_BYTES);
                    const uint32_t sb = sa + A_BYTES;
#pragma unroll
                    for (int kk = 0; kk < BK / 16; ++kk)
                        mma_bf16_pair(d_tmem, smem_desc_sw128(sa + kk * 32),
                                      smem_desc_sw128(sb + kk * 32), ((kb + u) | kk) != 0);
                }
                mma_commit_pair(&empty[s]);   // the group is free in both CTAs
                if (++s == GROUPS) {
                    s = 0;
                    ph ^= 1u;
                }
            }
            if (!ok) break;
            mma_commit_pair(&tfull[acc]);     // both halves of the accumulator are ready
            if (++acc == ACCS) {
                acc = 0;
                aph ^= 1u;
            }
        }
        // all MMAs issued by this thread have completed once `drain` fires
        mma_commit_local(drain);
        cm_mbar_wait(drain, 0, 100000000ull);
    } else if (warp >= 2) {
        // ---- epilogue (both CTAs): TMEM -> registers -> Ct ----
        const int q = warp & 3;                  // TMEM lane quarter of this warp
        const int row = q * 32 + lane;           // row of the CTA's tile
        int acc = 0;
        uint32_t aph = 0;
        for (int64_t p = first; p < g.pairs; p += stride) {
            // warp-uniform decisions: tcgen05.ld below is .sync.aligned
            if (__shfl_sync(0xffffffffu, *abort_flag, 0)) break;
            const bool ok = cm_mbar_wait(&tfull[acc], aph);
            if (!__all_sync(0xffffffffu, ok)) {
                if (lane == 0) fail();
                break;
            }
            tc_fence_after();
            const Tile x = tile_of(g, p, rank);
            const bool valid = row < x.rows;
            float *dst = g.Ct + (x.crow + row) * g.ldc + x.n0;
            const uint32_t taddr = tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(acc * BN);
#pragma unroll 1
            for (int c = 0; c < BN / 32; ++c) {
                float v[32];
                tmem_load32(taddr + c * 32, v);
                const int col = x.n0 + c * 32;
                if (valid && col < g.N) {
                    float *o = dst + c * 32;
                    if (col + 32 <= g.N && ((g.ldc & 3) == 0)) {
                        // streaming stores: Ct is written once and not read
                        // here, so it should not displace Bt from L2
#pragma unroll
                        for (int i = 0; i < 32; i += 4)
                            __stcs(reinterpret_cast<float4 *>(o + i),
                                   make_float4(v[i], v[i + 1], v[i + 2], v[i + 3]));
                    } else {
#pragma unroll
                        for (int i = 0; i < 32; ++i)
                            if (col + i < g.N) o[i] = v[i];
                    }
                }
            }
            tc_fence_before();
            mbar_arrive_cluster(map_to_rank(&tempty[acc], 0));   // release on the leader
            if (row < x.pad) {   // pad rows of the last systematic block past the tile
                float *z = dst + (int64_t)BM * g.ldc;
                for (int c = 0; c < BN && x.n0 + c < g.N; ++c) z[c] = 0.0f;
            }
            if (++acc == ACCS) {
                acc = 0;
                aph ^= 1u;
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    cluster_sync();   // neither CTA has a copy, commit or arrival left for the other
    if (warp == 1) {
        __syncwarp();
        tc_fence_after();
        asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;\n" ::"r"(tmem_base),
                     "r"(TMEM_COLS)
                     : "memory");
    }
}

}  // namespace

cudaError_t launch_coded_gemm(const CodeParams &cp, const uint16_t *A, int64_t lda,
                              const uint16_t *par, int64_t ldp, const uint16_t *Bt, int64_t ldb,
                              int N, float *Ct, int64_t ldc, int32_t *status, uint32_t only,
                              cudaStream_t s)
{
    CUtensorMap tmA, tmP, tmB;
    const uint64_t d = (uint64_t)cp.d;
    if (!cm_make_tmap_2d(&tmA, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, A, d, (uint64_t)cp.m,
                         (uint64_t)lda * 2, BK, BM, CU_TENSOR_MAP_SWIZZLE_128B) ||
        !cm_make_tmap_2d(&tmP, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, par, d,
                         (uint64_t)(cp.n - cp.k) * cp.L, (uint64_t)ldp * 2, BK, BM,
                         CU_TENSOR_MAP_SWIZZLE_128B) ||
        !cm_make_tmap_2d(&tmB, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, Bt, d, (uint64_t)N,
                         (uint64_t)ldb * 2, BK, BNH, CU_TENSOR_MAP_SWIZZLE_128B))
        return cudaErrorInvalidValue;
    GemmArgs g;
    g.Ct = Ct;
    g.ldc = ldc;
    g.status = status;
    g.kL = (int64_t)cp.k * cp.L;
    g.pL = (int64_t)(cp.n - cp.k) * cp.L;
    g.N = N;
    g.psys = (int)((cp.m + 2 * BM - 1) / (2 * BM));
    g.ppar = (int)((g.pL + 2 * BM - 1) / (2 * BM));
    g.ntiles = (N + BN - 1) / BN;
    g.kblocks = (int)((cp.d + BK - 1) / BK);
    g.pairs = (int64_t)(g.psys + g.ppar) * g.ntiles;
    g.L = cp.L;
    g.k = cp.k;
    g.nruns = 0;
    for (int j = 0; j <= CM_MAX_N; ++j) g.run_p0[j] = 0;
    for (int j = 0; j < CM_MAX_N; ++j) g.run_w[j] = g.run_cnt[j] = 0;
    if (only) {   // runs of consecutive workers of `only`, none across A | parity
        int32_t p0 = 0;
        for (int j = 0; j < cp.n;) {
            if (!((only >> j) & 1u)) {
                ++j;
                continue;
            }
            const int end = j < cp.k ? cp.k : cp.n;
            int c = 0;
            while (j + c < end && ((only >> (j + c)) & 1u)) ++c;
            g.run_w[g.nruns] = (int8_t)j;
            g.run_cnt[g.nruns] = (int8_t)c;
            g.run_p0[g.nruns++] = p0;
            p0 += (int32_t)((c * cp.L + 2 * BM - 1) / (2 * BM));
            j += c;
        }
        g.run_p0[g.nruns] = p0;
        g.pairs = (int64_t)p0 * g.ntiles;
    }
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 2;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = SMEM_BYTES;
    cfg.stream = s;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    // persistent: as many pairs as can be resident at once.  The shared-memory
    // limit belongs to the function in each device's context: set on every
    // call (about 0.2 us); the cluster occupancy is queried once per device.
    if (cudaFuncSetAttribute(gemm_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             SMEM_BYTES) != cudaSuccess)
        return cudaErrorInvalidConfiguration;
    static std::atomic<int> resident_of[64] = {};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return cudaErrorInvalidConfiguration;
    int resident = dev >= 0 && dev < 64 ? resident_of[dev].load(std::memory_order_relaxed) : 0;
    if (resident <= 0) {
        cudaLaunchConfig_t q = cfg;
        q.gridDim = dim3(2 * (unsigned)((cm_sm_count() + 1) / 2));
        int c = 0;
        if (cudaOccupancyMaxActiveClusters(&c, gemm_kernel, &q) != cudaSuccess)
            return cudaErrorInvalidConfiguration;
        resident = c;
        if (c > 0 && dev >= 0 && dev < 64) resident_of[dev].store(c, std::memory_order_relaxed);
    }
    int clusters = resident;
    if (clusters < 1) return cudaErrorInvalidConfiguration;
    if (clusters > g.pairs) clusters = (int)g.pairs;
    cfg.gridDim = dim3(2 * (unsigned)clusters);
    const cudaError_t e = cudaLaunchKernelEx(&cfg, gemm_kernel, tmA, tmP, tmB, g);
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
}
