// K8: the coded-shuffling planner on the device (Sec. IV).
//
// Computes, for the transition t -> t+1, exactly what the host planner
// (shuffle.cpp) computes -- the partition, Alg. 1's message plan, the
// decoding and commit programs and the cache update rule -- with the state
// (partition, cache masks, slot tables) resident in the caller's workspace,
// so that a transition needs no host work beyond reading back four counts.
// The definitions are the host planner's (see its header comment); the
// device version reaches the same result through selections and stable sorts:
//   partition     owner = rank of the row in (key, row) order / (q/n): a
//                 histogram of the top bits of the keys and its scan give
//                 every bucket its first rank; a bucket inside one owner's
//                 positions gives its rows that owner, and the few rows of
//                 the buckets across a boundary are ranked among themselves;
//   received      missing rows in (worker, row) order: a stable sort by
//                 worker of the rows in ascending order;
//   messages      received rows stably sorted by the set I (bit mask), i.e.
//                 (I, worker, row); row j of a worker's run in I goes to
//                 message row base(I) + j, entries ordered by worker;
//   cache update  the s - q/n candidates (worker, row) of smallest (key, row)
//                 of every worker: per worker a histogram of the top 16 key
//                 bits locates the bucket of its (s - q/n)-th candidate;
//                 candidates below it are kept, those in it ranked exactly;
//   commit        dropped slots of each worker, ascending, take its received
//                 rows in order.
// Radix sorts: 8-bit digits, one histogram launch for all passes of a sort
// and one launch per pass.  A pass takes tiles of 4096 items in the order of
// an atomic counter; a tile ranks its items stably (equal digits of a 32-item
// step by __match_any_sync, warps in order), publishes its digit counts, and
// finds its global digit offsets by looking back over the flags of the tiles
// before it (decoupled look-back: a tile's flag holds its count, then its
// inclusive prefix; a bounded wait, an error flag on time-out), then writes
// each digit's run to consecutive addresses through shared memory.
// Device scans: one launch, tiles of 4096 items per 1024-thread block taken
// in atomic-counter order, each tile's prefix by the same kind of look-back
// (warp 0 reads 32 predecessor flags at a time).
#include <cuda_runtime.h>
#include <stdint.h>

#include <algorithm>
#include <vector>

#include "cm_internal.cuh"
#include "shuffle_internal.h"

namespace {

constexpr int kSortThreads = 256;  // one radix tile per block: 8 warps
constexpr int kSortWarps = kSortThreads / 32;
constexpr int kSortIpt = 16;       // items per thread
constexpr int kTile = kSortThreads * kSortIpt;   // items per tile
constexpr int kMaxPasses = 2;      // 16-bit keys at most
constexpr int kSortSlots = 2;      // sorts per transition (own global histograms)
constexpr int kCBits = 16;         // bucket bits of the cache-update selection
// shared memory of a pass: the tile's keys and values in digit order, the
// per-warp digit counts, the tile's digit starts and global bases
constexpr int kSortSmem = kTile * 12 + (kSortWarps + 2) * 256 * 4 + 64;
// the totals array: T_COUNT counters read back by the host; the lengths of
// the two selections' boundary lists (kListP, kListC); per worker the
// cache-update bucket (kThr) and how many of its candidates to keep
// (kNeed); the tile and done counters of the running radix pass at kCtr;
// the global histograms of the radix sorts from word 64
constexpr int kListP = 8, kListC = 9, kThr = 16, kNeed = 32;
constexpr int kCtr = 56;
constexpr int kGhist = 64;
constexpr int kTotalsWords = kGhist + kSortSlots * kMaxPasses * 256;
constexpr int kScanBlock = 1024;
constexpr int kScanItems = 4 * kScanBlock;
constexpr int kMaxDeviceN = 16;    // dense tables over all 2^n worker sets

// slots of the small totals array
enum { T_R = 0, T_K, T_C, T_X, T_SETS, T_ERR, T_DUMMY, T_COUNT = 8 };

__device__ __forceinline__ uint64_t mix64(uint64_t seed, uint64_t index)
{
    uint64_t z = seed + index * 0x9E3779B97F4A7C15ull;
    z ^= z >> 30;
    z *= 0xBF58476D1CE4E5B9ull;
    z ^= z >> 27;
    z *= 0x94D049BB133111EBull;
    z ^= z >> 31;
    return z;
}

#define GS_LOOP(i, count)                                                                     \
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < (count);             \
         i += (int64_t)gridDim.x * blockDim.x)

unsigned grid_for(int64_t items)
{
    const int64_t want = (items + 255) / 256;
    const int64_t cap = (int64_t)cm_sm_count() * 8;
    return (unsigned)std::max<int64_t>(1, std::min(want, cap));
}

// ---- fills ----------------------------------------------------------------------------

__global__ void fill_i32(int32_t *p, int64_t count, int32_t v) { GS_LOOP(i, count) p[i] = v; }

// Zero up to 8 int32 regions in one launch.
struct ZeroList {
    int32_t *p[8];
    int64_t n[8];
    int k;
};

__global__ void zero_many_kernel(const ZeroList z)
{
    for (int r = 0; r < z.k; ++r) GS_LOOP(i, z.n[r]) z.p[r][i] = 0;
}

// ---- tile flags of the decoupled look-backs --------------------------------------------

// epoch (30 bits) << 34 | status << 32 | 32-bit value.  A flag whose epoch is
// not the running pass's has not been published yet; flags are never cleared.
constexpr uint64_t kFlagAgg = 1, kFlagInc = 2;   // the tile's own sum / its inclusive prefix
constexpr uint32_t kEpochMask = 0x3fffffffu;
constexpr int kLook = 16;   // tiles read together by one step of a radix look-back

__device__ __forceinline__ uint64_t flag_word(uint32_t epoch, uint64_t status, int32_t v)
{
    return ((uint64_t)(epoch & kEpochMask) << 34) | (status << 32) | (uint64_t)(uint32_t)v;
}
__device__ __forceinline__ bool flag_ready(uint64_t w, uint32_t epoch)
{
    return (uint32_t)(w >> 34) == (epoch & kEpochMask);
}
__device__ __forceinline__ uint64_t flag_status(uint64_t w) { return (w >> 32) & 3u; }
__device__ __forceinline__ int32_t flag_value(uint64_t w) { return (int32_t)(uint32_t)w; }

// Flags, epochs and counters shared by the look-back kernels of a planner
// workspace; the kernels run one after another on one stream.
struct LookBack {
    uint64_t *flags;
    int64_t nflags;
    int32_t *ctr;     // [0]: next tile, [1]: finished blocks (reset by the last one)
    int32_t *err;     // set on a look-back time-out
    uint32_t *epoch;  // host counter, one value per launch
};

uint32_t next_epoch(uint32_t *e)
{
    if (((++*e) & kEpochMask) == 0) ++*e;   // epoch 0 is the cleared flag
    return *e;
}

// ---- exclusive scan (int32) -----------------------------------------------------------

// Scan inputs and epilogues: the default reads an array and writes nothing
// more; a fused step generates its inputs or consumes (index, value,
// exclusive prefix) itself.
struct ArrayIn {
    const int32_t *p;
    __device__ int32_t operator()(int64_t i) const { return p[i]; }
};
struct NoEpilogue {
    __device__ void operator()(int64_t, int32_t, int32_t) const {}
};

// One pass: tiles of 4096 items in the order of an atomic counter; a tile
// scans itself, publishes its sum, and warp 0 looks back over the flags of
// the 32 tiles before it at a time for its prefix (bounded waits).  `out`
// (nullable) receives the exclusive prefixes.
template <class In, class Epi>
__global__ void __launch_bounds__(kScanBlock) scan_kernel(In in, Epi epi, int32_t *out,
                                                          int64_t count, int32_t *total,
                                                          uint64_t *flags, uint32_t epoch,
                                                          int32_t *ctr, int32_t *err)
{
    __shared__ int32_t warp_sums[32];
    __shared__ int32_t s_tile, s_prefix;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const bool multi = gridDim.x > 1;
    if (threadIdx.x == 0) s_tile = multi ? atomicAdd(&ctr[0], 1) : 0;
    __syncthreads();
    const int64_t tile = s_tile;
    const int64_t base = tile * kScanItems + 4 * (int64_t)threadIdx.x;
    int32_t v[4], sum = 0;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        v[k] = base + k < count ? in(base + k) : 0;
        sum += v[k];
    }
    int32_t x = sum;   // inclusive scan of the thread sums within the warp
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int32_t y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
    }
    if (lane == 31) warp_sums[warp] = x;
    __syncthreads();
    if (warp == 0) {
        int32_t w = warp_sums[lane];
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int32_t y = __shfl_up_sync(0xffffffffu, w, o);
            if (lane >= o) w += y;
        }
        warp_sums[lane] = w;   // inclusive over the warps; [31] = the tile's sum
        const int32_t agg = __shfl_sync(0xffffffffu, w, 31);
        int32_t pre = 0;
        if (multi) {
            if (lane == 0)
                atomicExch(reinterpret_cast<unsigned long long *>(flags + tile),
                           (unsigned long long)flag_word(epoch, tile ? kFlagAgg : kFlagInc, agg));
            int64_t t = tile - 1;
            uint32_t it = 0;
            while (t >= 0) {
                const int64_t idx = t - lane;
                const uint64_t f = idx >= 0 ? *(const volatile uint64_t *)(flags + idx)
                                            : flag_word(epoch, kFlagInc, 0);
                const bool ready = flag_ready(f, epoch);
                const unsigned incm = __ballot_sync(0xffffffffu, ready && flag_status(f) == kFlagInc);
                const unsigned notready = __ballot_sync(0xffffffffu, !ready);
                const int last = incm ? __ffs(incm) - 1 : 31;   // lanes [0, last] are summed
                const unsigned upto = last == 31 ? 0xffffffffu : ((2u << last) - 1u);
                if (notready & upto) {   // wait (bounded) and read the same tiles again
                    if (++it > (1u << 21) ||
                        __any_sync(0xffffffffu, *(volatile int32_t *)err != 0)) {
                        if (lane == 0) atomicExch(err, 1);
                        break;
                    }
                    __nanosleep(64);
                    continue;
                }
                int32_t part = lane <= last ? flag_value(f) : 0;
#pragma unroll
                for (int o = 16; o; o >>= 1) part += __shfl_xor_sync(0xffffffffu, part, o);
                pre += part;
                if (incm) break;
                t -= 32;
            }
            if (lane == 0 && tile > 0)
                atomicExch(reinterpret_cast<unsigned long long *>(flags + tile),
                           (unsigned long long)flag_word(epoch, kFlagInc, pre + agg));
        }
        if (lane == 0) {
            s_prefix = pre;
            if (total && tile == (count - 1) / kScanItems) *total = pre + agg;
        }
    }
    __syncthreads();
    int32_t excl = x - sum + (warp ? warp_sums[warp - 1] : 0) + s_prefix;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        if (base + k < count) {
            if (out) out[base + k] = excl;
            epi(base + k, v[k], excl);
        }
        excl += v[k];
    }
    if (multi && threadIdx.x == 0 && atomicAdd(&ctr[1], 1) == (int32_t)gridDim.x - 1) {
        ctr[0] = 0;
        ctr[1] = 0;
    }
}

int64_t up256(int64_t x) { return (x + 255) & ~(int64_t)255; }

// out[i] = in(0) + ... + in(i-1) for i < count (out nullable; an input
// array may be out), epi(i, in(i), out[i]) for every i; the sum of all of
// them goes to *total (device, nullable).  One launch.
template <class In, class Epi>
cudaError_t scan_fused(const LookBack &lb, In in, Epi epi, int32_t *out, int64_t count,
                       int32_t *total, cudaStream_t s)
{
    if (count <= 0) {
        if (total) fill_i32<<<1, 32, 0, s>>>(total, 1, 0);
        return cudaGetLastError();
    }
    const int64_t nb = (count + kScanItems - 1) / kScanItems;
    if (nb > lb.nflags || nb > INT32_MAX) return cudaErrorInvalidValue;
    const uint32_t epoch = nb > 1 ? next_epoch(lb.epoch) : 0;
    scan_kernel<In, Epi><<<(unsigned)nb, kScanBlock, 0, s>>>(in, epi, out, count, total, lb.flags,
                                                             epoch, lb.ctr, lb.err);
    return cudaGetLastError();
}

cudaError_t scan_exclusive(const LookBack &lb, const int32_t *in, int32_t *out, int64_t count,
                           int32_t *total, cudaStream_t s)
{
    return scan_fused(lb, ArrayIn{in}, NoEpilogue{}, out, count, total, s);
}

// ---- stable LSD radix sort (64-bit keys, int32 values) ---------------------------------

// Counts of every digit of every pass of a sort, summed into ghist[pass][256]
// (zero on entry).
__global__ void __launch_bounds__(256) radix_hist_kernel(const uint64_t *keys,
                                                         const int32_t *countp, int64_t cap,
                                                         int lo, int passes, int32_t *ghist)
{
    __shared__ int32_t h[kMaxPasses][256];
    for (int t = threadIdx.x; t < kMaxPasses * 256; t += blockDim.x) h[t / 256][t % 256] = 0;
    __syncthreads();
    const int64_t count = countp ? (int64_t)*countp : cap;
    GS_LOOP(i, count)
    {
        const uint64_t k = keys[i];
        for (int p = 0; p < passes; ++p) atomicAdd(&h[p][(k >> (lo + 8 * p)) & 255], 1);
    }
    __syncthreads();
    for (int t = threadIdx.x; t < passes * 256; t += blockDim.x)
        if (h[t / 256][t % 256]) atomicAdd(&ghist[t], h[t / 256][t % 256]);
}

// Exclusive scan over the block's 256 threads (one value each); returns the
// thread's exclusive prefix and leaves the total in *total.
__device__ __forceinline__ int32_t block_scan256(int32_t x, int32_t *wsum, int32_t *total)
{
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int32_t inc = x;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int32_t y = __shfl_up_sync(0xffffffffu, inc, o);
        if (lane >= o) inc += y;
    }
    if (lane == 31) wsum[warp] = inc;
    __syncthreads();
    int32_t before = 0, all = 0;
#pragma unroll
    for (int w = 0; w < kSortWarps; ++w) {
        const int32_t v = wsum[w];
        before += w < warp ? v : 0;
        all += v;
    }
    __syncthreads();
    *total = all;
    return before + inc - x;
}

// One pass: bits [shift, shift + 8) of the keys.  ctr[0] hands out tiles,
// ctr[1] counts finished blocks; the last block resets both.
__global__ void __launch_bounds__(kSortThreads)
radix_pass_kernel(const uint64_t *kin, const int32_t *vin, uint64_t *kout, int32_t *vout,
                  const int32_t *countp, int64_t cap, int shift, const int32_t *ghist,
                  uint64_t *flags, uint32_t epoch, int32_t *ctr, int32_t *err)
{
    extern __shared__ __align__(16) unsigned char smem[];
    uint64_t *sk = reinterpret_cast<uint64_t *>(smem);
    int32_t *sv = reinterpret_cast<int32_t *>(smem + kTile * 8);
    int32_t *wcnt = sv + kTile;                      // [warp][digit]
    int32_t *dstart = wcnt + kSortWarps * 256;       // tile-local start of each digit
    int32_t *gbase = dstart + 256;                   // global position of that start
    int32_t *misc = gbase + 256;                     // [0]: tile, [1..8]: warp sums
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, d = threadIdx.x;
    if (threadIdx.x == 0) misc[0] = atomicAdd(&ctr[0], 1);
    __syncthreads();
    const int64_t tile = misc[0];
    const int64_t count = countp ? (int64_t)*countp : cap;
    const int64_t beg = tile * kTile;
    if (beg < count) {
        const int nt = (int)(count - beg < kTile ? count - beg : kTile);
        // items w * 512 + 32 j + lane of the tile, in registers
        uint64_t k[kSortIpt];
        int32_t v[kSortIpt], r[kSortIpt];
#pragma unroll
        for (int j = 0; j < kSortIpt; ++j) {
            const int p = warp * 32 * kSortIpt + 32 * j + lane;
            k[j] = p < nt ? kin[beg + p] : 0;
            v[j] = p < nt ? vin[beg + p] : 0;
        }
        int32_t *mine = wcnt + warp * 256;
        for (int t = lane; t < 256; t += 32) mine[t] = 0;
        __syncwarp();
        const unsigned below = (1u << lane) - 1u;
#pragma unroll
        for (int j = 0; j < kSortIpt; ++j) {
            const bool valid = warp * 32 * kSortIpt + 32 * j + lane < nt;
            const int dg = valid ? (int)((k[j] >> shift) & 255) : 256;   // 256: not an item
            const unsigned peers = __match_any_sync(0xffffffffu, dg);
            r[j] = valid ? mine[dg] + __popc(peers & below) : 0;
            __syncwarp();
            if (valid && (peers & below) == 0) mine[dg] += __popc(peers);
            __syncwarp();
        }
        __syncthreads();
        // digit d: prefixes over the warps, its total, its tile-local start
        int32_t tot = 0;
#pragma unroll
        for (int w = 0; w < kSortWarps; ++w) {
            const int32_t c = wcnt[w * 256 + d];
            wcnt[w * 256 + d] = tot;
            tot += c;
        }
        // publish the tile's count of digit d (tile 0: its inclusive prefix,
        // from the digit's start over all keys) for the tiles after it
        int32_t gd = 0;
        uint64_t *f = flags + tile * 256 + d;
        if (tile == 0) {
            int32_t ga;
            gd = block_scan256(ghist[d], misc + 1, &ga);
            atomicExch(reinterpret_cast<unsigned long long *>(f),
                       (unsigned long long)flag_word(epoch, kFlagInc, gd + tot));
        } else {
            atomicExch(reinterpret_cast<unsigned long long *>(f),
                       (unsigned long long)flag_word(epoch, kFlagAgg, tot));
        }
        int32_t all;
        const int32_t ds = block_scan256(tot, misc + 1, &all);
        dstart[d] = ds;
        __syncthreads();
        // the tile in digit order in shared memory (the registers are free
        // before the look-back)
#pragma unroll
        for (int j = 0; j < kSortIpt; ++j) {
            if (warp * 32 * kSortIpt + 32 * j + lane < nt) {
                const int dg = (int)((k[j] >> shift) & 255);
                const int pos = dstart[dg] + wcnt[warp * 256 + dg] + r[j];
                sk[pos] = k[j];
                sv[pos] = v[j];
            }
        }
        if (tile > 0) {   // the counts of digit d in the tiles before this one
            // look back kLook tiles at a time: their flags are read together,
            // then summed newest first up to the first inclusive one; an
            // unpublished flag is read again (a bounded wait)
            int32_t excl = 0;
            int64_t t = tile - 1;
            uint32_t it = 0;
            while (t >= 0) {
                uint64_t w[kLook];
#pragma unroll
                for (int i = 0; i < kLook; ++i)
                    w[i] = t - i >= 0 ? *(const volatile uint64_t *)(flags + (t - i) * 256 + d)
                                      : flag_word(epoch, kFlagInc, 0);
                int used = kLook;
                bool done = false;
#pragma unroll
                for (int i = 0; i < kLook; ++i) {
                    if (done || used < kLook) continue;
                    if (!flag_ready(w[i], epoch)) {
                        used = i;   // not yet published: read again from tile t - i
                    } else {
                        excl += flag_value(w[i]);
                        if (flag_status(w[i]) == kFlagInc) done = true;
                    }
                }
                if (done) break;
                t -= used;
                if (used < kLook) {
                    // give up after about 0.1-1 s, or at once if another thread has
                    if (++it > (1u << 21) || *(volatile int32_t *)err) {
                        atomicExch(err, 1);
                        break;
                    }
                    __nanosleep(64);
                }
            }
            atomicExch(reinterpret_cast<unsigned long long *>(f),
                       (unsigned long long)flag_word(epoch, kFlagInc, excl + tot));
            gd = excl;
        }
        gbase[d] = gd;
        __syncthreads();
        // each digit's run out
        for (int p = threadIdx.x; p < nt; p += kSortThreads) {
            const uint64_t kk = sk[p];
            const int dg = (int)((kk >> shift) & 255);
            const int64_t g = (int64_t)gbase[dg] + (p - dstart[dg]);
            kout[g] = kk;
            vout[g] = sv[p];
        }
    }
    __syncthreads();
    if (threadIdx.x == 0 && atomicAdd(&ctr[1], 1) == (int32_t)gridDim.x - 1) {
        ctr[0] = 0;   // every block has taken its tile: ready for the next pass
        ctr[1] = 0;
    }
}

struct SortBufs {
    uint64_t *kA, *kB;
    int32_t *vA, *vB;
    int32_t *ghist;   // kSortSlots x kMaxPasses x 256, zero at the start of a transition
    LookBack lb;
};

// Stable sort of items [0, count) (count = *countp, or cap if countp is null)
// by bits [lo, hi) of their keys (at most kMaxPasses digits), using global
// histogram slot `slot`; on return the sorted keys and values are in
// (*k_out, *v_out), one of the two buffer pairs.
cudaError_t radix_sort(const SortBufs &b, const int32_t *countp, int64_t cap, int lo, int hi,
                       int slot, cudaStream_t s, uint64_t **k_out, int32_t **v_out)
{
    const int passes = (hi - lo + 7) / 8;
    if (passes < 1 || passes > kMaxPasses || slot < 0 || slot >= kSortSlots)
        return cudaErrorInvalidValue;
    const int64_t tiles = std::max<int64_t>(1, (cap + kTile - 1) / kTile);
    if (tiles * 256 > b.lb.nflags) return cudaErrorInvalidValue;
    int32_t *gh = b.ghist + slot * kMaxPasses * 256;
    uint64_t *ki = b.kA, *ko = b.kB;
    int32_t *vi = b.vA, *vo = b.vB;
    cudaError_t ea = cudaFuncSetAttribute(radix_pass_kernel,
                                          cudaFuncAttributeMaxDynamicSharedMemorySize, kSortSmem);
    if (ea != cudaSuccess) return ea;
    radix_hist_kernel<<<grid_for(cap), 256, 0, s>>>(ki, countp, cap, lo, passes, gh);
    for (int p = 0; p < passes; ++p) {
        const uint32_t epoch = next_epoch(b.lb.epoch);
        radix_pass_kernel<<<(unsigned)tiles, kSortThreads, kSortSmem, s>>>(
            ki, vi, ko, vo, countp, cap, lo + 8 * p, gh + p * 256, b.lb.flags, epoch, b.lb.ctr,
            b.lb.err);
        std::swap(ki, ko);
        std::swap(vi, vo);
    }
    *k_out = ki;
    *v_out = vi;
    return cudaGetLastError();
}

// ---- planner kernels --------------------------------------------------------------------

// ---- partition by selection ------------------------------------------------------------

__device__ __forceinline__ uint64_t part_key(uint64_t seed, int64_t t1, int64_t q, int64_t r)
{
    return mix64(seed, (uint64_t)t1 * (uint64_t)q + (uint64_t)r);
}

// rows per bucket of the top `bits` key bits (hist zero on entry)
__global__ void part_hist_kernel(int64_t q, uint64_t seed, int64_t t1, int bits, int32_t *hist)
{
    GS_LOOP(r, q) atomicAdd(&hist[part_key(seed, t1, q, r) >> (64 - bits)], 1);
}

// The owner of every row whose bucket's ranks [bstart, bstart + count) lie
// inside one owner's positions; the rows of the other buckets are listed.
__global__ void part_owner_kernel(int64_t q, uint64_t seed, int64_t t1, int bits, int64_t per,
                                  const int32_t *hist, const int32_t *bstart, int32_t *owner1,
                                  int32_t *list, int32_t *nlist)
{
    GS_LOOP(r, q)
    {
        const int64_t b = (int64_t)(part_key(seed, t1, q, r) >> (64 - bits));
        const int64_t lo = bstart[b], hi = lo + hist[b] - 1;
        if (lo / per == hi / per) owner1[r] = (int32_t)(lo / per);
        else list[atomicAdd(nlist, 1)] = (int32_t)r;
    }
}

// A listed row's rank: its bucket's first rank plus the listed rows of the
// same bucket before it in (key, row) order.
__global__ void part_rank_kernel(int64_t q, uint64_t seed, int64_t t1, int bits, int64_t per,
                                 const int32_t *bstart, const int32_t *list,
                                 const int32_t *nlist, int32_t *owner1)
{
    const int64_t m = *nlist;
    GS_LOOP(x, m)
    {
        const int32_t r = list[x];
        const uint64_t k = part_key(seed, t1, q, r), b = k >> (64 - bits);
        int64_t rank = bstart[b];
        for (int64_t y = 0; y < m; ++y) {
            const int32_t r2 = list[y];
            const uint64_t k2 = part_key(seed, t1, q, r2);
            if ((k2 >> (64 - bits)) == b && (k2 < k || (k2 == k && r2 < r))) ++rank;
        }
        owner1[r] = (int32_t)(rank / per);
    }
}

// ---- cache update by selection ---------------------------------------------------------

__device__ __forceinline__ uint64_t cache_key(uint64_t seed, int64_t t1, int n, int i, int64_t q,
                                              int64_t r)
{
    return mix64(seed, ((uint64_t)t1 * (uint64_t)n + (uint64_t)i) * (uint64_t)q + (uint64_t)r);
}

// Candidates of worker i: rows it caches outside its new set.  Counts per
// (worker, top kCBits key bits) (hist zero on entry).
__global__ void cand_hist_kernel(int64_t q, int n, int64_t t1, uint64_t seed,
                                 const int32_t *owner1, const uint64_t *cached0, int32_t *hist)
{
    GS_LOOP(r, q)
    {
        for (uint64_t b = cached0[r] & ~(1ull << owner1[r]); b; b &= b - 1) {
            const int i = __ffsll((long long)b) - 1;
            const uint64_t k = cache_key(seed, t1, n, i, q, r);
            atomicAdd(&hist[((int64_t)i << kCBits) + (int64_t)(k >> (64 - kCBits))], 1);
        }
    }
}

// One block per worker: the bucket that holds its keep-th candidate (thr)
// and how many of that bucket's candidates it keeps (need); thr = 2^kCBits
// when it keeps all, -1 when it keeps none.  Warp w sums its 2048 buckets
// (coalesced), the block scans the 32 sums, and the warp whose range holds
// the keep-th candidate walks its buckets 32 at a time.
__global__ void __launch_bounds__(1024) cand_threshold_kernel(const int32_t *hist, int64_t keep,
                                                              int32_t *thr, int32_t *need)
{
    constexpr int kChunk = (1 << kCBits) / 32;
    __shared__ int32_t wsum[32];
    const int i = blockIdx.x, lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int32_t *h = hist + ((int64_t)i << kCBits) + (int64_t)warp * kChunk;
    int32_t sum = 0;
    for (int j = lane; j < kChunk; j += 32) sum += h[j];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
    if (lane == 0) wsum[warp] = sum;
    __syncthreads();
    int64_t before = 0, total = 0;
    for (int w = 0; w < 32; ++w) {
        before += w < warp ? wsum[w] : 0;
        total += wsum[w];
    }
    if (threadIdx.x == 0) {
        if (keep <= 0) {
            thr[i] = -1;
            need[i] = 0;
        } else if (total <= keep) {
            thr[i] = 1 << kCBits;
            need[i] = 0;
        }
    }
    if (keep > 0 && total > keep && before < keep && keep <= before + sum) {
        int64_t run = before;   // candidates in the buckets before this step
        for (int j = 0; j < kChunk; j += 32) {
            const int32_t v = h[j + lane];
            int32_t inc = v;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int32_t y = __shfl_up_sync(0xffffffffu, inc, o);
                if (lane >= o) inc += y;
            }
            const unsigned hit = __ballot_sync(0xffffffffu, run + inc >= keep);
            if (hit) {
                const int f = __ffs(hit) - 1;
                if (lane == f) {
                    thr[i] = warp * kChunk + j + f;
                    need[i] = (int32_t)(keep - (run + inc - v));
                }
                break;
            }
            run += __shfl_sync(0xffffffffu, inc, 31);
        }
    }
}

// Candidates below their worker's bucket are kept (bits added to the new
// cache mask); those in it are listed.
__global__ void cand_classify_kernel(int64_t q, int n, int64_t t1, uint64_t seed,
                                     const int32_t *owner1, const uint64_t *cached0,
                                     const int32_t *thr, uint64_t *next, int32_t *lw,
                                     int32_t *lr, uint64_t *lk, int32_t *nlist)
{
    __shared__ int32_t sthr[kMaxDeviceN];
    if (threadIdx.x < n) sthr[threadIdx.x] = thr[threadIdx.x];
    __syncthreads();
    GS_LOOP(r, q)
    {
        uint64_t add = 0;
        for (uint64_t b = cached0[r] & ~(1ull << owner1[r]); b; b &= b - 1) {
            const int i = __ffsll((long long)b) - 1;
            const uint64_t k = cache_key(seed, t1, n, i, q, r);
            const int64_t bk = (int64_t)(k >> (64 - kCBits));
            if (bk < sthr[i]) {
                add |= 1ull << i;
            } else if (bk == sthr[i]) {
                const int32_t x = atomicAdd(nlist, 1);
                lw[x] = i;
                lr[x] = (int32_t)r;
                lk[x] = k;
            }
        }
        if (add) next[r] |= add;
    }
}

// A listed candidate is kept if fewer than need[i] listed candidates of its
// worker come before it in (key, row) order.
__global__ void cand_rank_kernel(const int32_t *nlist, const int32_t *lw, const int32_t *lr,
                                 const uint64_t *lk, const int32_t *need,
                                 unsigned long long *next)
{
    const int64_t m = *nlist;
    GS_LOOP(x, m)
    {
        const int i = lw[x];
        const int32_t r = lr[x];
        const uint64_t k = lk[x];
        int64_t rank = 0;
        for (int64_t y = 0; y < m; ++y)
            if (lw[y] == i && (lk[y] < k || (lk[y] == k && lr[y] < r))) ++rank;
        if (rank < need[i]) atomicOr(&next[r], 1ull << i);
    }
}

// Per row: missing from its new owner's cache?  Its set I; counts per
// (I, worker) and per worker.  The per-worker counters are aggregated in
// shared memory per block, and so are the (I, worker) counters when their
// table fits (`local` = 2^n n entries, else 0: global atomics).  The new
// cache masks start as the owner's bit.
__global__ void need_kernel(int64_t q, int n, const int32_t *owner1, const uint64_t *cached0,
                            uint64_t *rmask, uint64_t *next, int32_t *counts, int32_t *wcount,
                            int local)
{
    extern __shared__ int32_t sl[];
    __shared__ int32_t sw[kMaxDeviceN];
    if (threadIdx.x < kMaxDeviceN) sw[threadIdx.x] = 0;
    for (int i = threadIdx.x; i < local; i += blockDim.x) sl[i] = 0;
    __syncthreads();
    GS_LOOP(r, q)
    {
        const int i = owner1[r];
        const uint64_t bit = 1ull << i, have = cached0[r];
        const int nf = (have & bit) ? 0 : 1;
        rmask[r] = have | bit;
        next[r] = bit;
        if (nf) {
            const int64_t slot = (int64_t)(have | bit) * n + i;
            if (local) atomicAdd(&sl[slot], 1);
            else atomicAdd(&counts[slot], 1);
            atomicAdd(&sw[i], 1);
        }
    }
    __syncthreads();
    if (threadIdx.x < n) atomicAdd(&wcount[threadIdx.x], sw[threadIdx.x]);
    for (int i = threadIdx.x; i < local; i += blockDim.x)
        if (sl[i]) atomicAdd(&counts[i], sl[i]);
}

// Input of that scan: row r is missing from its new owner's cache.
struct MissingRow {
    const int32_t *owner1;
    const uint64_t *cached0;
    __device__ int32_t operator()(int64_t r) const
    {
        return (cached0[r] >> owner1[r]) & 1ull ? 0 : 1;
    }
};

// Epilogue of the scan of the missing flags: the missing rows compacted in
// row order, as (worker, row) keys of the sort by worker.
struct MissingToKeys {
    const int32_t *owner1;
    uint64_t *keys;
    int32_t *vals;
    __device__ void operator()(int64_t r, int32_t flag, int32_t pos) const
    {
        if (flag) {
            keys[pos] = (uint64_t)owner1[r];
            vals[pos] = (int32_t)r;
        }
    }
};



// The received rows (sorted by worker) stored, and keyed by their sets I for
// the sort into messages.
__global__ void mask_keys_kernel(const int32_t *countp, const int32_t *sorted,
                                 int32_t *recv_row, const uint64_t *rmask, uint64_t *keys,
                                 int32_t *vals)
{
    const int64_t count = *countp;
    GS_LOOP(v, count)
    {
        const int32_t r = sorted[v];
        recv_row[v] = r;
        keys[v] = rmask[r];
        vals[v] = (int32_t)v;
    }
}

__global__ void ell_kernel(int64_t nm, int n, const int32_t *counts, int32_t *ell, int32_t *sets)
{
    GS_LOOP(M, nm)
    {
        int32_t e = 0;
        for (int w = 0; w < n; ++w) e = max(e, counts[M * n + w]);
        ell[M] = e;
        if (e) atomicAdd(sets, 1);
    }
}

// Message row m: its set I (last I with base(I) <= m) and its number of
// entries (workers of I whose run is longer than m's position j).
__global__ void msgrow_kernel(int64_t q, int64_t nm, int n, const int32_t *msgbase,
                              const int32_t *Cp, const int32_t *counts, int32_t *earr,
                              uint64_t *msg_set)
{
    const int64_t C = *Cp;
    GS_LOOP(m, q + 1)
    {
        if (m < C) {
            int64_t lo = 0, hi = nm;   // first index with msgbase > m lies in (0, nm]
            while (lo < hi) {
                const int64_t mid = (lo + hi) / 2;
                if (msgbase[mid] > m) hi = mid;
                else lo = mid + 1;
            }
            const int64_t M = lo - 1;
            const int32_t j = (int32_t)(m - msgbase[M]);
            int32_t e = 0;
            for (int w = 0; w < n; ++w) e += counts[M * n + w] > j;
            earr[m] = e;
            msg_set[m] = (uint64_t)M;
        } else {
            earr[m] = 0;
        }
    }
}

__global__ void entries_kernel(const int32_t *Rp, int n, const int32_t *P, const int32_t *recv_row,
                               const int32_t *owner1, const uint64_t *rmask,
                               const int32_t *runstart, const int32_t *msgbase,
                               const int32_t *counts, const int32_t *enc_ptr, int32_t *enc_src,
                               int32_t *msg_worker, int32_t *dec_msg, int32_t *dec_dst,
                               int32_t *dx)
{
    const int64_t R = *Rp;
    GS_LOOP(k, R)
    {
        const int32_t v = P[k];
        const int32_t r = recv_row[v];
        const int w = owner1[r];
        const int64_t M = (int64_t)rmask[r];
        const int32_t j = (int32_t)(k - runstart[M * n + w]);
        const int32_t m = msgbase[M] + j;
        int32_t off = 0;
        for (int w2 = 0; w2 < w; ++w2) off += counts[M * n + w2] > j;
        const int32_t x = enc_ptr[m] + off;
        enc_src[x] = r;
        msg_worker[x] = w;
        dec_msg[x] = m;
        dec_dst[x] = v;
        dx[x] = enc_ptr[m + 1] - enc_ptr[m] - 1;
    }
}

__global__ void decslot_kernel(const int32_t *Rp, int64_t q, int64_t s, const int32_t *msg_worker,
                               const int32_t *dec_msg, const int32_t *enc_ptr,
                               const int32_t *enc_src, const int32_t *dec_ptr,
                               const int32_t *slot_of, int32_t *dec_slot, int32_t *err)
{
    const int64_t R = *Rp;
    GS_LOOP(x, R)
    {
        const int i = msg_worker[x];
        const int32_t m = dec_msg[x];
        int32_t at = dec_ptr[x];
        for (int32_t y = enc_ptr[m]; y < enc_ptr[m + 1]; ++y) {
            if (y == x) continue;
            const int32_t slot = slot_of[(int64_t)i * q + enc_src[y]];
            if (slot < 0) {
                atomicExch(err, 1);   // unreachable: every other row of I is cached at i
                continue;
            }
            dec_slot[at++] = (int32_t)(i * s + slot);
        }
    }
}

// Input of the scan of the dropped slots: slot g = i s + c of cache i is
// dropped when the new cache mask of its row lacks bit i (0 past the end).
struct DroppedSlot {
    int64_t ns, s;
    const int32_t *slot_row;
    const uint64_t *next;
    __device__ int32_t operator()(int64_t g) const
    {
        if (g >= ns) return 0;
        return (next[slot_row[g]] >> (int)(g / s)) & 1ull ? 0 : 1;
    }
};

__global__ void commit_kernel(int64_t ns, int64_t s, int64_t q, const int32_t *evrank,
                              const int32_t *recv_ptr,
                              const int32_t *recv_row, int32_t *com_dst, int32_t *slot_row,
                              int32_t *slot_of, int32_t *err)
{
    GS_LOOP(g, ns)
    {
        if (evrank[g + 1] == evrank[g]) continue;   // slot g is kept
        const int i = (int)(g / s);
        const int32_t e = evrank[g] - evrank[(int64_t)i * s];
        const int32_t v = recv_ptr[i] + e;
        if (v >= recv_ptr[i + 1]) {
            atomicExch(err, 2);   // unreachable: as many slots drop as rows arrive
            continue;
        }
        com_dst[v] = (int32_t)g;
        const int32_t old = slot_row[g], nr = recv_row[v];
        slot_of[(int64_t)i * q + old] = -1;
        slot_row[g] = nr;
        slot_of[(int64_t)i * q + nr] = (int32_t)(g - (int64_t)i * s);
    }
}

__global__ void check_kernel(int n, int64_t s, const int32_t *evrank, const int32_t *recv_ptr,
                             int32_t *err)
{
    GS_LOOP(i, n)
    {
        const int32_t dropped = evrank[(i + 1) * s] - evrank[i * s];
        if (dropped != recv_ptr[i + 1] - recv_ptr[i]) atomicExch(err, 3);   // unreachable
    }
}

// ---- workspace layout ----------------------------------------------------------------------

struct DevLayout {
    ShuffleLayout prog;       // the row programs, at the start (word offsets)
    int64_t owner[2], cached[2], slot_of;
    int64_t kA, kB, vA, vB, flags;
    int64_t rmask, recv_row, wcount, recv_ptr;
    int64_t counts, runstart, ell, msgbase, earr, msg_set, msg_worker, dx;
    int64_t cw, cr, ckey, evrank, totals;
    int64_t sel, pstart;      // selection histograms (partition, then cache update); scan
    int64_t flags_bytes;      // radix tile flags
    int64_t bytes;            // total
    int64_t capK, nm;
    int pbits;                // bucket bits of the partition selection
    int64_t sel_words;        // 2^pbits + n 2^kCBits
};

DevLayout device_layout(int32_t n, int64_t q, int64_t s)
{
    DevLayout D;
    D.prog = shuffle_layout(n, q, s);
    D.nm = (int64_t)1 << n;
    const int64_t ns = (int64_t)n * s;
    D.capK = std::max(q, ns);
    const int64_t tiles = std::max<int64_t>(1, (q + kTile - 1) / kTile);
    // about two rows per partition bucket
    int lg = 0;
    while (((int64_t)1 << lg) < q) ++lg;
    D.pbits = std::min(20, std::max(8, lg - 1));
    D.sel_words = ((int64_t)1 << D.pbits) + ((int64_t)n << kCBits);
    const int64_t scan_max = std::max({D.nm * n + 1, q + 1, (int64_t)1 << D.pbits, ns + 1});
    int64_t at = up256(D.prog.total * 4);
    auto take = [&](int64_t bytes) {
        const int64_t off = at;
        at = up256(at + bytes);
        return off;
    };
    D.owner[0] = take(4 * q);
    D.owner[1] = take(4 * q);
    D.cached[0] = take(8 * q);
    D.cached[1] = take(8 * q);
    D.slot_of = take(4 * (int64_t)n * q);
    D.kA = take(8 * q);
    D.kB = take(8 * q);
    D.vA = take(4 * q);
    D.vB = take(4 * q);
    // tile flags: a radix pass's 256 per tile, or a scan's one per 4096 items
    D.flags_bytes = 8 * std::max(256 * tiles, scan_max / kScanItems + 1);
    D.flags = take(D.flags_bytes);
    D.rmask = take(8 * q);
    D.recv_row = take(4 * q);
    D.wcount = take(4 * (n + 1));
    D.recv_ptr = take(4 * (n + 1));
    D.counts = take(4 * (D.nm * n + 1));
    D.runstart = take(4 * (D.nm * n + 1));
    D.ell = take(4 * (D.nm + 1));
    D.msgbase = take(4 * (D.nm + 1));
    D.earr = take(4 * (q + 1));
    D.msg_set = take(8 * q);
    D.msg_worker = take(4 * q);
    D.dx = take(4 * (q + 1));
    D.cw = take(4 * D.capK);
    D.cr = take(4 * D.capK);
    D.ckey = take(8 * D.capK);
    D.sel = take(4 * D.sel_words);
    D.pstart = take(4 * ((int64_t)1 << D.pbits));
    D.evrank = take(4 * (ns + 1));
    D.totals = take(4 * kTotalsWords);
    D.bytes = at;
    return D;
}

template <class T>
T *ptr(void *ws, int64_t byte_off)
{
    return reinterpret_cast<T *>(static_cast<unsigned char *>(ws) + byte_off);
}

int32_t *prog(void *ws, int64_t word_off) { return static_cast<int32_t *>(ws) + word_off; }

bool aligned16(const void *p) { return ((uintptr_t)p & 15u) == 0; }

cudaError_t put(void *dst, const void *src, size_t bytes, cudaStream_t s)
{
    if (!bytes) return cudaSuccess;
    return cudaMemcpyAsync(dst, src, bytes, cudaMemcpyHostToDevice, s);
}

cudaError_t get(void *dst, const void *src, size_t bytes)
{
    if (!bytes || !dst) return cudaSuccess;
    return cudaMemcpy(dst, src, bytes, cudaMemcpyDeviceToHost);
}

// The device planner's transition t -> t+1, all launches on `s`.
cudaError_t plan_on_device(cm_shuffle *S, void *ws, cudaStream_t s, int32_t *totals_host)
{
    const int32_t n = S->n;
    const int64_t q = S->q, sz = S->s, ns = (int64_t)n * sz;
    const DevLayout D = device_layout(n, q, sz);
    const int cur = S->dev_cur, nxt = cur ^ 1;
    const int64_t t1 = S->t + 1;
    const int64_t nm = D.nm;
    int32_t *owner1 = ptr<int32_t>(ws, D.owner[nxt]);
    uint64_t *cached0 = ptr<uint64_t>(ws, D.cached[cur]), *next = ptr<uint64_t>(ws, D.cached[nxt]);
    int32_t *slot_of = ptr<int32_t>(ws, D.slot_of);
    int32_t *slot_row = prog(ws, D.prog.fill_row);
    int32_t *totals = ptr<int32_t>(ws, D.totals);
    const LookBack lb{ptr<uint64_t>(ws, D.flags), D.flags_bytes / 8, totals + kCtr,
                      totals + T_ERR, &S->sort_epoch};
    SortBufs sb{ptr<uint64_t>(ws, D.kA), ptr<uint64_t>(ws, D.kB), ptr<int32_t>(ws, D.vA),
                ptr<int32_t>(ws, D.vB), totals + kGhist, lb};
    int32_t *counts = ptr<int32_t>(ws, D.counts), *wcount = ptr<int32_t>(ws, D.wcount);
    int32_t *ell = ptr<int32_t>(ws, D.ell);
    int32_t *dx = ptr<int32_t>(ws, D.dx);
    int32_t *phist = ptr<int32_t>(ws, D.sel), *pstart = ptr<int32_t>(ws, D.pstart);
    int32_t *chist = phist + ((int64_t)1 << D.pbits);
    cudaError_t e;
#define CK(x)                                      \
    do {                                           \
        if ((e = (x)) != cudaSuccess) return e;    \
    } while (0)
#define LAUNCHED() CK(cudaGetLastError())

    {
        const ZeroList z{{totals, counts, wcount, ell, dx, phist},
                         {kTotalsWords, nm * n + 1, n + 1, nm + 1, q + 1, D.sel_words},
                         6};
        zero_many_kernel<<<grid_for(D.sel_words + q), 256, 0, s>>>(z);
        LAUNCHED();
    }

    // partition: owner = rank in (key, row) order / (q/n), by selection
    part_hist_kernel<<<grid_for(q), 256, 0, s>>>(q, S->partition_seed, t1, D.pbits, phist);
    LAUNCHED();
    CK(scan_exclusive(lb, phist, pstart, (int64_t)1 << D.pbits, totals + T_DUMMY, s));
    part_owner_kernel<<<grid_for(q), 256, 0, s>>>(q, S->partition_seed, t1, D.pbits, S->per,
                                                  phist, pstart, owner1, sb.vA, totals + kListP);
    LAUNCHED();
    part_rank_kernel<<<64, 256, 0, s>>>(q, S->partition_seed, t1, D.pbits, S->per,
                                                 pstart, sb.vA, totals + kListP, owner1);
    LAUNCHED();

    // missing rows, their sets and the counters
    uint64_t *rmask = ptr<uint64_t>(ws, D.rmask);
    const int local = nm * n <= 8192 ? (int)(nm * n) : 0;   // 32 KB of shared counters
    need_kernel<<<grid_for(q), 256, sizeof(int32_t) * local, s>>>(
        q, n, owner1, cached0, rmask, next, counts, wcount, local);
    LAUNCHED();
    uint64_t *ko;
    int32_t *vo;
    // missing rows in row order, keyed by worker
    CK(scan_fused(lb, MissingRow{owner1, cached0}, MissingToKeys{owner1, sb.kA, sb.vA}, nullptr,
                  q, totals + T_R, s));

    // received order: (worker, row)
    int32_t *recv_row = ptr<int32_t>(ws, D.recv_row), *recv_ptr = ptr<int32_t>(ws, D.recv_ptr);
    CK(radix_sort(sb, totals + T_R, q, 0, 8, 0, s, &ko, &vo));
    CK(scan_exclusive(lb, wcount, recv_ptr, n + 1, totals + T_DUMMY, s));

    // message order: (I, worker, row); the sort's output (B) is stored as the
    // received rows and keyed into A
    if (vo == sb.vA) return cudaErrorInvalidValue;   // one pass: the result is in B
    mask_keys_kernel<<<grid_for(q), 256, 0, s>>>(totals + T_R, vo, recv_row, rmask, sb.kA, sb.vA);
    LAUNCHED();
    CK(radix_sort(sb, totals + T_R, q, 0, (n + 7) / 8 * 8, 1, s, &ko, &vo));
    const int32_t *P = vo;
    int32_t *runstart = ptr<int32_t>(ws, D.runstart), *msgbase = ptr<int32_t>(ws, D.msgbase);
    CK(scan_exclusive(lb, counts, runstart, nm * n + 1, totals + T_DUMMY, s));
    ell_kernel<<<grid_for(nm), 256, 0, s>>>(nm, n, counts, ell, totals + T_SETS);
    LAUNCHED();
    CK(scan_exclusive(lb, ell, msgbase, nm + 1, totals + T_C, s));
    int32_t *earr = ptr<int32_t>(ws, D.earr);
    uint64_t *msg_set = ptr<uint64_t>(ws, D.msg_set);
    msgrow_kernel<<<grid_for(q + 1), 256, 0, s>>>(q, nm, n, msgbase, totals + T_C, counts, earr,
                                                  msg_set);
    LAUNCHED();
    int32_t *enc_ptr = prog(ws, D.prog.enc_ptr), *enc_src = prog(ws, D.prog.enc_src);
    int32_t *dec_msg = prog(ws, D.prog.dec_msg), *dec_dst = prog(ws, D.prog.dec_dst);
    int32_t *dec_ptr = prog(ws, D.prog.dec_ptr), *dec_slot = prog(ws, D.prog.dec_slot);
    int32_t *com_dst = prog(ws, D.prog.com_dst);
    int32_t *msg_worker = ptr<int32_t>(ws, D.msg_worker);
    CK(scan_exclusive(lb, earr, enc_ptr, q + 1, totals + T_DUMMY, s));
    entries_kernel<<<grid_for(q), 256, 0, s>>>(totals + T_R, n, P, recv_row, owner1, rmask,
                                               runstart, msgbase, counts, enc_ptr, enc_src,
                                               msg_worker, dec_msg, dec_dst, dx);
    LAUNCHED();

    // decoding: the slots each received row subtracts (old slot tables)
    CK(scan_exclusive(lb, dx, dec_ptr, q + 1, totals + T_X, s));
    decslot_kernel<<<grid_for(q), 256, 0, s>>>(totals + T_R, q, sz, msg_worker, dec_msg, enc_ptr,
                                               enc_src, dec_ptr, slot_of, dec_slot,
                                               totals + T_ERR);
    LAUNCHED();

    // cache update rule: the s - q/n candidates of smallest (key, row) of
    // every worker kept, by selection
    int32_t *cw = ptr<int32_t>(ws, D.cw), *cr = ptr<int32_t>(ws, D.cr);
    uint64_t *ckey = ptr<uint64_t>(ws, D.ckey);
    cand_hist_kernel<<<grid_for(q), 256, 0, s>>>(q, n, t1, S->cache_seed, owner1, cached0, chist);
    LAUNCHED();
    cand_threshold_kernel<<<n, 1024, 0, s>>>(chist, sz - S->per, totals + kThr, totals + kNeed);
    LAUNCHED();
    cand_classify_kernel<<<grid_for(q), 256, 0, s>>>(q, n, t1, S->cache_seed, owner1, cached0,
                                                     totals + kThr, next, cw, cr, ckey,
                                                     totals + kListC);
    LAUNCHED();
    cand_rank_kernel<<<64, 256, 0, s>>>(totals + kListC, cw, cr, ckey, totals + kNeed,
                                                 reinterpret_cast<unsigned long long *>(next));
    LAUNCHED();

    // commit: dropped slots of each worker take its received rows in order
    int32_t *evrank = ptr<int32_t>(ws, D.evrank);
    CK(scan_fused(lb, DroppedSlot{ns, sz, slot_row, next}, NoEpilogue{}, evrank, ns + 1,
                  totals + T_DUMMY, s));
    commit_kernel<<<grid_for(ns), 256, 0, s>>>(ns, sz, q, evrank, recv_ptr, recv_row,
                                               com_dst, slot_row, slot_of, totals + T_ERR);
    check_kernel<<<1, 32, 0, s>>>(n, sz, evrank, recv_ptr, totals + T_ERR);
    LAUNCHED();
    CK(cudaMemcpyAsync(totals_host, totals, sizeof(int32_t) * T_COUNT, cudaMemcpyDeviceToHost, s));
    CK(cudaStreamSynchronize(s));
#undef CK
#undef LAUNCHED
    return cudaSuccess;
}

}  // namespace

cm_status shuffle_device_plan(const cm_shuffle *S, int32_t *msg_ptr, int32_t *msg_src,
                              int32_t *msg_worker, uint64_t *msg_set)
{
    const DevLayout D = device_layout(S->n, S->q, S->s);
    void *ws = S->device_ws;
    cudaError_t e = get(msg_ptr, prog(ws, D.prog.enc_ptr), 4 * (S->n_coded + 1));
    if (e == cudaSuccess) e = get(msg_src, prog(ws, D.prog.enc_src), 4 * S->n_recv);
    if (e == cudaSuccess) e = get(msg_worker, ptr<int32_t>(ws, D.msg_worker), 4 * S->n_recv);
    if (e == cudaSuccess) e = get(msg_set, ptr<uint64_t>(ws, D.msg_set), 8 * S->n_coded);
    return e == cudaSuccess ? CM_OK : CM_ECUDA;
}

cm_status shuffle_device_received(const cm_shuffle *S, int32_t *recv_ptr, int32_t *recv_row)
{
    const DevLayout D = device_layout(S->n, S->q, S->s);
    void *ws = S->device_ws;
    cudaError_t e = get(recv_ptr, ptr<int32_t>(ws, D.recv_ptr), 4 * (S->n + 1));
    if (e == cudaSuccess) e = get(recv_row, ptr<int32_t>(ws, D.recv_row), 4 * S->n_recv);
    return e == cudaSuccess ? CM_OK : CM_ECUDA;
}

cm_status shuffle_device_caches(const cm_shuffle *S, int32_t *owner, int32_t *slot_row)
{
    const DevLayout D = device_layout(S->n, S->q, S->s);
    void *ws = S->device_ws;
    cudaError_t e = get(owner, ptr<int32_t>(ws, D.owner[S->dev_cur]), 4 * S->q);
    if (e == cudaSuccess)
        e = get(slot_row, prog(ws, D.prog.fill_row), 4 * (int64_t)S->n * S->s);
    return e == cudaSuccess ? CM_OK : CM_ECUDA;
}

extern "C" {

size_t cm_shuffle_device_workspace_bytes(const cm_shuffle *S)
{
    if (!S || S->n > kMaxDeviceN) return 0;
    return (size_t)device_layout(S->n, S->q, S->s).bytes;
}

cm_status cm_shuffle_device_init(cm_shuffle *S, void *ws, size_t bytes, cm_stream_t stream)
{
    if (!S || !ws || !aligned16(ws) || S->device_ws || S->n > kMaxDeviceN) return CM_EINVAL;
    const DevLayout D = device_layout(S->n, S->q, S->s);
    if (bytes < (size_t)D.bytes) return CM_EINVAL;
    cudaStream_t s = (cudaStream_t)stream;
    const int64_t q = S->q;
    cudaError_t e = put(ptr<int32_t>(ws, D.owner[0]), S->owner.data(), 4 * q, s);
    if (e == cudaSuccess) e = put(ptr<uint64_t>(ws, D.cached[0]), S->cached.data(), 8 * q, s);
    if (e == cudaSuccess)
        e = put(ptr<int32_t>(ws, D.slot_of), S->slot_of.data(), 4 * (int64_t)S->n * q, s);
    if (e == cudaSuccess)
        e = put(prog(ws, D.prog.fill_row), S->slot_row.data(), 4 * S->slot_row.size(), s);
    // radix tile flags (tagged by S->sort_epoch) and the counters
    if (e == cudaSuccess)
        e = cudaMemsetAsync(ptr<unsigned char>(ws, D.flags), 0, D.flags_bytes, s);
    if (e == cudaSuccess) e = cudaMemsetAsync(ptr<int32_t>(ws, D.totals), 0, 4 * kTotalsWords, s);
    if (e == cudaSuccess && S->planned) {   // the current transition's programs and tables
        e = put(prog(ws, D.prog.enc_ptr), S->enc_ptr.data(), 4 * S->enc_ptr.size(), s);
        if (e == cudaSuccess) e = put(prog(ws, D.prog.enc_src), S->enc_src.data(), 4 * S->enc_src.size(), s);
        if (e == cudaSuccess) e = put(prog(ws, D.prog.dec_msg), S->dec_msg.data(), 4 * S->dec_msg.size(), s);
        if (e == cudaSuccess) e = put(prog(ws, D.prog.dec_ptr), S->dec_ptr.data(), 4 * S->dec_ptr.size(), s);
        if (e == cudaSuccess) e = put(prog(ws, D.prog.dec_slot), S->dec_slot.data(), 4 * S->dec_slot.size(), s);
        if (e == cudaSuccess) e = put(prog(ws, D.prog.dec_dst), S->dec_dst.data(), 4 * S->dec_dst.size(), s);
        if (e == cudaSuccess) e = put(prog(ws, D.prog.com_dst), S->com_dst.data(), 4 * S->com_dst.size(), s);
        if (e == cudaSuccess) e = put(ptr<int32_t>(ws, D.msg_worker), S->msg_worker.data(), 4 * S->msg_worker.size(), s);
        if (e == cudaSuccess) e = put(ptr<uint64_t>(ws, D.msg_set), S->msg_set.data(), 8 * S->msg_set.size(), s);
        if (e == cudaSuccess) e = put(ptr<int32_t>(ws, D.recv_row), S->recv_row.data(), 4 * S->recv_row.size(), s);
        if (e == cudaSuccess) e = put(ptr<int32_t>(ws, D.recv_ptr), S->recv_ptr.data(), 4 * S->recv_ptr.size(), s);
    }
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return CM_ECUDA;
    S->device_ws = ws;
    S->dev_cur = 0;
    S->sort_epoch = 0;
    S->uploaded_ws = ws;
    S->uploaded_t = S->t;
    return CM_OK;
}

cm_status cm_shuffle_device_next(cm_shuffle *S, void *ws, size_t bytes, cm_shuffle_stats *stats,
                                 cm_stream_t stream)
{
    if (!S || !ws || S->device_ws != ws) return CM_EINVAL;
    const DevLayout D = device_layout(S->n, S->q, S->s);
    if (bytes < (size_t)D.bytes) return CM_EINVAL;
    int32_t totals[T_COUNT] = {0};
    if (plan_on_device(S, ws, (cudaStream_t)stream, totals) != cudaSuccess) return CM_ECUDA;
    if (totals[T_ERR]) return CM_EINVAL;   // an internal inconsistency (not reachable)
    S->t += 1;
    S->dev_cur ^= 1;
    S->n_recv = totals[T_R];
    S->n_coded = totals[T_C];
    S->n_sub = totals[T_X];
    S->message_sets = totals[T_SETS];
    S->planned = true;
    S->uploaded_ws = ws;
    S->uploaded_t = S->t;
    if (stats) {
        stats->iteration = S->t;
        stats->message_sets = S->message_sets;
        stats->coded_rows = S->n_coded;
        stats->uncoded_rows = S->n_recv;
        stats->subtractions = S->n_sub;
    }
    return CM_OK;
}

}  // extern "C"
