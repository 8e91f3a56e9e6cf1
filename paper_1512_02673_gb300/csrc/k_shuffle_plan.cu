// K8: the coded-shuffling planner on the device (Sec. IV).
//
// Computes, for the transition t -> t+1, exactly what the host planner
// (shuffle.cpp) computes -- the partition, Alg. 1's message plan, the
// decoding and commit programs and the cache update rule -- with the state
// (partition, cache masks, slot tables) resident in the caller's workspace,
// so that a transition needs no host work beyond reading back four counts.
// The definitions are the host planner's (see its header comment); the
// device version reaches the same order through stable sorts:
//   partition     rows sorted by (key, row): a stable LSD radix sort of the
//                 rows (ascending) on the top 24 bits of their 64-bit keys,
//                 then each run of equal top bits sorted by (key, row);
//   received      missing rows in (worker, row) order: a stable sort by
//                 worker of the rows in ascending order;
//   messages      received rows stably sorted by the set I (bit mask), i.e.
//                 (I, worker, row); row j of a worker's run in I goes to
//                 message row base(I) + j, entries ordered by worker;
//   cache update  candidates (worker, row) stably sorted on the top key bits,
//                 then by worker, runs of equal (worker, top bits) by
//                 (key, row): the first s - q/n of each worker are kept;
//   commit        dropped slots of each worker, ascending, take its received
//                 rows in order.
// Radix passes: one warp per tile of 1024 items, 8-bit digits; a tile's
// histogram by shared-memory atomics, global offsets by an exclusive scan of
// the (digit, tile) matrix, and a stable scatter that ranks equal digits
// within each 32-item step by __match_any_sync, reorders the tile by digit in
// shared memory and writes each digit's run to consecutive addresses.
// Device scans: 4096 items per 1024-thread block, block sums scanned
// recursively.
#include <cuda_runtime.h>
#include <stdint.h>

#include <algorithm>
#include <vector>

#include "cm_internal.cuh"
#include "shuffle_internal.h"

namespace {

constexpr int kTile = 1024;        // items per warp in a radix pass
constexpr int kRadixWarps = 4;     // warps (tiles) per radix block
// shared memory of one warp's scatter: its tile's keys and values in digit
// order, and three 256-entry tables (local starts, running counts, global bases)
constexpr int kScatterWarpBytes = kTile * 12 + 3 * 256 * 4;
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

// ---- exclusive scan (int32) -----------------------------------------------------------

__global__ void __launch_bounds__(kScanBlock) scan_block_kernel(const int32_t *in, int32_t *out,
                                                                int64_t count,
                                                                int32_t *block_sums)
{
    __shared__ int32_t warp_sums[32];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int64_t base = (int64_t)blockIdx.x * kScanItems + 4 * (int64_t)threadIdx.x;
    int32_t v[4], sum = 0;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        v[k] = base + k < count ? in[base + k] : 0;
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
        warp_sums[lane] = w;
    }
    __syncthreads();
    int32_t excl = x - sum + (warp ? warp_sums[warp - 1] : 0);
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        if (base + k < count) out[base + k] = excl;
        excl += v[k];
    }
    if (threadIdx.x == kScanBlock - 1 && block_sums) block_sums[blockIdx.x] = excl;
}

__global__ void __launch_bounds__(kScanBlock) scan_add_kernel(int32_t *out, int64_t count,
                                                              const int32_t *offsets)
{
    const int32_t add = offsets[blockIdx.x];
    const int64_t base = (int64_t)blockIdx.x * kScanItems + 4 * (int64_t)threadIdx.x;
#pragma unroll
    for (int k = 0; k < 4; ++k)
        if (base + k < count) out[base + k] += add;
}

// The second pass when the block sums are few: every block sums the block
// sums before its own (at most kScanDirect of them, one or a few per thread)
// instead of waiting for a scan of them in a launch of its own, then adds
// that offset; the last block also writes the total.
constexpr int64_t kScanDirect = 4 * kScanBlock;

__global__ void __launch_bounds__(kScanBlock) scan_add_direct_kernel(int32_t *out, int64_t count,
                                                                     const int32_t *block_sums,
                                                                     int32_t *total)
{
    __shared__ int32_t warp_part[32];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int32_t part = 0;
    for (int64_t i = threadIdx.x; i < (int64_t)blockIdx.x; i += kScanBlock) part += block_sums[i];
#pragma unroll
    for (int o = 16; o; o >>= 1) part += __shfl_xor_sync(0xffffffffu, part, o);
    if (lane == 0) warp_part[warp] = part;
    __syncthreads();
    int32_t add = 0;
#pragma unroll 1
    for (int w = 0; w < kScanBlock / 32; ++w) add += warp_part[w];
    const int64_t base = (int64_t)blockIdx.x * kScanItems + 4 * (int64_t)threadIdx.x;
#pragma unroll
    for (int k = 0; k < 4; ++k)
        if (base + k < count) out[base + k] += add;
    if (total && threadIdx.x == 0 && blockIdx.x == gridDim.x - 1)
        *total = add + block_sums[blockIdx.x];
}

int64_t up256(int64_t x) { return (x + 255) & ~(int64_t)255; }

// out[i] = in[0] + ... + in[i-1] for i < count (in may be out); the sum of
// all of them goes to *total (device, nullable).  `scratch` holds the block
// sums of every level (count / 4096 + 512 words per level suffice).
cudaError_t scan_exclusive(const int32_t *in, int32_t *out, int64_t count, int32_t *scratch,
                           int32_t *total, cudaStream_t s)
{
    if (count <= 0) {
        if (total) fill_i32<<<1, 32, 0, s>>>(total, 1, 0);
        return cudaGetLastError();
    }
    const int64_t nb = (count + kScanItems - 1) / kScanItems;
    if (nb == 1) {
        scan_block_kernel<<<1, kScanBlock, 0, s>>>(in, out, count, total);
        return cudaGetLastError();
    }
    scan_block_kernel<<<(unsigned)nb, kScanBlock, 0, s>>>(in, out, count, scratch);
    if (nb <= kScanDirect) {
        scan_add_direct_kernel<<<(unsigned)nb, kScanBlock, 0, s>>>(out, count, scratch, total);
        return cudaGetLastError();
    }
    cudaError_t e = scan_exclusive(scratch, scratch, nb, scratch + up256(nb), total, s);
    if (e != cudaSuccess) return e;
    scan_add_kernel<<<(unsigned)nb, kScanBlock, 0, s>>>(out, count, scratch);
    return cudaGetLastError();
}

// ---- stable LSD radix sort (64-bit keys, int32 values) ---------------------------------

__global__ void radix_hist_kernel(const uint64_t *keys, const int32_t *countp, int64_t cap,
                                  int shift, int32_t *hist, int64_t tiles)
{
    __shared__ int32_t cnt[kRadixWarps][256];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int64_t tile = (int64_t)blockIdx.x * kRadixWarps + warp;
    for (int d = lane; d < 256; d += 32) cnt[warp][d] = 0;
    __syncwarp();
    if (tile >= tiles) return;
    const int64_t count = countp ? (int64_t)*countp : cap;
    const int64_t beg = tile * kTile, end = std::min(count, beg + kTile);
#pragma unroll 8
    for (int64_t i = beg + lane; i < end; i += 32) atomicAdd(&cnt[warp][(keys[i] >> shift) & 255], 1);
    __syncwarp();
    for (int d = lane; d < 256; d += 32) hist[(int64_t)d * tiles + tile] = cnt[warp][d];
}

// One warp per tile of 32 x 32 items: (1) the tile loaded into registers
// (lane l holds items l, 32 + l, ...; all loads in flight together), its digit
// counts and their exclusive scan (local starts); (2) every item placed,
// stably, at its digit's local start plus its rank in shared memory (equal
// digits of a 32-item step ranked by lane with __match_any_sync); (3) the
// tile written out in that digit order: a run of equal digits goes to
// consecutive global positions, so the writes coalesce.
__global__ void __launch_bounds__(32 * kRadixWarps)
radix_scatter_kernel(const uint64_t *kin, const int32_t *vin, uint64_t *kout, int32_t *vout,
                     const int32_t *countp, int64_t cap, int shift, const int32_t *offsets,
                     int64_t tiles)
{
    static_assert(kTile == 32 * 32, "a tile is 32 steps of 32 items");
    extern __shared__ __align__(16) unsigned char smem[];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    unsigned char *mine = smem + warp * kScatterWarpBytes;
    uint64_t *sk = reinterpret_cast<uint64_t *>(mine);
    int32_t *sv = reinterpret_cast<int32_t *>(mine + kTile * 8);
    int32_t *start = reinterpret_cast<int32_t *>(mine + kTile * 12);
    int32_t *run = start + 256;
    int32_t *base = run + 256;
    const int64_t tile = (int64_t)blockIdx.x * kRadixWarps + warp;
    if (tile >= tiles) return;
    const int64_t count = countp ? (int64_t)*countp : cap;
    const int64_t beg = tile * kTile, end = std::min(count, beg + kTile);
    const int nt = end > beg ? (int)(end - beg) : 0;
    for (int d = lane; d < 256; d += 32) {
        run[d] = 0;
        base[d] = offsets[(int64_t)d * tiles + tile];
    }
    uint64_t k[32];
    int32_t v[32];
#pragma unroll
    for (int j = 0; j < 32; ++j) {
        const int p = 32 * j + lane;
        k[j] = p < nt ? kin[beg + p] : 0;
        v[j] = p < nt ? vin[beg + p] : 0;
    }
    __syncwarp();
#pragma unroll
    for (int j = 0; j < 32; ++j)
        if (32 * j + lane < nt) atomicAdd(&run[(k[j] >> shift) & 255], 1);
    __syncwarp();
    {   // exclusive scan of the 256 counts: 8 per lane
        int32_t c[8], sum = 0;
#pragma unroll
        for (int q = 0; q < 8; ++q) {
            c[q] = run[8 * lane + q];
            sum += c[q];
        }
        int32_t x = sum;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int32_t y = __shfl_up_sync(0xffffffffu, x, o);
            if (lane >= o) x += y;
        }
        int32_t at = x - sum;
#pragma unroll
        for (int q = 0; q < 8; ++q) {
            start[8 * lane + q] = at;
            at += c[q];
        }
    }
    __syncwarp();
    for (int d = lane; d < 256; d += 32) run[d] = 0;
    __syncwarp();
    const unsigned below = (1u << lane) - 1u;
#pragma unroll
    for (int j = 0; j < 32; ++j) {
        if (32 * j >= nt) break;   // warp-uniform
        const bool valid = 32 * j + lane < nt;
        const int d = valid ? (int)((k[j] >> shift) & 255) : 256;   // 256: not an item
        const unsigned peers = __match_any_sync(0xffffffffu, d);
        if (valid) {
            const int pos = start[d] + run[d] + __popc(peers & below);
            sk[pos] = k[j];
            sv[pos] = v[j];
        }
        __syncwarp();
        if (valid && (peers & below) == 0) run[d] += __popc(peers);
        __syncwarp();
    }
    for (int p = lane; p < nt; p += 32) {
        const uint64_t kk = sk[p];
        const int d = (int)((kk >> shift) & 255);
        const int g = base[d] + (p - start[d]);
        kout[g] = kk;
        vout[g] = sv[p];
    }
}

struct SortBufs {
    uint64_t *kA, *kB;
    int32_t *vA, *vB;
    int32_t *hist, *scan;
};

// Stable sort of items [0, count) (count = *countp, or cap if countp is null)
// by bits [lo, hi) of their keys; on return the sorted keys and values are in
// (*k_out, *v_out), one of the two buffer pairs.
cudaError_t radix_sort(const SortBufs &b, const int32_t *countp, int64_t cap, int lo, int hi,
                       cudaStream_t s, uint64_t **k_out, int32_t **v_out)
{
    const int64_t tiles = std::max<int64_t>(1, (cap + kTile - 1) / kTile);
    const unsigned blocks = (unsigned)((tiles + kRadixWarps - 1) / kRadixWarps);
    uint64_t *ki = b.kA, *ko = b.kB;
    int32_t *vi = b.vA, *vo = b.vB;
    cudaError_t ea = cudaFuncSetAttribute(radix_scatter_kernel,
                                          cudaFuncAttributeMaxDynamicSharedMemorySize,
                                          kRadixWarps * kScatterWarpBytes);
    if (ea != cudaSuccess) return ea;
    for (int shift = lo; shift < hi; shift += 8) {
        radix_hist_kernel<<<blocks, 32 * kRadixWarps, 0, s>>>(ki, countp, cap, shift, b.hist, tiles);
        cudaError_t e = scan_exclusive(b.hist, b.hist, 256 * tiles, b.scan, nullptr, s);
        if (e != cudaSuccess) return e;
        radix_scatter_kernel<<<blocks, 32 * kRadixWarps, kRadixWarps * kScatterWarpBytes, s>>>(
            ki, vi, ko, vo, countp, cap, shift, b.hist, tiles);
        std::swap(ki, ko);
        std::swap(vi, vo);
    }
    *k_out = ki;
    *v_out = vi;
    return cudaGetLastError();
}

// ---- planner kernels --------------------------------------------------------------------

__global__ void partition_keys_kernel(uint64_t *keys, int32_t *vals, int64_t q, uint64_t seed,
                                      int64_t t1)
{
    GS_LOOP(r, q)
    {
        keys[r] = mix64(seed, (uint64_t)t1 * (uint64_t)q + (uint64_t)r);
        vals[r] = (int32_t)r;
    }
}

__global__ void owner_kernel(const int32_t *order, int64_t q, int64_t per, int32_t *owner1)
{
    GS_LOOP(pos, q) owner1[order[pos]] = (int32_t)(pos / per);
}

// Per row: missing from its new owner's cache?  Its set I, its candidate
// bits for the cache refill; counts per (I, worker), per worker and per
// candidate worker.  Counters of n bins are aggregated in shared memory.
// Per row: missing from its new owner's cache?  Its set I, its candidate
// bits for the cache refill; counts per (I, worker), per worker and per
// candidate worker.  The per-worker counters are aggregated in shared memory
// per block, and so are the (I, worker) counters when their table fits
// (`local` = 2^n n entries, else 0: global atomics).
__global__ void need_kernel(int64_t q, int n, const int32_t *owner1, const uint64_t *cached0,
                            uint64_t *rmask, int32_t *needflag, int32_t *ccnt_row, uint64_t *next,
                            int32_t *counts, int32_t *wcount, int32_t *ccount, int local)
{
    extern __shared__ int32_t sl[];
    __shared__ int32_t sw[kMaxDeviceN], sc[kMaxDeviceN];
    if (threadIdx.x < kMaxDeviceN) {
        sw[threadIdx.x] = 0;
        sc[threadIdx.x] = 0;
    }
    for (int i = threadIdx.x; i < local; i += blockDim.x) sl[i] = 0;
    __syncthreads();
    GS_LOOP(r, q)
    {
        const int i = owner1[r];
        const uint64_t bit = 1ull << i, have = cached0[r];
        const int nf = (have & bit) ? 0 : 1;
        const uint64_t cand = have & ~bit;
        needflag[r] = nf;
        rmask[r] = have | bit;
        next[r] = bit;
        ccnt_row[r] = __popcll(cand);
        if (nf) {
            const int64_t slot = (int64_t)(have | bit) * n + i;
            if (local) atomicAdd(&sl[slot], 1);
            else atomicAdd(&counts[slot], 1);
            atomicAdd(&sw[i], 1);
        }
        for (uint64_t b = cand; b; b &= b - 1) atomicAdd(&sc[__ffsll((long long)b) - 1], 1);
    }
    __syncthreads();
    if (threadIdx.x < n) {
        atomicAdd(&wcount[threadIdx.x], sw[threadIdx.x]);
        atomicAdd(&ccount[threadIdx.x], sc[threadIdx.x]);
    }
    for (int i = threadIdx.x; i < local; i += blockDim.x)
        if (sl[i]) atomicAdd(&counts[i], sl[i]);
}

__global__ void compact_kernel(int64_t q, const int32_t *flag, const int32_t *idx, int32_t *items)
{
    GS_LOOP(r, q) if (flag[r]) items[idx[r]] = (int32_t)r;
}

__global__ void worker_keys_kernel(const int32_t *countp, const int32_t *items,
                                   const int32_t *owner1, uint64_t *keys, int32_t *vals)
{
    const int64_t count = *countp;
    GS_LOOP(u, count)
    {
        keys[u] = (uint64_t)owner1[items[u]];
        vals[u] = items[u];
    }
}

__global__ void copy_i32_counted(const int32_t *countp, const int32_t *src, int32_t *dst)
{
    const int64_t count = *countp;
    GS_LOOP(u, count) dst[u] = src[u];
}

__global__ void mask_keys_kernel(const int32_t *countp, const int32_t *recv_row,
                                 const uint64_t *rmask, uint64_t *keys, int32_t *vals)
{
    const int64_t count = *countp;
    GS_LOOP(v, count)
    {
        keys[v] = rmask[recv_row[v]];
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

__global__ void cand_kernel(int64_t q, int n, int64_t t1, uint64_t seed, const int32_t *owner1,
                            const uint64_t *cached0, const int32_t *cbase, int32_t *cw,
                            int32_t *cr, uint64_t *ckey, uint64_t *keys, int32_t *vals)
{
    GS_LOOP(r, q)
    {
        uint64_t b = cached0[r] & ~(1ull << owner1[r]);
        int32_t c = cbase[r];
        for (; b; b &= b - 1, ++c) {
            const int i = __ffsll((long long)b) - 1;
            cw[c] = i;
            cr[c] = (int32_t)r;
            keys[c] = mix64(seed, ((uint64_t)t1 * (uint64_t)n + (uint64_t)i) * (uint64_t)q +
                                      (uint64_t)r);
            ckey[c] = keys[c];
            vals[c] = c;
        }
    }
}

__global__ void cand_worker_keys_kernel(const int32_t *Kp, const int32_t *vals, const int32_t *cw,
                                        uint64_t *keys)
{
    const int64_t K = *Kp;
    GS_LOOP(p, K) keys[p] = (uint64_t)cw[vals[p]];
}

// After a stable sort on the top 24 bits of the keys only, items whose top
// bits tie are adjacent and in their original order; each such run (short:
// keys are uniform 64-bit values) is put in full (key, row) order by the
// thread at its start.  `grp` (nullable) adds a group that must also tie
// (the worker of a candidate); keys and rows are read through the values
// (`key_of`, `row_of`: item id -> key / row; null: the sorted key array and
// the value itself).
__global__ void fixup_runs_kernel(const int32_t *countp, int64_t cap, const uint64_t *skeys,
                                  int32_t *vals, const uint64_t *key_of, const int32_t *row_of,
                                  const int32_t *grp)
{
    const int64_t count = countp ? (int64_t)*countp : cap;
    auto key = [&](int32_t v, int64_t p) { return key_of ? key_of[v] : skeys[p]; };
    auto row = [&](int32_t v) { return row_of ? row_of[v] : v; };
    auto top = [&](int32_t v, int64_t p) {
        return ((key(v, p) >> 40) << 8) | (uint64_t)(grp ? grp[v] : 0);
    };
    GS_LOOP(p, count)
    {
        const int32_t v0 = vals[p];
        const uint64_t t0 = top(v0, p);
        if (p > 0 && top(vals[p - 1], p - 1) == t0) continue;   // not a run start
        int64_t e = p + 1;
        while (e < count && top(vals[e], e) == t0) ++e;
        if (e - p < 2) continue;
        // insertion sort of vals[p, e) by (key, row); with key_of null the
        // keys move with the values
        for (int64_t i = p + 1; i < e; ++i) {
            const int32_t vi = vals[i];
            const uint64_t ki = key_of ? key_of[vi] : skeys[i];
            const int32_t ri = row(vi);
            int64_t j = i - 1;
            while (j >= p) {
                const int32_t vj = vals[j];
                const uint64_t kj = key_of ? key_of[vj] : skeys[j];
                if (kj < ki || (kj == ki && row(vj) < ri)) break;
                vals[j + 1] = vj;
                if (!key_of) const_cast<uint64_t *>(skeys)[j + 1] = kj;
                --j;
            }
            vals[j + 1] = vi;
            if (!key_of) const_cast<uint64_t *>(skeys)[j + 1] = ki;
        }
    }
}

__global__ void kept_kernel(const int32_t *Kp, int64_t keep, const int32_t *vals,
                            const int32_t *cw, const int32_t *cr, const int32_t *cstart,
                            unsigned long long *next)
{
    const int64_t K = *Kp;
    GS_LOOP(p, K)
    {
        const int32_t c = vals[p];
        const int i = cw[c];
        if (p - cstart[i] < keep) atomicOr(&next[cr[c]], 1ull << i);
    }
}

__global__ void evflag_kernel(int64_t ns, int64_t s, const int32_t *slot_row,
                              const uint64_t *next, int32_t *evflag)
{
    GS_LOOP(g, ns)
    {
        const int i = (int)(g / s);
        evflag[g] = (next[slot_row[g]] >> i) & 1ull ? 0 : 1;
    }
}

__global__ void commit_kernel(int64_t ns, int64_t s, int64_t q, const int32_t *evflag,
                              const int32_t *evrank, const int32_t *recv_ptr,
                              const int32_t *recv_row, int32_t *com_dst, int32_t *slot_row,
                              int32_t *slot_of, int32_t *err)
{
    GS_LOOP(g, ns)
    {
        if (!evflag[g]) continue;
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
    int64_t kA, kB, vA, vB, hist, scan;
    int64_t rmask, needflag, idx, items, recv_row, wcount, recv_ptr;
    int64_t counts, runstart, ell, msgbase, earr, msg_set, msg_worker, dx;
    int64_t ccnt_row, cbase, cw, cr, ckey, ccount, cstart, evflag, evrank, totals;
    int64_t bytes;            // total
    int64_t capK, nm;
};

DevLayout device_layout(int32_t n, int64_t q, int64_t s)
{
    DevLayout D;
    D.prog = shuffle_layout(n, q, s);
    D.nm = (int64_t)1 << n;
    const int64_t ns = (int64_t)n * s;
    D.capK = std::max(q, ns);
    const int64_t tiles = std::max<int64_t>(1, (D.capK + kTile - 1) / kTile);
    const int64_t scan_max = std::max({256 * tiles, D.capK + 1, D.nm * n + 1, q + 1});
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
    D.kA = take(8 * D.capK);
    D.kB = take(8 * D.capK);
    D.vA = take(4 * D.capK);
    D.vB = take(4 * D.capK);
    D.hist = take(4 * 256 * tiles);
    D.scan = take(4 * (scan_max / kScanItems + 8 * 256 + 1024));
    D.rmask = take(8 * q);
    D.needflag = take(4 * (q + 1));
    D.idx = take(4 * (q + 1));
    D.items = take(4 * q);
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
    D.ccnt_row = take(4 * (q + 1));
    D.cbase = take(4 * (q + 1));
    D.cw = take(4 * D.capK);
    D.cr = take(4 * D.capK);
    D.ckey = take(8 * D.capK);
    D.ccount = take(4 * (n + 1));
    D.cstart = take(4 * (n + 1));
    D.evflag = take(4 * (ns + 1));
    D.evrank = take(4 * (ns + 1));
    D.totals = take(4 * T_COUNT);
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
    int32_t *scan = ptr<int32_t>(ws, D.scan);
    SortBufs sb{ptr<uint64_t>(ws, D.kA), ptr<uint64_t>(ws, D.kB), ptr<int32_t>(ws, D.vA),
                ptr<int32_t>(ws, D.vB), ptr<int32_t>(ws, D.hist), scan};
    int32_t *counts = ptr<int32_t>(ws, D.counts), *wcount = ptr<int32_t>(ws, D.wcount);
    int32_t *ccount = ptr<int32_t>(ws, D.ccount), *ell = ptr<int32_t>(ws, D.ell);
    int32_t *dx = ptr<int32_t>(ws, D.dx);
    cudaError_t e;
#define CK(x)                                      \
    do {                                           \
        if ((e = (x)) != cudaSuccess) return e;    \
    } while (0)
#define LAUNCHED() CK(cudaGetLastError())

    fill_i32<<<1, 32, 0, s>>>(totals, T_COUNT, 0);
    fill_i32<<<grid_for(nm * n + 1), 256, 0, s>>>(counts, nm * n + 1, 0);
    fill_i32<<<1, 32, 0, s>>>(wcount, n + 1, 0);
    fill_i32<<<1, 32, 0, s>>>(ccount, n + 1, 0);
    fill_i32<<<grid_for(nm + 1), 256, 0, s>>>(ell, nm + 1, 0);
    fill_i32<<<grid_for(q + 1), 256, 0, s>>>(dx, q + 1, 0);
    LAUNCHED();

    // partition: rows sorted by (key, row)
    partition_keys_kernel<<<grid_for(q), 256, 0, s>>>(sb.kA, sb.vA, q, S->partition_seed, t1);
    LAUNCHED();
    uint64_t *ko;
    int32_t *vo;
    CK(radix_sort(sb, nullptr, q, 40, 64, s, &ko, &vo));   // top 24 bits, then the ties
    fixup_runs_kernel<<<grid_for(q), 256, 0, s>>>(nullptr, q, ko, vo, nullptr, nullptr, nullptr);
    LAUNCHED();
    owner_kernel<<<grid_for(q), 256, 0, s>>>(vo, q, S->per, owner1);
    LAUNCHED();

    // missing rows, their sets, the refill candidates and the counters
    uint64_t *rmask = ptr<uint64_t>(ws, D.rmask);
    int32_t *needflag = ptr<int32_t>(ws, D.needflag), *idx = ptr<int32_t>(ws, D.idx);
    int32_t *ccnt_row = ptr<int32_t>(ws, D.ccnt_row), *cbase = ptr<int32_t>(ws, D.cbase);
    const int local = nm * n <= 8192 ? (int)(nm * n) : 0;   // 32 KB of shared counters
    need_kernel<<<grid_for(q), 256, sizeof(int32_t) * local, s>>>(
        q, n, owner1, cached0, rmask, needflag, ccnt_row, next, counts, wcount, ccount, local);
    LAUNCHED();
    CK(scan_exclusive(needflag, idx, q, scan, totals + T_R, s));
    int32_t *items = ptr<int32_t>(ws, D.items);
    compact_kernel<<<grid_for(q), 256, 0, s>>>(q, needflag, idx, items);
    LAUNCHED();

    // received order: (worker, row)
    int32_t *recv_row = ptr<int32_t>(ws, D.recv_row), *recv_ptr = ptr<int32_t>(ws, D.recv_ptr);
    worker_keys_kernel<<<grid_for(q), 256, 0, s>>>(totals + T_R, items, owner1, sb.kA, sb.vA);
    LAUNCHED();
    CK(radix_sort(sb, totals + T_R, q, 0, 8, s, &ko, &vo));
    copy_i32_counted<<<grid_for(q), 256, 0, s>>>(totals + T_R, vo, recv_row);
    LAUNCHED();
    CK(scan_exclusive(wcount, recv_ptr, n + 1, scan, totals + T_DUMMY, s));

    // message order: (I, worker, row)
    mask_keys_kernel<<<grid_for(q), 256, 0, s>>>(totals + T_R, recv_row, rmask, sb.kA, sb.vA);
    LAUNCHED();
    CK(radix_sort(sb, totals + T_R, q, 0, (n + 7) / 8 * 8, s, &ko, &vo));
    const int32_t *P = vo;
    int32_t *runstart = ptr<int32_t>(ws, D.runstart), *msgbase = ptr<int32_t>(ws, D.msgbase);
    CK(scan_exclusive(counts, runstart, nm * n + 1, scan, totals + T_DUMMY, s));
    ell_kernel<<<grid_for(nm), 256, 0, s>>>(nm, n, counts, ell, totals + T_SETS);
    LAUNCHED();
    CK(scan_exclusive(ell, msgbase, nm + 1, scan, totals + T_C, s));
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
    CK(scan_exclusive(earr, enc_ptr, q + 1, scan, totals + T_DUMMY, s));
    entries_kernel<<<grid_for(q), 256, 0, s>>>(totals + T_R, n, P, recv_row, owner1, rmask,
                                               runstart, msgbase, counts, enc_ptr, enc_src,
                                               msg_worker, dec_msg, dec_dst, dx);
    LAUNCHED();

    // decoding: the slots each received row subtracts (old slot tables)
    CK(scan_exclusive(dx, dec_ptr, q + 1, scan, totals + T_X, s));
    decslot_kernel<<<grid_for(q), 256, 0, s>>>(totals + T_R, q, sz, msg_worker, dec_msg, enc_ptr,
                                               enc_src, dec_ptr, slot_of, dec_slot,
                                               totals + T_ERR);
    LAUNCHED();

    // cache update rule: candidates by (worker, key, row); the first s - q/n kept
    CK(scan_exclusive(ccnt_row, cbase, q, scan, totals + T_K, s));
    int32_t *cw = ptr<int32_t>(ws, D.cw), *cr = ptr<int32_t>(ws, D.cr);
    uint64_t *ckey = ptr<uint64_t>(ws, D.ckey);
    cand_kernel<<<grid_for(q), 256, 0, s>>>(q, n, t1, S->cache_seed, owner1, cached0, cbase, cw,
                                            cr, ckey, sb.kA, sb.vA);
    LAUNCHED();
    // by the top 24 bits of the key, then by worker (both stable), then each
    // run of equal (worker, top bits) in full (key, row) order
    CK(radix_sort(sb, totals + T_K, D.capK, 40, 64, s, &ko, &vo));
    {
        // the sort leaves its result in A or B: move it to A for the next one
        if (vo != sb.vA) {
            copy_i32_counted<<<grid_for(D.capK), 256, 0, s>>>(totals + T_K, vo, sb.vA);
            LAUNCHED();
        }
        cand_worker_keys_kernel<<<grid_for(D.capK), 256, 0, s>>>(totals + T_K, sb.vA, cw, sb.kA);
        LAUNCHED();
    }
    CK(radix_sort(sb, totals + T_K, D.capK, 0, 8, s, &ko, &vo));
    fixup_runs_kernel<<<grid_for(D.capK), 256, 0, s>>>(totals + T_K, D.capK, ko, vo, ckey, cr,
                                                        cw);
    LAUNCHED();
    int32_t *cstart = ptr<int32_t>(ws, D.cstart);
    CK(scan_exclusive(ccount, cstart, n + 1, scan, totals + T_DUMMY, s));
    kept_kernel<<<grid_for(D.capK), 256, 0, s>>>(totals + T_K, sz - S->per, vo, cw, cr, cstart,
                                                 reinterpret_cast<unsigned long long *>(next));
    LAUNCHED();

    // commit: dropped slots of each worker take its received rows in order
    int32_t *evflag = ptr<int32_t>(ws, D.evflag), *evrank = ptr<int32_t>(ws, D.evrank);
    fill_i32<<<1, 32, 0, s>>>(evflag + ns, 1, 0);
    evflag_kernel<<<grid_for(ns), 256, 0, s>>>(ns, sz, slot_row, next, evflag);
    LAUNCHED();
    CK(scan_exclusive(evflag, evrank, ns + 1, scan, totals + T_DUMMY, s));
    commit_kernel<<<grid_for(ns), 256, 0, s>>>(ns, sz, q, evflag, evrank, recv_ptr, recv_row,
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
