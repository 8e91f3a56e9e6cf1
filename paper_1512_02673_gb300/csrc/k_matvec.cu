// K2: the n worker products of coded mat-(multi-)vec (Sec. III-A protocol).
//
// Yt[j L + r][v] = sum_c A~_j[r][c] X[c][v] for every worker j < n, block row
// r < L and vector v < b <= 8.  Worker j < k reads its block in place from A
// (rows past m are virtual zeros); worker j >= k reads the parity buffer.
//
// Mapping.  A persistent grid (SMs x one resident CTA of 8 warps; 6 for
// single-round b = 1 launches).  Work unit = R consecutive block rows of one
// worker, owned by one warp; unit u
// belongs to the (u % nw)-th computed worker, so consecutive warps stream
// different workers and all workers progress together, as the n workers of
// the protocol do.  Normally all n workers are computed; when the survivors
// are known beforehand only those k are (the others' rows stay unwritten).
//
// Data movement.  The unit's rows stream through a per-warp ring of ST
// shared-memory slots of one 128-column step each, filled by 2-D TMA boxes of
// two steps (R rows x 256 columns, 1 KB contiguous per row) issued by the
// warp's lane 0.  Slots are guarded in groups of GS (2; 4 for the 12-slot
// ring of 4-row units and the 8-slot ring of the 6-warp CTAs): the boxes of
// steps (GS i, ..., GS i + GS - 1)
// complete on one mbarrier, so ST steps are in flight per warp without any
// per-lane copy work and the wait, the refill and the ring bookkeeping come
// once per GS steps.  Lane 0 refills a slot after
// a __syncwarp that follows every lane's reads of it: the warp barrier orders
// those reads before the copy is issued, and the slot is only ever written by
// TMA, so there is no generic-proxy write for a proxy fence to publish (one
// per step cost 3 % of the bandwidth at b = 8).  The tensor maps zero-fill
// whatever lies outside A or the parity buffer: the appended zero rows past m
// and the ragged column tail cost nothing.  Each coded element is read from
// HBM exactly once.  X is staged per chunk of columns by cp.async (double
// buffered, one CTA barrier per chunk) in a [vector][column] layout, so a
// lane's 4 columns of one vector are one conflict-free 128-bit load.
//
// Arithmetic.  Packed fp32x2 FMAs: accumulator pair (r, v) sums the even
// columns in its low half and the odd columns in its high half, so the pair
// (A[r][c], A[r][c+1]) from the ring multiplies (X[c][v], X[c+1][v]) from the
// X layout with no repacking.
//
// Precision.  After F steps (each half holds 2F terms) the halves are added
// and a transposing butterfly over the 32 lanes (each level sends half of the
// values, so V values cost V - V/32 shuffles) leaves every lane with complete
// fp32 partials over 128 F columns, which are added into fp64 accumulators.
// Results are fp64: decoding multiplies worker results by the entries of
// G_S^-1, so an fp32 rounding of them would be amplified.
//
// Waits.  The only spin is the mbarrier wait on a TMA step; it gives up after
// about 2 s, writes CM_ETIMEOUT to the status word and stops the warp's work
// (the CTA barriers stay matched), so a lost copy cannot hang the GPU.
#include "cm_internal.cuh"
#include "tma.cuh"

namespace {


template <int BP, int XF = 4096>
struct XCfg {
    // columns per staged X chunk (XF floats of X per buffer)
    static constexpr int CX = XF / BP;
    // floats between the [vector] rows of the smem layout: the 4-float pad
    // makes the staging stores of 32 consecutive (column, vector) elements hit
    // 32 distinct banks.
    static constexpr int GS = CX + 4;
    static constexpr int FLOATS = BP * GS;
};

template <int BP, int R, int ST, int W, int XF>
struct Smem {
    static constexpr int SLOT_FLOATS = R * 128;
    static constexpr int RING_BYTES = W * ST * SLOT_FLOATS * 4;
    static constexpr int X_BYTES = 2 * XCfg<BP, XF>::FLOATS * 4;
    static constexpr int BAR_BYTES = W * ST * 8;
    static constexpr int TOTAL = 1024 + RING_BYTES + X_BYTES + BAR_BYTES;   // + alignment slack
};

struct MatvecArgs {
    const float *X;
    double *Yt;
    int32_t *status;
    int64_t m, d, L;
    int32_t n, k, b;
    int32_t fast16;        // X chunks may be staged with 16-byte copies (b == 1)
    int64_t groups;        // total work units
    int32_t nw;            // workers computed: all n, or only the k survivors
    int8_t wmap[CM_MAX_N]; // computed worker slot -> worker index
};

// Column segments (matvec_kernel<..., SEGS = true>): CTA c sums the
// 128-column steps [s seg_steps, (s + 1) seg_steps) of every unit,
// s = c % nseg, into the partial results Yt + s part_stride; the CTAs of one
// segment share its units.  The instances without segments never read it.
struct SegArgs {
    int32_t nseg;
    int32_t seg_steps;
    int64_t part_stride;
};

__device__ __forceinline__ void cp_async16(float *dst, const float *src, int bytes)
{
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(cm_smem_u32(dst)),
                 "l"(src), "r"(bytes));
}

__device__ __forceinline__ void cp_async4(float *dst, const float *src, int bytes)
{
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;\n" ::"r"(cm_smem_u32(dst)),
                 "l"(src), "r"(bytes));
}

__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n"); }
__device__ __forceinline__ void cp_async_wait_all()
{
    asm volatile("cp.async.wait_group 0;\n" ::: "memory");
}

// Stage columns [c0, c0 + CX) of X into smem buffer xs as xs[v * GS + col]
// (zero past d and for padded vectors v >= b).
template <int BP, int XF, int kThreads>
__device__ __forceinline__ void stage_x(const MatvecArgs &a, float *xs, int64_t c0)
{
    using C = XCfg<BP, XF>;
    const int tid = threadIdx.x;
    const float *X = a.X;
    if (BP == 1 && a.fast16) {
        for (int u = tid; u < C::CX / 4; u += kThreads) {
            const int64_t col = c0 + 4 * u;
            const int64_t left = a.d - col;
            const int bytes = left >= 4 ? 16 : (left > 0 ? (int)left * 4 : 0);
            cp_async16(xs + 4 * u, bytes ? X + col : X, bytes);
        }
    } else if (kThreads % BP == 0) {
        // thread tid always stages vector v = tid % BP, columns tid / BP +
        // (kThreads / BP) i: pointers step, no per-element index arithmetic
        constexpr int CS = kThreads / BP;   // columns per sweep
        const int v = tid % BP;
        int col = tid / BP;
        float *dst = xs + v * C::GS + col;
        const float *src = X + (c0 + col) * a.b + v;
        const bool vin = v < a.b;
        const int64_t left = a.d - c0;      // columns of X from c0 on
#pragma unroll 4
        for (; col < C::CX; col += CS, dst += CS, src += (int64_t)CS * a.b) {
            const bool in = vin && col < left;
            cp_async4(dst, in ? src : X, in ? 4 : 0);
        }
    } else {
        for (int e = tid; e < C::CX * BP; e += kThreads) {
            const int col = e / BP, v = e % BP;
            const int64_t gc = c0 + col;
            const bool in = gc < a.d && v < a.b;
            cp_async4(xs + v * C::GS + col, in ? X + gc * a.b + v : X, in ? 4 : 0);
        }
    }
    cp_async_commit();
}

// Transposing butterfly: V fp32 values per lane -> max(1, V/32) complete sums
// per lane (see the header comment), added into acc64.
template <int V>
__device__ __forceinline__ void flush(float (&t)[V], double (&acc64)[V >= 32 ? V / 32 : 1],
                                      int lane)
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
}

// Add the halves of every packed pair, then flush.
template <int V>
__device__ __forceinline__ void flush_pairs(float2 (&acc)[V],
                                            double (&acc64)[V >= 32 ? V / 32 : 1], int lane)
{
    float t[V];
#pragma unroll
    for (int i = 0; i < V; ++i) {
        t[i] = acc[i].x + acc[i].y;
        acc[i] = make_float2(0.f, 0.f);
    }
    flush<V>(t, acc64, lane);
}

// Work unit g -> worker j, first block row rr0, and the TMA source of its
// rows: (map, row coordinate) in A or in the parity buffer.
struct Unit {
    int j;
    int64_t rr0;
    bool parity;
    int32_t y;
};

__device__ __forceinline__ Unit unit_of(const MatvecArgs &a, int64_t g, int R)
{
    Unit u;
    u.j = a.wmap[g % a.nw];
    u.rr0 = (g / a.nw) * R;
    u.parity = u.j >= a.k;
    u.y = (int32_t)(u.parity ? (int64_t)(u.j - a.k) * a.L + u.rr0 : (int64_t)u.j * a.L + u.rr0);
    return u;
}

// Lets a programmatic dependent launch (the decode of these products) start:
// its CTAs form their decode plan on SMs this grid leaves free, then wait
// for this grid to complete before they read any result.
__device__ __forceinline__ void griddep_launch_dependents()
{
    asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory");
}

template <int BP, int R, int ST, int F, int kWarps, int XF, bool SEGS>
__global__ void __launch_bounds__(kWarps * 32, 1)
matvec_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmP,
              const MatvecArgs a, const SegArgs sg)
{
    constexpr int kThreads = kWarps * 32;
    using C = XCfg<BP, XF>;
    using S = Smem<BP, R, ST, kWarps, XF>;
    static_assert(S::TOTAL <= 232448, "shared memory per CTA");
    constexpr int V = R * BP;
    constexpr int NH = V >= 32 ? V / 32 : 1;
    constexpr int IPC = C::CX / 128;   // steps per X chunk (a power of two)
    static_assert((IPC & (IPC - 1)) == 0, "steps per chunk");
    constexpr uint32_t STEP_BYTES = R * 128 * 4;
    extern __shared__ __align__(16) unsigned char smem_raw[];
    unsigned char *base = smem_raw + ((1024 - (cm_smem_u32(smem_raw) & 1023)) & 1023);
    float *rings = reinterpret_cast<float *>(base);
    float *xs = reinterpret_cast<float *>(base + S::RING_BYTES);
    uint64_t *bars = reinterpret_cast<uint64_t *>(base + S::RING_BYTES + S::X_BYTES);

    // slots per barrier group: 4 with the 12-slot ring, else 2 (3 groups of 2
    // for 6 slots; groups of 3 would leave two)
    constexpr int GS = ST % 4 == 0 && ST >= 8 ? 4 : 2;
    static_assert(ST % GS == 0 && IPC % GS == 0, "ring slots are guarded in groups");
    constexpr int NG = ST / GS;   // barrier groups per warp
    // A group's steps arrive in TMA boxes of R rows x 256 columns (two steps,
    // 1 KB contiguous per row): step u of a group sits in box u / 2 at column
    // offset 128 (u % 2), its rows 256 floats apart.  Against boxes of one
    // step (512 B per row) the DRAM sees twice the bytes per row access.
    constexpr int BOX_FLOATS = 2 * S::SLOT_FLOATS;
    const int lane = threadIdx.x & 31;
    const int warp = threadIdx.x >> 5;
    float *ring = rings + warp * (ST * S::SLOT_FLOATS);
    uint64_t *bar = bars + warp * NG;
    if (threadIdx.x < kWarps * NG) cm_mbar_init(&bars[threadIdx.x], 1);
    cm_fence_mbar_init();
    __syncthreads();

    // this CTA's column segment (SEGS): the first step, the steps, the
    // partial results; the CTAs of one segment share its units
    const int seg = SEGS ? (int)(blockIdx.x % sg.nseg) : 0;
    const int64_t total_warps = (int64_t)(SEGS ? gridDim.x / sg.nseg : gridDim.x) * kWarps;
    const int64_t gw = (int64_t)(SEGS ? blockIdx.x / sg.nseg : blockIdx.x) * kWarps + warp;
    const int rounds = (int)((a.groups + total_warps - 1) / total_warps);
    const int all_steps = (int)((a.d + 127) / 128);
    const int s0 = SEGS ? seg * sg.seg_steps : 0;
    const int steps = SEGS ? (all_steps - s0 < sg.seg_steps ? all_steps - s0 : sg.seg_steps)
                           : all_steps;
    const int64_t col0 = (int64_t)s0 * 128;
    const int nchunks = SEGS ? (steps * 128 + C::CX - 1) / C::CX
                             : (int)((a.d + C::CX - 1) / C::CX);
    double *const Yt = SEGS ? a.Yt + (int64_t)seg * sg.part_stride : a.Yt;
    // rounds in which this warp has a unit (a prefix: unit index grows with round)
    const int64_t my_rounds = gw < a.groups ? (a.groups - 1 - gw) / total_warps + 1 : 0;
    // A unit's steps go in groups of GS (the last one shorter when GS does
    // not divide the count); a group fills GS ring slots and completes on one
    // mbarrier.  Groups start at multiples of GS and chunks hold a multiple of
    // GS steps, so no group spans two X chunks.
    const int pairs_per_unit = (steps + GS - 1) / GS;
    const int64_t my_pairs = my_rounds * pairs_per_unit;

    // ---- producer state (lane 0): next group to load ----
    int64_t p_idx = 0;   // groups issued
    int p_g = 0, p_s = 0, p_round = 0;
    Unit pu = unit_of(a, gw, R);
    auto produce = [&]() {   // lane 0 only; loads the next group into ring group p_g
        const int nb = steps - p_s < GS ? steps - p_s : GS;
        // a box always lands whole (its columns past d read as zero; in a
        // column segment an odd last step reads, and ignores, the next one)
        if constexpr (GS == 2) {
            cm_mbar_arrive_expect_tx(&bar[p_g], 2 * STEP_BYTES);
            cm_tma_load_2d(ring + GS * p_g * S::SLOT_FLOATS, pu.parity ? &tmP : &tmA,
                           SEGS ? (int32_t)(col0 + 128 * p_s) : 128 * p_s, pu.y, &bar[p_g]);
        } else {
            const int nbox = (nb + 1) / 2;
            cm_mbar_arrive_expect_tx(&bar[p_g], nbox * 2 * STEP_BYTES);
            for (int u = 0; u < nbox; ++u)
                cm_tma_load_2d(ring + GS * p_g * S::SLOT_FLOATS + u * BOX_FLOATS,
                               pu.parity ? &tmP : &tmA,
                               SEGS ? (int32_t)(col0 + 128 * (p_s + 2 * u)) : 128 * (p_s + 2 * u),
                               pu.y, &bar[p_g]);
        }
        ++p_idx;
        p_g = p_g + 1 == NG ? 0 : p_g + 1;
        p_s += nb;
        if (p_s == steps) {
            p_s = 0;
            ++p_round;
            pu = unit_of(a, (int64_t)p_round * total_warps + gw, R);
        }
    };
    if (lane == 0)
        while (p_idx < my_pairs && p_idx < NG) produce();

    stage_x<BP, XF, kThreads>(a, xs, col0);
    griddep_launch_dependents();

    // ---- consumer ----
    int xbuf = 0;             // X buffer of the current chunk
    int64_t c_idx = 0;        // groups of this warp consumed so far
    int grp = 0;              // ring group of group c_idx
    uint32_t phase = 0;       // mbarrier phase parity of that group's current use
    bool failed = false;
    float2 acc[V];            // (even-column, odd-column) partial pairs
    double acc64[NH];
    // one 128-column step: the 4 columns of this lane, R rows, BP vectors
    auto step = [&](const float *ab, const float *xb) {
        float2 x01[BP], x23[BP];
#pragma unroll
        for (int v = 0; v < BP; ++v) {
            const float4 xv = *reinterpret_cast<const float4 *>(xb + v * C::GS);
            x01[v] = make_float2(xv.x, xv.y);
            x23[v] = make_float2(xv.z, xv.w);
        }
        // rows in groups of RH: all even-pair FMAs of the group, then all
        // odd-pair ones, so two updates of an accumulator sit RH * BP
        // instructions apart
        constexpr int RH = R >= 4 ? 4 : R;
#pragma unroll
        for (int r0 = 0; r0 < R; r0 += RH) {
            float4 av[RH];
#pragma unroll
            for (int r = 0; r < RH; ++r)
                av[r] = *reinterpret_cast<const float4 *>(ab + (r0 + r) * 256);
#pragma unroll
            for (int r = 0; r < RH; ++r)
#pragma unroll
                for (int v = 0; v < BP; ++v)
                    acc[(r0 + r) * BP + v] = __ffma2_rn(make_float2(av[r].x, av[r].y), x01[v],
                                                        acc[(r0 + r) * BP + v]);
#pragma unroll
            for (int r = 0; r < RH; ++r)
#pragma unroll
                for (int v = 0; v < BP; ++v)
                    acc[(r0 + r) * BP + v] = __ffma2_rn(make_float2(av[r].z, av[r].w), x23[v],
                                                        acc[(r0 + r) * BP + v]);
        }
    };
#pragma unroll 1
    for (int round = 0; round < rounds; ++round) {
        const bool has = round < my_rounds;
        const Unit cu = unit_of(a, (int64_t)round * total_warps + gw, R);
#pragma unroll
        for (int i = 0; i < V; ++i) acc[i] = make_float2(0.f, 0.f);
#pragma unroll
        for (int i = 0; i < NH; ++i) acc64[i] = 0.0;
        int fl = 0;
#pragma unroll 1
        for (int ch = 0; ch < nchunks; ++ch) {
            cp_async_wait_all();
            __syncthreads();   // X chunk visible; every warp is done with the other buffer
            if (ch + 1 < nchunks || round + 1 < rounds)
                stage_x<BP, XF, kThreads>(a, xs + (xbuf ^ 1) * C::FLOATS,
                                      col0 + (ch + 1 < nchunks ? (int64_t)(ch + 1) * C::CX : 0));
            const int ns = steps - ch * IPC < IPC ? steps - ch * IPC : IPC;
            if (has && !failed) {
                const float *xchunk = xs + xbuf * C::FLOATS + 4 * lane;
#pragma unroll
                for (int cs = 0; cs < IPC; cs += GS) {
                    if (cs >= ns || failed) break;
                    if (!cm_mbar_wait(&bar[grp], phase)) {
                        failed = true;
                        if (lane == 0 && a.status) *a.status = CM_ETIMEOUT;
                        break;
                    }
                    const float *ab = ring + GS * grp * S::SLOT_FLOATS + 4 * lane;
#pragma unroll
                    for (int u = 0; u < GS; ++u)
                        if (cs + u < ns)
                            step(ab + (u >> 1) * BOX_FLOATS + (u & 1) * 128,
                                 xchunk + (cs + u) * 128);
                    ++c_idx;
                    if (++grp == NG) {
                        grp = 0;
                        phase ^= 1u;
                    }
                    __syncwarp();   // every lane is done reading the group
                    if (lane == 0 && p_idx < my_pairs) produce();   // refill it
                    fl += ns - cs < GS ? ns - cs : GS;
                    if (fl >= F) {
                        flush_pairs<V>(acc, acc64, lane);
                        fl = 0;
                    }
                }
            }
            xbuf ^= 1;
        }
        if (has && !failed) {
            if (fl) flush_pairs<V>(acc, acc64, lane);
            const int64_t obase = (int64_t)cu.j * a.L + cu.rr0;
            if constexpr (V >= 32) {
#pragma unroll
                for (int i = 0; i < NH; ++i) {
                    const int vi = lane * NH + i;
                    const int r = vi / BP, v = vi % BP;
                    if (v < a.b && cu.rr0 + r < a.L) Yt[(obase + r) * a.b + v] = acc64[i];
                }
            } else {
                constexpr int SHIFT = V == 1 ? 5 : V == 2 ? 4 : V == 4 ? 3 : V == 8 ? 2 : 1;
                if ((lane & ((1 << SHIFT) - 1)) == 0) {
                    const int vi = lane >> SHIFT;
                    const int r = vi / BP, v = vi % BP;
                    if (v < a.b && cu.rr0 + r < a.L) Yt[(obase + r) * a.b + v] = acc64[0];
                }
            }
        }
    }
    cp_async_wait_all();
    // After a time-out, wait (bounded) for the copies still in flight before
    // the CTA's shared memory is released.
    if (failed && lane == 0) {
        for (int64_t i = c_idx; i < p_idx; ++i) {
            cm_mbar_wait(&bar[grp], phase, 100000000ull);
            if (++grp == NG) {
                grp = 0;
                phase ^= 1u;
            }
        }
    }
}

template <int BP, int R, int ST, int F, int kWarps, int XF = 4096>
cudaError_t launch_bp(MatvecArgs a, const SegArgs &sg, const float *A, int64_t lda,
                      const float *par, int64_t ldp, cudaStream_t s)
{
    constexpr int kThreads = kWarps * 32;
    using S = Smem<BP, R, ST, kWarps, XF>;
    auto kern = sg.nseg > 1 ? matvec_kernel<BP, R, ST, F, kWarps, XF, true>
                            : matvec_kernel<BP, R, ST, F, kWarps, XF, false>;
    CUtensorMap tmA, tmP;   // boxes of two steps: R rows x 256 columns
    if (!cm_make_tmap_2d(&tmA, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, A, a.d, a.m, lda * 4, 256, R,
                         CU_TENSOR_MAP_SWIZZLE_NONE) ||
        !cm_make_tmap_2d(&tmP, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, par, a.d,
                         (a.n - a.k) * a.L, ldp * 4, 256, R, CU_TENSOR_MAP_SWIZZLE_NONE))
        return cudaErrorInvalidValue;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         S::TOTAL);
    if (e != cudaSuccess) return e;
    a.groups = (a.L + R - 1) / R * a.nw;
    // CTAs per segment: as many as the SMs allow, no more than the units need
    const int64_t need = (a.groups + kWarps - 1) / kWarps;
    int64_t per_seg = (cm_sm_count() > 0 ? cm_sm_count() : 1) / sg.nseg;
    if (per_seg < 1) per_seg = 1;
    if (per_seg > need) per_seg = need;
    const int64_t grid = per_seg * sg.nseg;
    kern<<<(unsigned)grid, kThreads, S::TOTAL, s>>>(tmA, tmP, a, sg);
    return cudaGetLastError();
}

}  // namespace

// Rows per work unit for b = 1.  The persistent grid takes units in rounds of
// `warps`; a partly filled last round leaves the other warps idle, which on a
// small problem (a few rounds) costs up to a fifth of the time.  4-row units
// (with a ring twice as deep, the same bytes in flight) fill the rounds more
// evenly but add a round's X staging and ring start-up each time; measured on
// this part, they pay off when they fill the rounds at least 2 points better.
// (2-row units ran at two thirds of the bandwidth: per-step costs dominate.)
int matvec_rows_per_unit(int64_t L, int nw, int64_t warps)
{
    auto fill = [&](int R) {
        const int64_t units = (L + R - 1) / R * nw;
        const int64_t rounds = (units + warps - 1) / warps;
        return (double)units / (double)(rounds * warps);
    };
    return fill(4) >= fill(8) + 0.02 ? 4 : 8;
}

namespace {

MatvecArgs matvec_args(const CodeParams &cp, const float *X, int b, double *Yt, int32_t *status,
                       uint32_t only)
{
    MatvecArgs a = {};
    // workers to compute: all n, or the first k set bits of `only`
    a.nw = 0;
    for (int j = 0; j < cp.n; ++j)
        if (!only || (((only >> j) & 1u) && a.nw < cp.k)) a.wmap[a.nw++] = (int8_t)j;
    a.X = X;
    a.Yt = Yt;
    a.status = status;
    a.m = cp.m;
    a.d = cp.d;
    a.L = cp.L;
    a.n = cp.n;
    a.k = cp.k;
    a.b = b;
    a.groups = 0;
    a.fast16 = b == 1 && ((uintptr_t)X & 15u) == 0;
    return a;
}

// Rows per unit of the launch for these arguments (the kernel instance).
int unit_rows(const MatvecArgs &a)
{
    const int sms = cm_sm_count() > 0 ? cm_sm_count() : 1;
    if (a.b == 1) return matvec_rows_per_unit(a.L, a.nw, (int64_t)sms * 8);
    return 8;
}

cudaError_t dispatch(const MatvecArgs &a, const SegArgs &sg, const float *A, int64_t lda,
                     const float *par, int64_t ldp, cudaStream_t s)
{
    if (a.b == 1) {
        if (unit_rows(a) == 4) return launch_bp<1, 4, 12, 16, 8>(a, sg, A, lda, par, ldp, s);
        // Units that fit one round of 6-warp CTAs (e.g. the 800 units of
        // (25,23) at 5750 x 5750): 8-slot rings guarded in groups of four,
        // so each row is read 2 KB at a time (two adjacent boxes) with 32 KB
        // in flight per warp, in the same shared memory; 0.65 -> 0.74 of the
        // copy peak there.  With more rounds the 8-warp form stays ahead.
        const int sms = cm_sm_count() > 0 ? cm_sm_count() : 1;
        if (sg.nseg == 1 && (a.L + 7) / 8 * a.nw <= (int64_t)sms * 6)
            return launch_bp<1, 8, 8, 16, 6>(a, sg, A, lda, par, ldp, s);
        return launch_bp<1, 8, 6, 16, 8>(a, sg, A, lda, par, ldp, s);
    }
    if (a.b <= 4) return launch_bp<4, 8, 6, 16, 8>(a, sg, A, lda, par, ldp, s);
    return launch_bp<8, 8, 6, 64, 8>(a, sg, A, lda, par, ldp, s);
}

}  // namespace

// Column segments for the products of a decode that adds partial results.
// The persistent grid runs the units in rounds over its warps; when there are
// few units (few rows per worker, long rows: the 400 x 10000 regression of
// Sec. III-F has 70 units of 8 rows for 1216 warps), splitting every unit's
// columns into 2, 4 or 8 segments, each done by its own share of the CTAs,
// puts more warps to work.  The time is modelled as rounds x (T0 + steps of
// the segment), T0 = 5 steps the fixed cost of a unit (ring start-up, flush,
// result stores), fitted on this part: (25,23) at 5750 x 5750 ran equally
// fast whole (1 round of 45 steps) and in 4 segments (3 rounds of 12).  Taken
// only when the model drops by a tenth or more and every segment keeps at
// least 8 steps of 128 columns.
int matvec_segments(const CodeParams &cp, int b, uint32_t only)
{
    const MatvecArgs a = matvec_args(cp, nullptr, b, nullptr, nullptr, only);
    const int R = unit_rows(a);
    const int64_t units = (a.L + R - 1) / R * a.nw;
    const int sms = cm_sm_count() > 0 ? cm_sm_count() : 1;
    const int steps = (int)((cp.d + 127) / 128);
    auto cost = [&](int ns) {
        const int64_t warps = (int64_t)(sms / ns) * 8;
        const int seg_steps = (steps + ns - 1) / ns;
        return (double)((units + warps - 1) / warps) * (5.0 + seg_steps);
    };
    int best = 1;
    double best_c = cost(1);
    // whole rows in one round of 6-warp CTAs (see dispatch) ran 0.88 of the
    // time of the 8-warp form on (25,23) at 5750 x 5750
    if (b == 1 && R == 8 && units <= (int64_t)sms * 6) best_c *= 0.88;
    for (int ns = 2; ns <= 8; ns *= 2) {
        if (sms % ns || (steps + ns - 1) / ns < 8) break;
        const double c = cost(ns);
        if (c <= 0.9 * best_c) {
            best = ns;
            best_c = c;
        }
    }
    return best;
}

cudaError_t launch_matvec_split(const CodeParams &cp, const float *A, int64_t lda,
                                const float *par, int64_t ldp, const float *X, int b, double *Yt,
                                int32_t *status, uint32_t only, int nseg, int64_t part_stride,
                                cudaStream_t s)
{
    SegArgs sg;
    sg.nseg = nseg > 1 ? nseg : 1;
    sg.seg_steps = (int32_t)(((cp.d + 127) / 128 + sg.nseg - 1) / sg.nseg);
    sg.part_stride = part_stride;
    return dispatch(matvec_args(cp, X, b, Yt, status, only), sg, A, lda, par, ldp, s);
}

cudaError_t launch_matvec(const CodeParams &cp, const float *A, int64_t lda, const float *par,
                          int64_t ldp, const float *X, int b, double *Yt, int32_t *status,
                          uint32_t only, cudaStream_t s)
{
    const SegArgs whole = {1, (int32_t)((cp.d + 127) / 128), 0};
    return dispatch(matvec_args(cp, X, b, Yt, status, only), whole, A, lda, par, ldp, s);
}
