// K2: the n worker products of coded mat-(multi-)vec (Sec. III-A protocol).
//
// Yt[j L + r][v] = sum_c A~_j[r][c] X[c][v] for every worker j < n, block row
// r < L and vector v < b <= 8.  Worker j < k reads its block in place from A
// (rows past m are virtual zeros: never read, result 0); worker j >= k reads
// the parity buffer.
//
// Mapping.  A persistent grid (SMs x one resident CTA of 8 warps).  Work
// unit = a group of R consecutive block rows of one worker, owned by one warp;
// unit u belongs to worker u % n, so consecutive warps stream different
// workers and all n workers progress together, as the n workers of the
// protocol do.  The coded rows stream through a per-warp shared-memory ring
// of ST steps (R rows x 128 columns) filled by cp.async: lane l copies, and
// later reads back, only its own 16 bytes [4l, 4l+4) of every row, so a step
// is complete after cp.async.wait_group alone (no barrier, no spin) and
// ST-1 steps stay in flight per warp.  Each coded element is read from HBM
// exactly once.  The CTA's warps sweep the columns in lockstep through chunks
// of X staged by cp.async (double buffered, one barrier per chunk) in a
// [vector][column] layout, so a lane's 4 columns of one vector are one
// conflict-free 128-bit load.
//
// Arithmetic.  Packed fp32x2 FMAs: accumulator pair (r, v) sums the even
// columns in its low half and the odd columns in its high half, so the pair
// (A[r][c], A[r][c+1]) straight from the ring multiplies (X[c][v], X[c+1][v])
// straight from the X layout, with no repacking.
//
// Precision.  After F steps (each half holds 2F terms) the halves are added
// and a transposing butterfly over the 32 lanes (each level sends half of the
// values, so V values cost V - V/32 shuffles) leaves every lane with complete
// fp32 partials over 128 F columns, which are added into fp64 accumulators.
// Results are fp64: decoding multiplies worker results by the entries of
// G_S^-1, so an fp32 rounding of them would be amplified.
#include "cm_internal.cuh"

namespace {

constexpr int kWarps = 8;
constexpr int kThreads = kWarps * 32;

template <int BP>
struct XCfg {
    // columns per staged X chunk (16 KB of X per buffer)
    static constexpr int CX = 4096 / BP;
    // floats between the [vector] rows of the smem layout: the 4-float pad
    // makes the staging stores of 32 consecutive (column, vector) elements hit
    // 32 distinct banks.
    static constexpr int GS = CX + 4;
    static constexpr int FLOATS = BP * GS;
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

// Stage columns [c0, c0 + CX) of X into smem buffer xs as xs[v * GS + col]
// (zero past d and for padded vectors v >= b).
template <int BP>
__device__ __forceinline__ void stage_x(const MatvecArgs &a, float *xs, int64_t c0)
{
    using C = XCfg<BP>;
    const int tid = threadIdx.x;
    const float *X = a.X;
    if (BP == 1 && a.fast16) {
        for (int u = tid; u < C::CX / 4; u += kThreads) {
            const int64_t col = c0 + 4 * u;
            const int64_t left = a.d - col;
            const int bytes = left >= 4 ? 16 : (left > 0 ? (int)left * 4 : 0);
            cp_async16(xs + 4 * u, bytes ? X + col : a.A, bytes);
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

__device__ __forceinline__ uint64_t pack2(float lo, float hi)
{
    uint64_t r;
    asm("mov.b64 %0, {%1, %2};\n" : "=l"(r) : "f"(lo), "f"(hi));
    return r;
}

// d += a * b on both fp32 halves (round to nearest, no flush to zero)
__device__ __forceinline__ void fma2(uint64_t &d, uint64_t a, uint64_t b)
{
    asm("fma.rn.f32x2 %0, %1, %2, %0;\n" : "+l"(d) : "l"(a), "l"(b));
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

// cp.async.wait_group with a run-time count (the instruction takes an immediate)
__device__ __forceinline__ void cp_async_wait_upto(int n)
{
    switch (n) {
    case 0: asm volatile("cp.async.wait_group 0;\n" ::: "memory"); break;
    case 1: asm volatile("cp.async.wait_group 1;\n" ::: "memory"); break;
    case 2: asm volatile("cp.async.wait_group 2;\n" ::: "memory"); break;
    case 3: asm volatile("cp.async.wait_group 3;\n" ::: "memory"); break;
    case 4: asm volatile("cp.async.wait_group 4;\n" ::: "memory"); break;
    case 5: asm volatile("cp.async.wait_group 5;\n" ::: "memory"); break;
    case 6: asm volatile("cp.async.wait_group 6;\n" ::: "memory"); break;
    default: asm volatile("cp.async.wait_group 7;\n" ::: "memory"); break;
    }
}

// Rows of work unit g: R row pointers (NULL = virtual zero row or past L).
template <int R>
__device__ __forceinline__ void unit_rows(const MatvecArgs &a, int64_t g, const float *(&rowp)[R],
                                          int &j, int64_t &rr0)
{
    const bool has = g < a.groups;
    j = has ? (int)(g % a.n) : 0;
    rr0 = has ? (g / a.n) * R : 0;
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
}

// A streams into a per-warp ring of ST steps (R rows x 128 columns each) by
// cp.async: lane l copies, and later reads back, only its own 16 bytes of
// every row, so completion needs just cp.async.wait_group (no barrier, no
// spin).  ST-1 steps are in flight per warp while the warp computes.
template <int V>
__device__ __forceinline__ void flush_pairs(uint64_t (&acc)[V],
                                            double (&acc64)[V >= 32 ? V / 32 : 1], int lane)
{
    float t[V];
#pragma unroll
    for (int i = 0; i < V; ++i) {
        float lo, hi;
        asm("mov.b64 {%0, %1}, %2;\n" : "=f"(lo), "=f"(hi) : "l"(acc[i]));
        t[i] = lo + hi;
        acc[i] = 0ull;
    }
    flush<V>(t, acc64, lane);
}

template <int BP, int R, int ST, int F>
__global__ void __launch_bounds__(kThreads, 1)
matvec_kernel(const MatvecArgs a)
{
    using C = XCfg<BP>;
    constexpr int V = R * BP;
    constexpr int NH = V >= 32 ? V / 32 : 1;
    constexpr int IPC = C::CX / 128;   // steps per X chunk
    static_assert(ST >= 2 && ST <= 8, "ring depth");
    static_assert(IPC >= ST - 1, "an X chunk must outlast the ring");
    extern __shared__ __align__(16) float smem[];
    const int lane = threadIdx.x & 31;
    const int warp = threadIdx.x >> 5;
    float *ring = smem + 2 * C::FLOATS + warp * (ST * R * 128);
    const int64_t total_warps = (int64_t)gridDim.x * kWarps;
    const int64_t gw = (int64_t)blockIdx.x * kWarps + warp;
    const int64_t rounds = (a.groups + total_warps - 1) / total_warps;
    const int64_t steps = (a.d + 127) / 128;
    const int64_t nchunks = (a.d + C::CX - 1) / C::CX;
    const int64_t total = rounds * steps;

    // ---- issue side: A(step) for the flat step sequence of this warp ----
    int64_t is_round = 0, is_s = 0;
    int is_slot = 0;
    const float *irow[R];
    {
        int jj;
        int64_t r0;
        unit_rows<R>(a, gw, irow, jj, r0);
    }
    int since_x = 0;   // cp.async groups committed after the newest X group
    auto issue = [&]() {
        if (is_round < rounds) {
            const int64_t col = 128 * is_s + 4 * lane;
            const int64_t left = a.d - col;
            const int full = left >= 4 ? 16 : (left > 0 ? (int)left * 4 : 0);
            float *dst = ring + is_slot * (R * 128) + 4 * lane;
#pragma unroll
            for (int r = 0; r < R; ++r) {
                const int bytes = irow[r] ? full : 0;
                cp_async16(dst + r * 128, bytes ? irow[r] + col : a.A, bytes);
            }
            if (++is_s == steps) {
                is_s = 0;
                ++is_round;
                int jj;
                int64_t r0;
                unit_rows<R>(a, is_round * total_warps + gw, irow, jj, r0);
            }
            is_slot = is_slot + 1 == ST ? 0 : is_slot + 1;
        }
        cp_async_commit();
        ++since_x;
    };

    stage_x<BP>(a, smem, 0);
#pragma unroll 1
    for (int i = 0; i < ST - 1; ++i) issue();

    // ---- compute side ----
    int64_t xseq = 0;        // X chunks consumed so far (buffer = xseq & 1)
    int64_t round = 0, s = 0;
    int slot = 0, fl = 0, j = 0;
    int64_t rr0 = 0;
    bool has = false;
    uint64_t acc[V];   // packed (even-column, odd-column) partial pairs
    double acc64[NH];
#pragma unroll 1
    for (int64_t f = 0; f < total; ++f) {
        if (s == 0) {
            const int64_t g = round * total_warps + gw;
            has = g < a.groups;
            const float *dummy[R];
            unit_rows<R>(a, g, dummy, j, rr0);
#pragma unroll
            for (int i = 0; i < V; ++i) acc[i] = 0ull;
#pragma unroll
            for (int i = 0; i < NH; ++i) acc64[i] = 0.0;
            fl = 0;
        }
        issue();   // A(f + ST - 1)
        const int64_t cs = s % IPC;
        if (cs == 0) {
            // chunk start: X(this chunk) and A(f) complete, then make X visible
            cp_async_wait_upto(since_x < ST - 1 ? since_x : ST - 1);
            __syncthreads();   // also: every warp is done with the other X buffer
            const int64_t ch = s / IPC;
            const bool more = ch + 1 < nchunks || round + 1 < rounds;
            if (more) {
                stage_x<BP>(a, smem + ((xseq + 1) & 1) * C::FLOATS,
                            ch + 1 < nchunks ? (ch + 1) * C::CX : 0);
                since_x = 0;
            }
        } else {
            cp_async_wait_upto(ST - 1);
        }
        if (has) {
            const float *xb = smem + (xseq & 1) * C::FLOATS + 4 * ((int)cs * 32 + lane);
            const float *ab = ring + slot * (R * 128) + 4 * lane;
            uint64_t x01[BP], x23[BP];
#pragma unroll
            for (int v = 0; v < BP; ++v) {
                const float4 xv = *reinterpret_cast<const float4 *>(xb + v * C::GS);
                x01[v] = pack2(xv.x, xv.y);
                x23[v] = pack2(xv.z, xv.w);
            }
#pragma unroll
            for (int r = 0; r < R; ++r) {
                const float4 av = *reinterpret_cast<const float4 *>(ab + r * 128);
                const uint64_t a01 = pack2(av.x, av.y), a23 = pack2(av.z, av.w);
#pragma unroll
                for (int v = 0; v < BP; ++v) {
                    fma2(acc[r * BP + v], a01, x01[v]);
                    fma2(acc[r * BP + v], a23, x23[v]);
                }
            }
            if (++fl == F) {
                flush_pairs<V>(acc, acc64, lane);
                fl = 0;
            }
        }
        slot = slot + 1 == ST ? 0 : slot + 1;
        const bool chunk_end = cs == IPC - 1 || s == steps - 1;
        if (chunk_end) ++xseq;
        if (s == steps - 1) {
            if (has) {
                if (fl) flush_pairs<V>(acc, acc64, lane);
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
            s = 0;
            ++round;
        } else {
            ++s;
        }
    }
    cp_async_wait_all();
}

template <int BP, int R, int ST, int F>
cudaError_t launch_bp(MatvecArgs a, cudaStream_t s)
{
    using C = XCfg<BP>;
    auto kern = matvec_kernel<BP, R, ST, F>;
    const int smem = (2 * C::FLOATS + kWarps * ST * R * 128) * 4;
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
        return launch_bp<1, 4, 8, 16>(a, s);
    }
    a.fast16 = 0;
    if (b <= 4) return launch_bp<4, 8, 5, 16>(a, s);
    return launch_bp<8, 8, 5, 16>(a, s);
}
