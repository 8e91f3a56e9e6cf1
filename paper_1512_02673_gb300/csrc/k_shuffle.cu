// K7: coded shuffling data plane (Sec. IV) -- row programs on HBM-resident
// rows.
//
// One kernel runs every step of a transition: output row o is
//     out[dst(o)] = in0[first(o)]  (op)  in1[term(o, 0)]  (op)  in1[term(o, 1)] ...
// with (op) = + (encode: Alg. 1's sum of zero-padded blocks), - (decode by
// subtraction) or bitwise xor (both, exact), and with no terms it is a row
// copy (commit into the freed cache slots, and the initial cache fill).  A
// zero-padded block contributes no term, so a padded row of Alg. 1 costs
// nothing.  Rows are r 4-byte words with 16-byte aligned starts.
//
// Mapping: persistent grid (the resident blocks of every SM); row o goes to
// warp o mod W, which batches the program words of its next 32 rows.  Each
// lane owns U float4 columns
// of a column block of 32 U float4 and issues the U loads of a term together,
// so every warp keeps U x 512 bytes per term in flight.  Term row indices are
// read once per row by the lanes and broadcast by shuffles.  Every data byte
// is read once per use and written once (HBM bound; no reuse to stage).
#include <cuda_runtime.h>
#include <stdint.h>

#include "cm_internal.cuh"
#include "shuffle_internal.h"

namespace {

enum RowOp { ROW_SUM = 0, ROW_DIFF = 1, ROW_XOR = 2 };

struct RowProgram {
    int64_t rows;           // output rows
    const int32_t *ptr;     // rows + 1 term offsets (null: no terms)
    const int32_t *term;    // rows of in1
    const int32_t *first;   // row of in0 for each output row (null: row o)
    const int32_t *dst;     // output row for each output row (null: row o)
};

constexpr int kThreads = 256;
constexpr int kU = 2;

// Terms are read once (streaming); the first operand may be shared by
// adjacent output rows (a message row decoded by every worker of I).
__device__ __forceinline__ float4 ld4_once(const float *p)
{
    return __ldcs(reinterpret_cast<const float4 *>(p));
}

__device__ __forceinline__ float4 ld4_shared(const float *p)
{
    return __ldg(reinterpret_cast<const float4 *>(p));
}

template <int OP>
__device__ __forceinline__ float combine(float a, float b)
{
    if constexpr (OP == ROW_SUM) return a + b;
    else if constexpr (OP == ROW_DIFF) return a - b;
    else return __uint_as_float(__float_as_uint(a) ^ __float_as_uint(b));
}

template <int OP>
__device__ __forceinline__ void combine4(float4 &a, const float4 &b)
{
    a.x = combine<OP>(a.x, b.x);
    a.y = combine<OP>(a.y, b.y);
    a.z = combine<OP>(a.z, b.z);
    a.w = combine<OP>(a.w, b.w);
}

// Loads the U float4 columns of column block c0 of `row` that this lane owns
// (zeros past the row end).
__device__ __forceinline__ void load_block(float4 (&v)[kU], const float *row, int64_t c0,
                                           int64_t r4, int lane, bool shared)
{
#pragma unroll
    for (int u = 0; u < kU; ++u) {
        const int64_t c = c0 + u * 32 + lane;
        if (c < r4) v[u] = shared ? ld4_shared(row + 4 * c) : ld4_once(row + 4 * c);
        else v[u] = make_float4(0.f, 0.f, 0.f, 0.f);
    }
}

template <int OP, bool FIRST>
__global__ void __launch_bounds__(kThreads) row_program_kernel(
    RowProgram p, const float *__restrict__ in0, int64_t ld0, const float *__restrict__ in1,
    int64_t ld1, float *__restrict__ out, int64_t ldo, int64_t r)
{
    constexpr unsigned kAll = 0xffffffffu;
    const int lane = threadIdx.x & 31;
    const int64_t warp = (((int64_t)blockIdx.x * kThreads) + threadIdx.x) >> 5;
    const int64_t nwarps = ((int64_t)gridDim.x * kThreads) >> 5;
    const int64_t r4 = r >> 2;
    // Rows are dealt to warps round-robin (row o to warp o mod W), so that
    // neighbouring rows, which touch neighbouring messages and data rows,
    // are in flight together.  A warp reads the program words of its next 32
    // rows in one go (lane l: its l-th next row) and broadcasts them by
    // shuffles, and fetches the term indices of the next row while the
    // current row's data moves: a row waits on one memory latency, not three.
    for (int64_t base = warp; base < p.rows; base += 32 * nwarps) {
        const int64_t mine = base + lane * nwarps;
        const bool valid = mine < p.rows;
        const int cnt = (int)min((int64_t)32, (p.rows - base + nwarps - 1) / nwarps);
        int beg_l = 0, end_l = 0, first_l = 0, dst_l = 0;
        if (valid) {
            if (p.ptr) {
                beg_l = p.ptr[mine];
                end_l = p.ptr[mine + 1];
            }
            if (FIRST) first_l = p.first ? p.first[mine] : (int)mine;
            dst_l = p.dst ? p.dst[mine] : (int)mine;
        }
        // terms of row j: lane l holds terms l and 32 + l (nt <= 64)
        int next0 = 0, next1 = 0;
        if (p.ptr) {
            const int b = __shfl_sync(kAll, beg_l, 0);
            const int nj = __shfl_sync(kAll, end_l, 0) - b;
            next0 = lane < nj ? p.term[b + lane] : 0;
            next1 = 32 + lane < nj ? p.term[b + 32 + lane] : 0;
        }
        for (int j = 0; j < cnt; ++j) {
            const int t0 = next0, t1 = next1;
            const int beg = __shfl_sync(kAll, beg_l, j);
            const int nt = __shfl_sync(kAll, end_l, j) - beg;
            // j + 1 < cnt <= 32 keeps the shuffle source in range; lanes of an
            // out-of-range j + 1 read nothing (their nj comes out <= 0)
            const int jn = j + 1 < cnt ? j + 1 : j;
            const int bn = __shfl_sync(kAll, beg_l, jn);
            const int nn = j + 1 < cnt ? __shfl_sync(kAll, end_l, jn) - bn : 0;
            if (p.ptr) {
                next0 = lane < nn ? p.term[bn + lane] : 0;
                next1 = 32 + lane < nn ? p.term[bn + 32 + lane] : 0;
            }
            const float *src0 = nullptr;
            if constexpr (FIRST) src0 = in0 + (int64_t)__shfl_sync(kAll, first_l, j) * ld0;
            float *dst = out + (int64_t)__shfl_sync(kAll, dst_l, j) * ldo;
            const int e_begin = FIRST ? 0 : 1;
            for (int64_t c0 = 0; c0 < r4; c0 += 32 * kU) {
                float4 acc[kU];
                if constexpr (FIRST) {
                    load_block(acc, src0, c0, r4, lane, true);
                } else {   // a sum without in0 starts from its first term
                    const int row = __shfl_sync(kAll, t0, 0);
                    load_block(acc, in1 + (int64_t)row * ld1, c0, r4, lane, false);
                }
#pragma unroll 4
                for (int e = e_begin; e < nt; ++e) {
                    const int row = __shfl_sync(kAll, e < 32 ? t0 : t1, e & 31);
                    float4 v[kU];
                    load_block(v, in1 + (int64_t)row * ld1, c0, r4, lane, false);
#pragma unroll
                    for (int u = 0; u < kU; ++u) combine4<OP>(acc[u], v[u]);
                }
#pragma unroll
                for (int u = 0; u < kU; ++u) {
                    const int64_t c = c0 + u * 32 + lane;
                    if (c < r4) __stcs(reinterpret_cast<float4 *>(dst + 4 * c), acc[u]);
                }
            }
            // ragged tail of r % 4 words
            for (int64_t c = 4 * r4 + lane; c < r; c += 32) {
                float a = FIRST ? src0[c] : in1[(int64_t)p.term[beg] * ld1 + c];
                for (int e = e_begin; e < nt; ++e)
                    a = combine<OP>(a, in1[(int64_t)p.term[beg + e] * ld1 + c]);
                dst[c] = a;
            }
        }
    }
}

template <int OP, bool FIRST>
cudaError_t run(const RowProgram &p, const float *in0, int64_t ld0, const float *in1,
                int64_t ld1, float *out, int64_t ldo, int64_t r, cudaStream_t s)
{
    if (p.rows <= 0 || r <= 0) return cudaSuccess;
    const int64_t warps_per_block = kThreads / 32;
    const int64_t want = (p.rows + warps_per_block - 1) / warps_per_block;
    static int per_sm = 0;   // resident blocks per SM (one query per instantiation)
    if (per_sm == 0) {
        int b = 0;
        if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&b, row_program_kernel<OP, FIRST>,
                                                          kThreads, 0) != cudaSuccess || b < 1)
            b = 1;
        per_sm = b;
    }
    const int64_t cap = (int64_t)cm_sm_count() * per_sm;
    const int grid = (int)(want < cap ? want : cap);
    row_program_kernel<OP, FIRST><<<grid, kThreads, 0, s>>>(p, in0, ld0, in1, ld1, out, ldo, r);
    return cudaGetLastError();
}

bool aligned16(const void *p) { return ((uintptr_t)p & 15u) == 0; }

bool rows_ok(const void *p, int64_t ld, int64_t r)
{
    return p && aligned16(p) && ld >= r && ld % 4 == 0;
}

cm_status from_cuda(cudaError_t e) { return e == cudaSuccess ? CM_OK : CM_ECUDA; }

// The programs of the current transition in `ws`, or false if `ws` does not
// hold them (never uploaded, or uploaded before the last cm_shuffle_next).
bool current(const cm_shuffle *S, const void *ws) { return ws && S->uploaded_ws == ws && S->uploaded_t == S->t; }

const int32_t *at(const void *ws, int64_t words) { return static_cast<const int32_t *>(ws) + words; }

}  // namespace

extern "C" {

size_t cm_shuffle_workspace_bytes(const cm_shuffle *S)
{
    if (!S) return 0;
    return (size_t)shuffle_layout(S->n, S->q, S->s).total * sizeof(int32_t);
}

cm_status cm_shuffle_upload(cm_shuffle *S, void *ws, size_t bytes, cm_stream_t stream)
{
    if (!S || !ws || !aligned16(ws) || bytes < cm_shuffle_workspace_bytes(S)) return CM_EINVAL;
    if (S->device_ws) return CM_EINVAL;   // the device planner keeps its programs in place
    const ShuffleLayout L = shuffle_layout(S->n, S->q, S->s);
    cudaStream_t st = (cudaStream_t)stream;
    int32_t *w = static_cast<int32_t *>(ws);
    auto put = [&](int64_t off, const std::vector<int32_t> &v) -> cudaError_t {
        if (v.empty()) return cudaSuccess;
        return cudaMemcpyAsync(w + off, v.data(), v.size() * sizeof(int32_t),
                               cudaMemcpyHostToDevice, st);
    };
    cudaError_t e = put(L.fill_row, S->slot_row);
    if (e == cudaSuccess && S->planned) {
        if (e == cudaSuccess) e = put(L.enc_ptr, S->enc_ptr);
        if (e == cudaSuccess) e = put(L.enc_src, S->enc_src);
        if (e == cudaSuccess) e = put(L.dec_msg, S->dec_msg);
        if (e == cudaSuccess) e = put(L.dec_ptr, S->dec_ptr);
        if (e == cudaSuccess) e = put(L.dec_slot, S->dec_slot);
        if (e == cudaSuccess) e = put(L.dec_dst, S->dec_dst);
        if (e == cudaSuccess) e = put(L.com_dst, S->com_dst);
    }
    if (e != cudaSuccess) return CM_ECUDA;
    S->uploaded_ws = ws;
    S->uploaded_t = S->t;
    return CM_OK;
}

cm_status cm_shuffle_fill(const cm_shuffle *S, const void *ws, const void *A, int64_t lda,
                          int64_t r, void *caches, int64_t ldc, cm_stream_t stream)
{
    if (!S || !current(S, ws) || r < 1 || !rows_ok(A, lda, r) || !rows_ok(caches, ldc, r))
        return CM_EINVAL;
    const ShuffleLayout L = shuffle_layout(S->n, S->q, S->s);
    RowProgram p{(int64_t)S->n * S->s, nullptr, nullptr, at(ws, L.fill_row), nullptr};
    return from_cuda(run<ROW_SUM, true>(p, (const float *)A, lda, nullptr, 0, (float *)caches,
                                        ldc, r, (cudaStream_t)stream));
}

cm_status cm_shuffle_encode(const cm_shuffle *S, const void *ws, cm_shuffle_op op,
                            const void *A, int64_t lda, int64_t r, void *M, int64_t ldm,
                            cm_stream_t stream)
{
    if (!S || !S->planned || !current(S, ws) || r < 1 || !rows_ok(A, lda, r) ||
        !rows_ok(M, ldm, r))
        return CM_EINVAL;
    const ShuffleLayout L = shuffle_layout(S->n, S->q, S->s);
    RowProgram p{S->n_coded, at(ws, L.enc_ptr), at(ws, L.enc_src), nullptr,
                 nullptr};
    cudaStream_t st = (cudaStream_t)stream;
    if (op == CM_SHUFFLE_ADD)
        return from_cuda(run<ROW_SUM, false>(p, nullptr, 0, (const float *)A, lda, (float *)M,
                                             ldm, r, st));
    if (op == CM_SHUFFLE_XOR)
        return from_cuda(run<ROW_XOR, false>(p, nullptr, 0, (const float *)A, lda, (float *)M,
                                             ldm, r, st));
    return CM_EINVAL;
}

cm_status cm_shuffle_decode(const cm_shuffle *S, const void *ws, cm_shuffle_op op,
                            const void *M, int64_t ldm, const void *caches, int64_t ldc,
                            int64_t r, void *Rx, int64_t ldr, cm_stream_t stream)
{
    if (!S || !S->planned || !current(S, ws) || r < 1 || !rows_ok(M, ldm, r) ||
        !rows_ok(caches, ldc, r) || !rows_ok(Rx, ldr, r))
        return CM_EINVAL;
    const ShuffleLayout L = shuffle_layout(S->n, S->q, S->s);
    RowProgram p{S->n_recv, at(ws, L.dec_ptr), at(ws, L.dec_slot),
                 at(ws, L.dec_msg), at(ws, L.dec_dst)};
    cudaStream_t st = (cudaStream_t)stream;
    if (op == CM_SHUFFLE_ADD)
        return from_cuda(run<ROW_DIFF, true>(p, (const float *)M, ldm, (const float *)caches,
                                             ldc, (float *)Rx, ldr, r, st));
    if (op == CM_SHUFFLE_XOR)
        return from_cuda(run<ROW_XOR, true>(p, (const float *)M, ldm, (const float *)caches,
                                            ldc, (float *)Rx, ldr, r, st));
    return CM_EINVAL;
}

cm_status cm_shuffle_commit(const cm_shuffle *S, const void *ws, const void *Rx, int64_t ldr,
                            int64_t r, void *caches, int64_t ldc, cm_stream_t stream)
{
    if (!S || !S->planned || !current(S, ws) || r < 1 || !rows_ok(Rx, ldr, r) ||
        !rows_ok(caches, ldc, r))
        return CM_EINVAL;
    const ShuffleLayout L = shuffle_layout(S->n, S->q, S->s);
    RowProgram p{S->n_recv, nullptr, nullptr, nullptr, at(ws, L.com_dst)};
    return from_cuda(run<ROW_SUM, true>(p, (const float *)Rx, ldr, nullptr, 0,
                                        (float *)caches, ldc, r, (cudaStream_t)stream));
}

}  // extern "C"
