// Internal declarations shared by the libcm translation units.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/cm.h"

#define CM_MAX_N 32
#define CM_MAX_P 256   // (n-k) k <= 16 * 16 for n <= 32

enum CodeKind { CODE_GENERAL = 0, CODE_REPETITION = 1 };

struct cm_code {
    int32_t n, k;
    int64_t m, d, L;
    cm_dtype dt;
    int32_t kind;        // CodeKind
    float P[CM_MAX_P];   // (n-k) x k, row-major
};

// The code as a kernel parameter (passed by value; P lands in the constant
// parameter bank, read with uniform broadcast loads).
struct CodeParams {
    int32_t n, k;
    int64_t m, d, L;
    float P[CM_MAX_P];
};

inline CodeParams code_params(const cm_code *c)
{
    CodeParams p;
    p.n = c->n;
    p.k = c->k;
    p.m = c->m;
    p.d = c->d;
    p.L = c->L;
    for (int i = 0; i < CM_MAX_P; ++i) p.P[i] = c->P[i];
    return p;
}

// Number of SMs of the current device (cached per device).
int cm_sm_count();

// ---- launchers (return cudaSuccess or the launch error) --------------------
cudaError_t launch_encode_f32(const CodeParams &cp, const float *A, int64_t lda,
                              float *par, int64_t ldp, int32_t *status, cudaStream_t s);
cudaError_t launch_encode_bf16(const CodeParams &cp, const uint16_t *A, int64_t lda,
                               uint16_t *par, int64_t ldp, int32_t *status, cudaStream_t s);
// Rows per K2 work unit for b = 1 (8 or 4) given L, the computed workers
// and the warps of the persistent grid.
int matvec_rows_per_unit(int64_t L, int nw, int64_t warps);
// `only` = 0: all n workers; otherwise the workers of the first k set bits.
cudaError_t launch_matvec(const CodeParams &cp, const float *A, int64_t lda,
                          const float *par, int64_t ldp, const float *X, int b,
                          double *Yt, int32_t *status, uint32_t only, cudaStream_t s);
// Column segments (1, 2, 4 or 8) for products whose consumer adds partial
// results, and the products written as nseg partial results part_stride
// doubles apart (nseg = 1: launch_matvec).
int matvec_segments(const CodeParams &cp, int b, uint32_t only);
cudaError_t launch_matvec_split(const CodeParams &cp, const float *A, int64_t lda,
                                const float *par, int64_t ldp, const float *X, int b, double *Yt,
                                int32_t *status, uint32_t only, int nseg, int64_t part_stride,
                                cudaStream_t s);

// Decode epilogues (Sec. III-E: the two decodes of a gradient step).
enum DecodeMode { DEC_PLAIN = 0, DEC_RESIDUAL = 1, DEC_DESCENT = 2 };
// dependent: launched as a programmatic dependent of the kernel before it on
// the stream (the worker products), which it waits for before reading
// anything but its parameters; the plan then forms while the products end.
// nparts > 1: the products left that many partial results part_stride
// doubles apart (column segments, launch_matvec_split), summed on load.
cudaError_t launch_decode(const CodeParams &cp, const double *Yt, uint32_t survivors,
                          int b, float *Y, int32_t *status, int mode,
                          const float *lab, float eta, bool dependent, cudaStream_t s,
                          int nparts = 1, int64_t part_stride = 0);
cudaError_t launch_decode_mat(const CodeParams &cp, const float *Ct, int64_t ldc,
                              uint32_t survivors, int N, float *C, int64_t ldcc,
                              int32_t *status, cudaStream_t s);
cudaError_t launch_coded_gemm(const CodeParams &cp, const uint16_t *A, int64_t lda,
                              const uint16_t *par, int64_t ldp, const uint16_t *Bt, int64_t ldb,
                              int N, float *Ct, int64_t ldc, int32_t *status, uint32_t only,
                              cudaStream_t s);
