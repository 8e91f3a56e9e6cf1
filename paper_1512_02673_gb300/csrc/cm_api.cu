// C ABI of libcm: argument validation and dispatch to the kernels.
#include <cmath>
#include <cstdlib>
#include <cstring>

#include "cm_internal.cuh"

namespace {

bool aligned16(const void *p) { return ((uintptr_t)p & 15u) == 0; }

int popcount32(uint32_t x)
{
    int c = 0;
    for (; x; x &= x - 1) ++c;
    return c;
}

cm_status from_cuda(cudaError_t e) { return e == cudaSuccess ? CM_OK : CM_ECUDA; }

// The k workers a decode uses (written to *eff).  A general code decodes
// from any k results (Example "MDS codes"): the first k set bits.  A
// repetition code decodes from one result per block (Example "Repetition
// codes"): the lowest surviving replica of each block.
cm_status resolve_survivors(const cm_code *c, uint32_t survivors, uint32_t *eff)
{
    if (c->n < 32 && (survivors >> c->n)) return CM_EINVAL;
    if (c->kind == CODE_REPETITION) {
        uint32_t sel = 0;
        for (int i = 0; i < c->k; ++i) {
            int pick = -1;
            for (int j = i; j < c->n; j += c->k)
                if ((survivors >> j) & 1u) {
                    pick = j;
                    break;
                }
            if (pick < 0) return CM_ENOTDECODABLE;
            sel |= 1u << pick;
        }
        *eff = sel;
        return CM_OK;
    }
    if (popcount32(survivors) < c->k) return CM_ENOTDECODABLE;
    uint32_t sel = 0;
    int cnt = 0;
    for (int j = 0; j < c->n && cnt < c->k; ++j)
        if ((survivors >> j) & 1u) {
            sel |= 1u << j;
            ++cnt;
        }
    *eff = sel;
    return CM_OK;
}

cm_status check_survivors(const cm_code *c, uint32_t survivors)
{
    uint32_t eff;
    return resolve_survivors(c, survivors, &eff);
}

// Operand layout checks: base 16-byte aligned, leading dimension >= d and a
// multiple of 16 bytes.
bool layout_ok(const void *p, int64_t ld, int64_t d, int64_t elem)
{
    return p && aligned16(p) && ld >= d && (ld * elem) % 16 == 0;
}

}  // namespace

int cm_sm_count()
{
    static int cache[64] = {0};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0) return 0;
    if (dev < 64 && cache[dev]) return cache[dev];
    int sms = 0;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
        return 0;
    if (dev < 64) cache[dev] = sms;
    return sms;
}

extern "C" {

cm_status cm_code_create(int32_t n, int32_t k, int64_t m, int64_t d, cm_dtype dt,
                         const float *parity_host, cm_code **out)
{
    if (!out) return CM_EINVAL;
    *out = nullptr;
    if (k < 1 || n <= k || n > CM_MAX_N || m < 1 || d < 1 || !parity_host) return CM_EINVAL;
    if (dt != CM_F32 && dt != CM_BF16) return CM_EINVAL;
    if ((int64_t)(n - k) * k > CM_MAX_P) return CM_EINVAL;
    for (int i = 0; i < (n - k) * k; ++i)
        if (!std::isfinite(parity_host[i])) return CM_EINVAL;
    cm_code *c = (cm_code *)std::calloc(1, sizeof(cm_code));
    if (!c) return CM_ENOMEM;
    c->n = n;
    c->k = k;
    c->m = m;
    c->d = d;
    c->L = (m + k - 1) / k;   // zero rows appended up to k L (Sec. III-A footnote)
    c->dt = dt;
    c->kind = CODE_GENERAL;
    std::memcpy(c->P, parity_host, sizeof(float) * (n - k) * k);
    *out = c;
    return CM_OK;
}

cm_status cm_code_create_repetition(int32_t n, int32_t k, int64_t m, int64_t d, cm_dtype dt,
                                    cm_code **out)
{
    if (!out) return CM_EINVAL;
    *out = nullptr;
    if (k < 1 || n <= k || n > CM_MAX_N || n % k != 0) return CM_EINVAL;
    float P[CM_MAX_P];
    for (int p = 0; p < n - k; ++p)
        for (int i = 0; i < k; ++i) P[p * k + i] = (i == p % k) ? 1.f : 0.f;
    cm_status st = cm_code_create(n, k, m, d, dt, P, out);
    if (st == CM_OK) (*out)->kind = CODE_REPETITION;
    return st;
}

cm_status cm_select_decodable(const cm_code *c, uint32_t survivors, uint32_t *selected)
{
    if (!c || !selected) return CM_EINVAL;
    return resolve_survivors(c, survivors, selected);
}

void cm_code_destroy(cm_code *code) { std::free(code); }

int64_t cm_block_rows(const cm_code *code) { return code ? code->L : -1; }

cm_status cm_encode(const cm_code *c, const void *A, int64_t lda, void *par, int64_t ldp,
                    int32_t *dev_status, cm_stream_t stream)
{
    if (!c) return CM_EINVAL;
    int64_t es = c->dt == CM_F32 ? 4 : 2;
    if (!layout_ok(A, lda, c->d, es) || !layout_ok(par, ldp, c->d, es)) return CM_EINVAL;
    CodeParams cp = code_params(c);
    if (c->dt == CM_F32)
        return from_cuda(launch_encode_f32(cp, (const float *)A, lda, (float *)par, ldp,
                                           dev_status, (cudaStream_t)stream));
    return from_cuda(launch_encode_bf16(cp, (const uint16_t *)A, lda, (uint16_t *)par, ldp,
                                        dev_status, (cudaStream_t)stream));
}

cm_status cm_matvec(const cm_code *c, const float *A, int64_t lda, const float *par,
                    int64_t ldp, const float *X, int32_t b, double *Yt, int32_t *dev_status,
                    cm_stream_t stream)
{
    if (!c || c->dt != CM_F32) return CM_EINVAL;
    if (b < 1 || b > 8 || !X || !Yt) return CM_EINVAL;
    if (!layout_ok(A, lda, c->d, 4) || !layout_ok(par, ldp, c->d, 4)) return CM_EINVAL;
    if (((uintptr_t)X & 3u) || ((uintptr_t)Yt & 7u)) return CM_EINVAL;
    return from_cuda(launch_matvec(code_params(c), A, lda, par, ldp, X, b, Yt, dev_status, 0u,
                                   (cudaStream_t)stream));
}

cm_status cm_matvec_survivors(const cm_code *c, const float *A, int64_t lda, const float *par,
                              int64_t ldp, const float *X, int32_t b, uint32_t survivors,
                              double *Yt, int32_t *dev_status, cm_stream_t stream)
{
    if (!c || c->dt != CM_F32) return CM_EINVAL;
    uint32_t eff;
    cm_status st = resolve_survivors(c, survivors, &eff);
    if (st != CM_OK) return st;
    if (b < 1 || b > 8 || !X || !Yt) return CM_EINVAL;
    if (!layout_ok(A, lda, c->d, 4) || !layout_ok(par, ldp, c->d, 4)) return CM_EINVAL;
    if (((uintptr_t)X & 3u) || ((uintptr_t)Yt & 7u)) return CM_EINVAL;
    return from_cuda(launch_matvec(code_params(c), A, lda, par, ldp, X, b, Yt, dev_status,
                                   eff, (cudaStream_t)stream));
}

cm_status cm_decode(const cm_code *c, const double *Yt, uint32_t survivors, int32_t b,
                    float *Y, int32_t *dev_status, cm_stream_t stream)
{
    if (!c) return CM_EINVAL;
    uint32_t eff;
    cm_status st = resolve_survivors(c, survivors, &eff);
    if (st != CM_OK) return st;
    if (b < 1 || !Yt || !Y || ((uintptr_t)Yt & 7u) || ((uintptr_t)Y & 3u)) return CM_EINVAL;
    return from_cuda(launch_decode(code_params(c), Yt, eff, b, Y, dev_status,
                                   DEC_PLAIN, nullptr, 0.f, false, (cudaStream_t)stream));
}

// Partial results of the products that cm_matvec_decode may split into
// column segments: the largest count over both worker sets.
static int max_segments(const CodeParams &cp, int b)
{
    const uint32_t some = (uint32_t)((1ull << cp.k) - 1ull);   // k workers
    const int a = matvec_segments(cp, b, 0u), s = matvec_segments(cp, b, some);
    return a > s ? a : s;
}

size_t cm_matvec_decode_workspace_bytes(const cm_code *c, int32_t b)
{
    if (!c || b < 1 || b > 8) return 0;
    return sizeof(double) * (size_t)c->n * c->L * b * (size_t)max_segments(code_params(c), b);
}

cm_status cm_matvec_decode(const cm_code *c, const float *A, int64_t lda, const float *par,
                           int64_t ldp, const float *X, int32_t b, uint32_t survivors,
                           int32_t only_survivors, float *Y, void *ws, size_t ws_bytes,
                           int32_t *dev_status, cm_stream_t stream)
{
    if (!c || c->dt != CM_F32) return CM_EINVAL;
    uint32_t eff;
    cm_status st = resolve_survivors(c, survivors, &eff);
    if (st != CM_OK) return st;
    if (b < 1 || b > 8 || !X || !Y || ((uintptr_t)X & 3u) || ((uintptr_t)Y & 3u)) return CM_EINVAL;
    if (!layout_ok(A, lda, c->d, 4) || !layout_ok(par, ldp, c->d, 4)) return CM_EINVAL;
    if (!ws || ((uintptr_t)ws & 255u)) return CM_EINVAL;
    if (ws_bytes < cm_matvec_decode_workspace_bytes(c, b)) return CM_ENOMEM;
    const CodeParams cp = code_params(c);
    cudaStream_t s = (cudaStream_t)stream;
    double *Yt = (double *)ws;
    const uint32_t only = only_survivors ? eff : 0u;
    const int nseg = matvec_segments(cp, b, only);
    const int64_t part = (int64_t)c->n * c->L * b;
    if (launch_matvec_split(cp, A, lda, par, ldp, X, b, Yt, dev_status, only, nseg, part, s) !=
        cudaSuccess)
        return CM_ECUDA;
    return from_cuda(launch_decode(cp, Yt, eff, b, Y, dev_status, DEC_PLAIN, nullptr, 0.f, true, s,
                                   nseg, part));
}

// Workspace of a gradient step: stacked results of both products (fp64) and
// the residual z (fp32), each 256-byte aligned.
static size_t round256(size_t x) { return (x + 255) & ~(size_t)255; }

size_t cm_gd_workspace_bytes(const cm_code *cA, const cm_code *cAT)
{
    if (!cA || !cAT) return 0;
    return round256(cm_matvec_decode_workspace_bytes(cA, 1)) +
           round256(sizeof(float) * (size_t)cA->m) +
           round256(cm_matvec_decode_workspace_bytes(cAT, 1));
}

namespace {

// Sec. III-E: the master multicasts x, decodes A x from any k1 results,
// forms z = A x - y, multicasts it, decodes A^T z from any k2 results and
// steps x <- x - eta A^T z.  Each decode writes the residual or the step
// itself and is launched as a programmatic dependent of its products.
cm_status gd_step(const cm_code *cA, const float *A, int64_t lda, const float *PA, int64_t ldpa,
                  const cm_code *cAT, const float *AT, int64_t ldat, const float *PAT,
                  int64_t ldpat, const float *y, float *x, float eta, uint32_t surv_A,
                  uint32_t surv_AT, void *ws, size_t ws_bytes, int32_t *dev_status,
                  cm_stream_t stream, bool only)
{
    if (!cA || !cAT || cA->dt != CM_F32 || cAT->dt != CM_F32) return CM_EINVAL;
    if (cAT->m != cA->d || cAT->d != cA->m || cAT->n != cA->n) return CM_EINVAL;
    uint32_t effA, effAT;
    cm_status st = resolve_survivors(cA, surv_A, &effA);
    if (st != CM_OK) return st;
    st = resolve_survivors(cAT, surv_AT, &effAT);
    if (st != CM_OK) return st;
    if (!layout_ok(A, lda, cA->d, 4) || !layout_ok(PA, ldpa, cA->d, 4) ||
        !layout_ok(AT, ldat, cAT->d, 4) || !layout_ok(PAT, ldpat, cAT->d, 4))
        return CM_EINVAL;
    if (!y || !x || ((uintptr_t)y & 3u) || ((uintptr_t)x & 3u) || !std::isfinite(eta))
        return CM_EINVAL;
    if (!ws || ((uintptr_t)ws & 255u)) return CM_EINVAL;
    if (ws_bytes < cm_gd_workspace_bytes(cA, cAT)) return CM_ENOMEM;
    char *w = (char *)ws;
    double *ytA = (double *)w;
    w += round256(cm_matvec_decode_workspace_bytes(cA, 1));
    float *z = (float *)w;
    w += round256(sizeof(float) * (size_t)cA->m);
    double *ytAT = (double *)w;
    cudaStream_t s = (cudaStream_t)stream;
    CodeParams pA = code_params(cA), pAT = code_params(cAT);
    const uint32_t onlyA = only ? effA : 0u, onlyAT = only ? effAT : 0u;
    const int segA = matvec_segments(pA, 1, onlyA), segAT = matvec_segments(pAT, 1, onlyAT);
    const int64_t partA = (int64_t)cA->n * cA->L, partAT = (int64_t)cAT->n * cAT->L;
    if (launch_matvec_split(pA, A, lda, PA, ldpa, x, 1, ytA, dev_status, onlyA, segA, partA, s) !=
        cudaSuccess)
        return CM_ECUDA;
    if (launch_decode(pA, ytA, effA, 1, z, dev_status, DEC_RESIDUAL, y, 0.f, true, s, segA,
                      partA) != cudaSuccess)
        return CM_ECUDA;
    if (launch_matvec_split(pAT, AT, ldat, PAT, ldpat, z, 1, ytAT, dev_status, onlyAT, segAT,
                            partAT, s) != cudaSuccess)
        return CM_ECUDA;
    if (launch_decode(pAT, ytAT, effAT, 1, x, dev_status, DEC_DESCENT, nullptr, eta, true, s,
                      segAT, partAT) != cudaSuccess)
        return CM_ECUDA;
    return CM_OK;
}

}  // namespace

cm_status cm_gd_step(const cm_code *cA, const float *A, int64_t lda, const float *PA,
                     int64_t ldpa, const cm_code *cAT, const float *AT, int64_t ldat,
                     const float *PAT, int64_t ldpat, const float *y, float *x, float eta,
                     uint32_t surv_A, uint32_t surv_AT, void *ws, size_t ws_bytes,
                     int32_t *dev_status, cm_stream_t stream)
{
    return gd_step(cA, A, lda, PA, ldpa, cAT, AT, ldat, PAT, ldpat, y, x, eta, surv_A, surv_AT,
                   ws, ws_bytes, dev_status, stream, false);
}

cm_status cm_gd_step_survivors(const cm_code *cA, const float *A, int64_t lda, const float *PA,
                               int64_t ldpa, const cm_code *cAT, const float *AT, int64_t ldat,
                               const float *PAT, int64_t ldpat, const float *y, float *x,
                               float eta, uint32_t surv_A, uint32_t surv_AT, void *ws,
                               size_t ws_bytes, int32_t *dev_status, cm_stream_t stream)
{
    return gd_step(cA, A, lda, PA, ldpa, cAT, AT, ldat, PAT, ldpat, y, x, eta, surv_A, surv_AT,
                   ws, ws_bytes, dev_status, stream, true);
}

cm_status cm_coded_gemm(const cm_code *c, const void *A, int64_t lda, const void *par,
                        int64_t ldp, const void *Bt, int64_t ldb, int32_t N, float *Ct,
                        int64_t ldc, int32_t *dev_status, cm_stream_t stream)
{
    if (!c || c->dt != CM_BF16) return CM_EINVAL;
    if (N < 1) return CM_EINVAL;
    if (!layout_ok(A, lda, c->d, 2) || !layout_ok(par, ldp, c->d, 2) ||
        !layout_ok(Bt, ldb, c->d, 2))
        return CM_EINVAL;
    if (!Ct || ((uintptr_t)Ct & 15u) || ldc < N) return CM_EINVAL;
    return from_cuda(launch_coded_gemm(code_params(c), (const uint16_t *)A, lda,
                                       (const uint16_t *)par, ldp, (const uint16_t *)Bt, ldb,
                                       N, Ct, ldc, dev_status, 0u, (cudaStream_t)stream));
}

cm_status cm_coded_gemm_survivors(const cm_code *c, const void *A, int64_t lda, const void *par,
                                  int64_t ldp, const void *Bt, int64_t ldb, int32_t N,
                                  uint32_t survivors, float *Ct, int64_t ldc,
                                  int32_t *dev_status, cm_stream_t stream)
{
    if (!c || c->dt != CM_BF16) return CM_EINVAL;
    uint32_t eff;
    cm_status st = resolve_survivors(c, survivors, &eff);
    if (st != CM_OK) return st;
    if (N < 1) return CM_EINVAL;
    if (!layout_ok(A, lda, c->d, 2) || !layout_ok(par, ldp, c->d, 2) ||
        !layout_ok(Bt, ldb, c->d, 2))
        return CM_EINVAL;
    if (!Ct || ((uintptr_t)Ct & 15u) || ldc < N) return CM_EINVAL;
    return from_cuda(launch_coded_gemm(code_params(c), (const uint16_t *)A, lda,
                                       (const uint16_t *)par, ldp, (const uint16_t *)Bt, ldb,
                                       N, Ct, ldc, dev_status, eff, (cudaStream_t)stream));
}

cm_status cm_decode_mat(const cm_code *c, const float *Ct, int64_t ldc, uint32_t survivors,
                        int32_t N, float *C, int64_t ldcc, int32_t *dev_status,
                        cm_stream_t stream)
{
    if (!c) return CM_EINVAL;
    uint32_t eff;
    cm_status st = resolve_survivors(c, survivors, &eff);
    if (st != CM_OK) return st;
    if (N < 1 || !Ct || !C || ldc < N || ldcc < N || ((uintptr_t)Ct & 3u) ||
        ((uintptr_t)C & 3u))
        return CM_EINVAL;
    if (C == Ct && ldcc != ldc) return CM_EINVAL;
    return from_cuda(launch_decode_mat(code_params(c), Ct, ldc, eff, N, C, ldcc,
                                       dev_status, (cudaStream_t)stream));
}

cm_status cm_matmat(const cm_code *c, const void *A, int64_t lda, const void *par,
                    int64_t ldp, const void *Bt, int64_t ldb, int32_t N, float *Ct,
                    int64_t ldc, uint32_t survivors, float *C, int64_t ldcc,
                    int32_t *dev_status, cm_stream_t stream)
{
    if (!c) return CM_EINVAL;
    cm_status st = check_survivors(c, survivors);
    if (st != CM_OK) return st;
    st = cm_coded_gemm(c, A, lda, par, ldp, Bt, ldb, N, Ct, ldc, dev_status, stream);
    if (st != CM_OK) return st;
    return cm_decode_mat(c, Ct, ldc, survivors, N, C, ldcc, dev_status, stream);
}

const char *cm_status_string(cm_status s)
{
    switch (s) {
    case CM_OK: return "ok";
    case CM_EINVAL: return "invalid argument, shape, alignment or dtype";
    case CM_ENOTDECODABLE: return "fewer than k survivors: not decodable";
    case CM_ESINGULAR: return "singular generator submatrix G_S";
    case CM_ECUDA: return "CUDA launch or query failed";
    case CM_ENOMEM: return "out of memory or workspace too small";
    case CM_ETIMEOUT: return "bounded device wait gave up";
    case CM_EUNSUPPORTED: return "unsupported request";
    }
    return "unknown status";
}

}  // extern "C"
