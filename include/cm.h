/*
 * cm.h -- C ABI of libcm, MDS-coded matrix multiplication on one GB300 GPU.
 *
 * Method: Lee, Lam, Pedarsani, Papailiopoulos, Ramchandran, "Speeding Up
 * Distributed Machine Learning Using Codes", Sec. III.  A data matrix A
 * (m x d) is split by rows into k blocks A_0..A_{k-1} of L = ceil(m/k) rows
 * (zero rows appended, Sec. III-A footnote); a systematic (n,k) code with
 * generator G = [I_k; P] turns them into n coded blocks
 * A~_j = sum_i G[j][i] A_i (Sec. III-A).  The n block products A~_j X are the
 * n simulated workers; from ANY k of the n results the product A X is
 * recovered (Example "MDS codes", Sec. III-B).  Straggler sets follow the
 * shifted-exponential runtime model (Sec. III-C, III-D).  The same machinery
 * runs coded gradient descent for linear regression (Sec. III-E).
 *
 * Conventions for every call:
 *  - Matrices are row-major.  "Stacked" results hold worker j's block in rows
 *    [j L, (j+1) L).  Worker j < k is systematic: its coded block is A_j
 *    itself, read in place from the caller's A (rows >= m are virtual zero
 *    rows, never read); workers j >= k are parity blocks held in a separate
 *    (n-k) L x d "parity" buffer.
 *  - Device pointers are CUDA device memory (or managed memory) of the
 *    current device.  The caller allocates and frees every device buffer; the
 *    library allocates no device memory and keeps no global state, so calls
 *    on distinct objects are thread-safe.  A cm_code is a small immutable
 *    host object.
 *  - Every GPU call is asynchronous on the given stream (NULL = legacy
 *    default stream).  Argument errors are returned synchronously and nothing
 *    is launched.  CM_ECUDA is returned when a launch fails.  Conditions only
 *    the device can see (a singular system, a bounded wait that gave up) are
 *    written to the optional int32 device word *dev_status after the stream
 *    reaches the kernel; the library only ever writes error codes there
 *    (never CM_OK), so the caller clears it beforehand.
 *  - Alignment: A, parity and (for cm_matmat) B start on 16-byte boundaries
 *    and their leading dimensions are multiples of 16 bytes (4 fp32 or 8 bf16
 *    elements); X, Y and Yt have no alignment requirement beyond their type.
 *  - No call traps, aborts or exits the process.
 */
#ifndef CM_H
#define CM_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    CM_OK = 0,
    CM_EINVAL = -1,          /* bad argument, shape, alignment or dtype */
    CM_ENOTDECODABLE = -2,   /* fewer than k survivors */
    CM_ESINGULAR = -3,       /* G_S is singular (device-detected) */
    CM_ECUDA = -4,           /* a CUDA launch or query failed */
    CM_ENOMEM = -5,          /* host allocation failed, or workspace too small */
    CM_ETIMEOUT = -6,        /* a bounded device wait gave up */
    CM_EUNSUPPORTED = -7     /* valid request the library does not handle */
} cm_status;

typedef enum { CM_F32 = 0, CM_BF16 = 1 } cm_dtype;

typedef struct cm_code cm_code;          /* opaque, immutable after create */
typedef struct CUstream_st *cm_stream_t; /* same type as cudaStream_t */

/* Build an (n,k) systematic code for an m x d data matrix of type dt
 * (Sec. III-A).  parity_host is the (n-k) x k block P of G = [I_k; P], fp32,
 * row-major, on the host; it is copied.  Any P whose square submatrices are
 * all nonsingular gives an MDS code; a Gaussian P does with probability 1.
 * Requires 1 <= k < n <= 32, m >= 1, d >= 1, finite P.  No CUDA call. */
cm_status cm_code_create(int32_t n, int32_t k, int64_t m, int64_t d, cm_dtype dt,
                         const float *parity_host, cm_code **out);
void cm_code_destroy(cm_code *code);

/* The n/k-repetition code of Sec. III-B (Example "Repetition codes"): every
 * data block is replicated n/k times; worker j holds block j mod k (workers
 * j < k are the systematic copies), i.e. P[p][i] = 1 if i == p mod k else 0.
 * Requires n % k == 0.  Its decodable sets are the products of the replica
 * groups {i, i+k, i+2k, ...}: decoding uses the lowest surviving replica of
 * each block.  No CUDA call. */
cm_status cm_code_create_repetition(int32_t n, int32_t k, int64_t m, int64_t d, cm_dtype dt,
                                    cm_code **out);

/* The k workers a decode of this code uses for the given survivor mask:
 * the first k set bits for a general (MDS) code, the lowest surviving
 * replica of each block for a repetition code.  CM_ENOTDECODABLE when the
 * survivors hold no decodable set. */
cm_status cm_select_decodable(const cm_code *code, uint32_t survivors, uint32_t *selected);

/* L = ceil(m / k), the rows per block after zero padding (Sec. III-A
 * footnote); -1 for a NULL code. */
int64_t cm_block_rows(const cm_code *code);

/* Encoding (Sec. III-A): parity block p (rows [p L, (p+1) L) of parity_out,
 * leading dimension ldp) = sum_i P[p][i] A_i, for p = 0..n-k-1, in one pass
 * over A (n - k <= 16; larger counts take one pass per 16 parity blocks).
 * A is m x d with leading dimension lda, of the code's dtype (fp32, or bf16
 * with fp32 accumulation and round-to-nearest-even output).  parity_out must
 * not overlap A.  A bounded wait that gives up writes CM_ETIMEOUT to
 * *dev_status (nullable). */
cm_status cm_encode(const cm_code *code, const void *A, int64_t lda,
                    void *parity_out, int64_t ldp, int32_t *dev_status, cm_stream_t stream);

/* The n worker products (Sec. III-A protocol): Yt[j L + r][v] =
 * sum_c A~_j[r][c] X[c][v] for every worker j, row r < L and vector v < b,
 * all workers concurrently.  fp32 code only.  X is d x b fp32 (row-major,
 * vectors contiguous per row), 1 <= b <= 8.  Yt is n L x b fp64: each sum is
 * formed from short fp32 partial sums combined in fp64, so decoding does not
 * amplify an fp32 rounding of the results.  A bounded wait inside the kernel
 * that gives up writes CM_ETIMEOUT to *dev_status (nullable); Yt is then
 * incomplete. */
cm_status cm_matvec(const cm_code *code, const float *A, int64_t lda,
                    const float *parity, int64_t ldp, const float *X, int32_t b,
                    double *Yt, int32_t *dev_status, cm_stream_t stream);

/* cm_matvec restricted to the survivors: when the straggler set is known
 * before the products run, only the workers that cm_decode will read (the
 * first k set bits of `survivors`) are computed, saving (n-k)/n of the reads
 * (the MDS run ends at the k-th arrival, eq. for the MDS runtime, so the
 * stragglers' work is never used).  Rows of the other workers in Yt are left
 * unwritten.  Same layout, precision and errors as cm_matvec; fewer than k
 * survivors returns CM_ENOTDECODABLE. */
cm_status cm_matvec_survivors(const cm_code *code, const float *A, int64_t lda,
                              const float *parity, int64_t ldp, const float *X, int32_t b,
                              uint32_t survivors, double *Yt, int32_t *dev_status,
                              cm_stream_t stream);

/* Straggler draw (Sec. III-C, III-D; eq. for the MDS runtime).  Host only.
 * Worker j's time in round `counter` is T_j = (shift + E_j / rate) / k with
 * E_j = -log(1 - U_j), U_j = (z_j >> 11) 2^-53, z_j the SplitMix64 output
 * (Steele, Lea, Flood 2014) of the Weyl state
 * seed + (counter n + j + 1) 0x9E3779B97F4A7C15.  The coded run ends at the
 * k-th arrival, so the survivors are the k workers with the smallest T_j,
 * ranked on the integers (z_j >> 11, j) (ties go to the lower index).
 * *survivors receives the bitmask (bit j = worker j survives), exactly k
 * bits; times (nullable, n entries) receives the T_j.  1 <= k <= n <= 32,
 * rate > 0. */
cm_status cm_draw_erasures(uint64_t seed, uint64_t counter, int32_t n, int32_t k,
                           double shift, double rate, uint32_t *survivors,
                           double *times);

/* Decoding (Sec. III-A last paragraph; Example "MDS codes").  S = the first
 * k set bits of `survivors` (ascending; extra survivors are ignored, which
 * favours the systematic workers).  The surviving results satisfy
 * Yt_S = G_S Z with Z the uncoded block products.  One launch: every CTA
 * inverts G_S in fp64 in its own shared memory (the k-e unit rows of
 * surviving systematic workers are eliminated first, then Gauss-Jordan with
 * partial pivoting on the e x e block Q of the missing systematic columns,
 * in the registers of one warp for e <= 4, of four for e <= 16; adj(Q) /
 * det Q for e <= 2) and applies the rows of G_S^-1 for the e missing
 * systematic blocks to the k surviving results, as Q^-1 (Yt_par - P_sys
 * Yt_sys) with the second factor formed while the inversion runs
 * (double-float arithmetic, about 2^-44 relative per term); surviving
 * systematic blocks pass through.  The launch is a
 * programmatic dependent of the kernel before it on `stream`: the eliminating
 * warps start from the kernel parameters at once and the others wait for the
 * earlier grids before reading Yt, so after cm_matvec on the same stream the
 * inversion overlaps the products' last round (after any other kernel the
 * wait returns at once).  Nothing is kept between calls.  Y (m x b
 * fp32) is the concatenation of the k decoded blocks without the appended
 * zero rows.  Returns CM_ENOTDECODABLE when fewer than k bits are set; a
 * singular G_S (a zero pivot, or ||Q|| ||Q^-1|| beyond 1 / (64 eps) for the
 * e x e block) writes CM_ESINGULAR to *dev_status (nullable) and leaves the
 * missing blocks of Y unwritten (surviving systematic blocks are still
 * copied). */
cm_status cm_decode(const cm_code *code, const double *Yt, uint32_t survivors,
                    int32_t b, float *Y, int32_t *dev_status, cm_stream_t stream);

/* Workspace bytes cm_matvec_decode needs for b vectors (the stacked results,
 * n L b fp64 per column segment; 0 on a bad code or b outside 1..8). */
size_t cm_matvec_decode_workspace_bytes(const cm_code *code, int32_t b);

/* The worker products and the decode in one call (Sec. III-A: the master
 * needs only the first k results, and decoding is a fixed linear map of
 * them): Y = A X (m x b fp32), the result of cm_matvec (or
 * cm_matvec_survivors) followed by cm_decode.  On small problems, whose
 * units fill the persistent grid poorly, the products are split into 2, 4
 * or 8 column segments done by separate shares of the SMs, and the decode
 * adds the segments' fp64 partial sums as it loads them (Y then differs from
 * the two calls' by the products' own rounding, short fp32 partial sums
 * being flushed at other columns).  The decode is launched as a
 * programmatic dependent of the products: its CTAs start on the SMs the
 * products leave free in their last round, form the rows of G_S^-1 (the fp64
 * elimination of cm_decode) from the kernel parameters alone, and wait for
 * the products only before they read a result, so the decode's launch and
 * inversion overlap the products' tail.  only_survivors = 0: all n workers
 * compute (the protocol of Sec. III-A); 1: only the k used workers compute
 * (the stragglers known beforehand), reading (n-k)/n fewer bytes.  S is the
 * first k set bits of `survivors` (for a repetition code, the first survivor
 * of each block), as for cm_decode.  ws is caller device memory of at least
 * cm_matvec_decode_workspace_bytes(code, b) bytes, 256-byte aligned, which
 * receives the stacked worker results (n L x b fp64 per column segment;
 * rows of workers that did not compute are left unwritten).  Two launches.
 * Errors as cm_matvec and cm_decode; CM_ENOMEM for a short workspace. */
cm_status cm_matvec_decode(const cm_code *code, const float *A, int64_t lda,
                           const float *parity, int64_t ldp, const float *X, int32_t b,
                           uint32_t survivors, int32_t only_survivors, float *Y, void *ws,
                           size_t ws_bytes, int32_t *dev_status, cm_stream_t stream);

/* Workspace bytes cm_gd_step needs for this pair of codes (0 on bad codes). */
size_t cm_gd_workspace_bytes(const cm_code *code_A, const cm_code *code_AT);

/* One iteration of coded gradient descent for linear regression (Sec. III-E):
 * x <- x - eta A^T (A x - y).  The first product uses code_A (m x d) on A and
 * its parity PA with survivors surv_A; the result decodes to z = A x - y.
 * The second uses code_AT (d x m) on AT = A^T (row-major d x m, i.e. the
 * column split of A, Sec. III-E) and its parity PAT with survivors surv_AT;
 * the result decodes to the gradient g = A^T z and x -= eta g.  x (d fp32) is
 * updated in place.  All n workers compute each product (the protocol of
 * Sec. III-A); each decode writes z or the step itself and is launched as a
 * programmatic dependent of its products, as in cm_matvec_decode.  ws is
 * caller device memory of at least cm_gd_workspace_bytes(code_A, code_AT)
 * bytes (holds both stacked results and z), 256-byte aligned.  Four launches
 * on `stream`. */
cm_status cm_gd_step(const cm_code *code_A, const float *A, int64_t lda,
                     const float *PA, int64_t ldpa,
                     const cm_code *code_AT, const float *AT, int64_t ldat,
                     const float *PAT, int64_t ldpat,
                     const float *y, float *x, float eta,
                     uint32_t surv_A, uint32_t surv_AT,
                     void *ws, size_t ws_bytes, int32_t *dev_status,
                     cm_stream_t stream);

/* cm_gd_step with only the k used workers of each product computing (the
 * straggler sets known before the products run, Sec. III-A: the master needs
 * only k results).  Same arguments, workspace and result. */
cm_status cm_gd_step_survivors(const cm_code *code_A, const float *A, int64_t lda,
                               const float *PA, int64_t ldpa,
                               const cm_code *code_AT, const float *AT, int64_t ldat,
                               const float *PAT, int64_t ldpat,
                               const float *y, float *x, float eta,
                               uint32_t surv_A, uint32_t surv_AT,
                               void *ws, size_t ws_bytes, int32_t *dev_status,
                               cm_stream_t stream);

/* Size of the fixed device scratch array behind cm_gd_step_noalloc: 4 MiB. */
#define CM_GD_STATIC_SCRATCH_BYTES (4u << 20)

/* cm_gd_step without a caller workspace (the paper has no counterpart: this
 * is a service for callers that cannot allocate device memory, e.g. a
 * plug-in inside an application that owns all device memory through its own
 * pool, or a loop that must not call cudaMalloc / cudaFree because they can
 * synchronize the device).  Same arguments and result as cm_gd_step minus
 * ws / ws_bytes; the workspace is a file-scope device array of
 * CM_GD_STATIC_SCRATCH_BYTES held by every GPU that loads the library until
 * the process exits.  The call allocates nothing.  Returns CM_ENOMEM when
 * cm_gd_workspace_bytes(code_A, code_AT) exceeds the array.  The first call
 * on a device looks up the array's device address (with that device
 * current) and keeps it for that device's current CUDA context; a call made
 * under another context of the device (after cudaDeviceReset, or in a
 * context the caller created) looks it up again.  Make the first call in
 * each context before any stream capture.
 * All calls on a device share the array and it keeps the last call's
 * contents (nothing in it needs to start at zero); calls whose kernels
 * overlap on the GPU race on it. */
cm_status cm_gd_step_noalloc(const cm_code *code_A, const float *A, int64_t lda,
                             const float *PA, int64_t ldpa,
                             const cm_code *code_AT, const float *AT, int64_t ldat,
                             const float *PAT, int64_t ldpat,
                             const float *y, float *x, float eta,
                             uint32_t surv_A, uint32_t surv_AT, int32_t *dev_status,
                             cm_stream_t stream);

/* Coded matrix-matrix products (the s-column X of the Sec. I-A example) on
 * tensor cores: Ct[j L + r][c] = sum_t A~_j[r][t] B[t][c] for all n workers,
 * bf16 inputs, fp32 accumulation in tensor memory, fp32 output.  bf16 code
 * only.  B is passed transposed: Bt is N x d bf16 (row-major, leading
 * dimension ldb), i.e. each column of B contiguous.  Ct is n L x N fp32 with
 * leading dimension ldc (16-byte aligned base).  Any N >= 1 (the ragged last
 * column tile and K tail read zeros).  A bounded wait that gives up writes
 * CM_ETIMEOUT to *dev_status (nullable). */
cm_status cm_coded_gemm(const cm_code *code, const void *A, int64_t lda,
                        const void *parity, int64_t ldp, const void *Bt, int64_t ldb,
                        int32_t N, float *Ct, int64_t ldc, int32_t *dev_status,
                        cm_stream_t stream);

/* The coded matrix-matrix products of the k workers that cm_decode_mat will
 * read (the first k set bits of `survivors`; for a repetition code the
 * first survivor of each block), when the stragglers are known before the
 * products run (Sec. III-A: the master needs only k results).  Arguments
 * and layout as cm_coded_gemm; the blocks of the other workers in Ct are not
 * written.  The computed blocks equal cm_coded_gemm's bit for bit.  Returns
 * CM_ENOTDECODABLE when the survivors cannot be decoded. */
cm_status cm_coded_gemm_survivors(const cm_code *code, const void *A, int64_t lda,
                                  const void *parity, int64_t ldp, const void *Bt, int64_t ldb,
                                  int32_t N, uint32_t survivors, float *Ct, int64_t ldc,
                                  int32_t *dev_status, cm_stream_t stream);

/* Decoding of matrix results: as cm_decode with b = N columns of fp32
 * stacked results Ct (leading dimension ldc) into C (m x N fp32, leading
 * dimension ldcc).  The decode coefficients are formed in fp64 in each CTA as
 * for cm_decode and applied in fp32.  C may alias Ct (C == Ct, ldcc == ldc): surviving systematic
 * blocks are then already in place and only the missing ones are written. */
cm_status cm_decode_mat(const cm_code *code, const float *Ct, int64_t ldc,
                        uint32_t survivors, int32_t N, float *C, int64_t ldcc,
                        int32_t *dev_status, cm_stream_t stream);

/* cm_coded_gemm followed by cm_decode_mat on the same stream. */
cm_status cm_matmat(const cm_code *code, const void *A, int64_t lda,
                    const void *parity, int64_t ldp, const void *Bt, int64_t ldb,
                    int32_t N, float *Ct, int64_t ldc, uint32_t survivors,
                    float *C, int64_t ldcc, int32_t *dev_status, cm_stream_t stream);

/* Self-test of the bounded device wait that cm_matvec and cm_coded_gemm use
 * for their TMA pipelines (no counterpart in the paper: failure detection).
 * Launches one warp that waits on an mbarrier nothing arrives at, giving up
 * after limit_ns nanoseconds (1 .. 2e9); the kernel then writes CM_ETIMEOUT
 * to *dev_status and returns, and the context stays usable. */
cm_status cm_selftest_bounded_wait(int32_t *dev_status, uint64_t limit_ns, cm_stream_t stream);

/* ---- runtime model (Sec. III-B, III-C, III-D), host only ----------------
 * A job split k ways runs each task for T = (shift + E / rate) / k, E ~ Exp(1)
 * (the shifted-exponential mother distribution F(t) = 1 - e^{-rate (t - shift)}
 * scaled by the split, P(T <= t) = F(k t)).  The overall runtime is the max of
 * the n tasks for an uncoded job (split n ways, eq. for the uncoded runtime),
 * the max over blocks of the min over replicas for an n/k-repetition code
 * (eq. for the repetition runtime), and the k-th arrival for an (n,k) MDS
 * code (eq. for the MDS runtime). */
typedef enum { CM_SCHEME_UNCODED = 0, CM_SCHEME_REPETITION = 1, CM_SCHEME_MDS = 2 } cm_scheme;

/* Expected overall runtime, exact harmonic-number form of Sec. III-D:
 * uncoded (shift + H_n/rate)/n; repetition (shift + (k/n) H_k/rate)/k;
 * MDS (shift + (H_n - H_{n-k})/rate)/k.  k is ignored for the uncoded
 * scheme; repetition needs n % k == 0. */
cm_status cm_runtime_mean(cm_scheme scheme, int32_t n, int32_t k, double shift, double rate,
                          double *mean);

/* Distribution P(T_overall <= t) at `count` points (eqs. for F_uncoded,
 * F_rep and F_MDS; the MDS one as the binomial tail equal to its integral
 * form). */
cm_status cm_runtime_cdf(cm_scheme scheme, int32_t n, int32_t k, double shift, double rate,
                         const double *t, int64_t count, double *F);

/* Monte-Carlo overall runtimes of `count` rounds (counters counter0 ..),
 * drawn exactly as cm_draw_erasures draws worker times (n <= 32). */
cm_status cm_runtime_simulate(cm_scheme scheme, int32_t n, int32_t k, double shift, double rate,
                              uint64_t seed, uint64_t counter0, int64_t count, double *T);

/* Lemma on optimal MDS-coded algorithms: k* = (1 + 1/W_{-1}(-e^{-rate-1})) n
 * minimises the expected MDS runtime (log form of the harmonic numbers), and
 * n T* = gamma* = -W_{-1}(-e^{-rate-1}) / rate (W_{-1}: the lower branch of
 * the Lambert W function). */
cm_status cm_optimal_mds_k(int32_t n, double rate, double *k_star, double *gamma_star);

/* ---- coded shuffling (Sec. IV) --------------------------------------------
 * q data rows of r 4-byte words are reshuffled across n workers before every
 * iteration: a uniformly random partition into sets S_i of q/n rows (Sec.
 * IV-A).  Worker i has a cache of s rows (q/n <= s <= q) holding S_i plus
 * s - q/n rows kept by the cache update rule: drawn without replacement from
 * its previous cache outside the new S_i (Sec. IV-B).  For the transition
 * t -> t+1 the master sends, for every worker set I with |I| >= 2, the sum of
 * the zero-padded blocks A(S_i^{t+1} & C~_{I\{i}}), i in I, where C~_J is the
 * set of rows cached at every worker of J and at no other (Alg. 1); each
 * worker recovers its missing rows by subtracting the rows it caches (the
 * decoding algorithm of Sec. IV-B).
 *
 * A cm_shuffle is a host object: the master's planner.  It holds the
 * partition, the caches (as n x s slot tables: slot c of worker i holds data
 * row slot_row[i s + c]) and the row programs of the last transition.  The
 * data plane runs on the device on caller-owned buffers:
 *   A       q x r data rows (leading dimension lda words)
 *   caches  n s x r: slot c of worker i is row i s + c (leading dimension ldc)
 *   M       coded message rows, >= coded_rows x r (leading dimension ldm)
 *   Rx      received rows, >= uncoded_rows x r (leading dimension ldr): the
 *           rows of S_i^{t+1} missing from cache i, for worker 0, 1, ... in
 *           ascending data-row order (cm_shuffle_received lists them).
 * Every device buffer starts on a 16-byte boundary and its leading dimension
 * is a multiple of 4 words; any r >= 1.  Nothing runs in place: M, Rx and
 * the caches are distinct buffers.
 *
 * Sums: CM_SHUFFLE_ADD adds and subtracts the rows as fp32 reals, the
 * arithmetic of the paper (decoded rows then carry fp32 rounding of the sum);
 * CM_SHUFFLE_XOR combines the 32-bit words by exclusive or, a sum in which
 * every element is its own negative, so decoding is exact for any data.
 *
 * Random draws are SplitMix64 outputs (state = seed + index
 * 0x9E3779B97F4A7C15, then the standard finaliser): iteration t's partition
 * orders rows by (key(partition_seed, t q + r), r) and gives the positions
 * [i q/n, (i+1) q/n) to worker i; a cache refill of worker i at iteration t
 * keeps the s - q/n candidates with the smallest (key(cache_seed,
 * (t n + i) q + r), r).  Iteration 0's caches refill from all rows outside
 * S_i^0. */
typedef struct cm_shuffle cm_shuffle;

typedef enum { CM_SHUFFLE_ADD = 0, CM_SHUFFLE_XOR = 1 } cm_shuffle_op;

typedef struct {
    int64_t iteration;      /* t of the current partition and caches */
    int64_t message_sets;   /* sets I with a non-empty message in the last transition */
    int64_t coded_rows;     /* rows the coded scheme sends (the realised R_c) */
    int64_t uncoded_rows;   /* rows missing from their new owner's cache (realised R_u) */
    int64_t subtractions;   /* cached rows the workers subtract while decoding */
} cm_shuffle_stats;

/* Draws iteration 0 (partition and caches).  2 <= n <= 64, q % n == 0,
 * q/n <= s <= q and n q < 2^31; else CM_EINVAL.  CM_ENOMEM if the host tables
 * (about 4 n q + 16 q bytes) cannot be allocated. */
cm_status cm_shuffle_create(int32_t n, int64_t q, int64_t s, uint64_t partition_seed,
                            uint64_t cache_seed, cm_shuffle **out);
void cm_shuffle_destroy(cm_shuffle *shuffle);

/* Host planning of the transition t -> t+1: draws the next partition, plans
 * Alg. 1's messages and the decoding, applies the cache update rule and
 * assigns the received rows to the freed cache slots.  stats is nullable. */
cm_status cm_shuffle_next(cm_shuffle *shuffle, cm_shuffle_stats *stats);

/* Statistics of the last transition (zeros before the first). */
cm_status cm_shuffle_query(const cm_shuffle *shuffle, cm_shuffle_stats *stats);

/* The messages of the last transition: message row m sums data rows
 * msg_src[msg_ptr[m] .. msg_ptr[m+1]) (coded_rows + 1 offsets; uncoded_rows
 * rows), row x needed by worker msg_worker[x]; msg_set[m] is the bit mask of
 * its I.  Any output may be NULL.  CM_EINVAL before the first transition. */
cm_status cm_shuffle_plan(const cm_shuffle *shuffle, int32_t *msg_ptr, int32_t *msg_src,
                          int32_t *msg_worker, uint64_t *msg_set);

/* Layout of Rx: worker i's received rows are rows [recv_ptr[i], recv_ptr[i+1])
 * (n + 1 offsets), holding data rows recv_row[...] in ascending order. */
cm_status cm_shuffle_received(const cm_shuffle *shuffle, int32_t *recv_ptr, int32_t *recv_row);

/* The current partition (owner[r] = i for r in S_i, q entries) and cache
 * slot tables (n s entries).  Either output may be NULL. */
cm_status cm_shuffle_caches(const cm_shuffle *shuffle, int32_t *owner, int32_t *slot_row);

/* Communication rates of the coded shuffling rate theorem, in data rows per
 * iteration: R_c = sum_{i=2}^{n} C(n,i) (q/n) ((i-1)/n) p^{i-2} (1-p)^{n-i+1},
 * p = (s - q/n)/(q - q/n) (the sum its proof evaluates; equal to the closed
 * form q/(np)^2 ((1-p)^{n+1} + (n-1) p (1-p) - (1-p)^2)), and the uncoded
 * rate R_u = q (1 - s/q) (eq. for R_u).  Host only. */
cm_status cm_shuffle_rates(int32_t n, double q, double s, double *coded, double *uncoded);

/* Bytes of device workspace for the row programs of any transition of this
 * instance (about 4 q (n + 5) + 4 n s). */
size_t cm_shuffle_workspace_bytes(const cm_shuffle *shuffle);

/* Copies the current row programs (and slot tables) into `workspace` (16-byte
 * aligned, >= cm_shuffle_workspace_bytes) on `stream`.  The host tables may
 * change once this returns.  Every data-plane call below checks that the
 * workspace it is given holds the programs of the current transition and
 * returns CM_EINVAL otherwise. */
cm_status cm_shuffle_upload(cm_shuffle *shuffle, void *workspace, size_t bytes,
                            cm_stream_t stream);

/* Loads every cache from A by its slot table: caches[i s + c] = A[slot_row[i s + c]]. */
cm_status cm_shuffle_fill(const cm_shuffle *shuffle, const void *workspace, const void *A,
                          int64_t lda, int64_t r, void *caches, int64_t ldc,
                          cm_stream_t stream);

/* Alg. 1 (master): M[m] = sum of the data rows of message row m (zero-padded
 * blocks contribute nothing).  Needs a planned transition. */
cm_status cm_shuffle_encode(const cm_shuffle *shuffle, const void *workspace, cm_shuffle_op op,
                            const void *A, int64_t lda, int64_t r, void *M, int64_t ldm,
                            cm_stream_t stream);

/* Decoding by subtraction (workers): every received row = its message row
 * minus the other rows of that message row, read from the receiving
 * worker's cache before the transition (the caches must still hold C^t). */
cm_status cm_shuffle_decode(const cm_shuffle *shuffle, const void *workspace, cm_shuffle_op op,
                            const void *M, int64_t ldm, const void *caches, int64_t ldc,
                            int64_t r, void *Rx, int64_t ldr, cm_stream_t stream);

/* ---- the planner on the device ---------------------------------------------
 * The same plan as cm_shuffle_next (bit for bit: partition, messages,
 * programs, cache update, slot tables), computed on the GPU with the state
 * resident in a caller-owned workspace, for n <= 16.  After
 * cm_shuffle_device_init the instance is in device mode: cm_shuffle_next and
 * cm_shuffle_upload return CM_EINVAL, cm_shuffle_device_next plans each
 * transition, the data-plane calls take this workspace, and cm_shuffle_plan,
 * cm_shuffle_received and cm_shuffle_caches copy their tables out of it
 * (synchronously). */

/* Bytes of device workspace for the device planner (0 if n > 16): the row
 * programs of cm_shuffle_workspace_bytes first, then the resident state and
 * scratch (about 4 q (n + 21) + 4 n s + 16 max(q, n s) + 8 n 2^n + 2^18 n
 * bytes). */
size_t cm_shuffle_device_workspace_bytes(const cm_shuffle *shuffle);

/* Moves the current host state (and, after a transition, its programs) into
 * `workspace` (16-byte aligned, >= cm_shuffle_device_workspace_bytes) and
 * switches the instance to device mode.  Synchronises `stream`. */
cm_status cm_shuffle_device_init(cm_shuffle *shuffle, void *workspace, size_t bytes,
                                 cm_stream_t stream);

/* Plans the transition t -> t+1 on the device (about 26 launches on
 * `stream`), then reads back its counts (synchronising `stream`); stats is
 * nullable.  The programs are then in place for cm_shuffle_encode, _decode
 * and _commit. */
cm_status cm_shuffle_device_next(cm_shuffle *shuffle, void *workspace, size_t bytes,
                                 cm_shuffle_stats *stats, cm_stream_t stream);

/* Cache update (workers): writes every received row into the cache slot it
 * takes over, turning the caches C^t into C^{t+1}.  Run after the decode of
 * the same transition. */
cm_status cm_shuffle_commit(const cm_shuffle *shuffle, const void *workspace, const void *Rx,
                            int64_t ldr, int64_t r, void *caches, int64_t ldc,
                            cm_stream_t stream);

/* Static description of a status code. */
const char *cm_status_string(cm_status s);

#ifdef __cplusplus
}
#endif
#endif /* CM_H */
