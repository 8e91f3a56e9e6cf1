/*
 * oracle.c -- plain fp64 CPU oracle for MDS-coded matrix multiplication
 * (Lee, Lam, Pedarsani, Papailiopoulos, Ramchandran, "Speeding Up Distributed
 * Machine Learning Using Codes", Sec. III).
 *
 * TEST INFRASTRUCTURE.  Only the test suite, the smoke check and the
 * benchmark's CPU-baseline leg may load this library.  The CUDA library never
 * links, includes or calls it, and the two share no source, header, table or
 * helper.
 *
 * Every function works in fp64 with plain loops, following the definitions
 * of Sec. III in the paper's order.  OpenMP splits independent output rows
 * across threads and never changes a result.
 *
 * Layout conventions (shared with the callers, not with the CUDA library):
 * matrices are row-major; A is m x d with leading dimension lda; X is d x b;
 * the code is (n, k) with generator G = [I_k; P], P the (n-k) x k parity
 * block; L = ceil(m / k) is the block height; coded block j (0-based) is
 * rows [j L, (j+1) L) of the stacked n L x d coded matrix.
 *
 * Status codes returned here: 0 ok, -1 bad argument, -2 fewer than k
 * survivors, -3 singular system.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

int or_num_threads(void)
{
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

/* Threads for the parallel loops that follow (timing only; no arithmetic
 * depends on it: every loop splits independent outputs). */
void or_set_threads(int threads)
{
#ifdef _OPENMP
    if (threads > 0) omp_set_num_threads(threads);
#else
    (void)threads;
#endif
}

/* Sec. III-A, footnote on zero padding: when m is not a multiple of k, zero
 * rows are appended so that A splits into k equal blocks of L = ceil(m/k). */
int64_t or_block_rows(int64_t m, int32_t k)
{
    if (k <= 0 || m < 0) return -1;
    return (m + k - 1) / k;
}

/* Row r of data block i of the zero-padded A, or NULL for an appended zero row. */
static const float *data_row(const float *A, int64_t lda, int64_t m, int64_t L,
                             int32_t i, int64_t r)
{
    int64_t g = (int64_t)i * L + r;
    return g < m ? A + g * lda : NULL;
}

/* Element (i, j) of G = [I_k; P], 0-based. */
static double gen_entry(int32_t k, const double *P, int32_t row, int32_t col)
{
    if (row < k) return row == col ? 1.0 : 0.0;
    return P[(int64_t)(row - k) * k + col];
}

/* Sec. III-A: applying the (n,k) code to each element of the k blocks gives
 * coded block j = sum_i G[j][i] A_i; with a systematic code the first k coded
 * blocks are the data blocks themselves, so only the n-k parity blocks
 * sum_i P[p][i] A_i are formed here.  parity is (n-k) L x d, row-major.
 * absbound (nullable) receives sum_i |P[p][i]| |A_i| per element, the scale
 * of the rounding error of any floating-point evaluation of that sum. */
int or_encode(int32_t n, int32_t k, int64_t m, int64_t d, const double *P,
              const float *A, int64_t lda, double *parity, double *absbound)
{
    if (k < 1 || n <= k || m < 1 || d < 1 || lda < d) return -1;
    int64_t L = or_block_rows(m, k);
    int64_t rows = (int64_t)(n - k) * L;
#pragma omp parallel for schedule(static)
    for (int64_t pr = 0; pr < rows; ++pr) {
        int32_t p = (int32_t)(pr / L);
        int64_t r = pr % L;
        double *out = parity + pr * d;
        double *ab = absbound ? absbound + pr * d : NULL;
        for (int64_t c = 0; c < d; ++c) {
            out[c] = 0.0;
            if (ab) ab[c] = 0.0;
        }
        for (int32_t i = 0; i < k; ++i) {
            const float *a = data_row(A, lda, m, L, i, r);
            if (!a) continue;
            double g = P[(int64_t)p * k + i];
            for (int64_t c = 0; c < d; ++c) {
                out[c] += g * (double)a[c];
                if (ab) ab[c] += fabs(g) * fabs((double)a[c]);
            }
        }
    }
    return 0;
}

/* The computation the coded algorithm reaches (Sec. I-A example, Sec. III-A
 * last paragraph): Y = A X, with Y m x b in fp64. */
int or_matmul(int64_t m, int64_t d, int32_t b, const float *A, int64_t lda,
              const float *X, double *Y)
{
    if (m < 1 || d < 1 || b < 1 || lda < d) return -1;
#pragma omp parallel for schedule(static)
    for (int64_t r = 0; r < m; ++r) {
        const float *a = A + r * lda;
        double *y = Y + r * b;
        for (int32_t v = 0; v < b; ++v) y[v] = 0.0;
        for (int64_t c = 0; c < d; ++c) {
            double av = (double)a[c];
            for (int32_t v = 0; v < b; ++v) y[v] += av * (double)X[c * b + v];
        }
    }
    return 0;
}

/* Sec. III-A protocol: worker j computes its local product, coded block j
 * times X.  Workers j < k hold the data blocks (appended rows are zero);
 * workers j >= k hold the given parity blocks (fp32, ldp-strided).  Output
 * Yt is the stacked n L x b matrix of all worker results, fp64. */
int or_worker_outputs(int32_t n, int32_t k, int64_t m, int64_t d, int32_t b,
                      const float *A, int64_t lda, const float *parity, int64_t ldp,
                      const float *X, double *Yt)
{
    if (k < 1 || n <= k || m < 1 || d < 1 || b < 1 || lda < d || ldp < d) return -1;
    int64_t L = or_block_rows(m, k);
    int64_t rows = (int64_t)n * L;
#pragma omp parallel for schedule(static)
    for (int64_t jr = 0; jr < rows; ++jr) {
        int32_t j = (int32_t)(jr / L);
        int64_t r = jr % L;
        const float *a = j < k ? data_row(A, lda, m, L, j, r)
                               : parity + ((int64_t)(j - k) * L + r) * ldp;
        double *y = Yt + jr * b;
        for (int32_t v = 0; v < b; ++v) y[v] = 0.0;
        if (!a) continue;
        for (int64_t c = 0; c < d; ++c) {
            double av = (double)a[c];
            for (int32_t v = 0; v < b; ++v) y[v] += av * (double)X[c * b + v];
        }
    }
    return 0;
}

/* Same worker products with fp64 parity blocks (the exact code of or_encode). */
int or_worker_outputs_f64(int32_t n, int32_t k, int64_t m, int64_t d, int32_t b,
                          const float *A, int64_t lda, const double *parity, int64_t ldp,
                          const float *X, double *Yt)
{
    if (k < 1 || n <= k || m < 1 || d < 1 || b < 1 || lda < d || ldp < d) return -1;
    int64_t L = or_block_rows(m, k);
    int64_t rows = (int64_t)n * L;
#pragma omp parallel for schedule(static)
    for (int64_t jr = 0; jr < rows; ++jr) {
        int32_t j = (int32_t)(jr / L);
        int64_t r = jr % L;
        double *y = Yt + jr * b;
        for (int32_t v = 0; v < b; ++v) y[v] = 0.0;
        if (j < k) {
            const float *a = data_row(A, lda, m, L, j, r);
            if (!a) continue;
            for (int64_t c = 0; c < d; ++c)
                for (int32_t v = 0; v < b; ++v) y[v] += (double)a[c] * (double)X[c * b + v];
        } else {
            const double *a = parity + ((int64_t)(j - k) * L + r) * ldp;
            for (int64_t c = 0; c < d; ++c)
                for (int32_t v = 0; v < b; ++v) y[v] += a[c] * (double)X[c * b + v];
        }
    }
    return 0;
}

/* bf16 values are the upper 16 bits of an fp32; widening is exact. */
static double bf16_to_double(uint16_t h)
{
    uint32_t u = (uint32_t)h << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

/* Same as or_encode for bf16 data (raw bf16 bits), result in fp64. */
int or_encode_bf16(int32_t n, int32_t k, int64_t m, int64_t d, const double *P,
                   const uint16_t *A, int64_t lda, double *parity, double *absbound)
{
    if (k < 1 || n <= k || m < 1 || d < 1 || lda < d) return -1;
    int64_t L = or_block_rows(m, k);
    int64_t rows = (int64_t)(n - k) * L;
#pragma omp parallel for schedule(static)
    for (int64_t pr = 0; pr < rows; ++pr) {
        int32_t p = (int32_t)(pr / L);
        int64_t r = pr % L;
        double *out = parity + pr * d;
        double *ab = absbound ? absbound + pr * d : NULL;
        for (int64_t c = 0; c < d; ++c) {
            out[c] = 0.0;
            if (ab) ab[c] = 0.0;
        }
        for (int32_t i = 0; i < k; ++i) {
            int64_t g = (int64_t)i * L + r;
            if (g >= m) continue;
            const uint16_t *a = A + g * lda;
            double coef = P[(int64_t)p * k + i];
            for (int64_t c = 0; c < d; ++c) {
                double av = bf16_to_double(a[c]);
                out[c] += coef * av;
                if (ab) ab[c] += fabs(coef) * fabs(av);
            }
        }
    }
    return 0;
}

/* Worker products for the matrix-matrix variant (Sec. I-A: X may have s
 * columns), on bf16 coded blocks: C~_j = A~_j B in fp64.  B is d x N bf16. */
int or_worker_outputs_bf16(int32_t n, int32_t k, int64_t m, int64_t d, int32_t N,
                           const uint16_t *A, int64_t lda, const uint16_t *parity,
                           int64_t ldp, const uint16_t *B, double *Ct)
{
    if (k < 1 || n <= k || m < 1 || d < 1 || N < 1 || lda < d || ldp < d) return -1;
    int64_t L = or_block_rows(m, k);
    int64_t rows = (int64_t)n * L;
#pragma omp parallel for schedule(static)
    for (int64_t jr = 0; jr < rows; ++jr) {
        int32_t j = (int32_t)(jr / L);
        int64_t r = jr % L;
        const uint16_t *a = NULL;
        if (j < k) {
            int64_t g = (int64_t)j * L + r;
            if (g < m) a = A + g * lda;
        } else {
            a = parity + ((int64_t)(j - k) * L + r) * ldp;
        }
        double *y = Ct + jr * N;
        for (int32_t v = 0; v < N; ++v) y[v] = 0.0;
        if (!a) continue;
        for (int64_t c = 0; c < d; ++c) {
            double av = bf16_to_double(a[c]);
            if (av == 0.0) continue;
            const uint16_t *brow = B + c * N;
            for (int32_t v = 0; v < N; ++v) y[v] += av * bf16_to_double(brow[v]);
        }
    }
    return 0;
}

/* ---- straggler model (Sec. III-C, III-D) ------------------------------- */

/* SplitMix64 output function (Steele, Lea and Flood, "Fast splittable
 * pseudorandom number generators", OOPSLA 2014): the published
 * finaliser applied to a Weyl-sequence state. */
static uint64_t splitmix64_mix(uint64_t z)
{
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
    return z ^ (z >> 31);
}

/* The i-th output (i >= 1) of the SplitMix64 stream started at state seed. */
uint64_t or_splitmix64(uint64_t seed, uint64_t i)
{
    return splitmix64_mix(seed + i * 0x9E3779B97F4A7C15ULL);
}

/* Sec. III-C/III-D: each of the n tasks of a k-way split runs for a time
 * distributed as the mother distribution scaled by 1/k, P(T_j <= t) = F(k t),
 * with the shifted exponential mother F(t) = 1 - exp(-mu (t - shift)).  So
 * T_j = (shift + E_j / mu) / k with E_j ~ Exp(1), drawn by inversion from the
 * 53-bit uniform U_j = (z_j >> 11) 2^-53, E_j = -log(1 - U_j).  Worker j's
 * draw in round `counter` is output (counter n + j + 1) of the stream at
 * `seed`.  An MDS-coded run ends at the k-th arrival (eq. for the MDS
 * runtime, T_(k)), so the survivors are the k workers with the smallest
 * T_j.  Since T_j increases with (z_j >> 11), the ranking compares those
 * integers, ties going to the lower worker index; the times are reported
 * only.  Writes the survivor bitmask (bit j = worker j) and, if non-NULL,
 * the n times. */
int or_draw_erasures(uint64_t seed, uint64_t counter, int32_t n, int32_t k,
                     double shift, double rate, uint32_t *survivors, double *times)
{
    if (n < 1 || n > 32 || k < 1 || k > n || !(rate > 0.0)) return -1;
    uint64_t key[32];
    for (int32_t j = 0; j < n; ++j) {
        uint64_t z = or_splitmix64(seed, counter * (uint64_t)n + (uint64_t)j + 1);
        key[j] = z >> 11;
        if (times) {
            double u = (double)key[j] * 0x1.0p-53;
            double e = -log1p(-u);
            times[j] = (shift + e / rate) / (double)k;
        }
    }
    uint32_t mask = 0;
    for (int32_t j = 0; j < n; ++j) {
        /* rank of worker j = number of workers strictly ahead of it */
        int32_t ahead = 0;
        for (int32_t i = 0; i < n; ++i)
            if (key[i] < key[j] || (key[i] == key[j] && i < j)) ++ahead;
        if (ahead < k) mask |= 1u << j;
    }
    *survivors = mask;
    return 0;
}

/* ---- decoding (Sec. III-A, Example "MDS codes") ---------------------------
 * Any k of the n results determine A X: with S the surviving workers, the k
 * results satisfy Yt_S = G_S Z, where G_S is the k x k submatrix of G on rows
 * S and Z stacks the k uncoded block products A_i X.  The oracle solves this
 * system by Gaussian elimination with partial pivoting and back substitution
 * in fp64, then concatenates the blocks (dropping appended zero rows).  When
 * more than k workers survive, the k lowest indices are used. */
static int survivor_list(int32_t n, int32_t k, uint32_t mask, int32_t *S)
{
    int32_t cnt = 0;
    for (int32_t j = 0; j < n && cnt < k; ++j)
        if (mask & (1u << j)) S[cnt++] = j;
    return cnt == k ? 0 : -2;
}

int or_decode(int32_t n, int32_t k, int64_t m, int64_t b, const double *P,
              uint32_t survivors, const double *Yt, double *Y)
{
    if (k < 1 || n <= k || n > 32 || m < 1 || b < 1) return -1;
    if (n < 32 && (survivors >> n)) return -1;
    int32_t S[32];
    if (survivor_list(n, k, survivors, S)) return -2;
    int64_t L = or_block_rows(m, k);
    int64_t w = L * b;                       /* right-hand-side width per block */
    double *G = malloc(sizeof(double) * k * k);
    double *R = malloc(sizeof(double) * k * w);
    if (!G || !R) { free(G); free(R); return -1; }
    for (int32_t a = 0; a < k; ++a) {
        for (int32_t c = 0; c < k; ++c) G[a * k + c] = gen_entry(k, P, S[a], c);
        memcpy(R + a * w, Yt + (int64_t)S[a] * w, sizeof(double) * w);
    }
    int status = 0;
    for (int32_t c = 0; c < k && !status; ++c) {
        int32_t piv = c;
        for (int32_t a = c + 1; a < k; ++a)
            if (fabs(G[a * k + c]) > fabs(G[piv * k + c])) piv = a;
        if (!(fabs(G[piv * k + c]) > 0.0)) { status = -3; break; }
        if (piv != c) {
            for (int32_t t = 0; t < k; ++t) {
                double tmp = G[c * k + t]; G[c * k + t] = G[piv * k + t]; G[piv * k + t] = tmp;
            }
            for (int64_t t = 0; t < w; ++t) {
                double tmp = R[c * w + t]; R[c * w + t] = R[piv * w + t]; R[piv * w + t] = tmp;
            }
        }
        for (int32_t a = c + 1; a < k; ++a) {
            double f = G[a * k + c] / G[c * k + c];
            if (f == 0.0) continue;
            for (int32_t t = c; t < k; ++t) G[a * k + t] -= f * G[c * k + t];
            for (int64_t t = 0; t < w; ++t) R[a * w + t] -= f * R[c * w + t];
        }
    }
    if (!status) {
        /* back substitution, in place in R: block c of Z */
        for (int32_t c = k - 1; c >= 0; --c) {
            for (int32_t t = c + 1; t < k; ++t) {
                double g = G[c * k + t];
                if (g == 0.0) continue;
                for (int64_t u = 0; u < w; ++u) R[c * w + u] -= g * R[t * w + u];
            }
            double inv = G[c * k + c];
            for (int64_t u = 0; u < w; ++u) R[c * w + u] /= inv;
        }
        /* concatenation: Y = [Z_0; Z_1; ...] truncated to the m real rows */
        memcpy(Y, R, sizeof(double) * m * b);
    }
    free(G);
    free(R);
    return status;
}

/* fp64 inverse of G_S by the same elimination (identity right-hand side);
 * used to report the conditioning of each decode. */
int or_generator_inverse(int32_t n, int32_t k, const double *P, uint32_t survivors,
                         double *Ginv)
{
    if (k < 1 || n <= k || n > 32) return -1;
    int32_t S[32];
    if (survivor_list(n, k, survivors, S)) return -2;
    /* Solve G_S Z = I by treating the identity as k "blocks" of width k. */
    double *G = malloc(sizeof(double) * k * k);
    double *R = malloc(sizeof(double) * k * k);
    if (!G || !R) { free(G); free(R); return -1; }
    for (int32_t a = 0; a < k; ++a)
        for (int32_t c = 0; c < k; ++c) {
            G[a * k + c] = gen_entry(k, P, S[a], c);
            R[a * k + c] = a == c ? 1.0 : 0.0;
        }
    int status = 0;
    for (int32_t c = 0; c < k; ++c) {
        int32_t piv = c;
        for (int32_t a = c + 1; a < k; ++a)
            if (fabs(G[a * k + c]) > fabs(G[piv * k + c])) piv = a;
        if (!(fabs(G[piv * k + c]) > 0.0)) { status = -3; break; }
        for (int32_t t = 0; t < k; ++t) {
            double tmp = G[c * k + t]; G[c * k + t] = G[piv * k + t]; G[piv * k + t] = tmp;
            tmp = R[c * k + t]; R[c * k + t] = R[piv * k + t]; R[piv * k + t] = tmp;
        }
        for (int32_t a = c + 1; a < k; ++a) {
            double f = G[a * k + c] / G[c * k + c];
            for (int32_t t = 0; t < k; ++t) {
                G[a * k + t] -= f * G[c * k + t];
                R[a * k + t] -= f * R[c * k + t];
            }
        }
    }
    if (!status) {
        for (int32_t c = k - 1; c >= 0; --c) {
            for (int32_t t = c + 1; t < k; ++t)
                for (int32_t u = 0; u < k; ++u) R[c * k + u] -= G[c * k + t] * R[t * k + u];
            for (int32_t u = 0; u < k; ++u) R[c * k + u] /= G[c * k + c];
        }
        memcpy(Ginv, R, sizeof(double) * k * k);
    }
    free(G);
    free(R);
    return status;
}

/* ---- gradient descent (Sec. III-E) -----------------------------------------
 * Linear regression min 0.5 ||A x - y||^2 by the exact-gradient iteration
 * x_{t+1} = x_t - eta A^T (A x_t - y) (eq. for the exact gradient step).  The
 * coded variant decodes both products exactly, so its iterates are these
 * iterates whatever the erasure sets; the oracle runs the plain iteration.
 * x holds x_0 on entry and x_iters on return. */
int or_gd(int64_t m, int64_t d, const float *A, int64_t lda, const float *y,
          double eta, int32_t iters, double *x)
{
    if (m < 1 || d < 1 || lda < d || iters < 0) return -1;
    double *z = malloc(sizeof(double) * m);
    double *g = malloc(sizeof(double) * d);
    if (!z || !g) { free(z); free(g); return -1; }
    for (int32_t t = 0; t < iters; ++t) {
        /* z = A x - y */
#pragma omp parallel for schedule(static)
        for (int64_t r = 0; r < m; ++r) {
            const float *a = A + r * lda;
            double s = 0.0;
            for (int64_t c = 0; c < d; ++c) s += (double)a[c] * x[c];
            z[r] = s - (double)y[r];
        }
        /* g = A^T z: every g[c] sums over r = 0, 1, ..., m-1 in order; each
         * thread owns a slab of columns and streams the rows through it. */
        const int64_t slab = 256;
#pragma omp parallel for schedule(static)
        for (int64_t c0 = 0; c0 < d; c0 += slab) {
            int64_t c1 = c0 + slab < d ? c0 + slab : d;
            for (int64_t c = c0; c < c1; ++c) g[c] = 0.0;
            for (int64_t r = 0; r < m; ++r) {
                const float *a = A + r * lda;
                double zr = z[r];
                for (int64_t c = c0; c < c1; ++c) g[c] += (double)a[c] * zr;
            }
        }
        for (int64_t c = 0; c < d; ++c) x[c] -= eta * g[c];
    }
    free(z);
    free(g);
    return 0;
}

/* ---- runtime model (Sec. III-B, III-C, III-D) ---------------------------------
 * Overall runtime of one round under the shifted-exponential model, from the
 * same worker draws as or_draw_erasures.  scheme 0: uncoded, the job split n
 * ways and the round ends with the last task (eq. for the uncoded runtime);
 * scheme 1: n/k-repetition, block i held by workers i, i+k, i+2k, ... and the
 * round ends when every block has one finished replica (eq. for the
 * repetition runtime); scheme 2: (n,k) MDS, the round ends at the k-th
 * arrival (eq. for the MDS runtime).  Writes `count` runtimes. */
int or_runtime_simulate(int32_t scheme, int32_t n, int32_t k, double shift, double rate,
                        uint64_t seed, uint64_t counter0, int64_t count, double *T)
{
    if (n < 1 || n > 32 || !(rate > 0.0) || scheme < 0 || scheme > 2) return -1;
    if (scheme != 0 && (k < 1 || k > n)) return -1;
    if (scheme == 1 && n % k) return -1;
    int32_t split = scheme == 0 ? n : k;
    for (int64_t c = 0; c < count; ++c) {
        double t[32];
        for (int32_t j = 0; j < n; ++j) {
            uint64_t z = or_splitmix64(seed, (counter0 + (uint64_t)c) * (uint64_t)n + (uint64_t)j + 1);
            double u = (double)(z >> 11) * 0x1.0p-53;
            t[j] = (shift - log1p(-u) / rate) / (double)split;
        }
        double r;
        if (scheme == 0) {
            r = t[0];
            for (int32_t j = 1; j < n; ++j) if (t[j] > r) r = t[j];
        } else if (scheme == 1) {
            r = 0.0;
            for (int32_t i = 0; i < k; ++i) {
                double g = t[i];
                for (int32_t j = i + k; j < n; j += k) if (t[j] < g) g = t[j];
                if (g > r) r = g;
            }
        } else {
            /* k-th smallest by counting: the time with exactly k-1 smaller ones */
            r = 0.0;
            for (int32_t j = 0; j < n; ++j) {
                int32_t below = 0, tie = 0;
                for (int32_t i = 0; i < n; ++i) {
                    if (t[i] < t[j]) ++below;
                    else if (t[i] == t[j] && i < j) ++tie;
                }
                if (below + tie == k - 1) r = t[j];
            }
        }
        T[c] = r;
    }
    return 0;
}

/* Example "Repetition codes": the decodable sets of an n/k-repetition code are
 * the products of the replica groups; this picks, for every block i, the
 * lowest surviving worker among i, i+k, i+2k, ...  Returns -2 if some block
 * has no surviving replica. */
int or_repetition_select(int32_t n, int32_t k, uint32_t survivors, uint32_t *selected)
{
    if (k < 1 || n <= k || n > 32 || n % k) return -1;
    uint32_t sel = 0;
    for (int32_t i = 0; i < k; ++i) {
        int32_t pick = -1;
        for (int32_t j = i; j < n && pick < 0; j += k)
            if (survivors & (1u << j)) pick = j;
        if (pick < 0) return -2;
        sel |= 1u << pick;
    }
    *selected = sel;
    return 0;
}
