/*
 * whtmix_oracle.c -- CPU oracle for the WHTMix token mixer.  TEST INFRASTRUCTURE ONLY.
 *
 * Only the tests, the smoke check and the bench's CPU-baseline / reference legs may load this
 * file's library.  It shares no code with the CUDA path and is deliberately plain and slow:
 * float64 arithmetic (uint32 with wrap-around for the integer mode), single-threaded, the
 * textbook radix-2 fast Walsh-Hadamard transform applied along rows, then along columns.
 *
 * What it computes (paper Section III-B, Eq. 1-4, "Walsh-Hadamard Token Mixer"):
 *   H_n is the n x n Sylvester-Hadamard matrix, (H_n)_{ij} = (-1)^{popcount(i & j)}, n = 2^k;
 *   the orthonormal transform is H_n / sqrt(n), which is symmetric and its own inverse.
 *   For one plane X [N, C] (tokens x channels) and a gain matrix G [N, C]:
 *       Y = H_N ( G (.) (H_N X H_C) ) H_C / (N C)                               (floating point)
 *       Y = H_N ( G (.) (H_N X H_C) ) H_C            mod 2^32                 (integer mode)
 *   The paper's separable log-domain gains are the rank-1 case G = exp(g_t) exp(g_c)^T; its
 *   channel mix (Eq. 2) and token mix (Eq. 3) act on different axes and commute, so the 2D
 *   form with one elementwise gain is the same map.  The orthonormal 1/sqrt(n) factors of the
 *   four transforms multiply to 1/(N C), applied once at the gain step.  W_in / W_out (Eq. 1
 *   and Eq. 4) are dense projections outside this map.
 *
 * Backward (not printed in the paper, which trains the block: Section IV-A; it follows from the
 * map being linear in X and in G, with H symmetric):
 *       dX_b = H_N ( G (.) (H_N dY_b H_C) ) H_C / (N C)
 *       dG   = sum_{b = 0, 1, ..., B-1} (H_N X_b H_C) (.) (H_N dY_b H_C) / (N C)
 *   (integer mode: no 1/(N C), mod 2^32).
 *
 * Layout: X, Y, dY, dX are row-major [B, N, C] (c fastest); G and dG are row-major [N, C].
 * N and C must be powers of two (the paper zero-pads the token axis to the next power of two
 * before the transform; padding is the caller's job here).
 *
 * Threads: single-threaded unless oracle_set_threads(k > 1) is called, which only the timed
 * all-core CPU baseline does.  The threaded mode splits work whose pieces are independent -- the
 * token rows of a row transform, blocks of channel columns of a column transform, the elements
 * of the gain step -- so every element goes through exactly the same additions in the same order
 * and the results are bit-identical to the single-threaded ones.
 */
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

static int g_threads = 1;

/* Number of OpenMP threads the next calls use (1: the plain single-threaded loops).  Returns the
 * count in effect (always 1 when built without OpenMP). */
int oracle_set_threads(int k) {
#ifdef _OPENMP
    g_threads = k < 1 ? 1 : k;
#else
    (void)k;
    g_threads = 1;
#endif
    return g_threads;
}

static int is_pow2(int64_t n) { return n > 0 && (n & (n - 1)) == 0; }

/* In-place unnormalised FWHT of n = 2^k values spaced `stride` apart, natural (Sylvester)
 * order: for h = 1, 2, 4, ..., n/2, every pair (j, j + h) inside each block of 2h becomes
 * (a + b, a - b).  (Fino & Algazi, IEEE Trans. Computers, 1976.) */
void oracle_fwht_f64(double *v, int64_t n, int64_t stride) {
    for (int64_t h = 1; h < n; h *= 2)
        for (int64_t i = 0; i < n; i += 2 * h)
            for (int64_t j = i; j < i + h; ++j) {
                double a = v[j * stride], b = v[(j + h) * stride];
                v[j * stride] = a + b;
                v[(j + h) * stride] = a - b;
            }
}

void oracle_fwht_u32(uint32_t *v, int64_t n, int64_t stride) {
    for (int64_t h = 1; h < n; h *= 2)
        for (int64_t i = 0; i < n; i += 2 * h)
            for (int64_t j = i; j < i + h; ++j) {
                uint32_t a = v[j * stride], b = v[(j + h) * stride];
                v[j * stride] = a + b;
                v[(j + h) * stride] = a - b;
            }
}

/* The same column transform as applying oracle_fwht_f64 to each of the C columns (stride C):
 * every butterfly pairs row j with row j + h; the channel loop is innermost only so that the
 * rows are walked contiguously.  Each element sees exactly the same additions. */
static void fwht_columns_f64(double *a, int64_t N, int64_t C) {
    for (int64_t h = 1; h < N; h *= 2)
        for (int64_t i = 0; i < N; i += 2 * h)
            for (int64_t j = i; j < i + h; ++j) {
                double *r0 = a + j * C, *r1 = a + (j + h) * C;
                for (int64_t c = 0; c < C; ++c) {
                    double p = r0[c], q = r1[c];
                    r0[c] = p + q;
                    r1[c] = p - q;
                }
            }
}

static void fwht_columns_u32(uint32_t *a, int64_t N, int64_t C) {
    for (int64_t h = 1; h < N; h *= 2)
        for (int64_t i = 0; i < N; i += 2 * h)
            for (int64_t j = i; j < i + h; ++j) {
                uint32_t *r0 = a + j * C, *r1 = a + (j + h) * C;
                for (int64_t c = 0; c < C; ++c) {
                    uint32_t p = r0[c], q = r1[c];
                    r0[c] = p + q;
                    r1[c] = p - q;
                }
            }
}

/* Threaded column transform: each thread takes whole blocks of 8 adjacent channel columns (one
 * 64-byte line of doubles per row) through all the stages; a column sees the same butterflies in
 * the same order as in fwht_columns_f64. */
static void fwht_columns_par_f64(double *a, int64_t N, int64_t C) {
    const int64_t nblk = (C + 7) / 8;
#pragma omp parallel for num_threads(g_threads) schedule(static)
    for (int64_t blk = 0; blk < nblk; ++blk) {
        const int64_t c0 = 8 * blk, c1 = c0 + 8 < C ? c0 + 8 : C;
        for (int64_t h = 1; h < N; h *= 2)
            for (int64_t i = 0; i < N; i += 2 * h)
                for (int64_t j = i; j < i + h; ++j) {
                    double *r0 = a + j * C, *r1 = a + (j + h) * C;
                    for (int64_t c = c0; c < c1; ++c) {
                        double p = r0[c], q = r1[c];
                        r0[c] = p + q;
                        r1[c] = p - q;
                    }
                }
    }
}

static void fwht_rows_f64(double *a, int64_t N, int64_t C) {
#pragma omp parallel for num_threads(g_threads) schedule(static) if (g_threads > 1)
    for (int64_t n = 0; n < N; ++n) oracle_fwht_f64(a + n * C, C, 1);
}

/* A <- H_N A H_C: the channel transform on every token row (Eq. 2's H_C), then the token
 * transform on every channel column (Eq. 3's H_N). */
static void wht2d_f64(double *a, int64_t N, int64_t C) {
    fwht_rows_f64(a, N, C);
    if (g_threads > 1)
        fwht_columns_par_f64(a, N, C);
    else
        fwht_columns_f64(a, N, C);
}

static void wht2d_u32(uint32_t *a, int64_t N, int64_t C) {
    for (int64_t n = 0; n < N; ++n) oracle_fwht_u32(a + n * C, C, 1);
    fwht_columns_u32(a, N, C);
}

/* Inverse order of the same two transforms (columns, then rows); H is its own inverse up to
 * the scale, so only the order differs. */
static void wht2d_inv_f64(double *a, int64_t N, int64_t C) {
    if (g_threads > 1)
        fwht_columns_par_f64(a, N, C);
    else
        fwht_columns_f64(a, N, C);
    fwht_rows_f64(a, N, C);
}

static void wht2d_inv_u32(uint32_t *a, int64_t N, int64_t C) {
    fwht_columns_u32(a, N, C);
    for (int64_t n = 0; n < N; ++n) oracle_fwht_u32(a + n * C, C, 1);
}

/* Public entry: the 2D transform alone, out = H_N X H_C (unnormalised), per plane. */
int oracle_wht2d_f64(const double *x, double *out, int64_t B, int64_t N, int64_t C) {
    if (!is_pow2(N) || !is_pow2(C) || B < 0) return 2;
    const int64_t L = N * C;
    memcpy(out, x, (size_t)(B * L) * sizeof(double));
    for (int64_t b = 0; b < B; ++b) wht2d_f64(out + b * L, N, C);
    return 0;
}

/* Forward mixer, floating point: Y_b = H_N (G (.) H_N X_b H_C) H_C / (N C), per plane b. */
int oracle_forward_f64(const double *x, const double *g, double *y, int64_t B, int64_t N, int64_t C) {
    if (!is_pow2(N) || !is_pow2(C) || B < 0) return 2;
    const int64_t L = N * C;
    const double inv_l = 1.0 / (double)L;
    for (int64_t b = 0; b < B; ++b) {
        double *a = y + b * L;
        memcpy(a, x + b * L, (size_t)L * sizeof(double));
        wht2d_f64(a, N, C);                                   /* (i), (ii)  */
#pragma omp parallel for num_threads(g_threads) schedule(static) if (g_threads > 1)
        for (int64_t i = 0; i < L; ++i) a[i] = a[i] * g[i] * inv_l; /* (iii) gain and 1/(NC) */
        wht2d_inv_f64(a, N, C);                               /* (iv), (v)  */
    }
    return 0;
}

/* Forward mixer, integer mode: unnormalised, every operation mod 2^32. */
int oracle_forward_u32(const uint32_t *x, const uint32_t *g, uint32_t *y, int64_t B, int64_t N, int64_t C) {
    if (!is_pow2(N) || !is_pow2(C) || B < 0) return 2;
    const int64_t L = N * C;
    for (int64_t b = 0; b < B; ++b) {
        uint32_t *a = y + b * L;
        memcpy(a, x + b * L, (size_t)L * sizeof(uint32_t));
        wht2d_u32(a, N, C);
        for (int64_t i = 0; i < L; ++i) a[i] = a[i] * g[i];
        wht2d_inv_u32(a, N, C);
    }
    return 0;
}

/* Backward, floating point.  dx may not alias x or dy; dg is [N, C] and is overwritten. */
int oracle_backward_f64(const double *x, const double *g, const double *dy, double *dx, double *dg,
                        int64_t B, int64_t N, int64_t C) {
    if (!is_pow2(N) || !is_pow2(C) || B < 0) return 2;
    const int64_t L = N * C;
    const double inv_l = 1.0 / (double)L;
    double *u = (double *)malloc((size_t)L * sizeof(double));
    if (!u) return 6;
    for (int64_t i = 0; i < L; ++i) dg[i] = 0.0;
    for (int64_t b = 0; b < B; ++b) {
        double *v = dx + b * L;
        memcpy(u, x + b * L, (size_t)L * sizeof(double));
        memcpy(v, dy + b * L, (size_t)L * sizeof(double));
        wht2d_f64(u, N, C);                                   /* H X_b H   */
        wht2d_f64(v, N, C);                                   /* H dY_b H  */
#pragma omp parallel for num_threads(g_threads) schedule(static) if (g_threads > 1)
        for (int64_t i = 0; i < L; ++i) {
            dg[i] += u[i] * v[i] * inv_l;                     /* b ascending */
            v[i] = v[i] * g[i] * inv_l;
        }
        wht2d_inv_f64(v, N, C);                               /* dX_b */
    }
    free(u);
    return 0;
}

int oracle_backward_u32(const uint32_t *x, const uint32_t *g, const uint32_t *dy, uint32_t *dx,
                        uint32_t *dg, int64_t B, int64_t N, int64_t C) {
    if (!is_pow2(N) || !is_pow2(C) || B < 0) return 2;
    const int64_t L = N * C;
    uint32_t *u = (uint32_t *)malloc((size_t)L * sizeof(uint32_t));
    if (!u) return 6;
    for (int64_t i = 0; i < L; ++i) dg[i] = 0u;
    for (int64_t b = 0; b < B; ++b) {
        uint32_t *v = dx + b * L;
        memcpy(u, x + b * L, (size_t)L * sizeof(uint32_t));
        memcpy(v, dy + b * L, (size_t)L * sizeof(uint32_t));
        wht2d_u32(u, N, C);
        wht2d_u32(v, N, C);
        for (int64_t i = 0; i < L; ++i) {
            dg[i] += u[i] * v[i];
            v[i] = v[i] * g[i];
        }
        wht2d_inv_u32(v, N, C);
    }
    free(u);
    return 0;
}
