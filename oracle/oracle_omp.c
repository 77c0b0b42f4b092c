/*
 * All-core CPU baseline: the oracle's BICG loops (oracle.c) spread over
 * every host core with OpenMP.
 *
 * TEST INFRASTRUCTURE ONLY, like oracle.c: only the CPU-baseline leg of the
 * benchmark (and the test that checks this file against oracle.c) uses it.
 * It shares nothing with the CUDA library, and nothing with oracle.c but
 * the definitions it restates.
 *
 * Same definition and precision rules as oracle.c (BICG, Table 1 / Table 2:
 * q = A p, s = A^T r; double sums for f32, Dot2 for f64, sums modulo 2^64
 * for i32), and every output is summed in the same order as there, so the
 * results are oracle.c's bit for bit:
 *   q  rows split between threads; row i's terms in ascending column order;
 *   s  blocks of kColBlock columns split between threads; each column's
 *      terms in ascending row order.
 * A is therefore read twice (once for q, once for s).  Build: C99 with
 * -fopenmp, -O2 -fno-fast-math -ffp-contract=off.
 */
#include <math.h>
#include <omp.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define OMP_OK 0
#define OMP_EINVAL 1
#define OMP_ENOMEM 2

static const int64_t kColBlock = 256;

static int omp_check(int64_t M, int64_t N, int64_t lda, const void *A, const void *p,
                     const void *r, const void *q, const void *s)
{
    if (M < 0 || N < 0) return OMP_EINVAL;
    if (lda < N || lda < 1) return OMP_EINVAL;
    if (M > 0 && N > 0 && (A == NULL || p == NULL || r == NULL)) return OMP_EINVAL;
    if (M > 0 && q == NULL) return OMP_EINVAL;
    if (N > 0 && s == NULL) return OMP_EINVAL;
    return OMP_OK;
}

/* Threads a parallel region of this library uses. */
int oracle_omp_threads(void) { return omp_get_max_threads(); }

int oracle_omp_dualmv_f32(int64_t M, int64_t N, const float *A, int64_t lda,
                          const float *p, const float *r, double *q, double *s)
{
    int rc = omp_check(M, N, lda, A, p, r, q, s);
    if (rc) return rc;
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < M; ++i) {
        double qi = 0.0;
        for (int64_t j = 0; j < N; ++j) qi += (double)A[i * lda + j] * (double)p[j];
        q[i] = qi;
    }
    const int64_t nb = (N + kColBlock - 1) / kColBlock;
#pragma omp parallel for schedule(static)
    for (int64_t b = 0; b < nb; ++b) {
        const int64_t j0 = b * kColBlock, j1 = j0 + kColBlock < N ? j0 + kColBlock : N;
        for (int64_t j = j0; j < j1; ++j) s[j] = 0.0;
        for (int64_t i = 0; i < M; ++i) {
            const double ri = (double)r[i];
            for (int64_t j = j0; j < j1; ++j) s[j] += (double)A[i * lda + j] * ri;
        }
    }
    return OMP_OK;
}

/* Knuth's TwoSum and the FMA TwoProduct, as in oracle.c. */
static void two_sum(double x, double y, double *sum, double *err)
{
    const double t = x + y;
    const double z = t - x;
    *err = (x - (t - z)) + (y - z);
    *sum = t;
}

static void two_prod(double x, double y, double *prod, double *err)
{
    const double t = x * y;
    *err = fma(x, y, -t);
    *prod = t;
}

int oracle_omp_dualmv_f64(int64_t M, int64_t N, const double *A, int64_t lda,
                          const double *p, const double *r, double *q, double *s)
{
    int rc = omp_check(M, N, lda, A, p, r, q, s);
    if (rc) return rc;
    double *s_lo = NULL;
    if (N > 0) {
        s_lo = (double *)malloc((size_t)N * sizeof(double));
        if (s_lo == NULL) return OMP_ENOMEM;
    }
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < M; ++i) {
        double hi = 0.0, lo = 0.0, prod, perr, sum, serr;
        for (int64_t j = 0; j < N; ++j) {
            two_prod(A[i * lda + j], p[j], &prod, &perr);
            two_sum(hi, prod, &sum, &serr);
            hi = sum;
            lo = lo + (perr + serr);
        }
        q[i] = hi + lo;
    }
    const int64_t nb = (N + kColBlock - 1) / kColBlock;
#pragma omp parallel for schedule(static)
    for (int64_t b = 0; b < nb; ++b) {
        const int64_t j0 = b * kColBlock, j1 = j0 + kColBlock < N ? j0 + kColBlock : N;
        for (int64_t j = j0; j < j1; ++j) { s[j] = 0.0; s_lo[j] = 0.0; }
        for (int64_t i = 0; i < M; ++i) {
            const double ri = r[i];
            for (int64_t j = j0; j < j1; ++j) {
                double prod, perr, sum, serr;
                two_prod(A[i * lda + j], ri, &prod, &perr);
                two_sum(s[j], prod, &sum, &serr);
                s[j] = sum;
                s_lo[j] = s_lo[j] + (perr + serr);
            }
        }
        for (int64_t j = j0; j < j1; ++j) s[j] = s[j] + s_lo[j];
    }
    free(s_lo);
    return OMP_OK;
}

int oracle_omp_dualmv_i32(int64_t M, int64_t N, const int32_t *A, int64_t lda,
                          const int32_t *p, const int32_t *r, int64_t *q, int64_t *s)
{
    int rc = omp_check(M, N, lda, A, p, r, q, s);
    if (rc) return rc;
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < M; ++i) {
        uint64_t qi = 0u;
        for (int64_t j = 0; j < N; ++j)
            qi += (uint64_t)((int64_t)A[i * lda + j] * (int64_t)p[j]);
        memcpy(&q[i], &qi, sizeof qi);
    }
    const int64_t nb = (N + kColBlock - 1) / kColBlock;
#pragma omp parallel for schedule(static)
    for (int64_t b = 0; b < nb; ++b) {
        const int64_t j0 = b * kColBlock, j1 = j0 + kColBlock < N ? j0 + kColBlock : N;
        uint64_t acc[256];
        for (int64_t j = j0; j < j1; ++j) acc[j - j0] = 0u;
        for (int64_t i = 0; i < M; ++i) {
            const int64_t ri = (int64_t)r[i];
            for (int64_t j = j0; j < j1; ++j)
                acc[j - j0] += (uint64_t)((int64_t)A[i * lda + j] * ri);
        }
        for (int64_t j = j0; j < j1; ++j) memcpy(&s[j], &acc[j - j0], sizeof(uint64_t));
    }
    return OMP_OK;
}
