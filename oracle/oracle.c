/*
 * CPU oracle for the fused dual matrix-vector product (PolyBench BICG).
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product path links, loads or
 * calls this file: only the test suite, the package smoke check and the
 * CPU-baseline leg of the benchmark use it.  It shares no code, header,
 * table or helper with the CUDA library.
 *
 * What it computes.  The paper optimises the PolyBench BICG kernel (Table 1,
 * row "BICG", NVIDIA platform; Table 2, row "BICG", DCU platform; Section 4.2)
 * but prints no formula for it.  The definition used here is the standard
 * BiCG sub-kernel of PolyBench:
 *
 *     q_i = sum_{j=0}^{N-1} A[i*lda + j] * p_j        (i = 0..M-1)
 *     s_j = sum_{i=0}^{M-1} A[i*lda + j] * r_i        (j = 0..N-1)
 *
 * A is M x N, row-major, with leading dimension lda >= N.  Columns
 * N..lda-1 of each row (padding) are never read.  Both sums run in
 * ascending index order, one term at a time, with no blocking.
 *
 * Precision of each flavour:
 *   f32 -> every product of two floats is exact in double, and the sum is
 *          kept in double; the result is returned in double (not rounded
 *          back to float) so that it is a better reference than the float
 *          result under test.
 *   f64 -> compensated dot product "Dot2" (Ogita, Rump and Oishi,
 *          "Accurate sum and dot product", SIAM J. Sci. Comput. 26(6),
 *          2005): each product is split exactly with an FMA (TwoProduct),
 *          each addition exactly with Knuth's TwoSum, and the error terms
 *          are summed separately and added once at the end.  The result is
 *          as accurate as if computed in twice the working precision and
 *          then rounded.
 *   i32 -> products formed exactly in 64 bits, sums taken modulo 2^64
 *          (two's complement wrap), returned as int64.  Modular addition is
 *          associative, so any summation order gives the same bits.
 *
 * Also provided: the magnitude sums  sum_j |A_ij||p_j|  and
 * sum_i |A_ij||r_i|  in double, the denominators of the parity metric
 * max |err| / sum |A||x|; and two more PolyBench kernels of the paper's
 * tables built from the same products, with the same precision rules:
 *     GESUMMV  y = alpha (A x) + beta (B x)       (Table 1, Table 2)
 *     ATAX     y = A^T (A x)                      (Table 1)
 *     GEMVER   A_hat = A + u1 v1^T + u2 v2^T, x = x + beta A_hat^T y + z,
 *              w = w + alpha A_hat x              (Table 1, Table 2)
 *
 * Build: plain C99, -O2 -fno-fast-math -ffp-contract=off, so the compiler
 * neither reassociates the sums nor fuses a multiply into an add.
 *
 * Return codes: 0 success, 1 invalid argument, 2 out of host memory.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define ORACLE_OK 0
#define ORACLE_EINVAL 1
#define ORACLE_ENOMEM 2

static int oracle_check(int64_t M, int64_t N, int64_t lda, const void *A,
                        const void *p, const void *r, const void *q,
                        const void *s)
{
    if (M < 0 || N < 0) return ORACLE_EINVAL;
    if (lda < N || lda < 1) return ORACLE_EINVAL;
    if (M > 0 && N > 0 && (A == NULL || p == NULL || r == NULL)) return ORACLE_EINVAL;
    if (M > 0 && q == NULL) return ORACLE_EINVAL;
    if (N > 0 && s == NULL) return ORACLE_EINVAL;
    return ORACLE_OK;
}

/* ---------------------------------------------------------------- f32 --- */

/* BICG (Table 1 / Table 2) on float inputs, double accumulation. */
int oracle_dualmv_f32(int64_t M, int64_t N, const float *A, int64_t lda,
                      const float *p, const float *r, double *q, double *s)
{
    int rc = oracle_check(M, N, lda, A, p, r, q, s);
    if (rc) return rc;
    for (int64_t j = 0; j < N; ++j) s[j] = 0.0;
    for (int64_t i = 0; i < M; ++i) {
        double qi = 0.0;
        const double ri = (double)r[i];
        for (int64_t j = 0; j < N; ++j) {
            const double a = (double)A[i * lda + j];
            qi += a * (double)p[j];
            s[j] += a * ri;
        }
        q[i] = qi;
    }
    return ORACLE_OK;
}

/* ---------------------------------------------------------------- f64 --- */

/* Knuth's TwoSum: x + y = *sum + *err exactly, *sum = fl(x + y). */
static void two_sum(double x, double y, double *sum, double *err)
{
    const double t = x + y;
    const double z = t - x;
    *err = (x - (t - z)) + (y - z);
    *sum = t;
}

/* TwoProduct with a fused multiply-add: x * y = *prod + *err exactly. */
static void two_prod(double x, double y, double *prod, double *err)
{
    const double t = x * y;
    *err = fma(x, y, -t);
    *prod = t;
}

/* BICG (Table 1 / Table 2) on double inputs, Dot2 accumulation.  Each output
 * keeps a running sum (hi) and a running sum of the exact error terms (lo);
 * the result is hi + lo, rounded once. */
int oracle_dualmv_f64(int64_t M, int64_t N, const double *A, int64_t lda,
                      const double *p, const double *r, double *q, double *s)
{
    int rc = oracle_check(M, N, lda, A, p, r, q, s);
    if (rc) return rc;
    double *s_lo = NULL;
    if (N > 0) {
        s_lo = (double *)malloc((size_t)N * sizeof(double));
        if (s_lo == NULL) return ORACLE_ENOMEM;
        for (int64_t j = 0; j < N; ++j) { s[j] = 0.0; s_lo[j] = 0.0; }
    }
    for (int64_t i = 0; i < M; ++i) {
        double q_hi = 0.0, q_lo = 0.0;
        const double ri = r[i];
        for (int64_t j = 0; j < N; ++j) {
            const double a = A[i * lda + j];
            double prod, perr, sum, serr;
            /* row i of A times p */
            two_prod(a, p[j], &prod, &perr);
            two_sum(q_hi, prod, &sum, &serr);
            q_hi = sum;
            q_lo = q_lo + (perr + serr);
            /* column j of A times r */
            two_prod(a, ri, &prod, &perr);
            two_sum(s[j], prod, &sum, &serr);
            s[j] = sum;
            s_lo[j] = s_lo[j] + (perr + serr);
        }
        q[i] = q_hi + q_lo;
    }
    for (int64_t j = 0; j < N; ++j) s[j] = s[j] + s_lo[j];
    free(s_lo);
    return ORACLE_OK;
}

/* ---------------------------------------------------------------- i32 --- */

/* BICG (Table 1 / Table 2) on int32 inputs: exact 64-bit products, sums
 * modulo 2^64.  The arithmetic is done on uint64_t, where wrap-around is
 * defined, and the bits are returned as int64. */
int oracle_dualmv_i32(int64_t M, int64_t N, const int32_t *A, int64_t lda,
                      const int32_t *p, const int32_t *r, int64_t *q,
                      int64_t *s)
{
    int rc = oracle_check(M, N, lda, A, p, r, q, s);
    if (rc) return rc;
    uint64_t *s_acc = NULL;
    if (N > 0) {
        s_acc = (uint64_t *)malloc((size_t)N * sizeof(uint64_t));
        if (s_acc == NULL) return ORACLE_ENOMEM;
        for (int64_t j = 0; j < N; ++j) s_acc[j] = 0u;
    }
    for (int64_t i = 0; i < M; ++i) {
        uint64_t qi = 0u;
        const int64_t ri = (int64_t)r[i];
        for (int64_t j = 0; j < N; ++j) {
            const int64_t a = (int64_t)A[i * lda + j];
            qi += (uint64_t)(a * (int64_t)p[j]);
            s_acc[j] += (uint64_t)(a * ri);
        }
        memcpy(&q[i], &qi, sizeof qi);
    }
    for (int64_t j = 0; j < N; ++j) memcpy(&s[j], &s_acc[j], sizeof(uint64_t));
    free(s_acc);
    return ORACLE_OK;
}

/* ------------------------------------------------- parity denominators --- */

/* qa_i = sum_j |A_ij| |p_j|,  sa_j = sum_i |A_ij| |r_i|, in double.  These
 * scale the error of each output in the parity metric. */
int oracle_absdot_f32(int64_t M, int64_t N, const float *A, int64_t lda,
                      const float *p, const float *r, double *qa, double *sa)
{
    int rc = oracle_check(M, N, lda, A, p, r, qa, sa);
    if (rc) return rc;
    for (int64_t j = 0; j < N; ++j) sa[j] = 0.0;
    for (int64_t i = 0; i < M; ++i) {
        double acc = 0.0;
        const double ri = fabs((double)r[i]);
        for (int64_t j = 0; j < N; ++j) {
            const double a = fabs((double)A[i * lda + j]);
            acc += a * fabs((double)p[j]);
            sa[j] += a * ri;
        }
        qa[i] = acc;
    }
    return ORACLE_OK;
}

int oracle_absdot_f64(int64_t M, int64_t N, const double *A, int64_t lda,
                      const double *p, const double *r, double *qa, double *sa)
{
    int rc = oracle_check(M, N, lda, A, p, r, qa, sa);
    if (rc) return rc;
    for (int64_t j = 0; j < N; ++j) sa[j] = 0.0;
    for (int64_t i = 0; i < M; ++i) {
        double acc = 0.0;
        const double ri = fabs(r[i]);
        for (int64_t j = 0; j < N; ++j) {
            const double a = fabs(A[i * lda + j]);
            acc += a * fabs(p[j]);
            sa[j] += a * ri;
        }
        qa[i] = acc;
    }
    return ORACLE_OK;
}

/* ---------------------------------------------------- trimmed mean ------ */

/* Eq. 3 of the paper (Section 3.2): sort the R timings ascending, drop the k
 * lowest and the k highest, and average the rest.  Requires R > 2k.  The
 * input array is sorted in place (insertion sort: R is small). */
int oracle_trimmed_mean(double *t, int64_t R, int64_t k, double *out)
{
    if (t == NULL || out == NULL || k < 0 || R <= 2 * k) return ORACLE_EINVAL;
    for (int64_t a = 1; a < R; ++a) {
        const double key = t[a];
        int64_t b = a - 1;
        while (b >= 0 && t[b] > key) { t[b + 1] = t[b]; --b; }
        t[b + 1] = key;
    }
    double sum = 0.0;
    for (int64_t i = k; i < R - k; ++i) sum += t[i];
    *out = sum / (double)(R - 2 * k);
    return ORACLE_OK;
}

/* ------------------------------------------------------------- GESUMMV --- */

/* GESUMMV (Table 1 / Table 2): tmp = A x, yb = B x, y = alpha tmp + beta yb,
 * with A and B M x N (leading dimensions lda, ldb >= N).  Float inputs:
 * exact double products summed in double, result in double. */
int oracle_gesummv_f32(int64_t M, int64_t N, double alpha, const float *A, int64_t lda,
                       double beta, const float *B, int64_t ldb, const float *x, double *y)
{
    if (M < 0 || N < 0 || lda < N || ldb < N || lda < 1 || ldb < 1) return ORACLE_EINVAL;
    if (M > 0 && (y == NULL || (N > 0 && (A == NULL || B == NULL || x == NULL))))
        return ORACLE_EINVAL;
    for (int64_t i = 0; i < M; ++i) {
        double ta = 0.0, tb = 0.0;
        for (int64_t j = 0; j < N; ++j) {
            ta += (double)A[i * lda + j] * (double)x[j];
            tb += (double)B[i * ldb + j] * (double)x[j];
        }
        y[i] = alpha * ta + beta * tb;
    }
    return ORACLE_OK;
}

/* Double inputs: each dot product with Dot2, then alpha tmp + beta yb. */
int oracle_gesummv_f64(int64_t M, int64_t N, double alpha, const double *A, int64_t lda,
                       double beta, const double *B, int64_t ldb, const double *x, double *y)
{
    if (M < 0 || N < 0 || lda < N || ldb < N || lda < 1 || ldb < 1) return ORACLE_EINVAL;
    if (M > 0 && (y == NULL || (N > 0 && (A == NULL || B == NULL || x == NULL))))
        return ORACLE_EINVAL;
    for (int64_t i = 0; i < M; ++i) {
        double a_hi = 0.0, a_lo = 0.0, b_hi = 0.0, b_lo = 0.0;
        for (int64_t j = 0; j < N; ++j) {
            double prod, perr, sum, serr;
            two_prod(A[i * lda + j], x[j], &prod, &perr);
            two_sum(a_hi, prod, &sum, &serr);
            a_hi = sum;
            a_lo = a_lo + (perr + serr);
            two_prod(B[i * ldb + j], x[j], &prod, &perr);
            two_sum(b_hi, prod, &sum, &serr);
            b_hi = sum;
            b_lo = b_lo + (perr + serr);
        }
        y[i] = alpha * (a_hi + a_lo) + beta * (b_hi + b_lo);
    }
    return ORACLE_OK;
}

/* ---------------------------------------------------------------- ATAX --- */

/* ATAX (Table 1): tmp = A x (length M), y = A^T tmp (length N).  Float
 * inputs: both products in double, tmp kept in double. */
int oracle_atax_f32(int64_t M, int64_t N, const float *A, int64_t lda, const float *x,
                    double *y)
{
    if (M < 0 || N < 0 || lda < N || lda < 1) return ORACLE_EINVAL;
    if (N > 0 && (y == NULL || (M > 0 && (A == NULL || x == NULL)))) return ORACLE_EINVAL;
    for (int64_t j = 0; j < N; ++j) y[j] = 0.0;
    for (int64_t i = 0; i < M; ++i) {
        double tmp = 0.0;
        for (int64_t j = 0; j < N; ++j) tmp += (double)A[i * lda + j] * (double)x[j];
        for (int64_t j = 0; j < N; ++j) y[j] += (double)A[i * lda + j] * tmp;
    }
    return ORACLE_OK;
}

/* Double inputs: tmp_i with Dot2 (rounded to double), then each y_j with
 * Dot2 over i of A_ij tmp_i. */
int oracle_atax_f64(int64_t M, int64_t N, const double *A, int64_t lda, const double *x,
                    double *y)
{
    if (M < 0 || N < 0 || lda < N || lda < 1) return ORACLE_EINVAL;
    if (N > 0 && (y == NULL || (M > 0 && (A == NULL || x == NULL)))) return ORACLE_EINVAL;
    double *y_lo = NULL;
    if (N > 0) {
        y_lo = (double *)malloc((size_t)N * sizeof(double));
        if (y_lo == NULL) return ORACLE_ENOMEM;
        for (int64_t j = 0; j < N; ++j) { y[j] = 0.0; y_lo[j] = 0.0; }
    }
    for (int64_t i = 0; i < M; ++i) {
        double t_hi = 0.0, t_lo = 0.0;
        for (int64_t j = 0; j < N; ++j) {
            double prod, perr, sum, serr;
            two_prod(A[i * lda + j], x[j], &prod, &perr);
            two_sum(t_hi, prod, &sum, &serr);
            t_hi = sum;
            t_lo = t_lo + (perr + serr);
        }
        const double tmp = t_hi + t_lo;
        for (int64_t j = 0; j < N; ++j) {
            double prod, perr, sum, serr;
            two_prod(A[i * lda + j], tmp, &prod, &perr);
            two_sum(y[j], prod, &sum, &serr);
            y[j] = sum;
            y_lo[j] = y_lo[j] + (perr + serr);
        }
    }
    for (int64_t j = 0; j < N; ++j) y[j] = y[j] + y_lo[j];
    free(y_lo);
    return ORACLE_OK;
}

/* -------------------------------------------------------------- GEMVER --- */

/* GEMVER (Table 1 / Table 2):  A_hat = A + u1 v1^T + u2 v2^T;
 * x = x + beta A_hat^T y + z;  w = w + alpha A_hat x.
 * Float inputs: everything in double (A_hat_ij = a + u1 v1 + u2 v2 summed
 * left to right from exact products), A_hat returned in ahat (M x N, row
 * stride N), x and w returned in xo and wo (double). */
int oracle_gemver_f32(int64_t M, int64_t N, double alpha, double beta, const float *A,
                      int64_t lda, const float *u1, const float *v1, const float *u2,
                      const float *v2, const float *w, const float *x, const float *y,
                      const float *z, double *ahat, double *wo, double *xo)
{
    if (M < 0 || N < 0 || lda < N || lda < 1) return ORACLE_EINVAL;
    for (int64_t i = 0; i < M; ++i)
        for (int64_t j = 0; j < N; ++j)
            ahat[i * N + j] = (double)A[i * lda + j] + (double)u1[i] * (double)v1[j]
                              + (double)u2[i] * (double)v2[j];
    for (int64_t j = 0; j < N; ++j) {
        double acc = 0.0;
        for (int64_t i = 0; i < M; ++i) acc += ahat[i * N + j] * (double)y[i];
        xo[j] = (double)x[j] + beta * acc + (double)z[j];
    }
    for (int64_t i = 0; i < M; ++i) {
        double acc = 0.0;
        for (int64_t j = 0; j < N; ++j) acc += ahat[i * N + j] * xo[j];
        wo[i] = (double)w[i] + alpha * acc;
    }
    return ORACLE_OK;
}

/* Double inputs: each A_hat entry as a compensated sum of a, TwoProduct(u1,
 * v1) and TwoProduct(u2, v2), rounded once; both products with Dot2 on the
 * rounded A_hat (and on the rounded new x). */
int oracle_gemver_f64(int64_t M, int64_t N, double alpha, double beta, const double *A,
                      int64_t lda, const double *u1, const double *v1, const double *u2,
                      const double *v2, const double *w, const double *x, const double *y,
                      const double *z, double *ahat, double *wo, double *xo)
{
    if (M < 0 || N < 0 || lda < N || lda < 1) return ORACLE_EINVAL;
    for (int64_t i = 0; i < M; ++i)
        for (int64_t j = 0; j < N; ++j) {
            double p1, e1, p2, e2, s1, t1, s2, t2;
            two_prod(u1[i], v1[j], &p1, &e1);
            two_prod(u2[i], v2[j], &p2, &e2);
            two_sum(A[i * lda + j], p1, &s1, &t1);
            two_sum(s1, p2, &s2, &t2);
            ahat[i * N + j] = s2 + ((t1 + t2) + (e1 + e2));
        }
    for (int64_t j = 0; j < N; ++j) {
        double hi = 0.0, lo = 0.0;
        for (int64_t i = 0; i < M; ++i) {
            double prod, perr, sum, serr;
            two_prod(ahat[i * N + j], y[i], &prod, &perr);
            two_sum(hi, prod, &sum, &serr);
            hi = sum;
            lo = lo + (perr + serr);
        }
        xo[j] = x[j] + beta * (hi + lo) + z[j];
    }
    for (int64_t i = 0; i < M; ++i) {
        double hi = 0.0, lo = 0.0;
        for (int64_t j = 0; j < N; ++j) {
            double prod, perr, sum, serr;
            two_prod(ahat[i * N + j], xo[j], &prod, &perr);
            two_sum(hi, prod, &sum, &serr);
            hi = sum;
            lo = lo + (perr + serr);
        }
        wo[i] = w[i] + alpha * (hi + lo);
    }
    return ORACLE_OK;
}
