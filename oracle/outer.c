/*
 * The two rank-one updates of the oracle's column sweep, as plain C loops.
 * Test infrastructure for the fp64 oracle (oracle/realq.py); not product code.
 *
 * After quantizing column j the sweep of Eq. (gptq_update) applies
 *     W[:, j+1:]        -= (delta_j / [H^-1]_jj) [H^-1]_{j, j+1:}        (compensation)
 *     H^-1[j+1:, j+1:]  -= H^-1_{j+1:, j} H^-1_{j, j+1:} / [H^-1]_jj      (Schur downdate)
 * immediately to every remaining column.  numpy evaluates each as an outer
 * product followed by an in-place subtraction; these loops do the same
 * operations on every element in the same order (one rounded product, for
 * the downdate one rounded division, then one rounded subtraction), with no
 * fused multiply-add (built with -ffp-contract=off), so the results are the
 * same bits.  Rows are independent and are shared among OpenMP threads.
 */
#include <stdint.h>

/* A[i][k] -= u[i] * v[k]          for 0 <= i < rows, 0 <= k < cols (compensation; u already divided) */
void realq_oracle_outer_sub(int64_t rows, int64_t cols, double *A, int64_t lda, const double *u,
                            int64_t ustride, const double *v) {
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < rows; ++i) {
        const double ui = u[i * ustride];
        double *a = A + i * lda;
        for (int64_t k = 0; k < cols; ++k) {
            const double p = ui * v[k];
            a[k] = a[k] - p;
        }
    }
}

/* A[i][k] -= (u[i] * v[k]) / d    for 0 <= i < rows, 0 <= k < cols (downdate) */
void realq_oracle_outer_sub_div(int64_t rows, int64_t cols, double *A, int64_t lda, const double *u,
                                int64_t ustride, const double *v, double d) {
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < rows; ++i) {
        const double ui = u[i * ustride];
        double *a = A + i * lda;
        for (int64_t k = 0; k < cols; ++k) {
            const double p = ui * v[k];
            const double q = p / d;
            a[k] = a[k] - q;
        }
    }
}
