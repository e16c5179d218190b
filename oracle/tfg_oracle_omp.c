/*
 * tfg_oracle_omp.c -- the oracle's row functions run on all host cores.
 *
 * TEST INFRASTRUCTURE ONLY (a CPU baseline for the benchmark, not a parity
 * oracle).  It adds no arithmetic of its own: it calls the unchanged row
 * functions of tfg_oracle.c (oracle_aggregate_rows,
 * oracle_edge_softmax_rows) on contiguous blocks of target rows, one block
 * per OpenMP task.  Rows are independent once the edges are grouped by
 * target (the reduce key of Section 2.1.2), so the blocks write disjoint
 * output rows and the results equal the single-threaded ones exactly.
 * Built together with tfg_oracle.c into a separate library with -fopenmp.
 */
#include <stdint.h>

#ifdef _OPENMP
#include <omp.h>
#endif

int oracle_aggregate_rows(int reduce, int64_t n, const int32_t *rowptr, const int32_t *col,
                          const int32_t *perm, const double *w, const double *x, int64_t f,
                          const double *self_w, const int64_t *rows, int64_t nrows,
                          double *out, double *absout);
int oracle_edge_softmax_rows(int64_t n, const int32_t *rowptr, const int32_t *col,
                             const double *x, int h, int c, const double *a_src,
                             const double *a_dst, double slope, const int64_t *rows,
                             int64_t nrows, double *out, double *alpha_rows, double *absout);

#define BLOCK 128

/* Number of threads a parallel region of this library uses. */
int oracle_omp_threads(void)
{
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

/* oracle_aggregate_rows over all n rows; out/absout are [n, f]. */
int oracle_omp_aggregate_all(int reduce, int64_t n, const int32_t *rowptr, const int32_t *col,
                             const int32_t *perm, const double *w, const double *x, int64_t f,
                             const double *self_w, double *out, double *absout)
{
    int rc = 0;
#pragma omp parallel for schedule(dynamic, 1) reduction(| : rc)
    for (int64_t r0 = 0; r0 < n; r0 += BLOCK) {
        int64_t rows[BLOCK];
        const int64_t nr = n - r0 < BLOCK ? n - r0 : BLOCK;
        for (int64_t i = 0; i < nr; ++i) rows[i] = r0 + i;
        rc |= -oracle_aggregate_rows(reduce, n, rowptr, col, perm, w, x, f, self_w, rows, nr,
                                     out + r0 * f, absout + r0 * f);
    }
    return -rc;
}

/* oracle_edge_softmax_rows over all n rows (no alpha); out/absout [n, h*c]. */
int oracle_omp_edge_softmax_all(int64_t n, const int32_t *rowptr, const int32_t *col,
                                const double *x, int h, int c, const double *a_src,
                                const double *a_dst, double slope, double *out, double *absout)
{
    const int64_t f = (int64_t)h * c;
    int rc = 0;
#pragma omp parallel for schedule(dynamic, 1) reduction(| : rc)
    for (int64_t r0 = 0; r0 < n; r0 += BLOCK) {
        int64_t rows[BLOCK];
        const int64_t nr = n - r0 < BLOCK ? n - r0 : BLOCK;
        for (int64_t i = 0; i < nr; ++i) rows[i] = r0 + i;
        rc |= -oracle_edge_softmax_rows(n, rowptr, col, x, h, c, a_src, a_dst, slope, rows, nr,
                                        out + r0 * f, (double *)0, absout + r0 * f);
    }
    return -rc;
}
