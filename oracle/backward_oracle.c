/*
 * backward_oracle.c -- double-precision CPU oracle for the backward passes
 * of the row-wise operator family (softmax, log-softmax, LayerNorm,
 * RMSNorm) over dense rows.
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the oracle, not the product: only
 * the test suite, the smoke check and the benchmark's CPU-baseline leg may
 * load it.  It shares no code, header, table or constant with the CUDA
 * library, and it never includes anything from it.
 *
 * Source of the definitions.  The paper names the forward family only
 * through its running-example kernels (§2.1) and states no backward pass.
 * The backward passes here are the analytic derivatives (chain rule) of the
 * forward definitions the oracle already uses, for an upstream gradient dy
 * of the output:
 *
 *   softmax      given y = softmax(x):     s = sum_j dy_j y_j
 *                                          dx_j = y_j (dy_j - s)
 *   log-softmax  given y = logsoftmax(x):  s = sum_j dy_j
 *                                          dx_j = dy_j - exp(y_j) s
 *   LayerNorm    given x, gamma:  mu, var (biased), rstd = 1/sqrt(var + eps),
 *                xhat_j = (x_j - mu) rstd, g_j = dy_j gamma_j,
 *                a = sum_j g_j / n, b = sum_j g_j xhat_j / n,
 *                dx_j = rstd (g_j - a - xhat_j b),
 *                dgamma_j = sum over rows of dy_j xhat_j,
 *                dbeta_j  = sum over rows of dy_j
 *   RMSNorm      given x, gamma:  rstd = 1/sqrt(sum_j x_j^2 / n + eps),
 *                xhat_j = x_j rstd, g_j = dy_j gamma_j,
 *                b = sum_j g_j xhat_j / n,
 *                dx_j = rstd (g_j - xhat_j b),
 *                dgamma_j = sum over rows of dy_j xhat_j
 *
 * The norm statistics are recomputed from x exactly as the forward oracle
 * computes them (two passes, left-to-right sums in double).  Every sum is a
 * plain left-to-right loop; the column sums run over rows in row order
 * after the (optionally threaded) row loop, so threading never changes a
 * result.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>

/* ---- one row ------------------------------------------------------------ */

static void softmax_bwd_row(const double *y, const double *dy, double *dx,
                            int64_t n)
{
    double s = 0.0;
    for (int64_t j = 0; j < n; ++j)
        s += dy[j] * y[j];
    for (int64_t j = 0; j < n; ++j)
        dx[j] = y[j] * (dy[j] - s);
}

static void logsoftmax_bwd_row(const double *y, const double *dy, double *dx,
                               int64_t n)
{
    double s = 0.0;
    for (int64_t j = 0; j < n; ++j)
        s += dy[j];
    for (int64_t j = 0; j < n; ++j)
        dx[j] = dy[j] - exp(y[j]) * s;
}

/* mean and 1/sqrt(var + eps) of a row, as the forward LayerNorm forms them */
static void layernorm_stats(const double *x, int64_t n, double eps,
                            double *mu_out, double *rstd_out)
{
    double sum = 0.0;
    for (int64_t j = 0; j < n; ++j)
        sum += x[j];
    const double mu = sum / (double)n;
    double sq = 0.0;
    for (int64_t j = 0; j < n; ++j)
        sq += (x[j] - mu) * (x[j] - mu);
    *mu_out = mu;
    *rstd_out = 1.0 / sqrt(sq / (double)n + eps);
}

static double rmsnorm_rstd(const double *x, int64_t n, double eps)
{
    double sq = 0.0;
    for (int64_t j = 0; j < n; ++j)
        sq += x[j] * x[j];
    return 1.0 / sqrt(sq / (double)n + eps);
}

static void layernorm_bwd_row(const double *x, const double *dy,
                              const double *gamma, double *dx, int64_t n,
                              double mu, double rstd)
{
    double sg = 0.0, sgx = 0.0;
    for (int64_t j = 0; j < n; ++j) {
        const double g = dy[j] * gamma[j];
        sg += g;
        sgx += g * ((x[j] - mu) * rstd);
    }
    const double a = sg / (double)n;
    const double b = sgx / (double)n;
    for (int64_t j = 0; j < n; ++j) {
        const double xhat = (x[j] - mu) * rstd;
        dx[j] = rstd * (dy[j] * gamma[j] - a - xhat * b);
    }
}

static void rmsnorm_bwd_row(const double *x, const double *dy,
                            const double *gamma, double *dx, int64_t n,
                            double rstd)
{
    double sgx = 0.0;
    for (int64_t j = 0; j < n; ++j)
        sgx += dy[j] * gamma[j] * (x[j] * rstd);
    const double b = sgx / (double)n;
    for (int64_t j = 0; j < n; ++j)
        dx[j] = rstd * (dy[j] * gamma[j] - (x[j] * rstd) * b);
}

/* ---- dense rows x cols, contiguous -------------------------------------- */

void oracle_softmax_backward(const double *y, const double *dy, double *dx,
                             int64_t rows, int64_t cols, int nthreads)
{
    (void)nthreads;
#pragma omp parallel for schedule(dynamic, 8) num_threads(nthreads)
    for (int64_t r = 0; r < rows; ++r)
        softmax_bwd_row(y + r * cols, dy + r * cols, dx + r * cols, cols);
}

void oracle_logsoftmax_backward(const double *y, const double *dy, double *dx,
                                int64_t rows, int64_t cols, int nthreads)
{
    (void)nthreads;
#pragma omp parallel for schedule(dynamic, 8) num_threads(nthreads)
    for (int64_t r = 0; r < rows; ++r)
        logsoftmax_bwd_row(y + r * cols, dy + r * cols, dx + r * cols, cols);
}

/* dgamma / dbeta may be NULL (not wanted).  Returns 0, or -1 when the
 * per-row statistics buffer could not be allocated. */
int oracle_layernorm_backward(const double *x, const double *dy,
                              const double *gamma, double *dx, double *dgamma,
                              double *dbeta, int64_t rows, int64_t cols,
                              double eps, int nthreads)
{
    (void)nthreads;
    double *st = (double *)malloc(sizeof(double) * 2 * (size_t)(rows > 0 ? rows : 1));
    if (!st)
        return -1;
#pragma omp parallel for schedule(dynamic, 8) num_threads(nthreads)
    for (int64_t r = 0; r < rows; ++r) {
        layernorm_stats(x + r * cols, cols, eps, &st[2 * r], &st[2 * r + 1]);
        layernorm_bwd_row(x + r * cols, dy + r * cols, gamma, dx + r * cols,
                          cols, st[2 * r], st[2 * r + 1]);
    }
    for (int64_t j = 0; j < cols; ++j) {
        double sg = 0.0, sb = 0.0;
        for (int64_t r = 0; r < rows; ++r) {
            const double xhat = (x[r * cols + j] - st[2 * r]) * st[2 * r + 1];
            sg += dy[r * cols + j] * xhat;
            sb += dy[r * cols + j];
        }
        if (dgamma)
            dgamma[j] = sg;
        if (dbeta)
            dbeta[j] = sb;
    }
    free(st);
    return 0;
}

int oracle_rmsnorm_backward(const double *x, const double *dy,
                            const double *gamma, double *dx, double *dgamma,
                            int64_t rows, int64_t cols, double eps,
                            int nthreads)
{
    (void)nthreads;
    double *rs = (double *)malloc(sizeof(double) * (size_t)(rows > 0 ? rows : 1));
    if (!rs)
        return -1;
#pragma omp parallel for schedule(dynamic, 8) num_threads(nthreads)
    for (int64_t r = 0; r < rows; ++r) {
        rs[r] = rmsnorm_rstd(x + r * cols, cols, eps);
        rmsnorm_bwd_row(x + r * cols, dy + r * cols, gamma, dx + r * cols,
                        cols, rs[r]);
    }
    if (dgamma) {
        for (int64_t j = 0; j < cols; ++j) {
            double sg = 0.0;
            for (int64_t r = 0; r < rows; ++r)
                sg += dy[r * cols + j] * (x[r * cols + j] * rs[r]);
            dgamma[j] = sg;
        }
    }
    free(rs);
    return 0;
}
