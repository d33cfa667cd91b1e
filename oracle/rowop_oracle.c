/*
 * rowop_oracle.c -- double-precision CPU oracle for the row-wise
 * reduce-then-normalise operator family (softmax, log-softmax, LayerNorm,
 * RMSNorm) over dense rows and over ragged rows given by CSR offsets.
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the oracle, not the product: only
 * the test suite, the smoke check and the benchmark's CPU-baseline leg may
 * load it.  It shares no code, header, table or constant with the CUDA
 * library, and it never includes anything from it.
 *
 * Source of the definitions.  The paper names this family only through its
 * running-example kernel names (small_row_kernel, medium_row_kernel,
 * large_row_kernel, launch_by_rows, BLOCK_ROWS; the listing style of §2.1
 * "A Running Example") and never writes the operators out.  The oracle
 * therefore takes the textbook definitions, in the PyTorch convention:
 *
 *   softmax      m = max_j x_j ; s = sum_j exp(x_j - m) ; y_j = exp(x_j - m) / s
 *   log-softmax  y_j = (x_j - m) - log(s)
 *   LayerNorm    mu = sum_j x_j / n ; var = sum_j (x_j - mu)^2 / n  (biased)
 *                y_j = (x_j - mu) / sqrt(var + eps) * gamma_j + beta_j
 *   RMSNorm      ms = sum_j x_j^2 / n ; y_j = x_j / sqrt(ms + eps) * gamma_j
 *   ragged       row i is x[off[i] .. off[i+1]); gamma_j / beta_j are indexed
 *                by the column j inside the row.
 *
 * Every sum is a plain left-to-right loop in double.  Rows are independent;
 * the optional OpenMP pragma only spreads whole rows over threads and does
 * not change any row's arithmetic.
 *
 * Row-length dispatch rule (launch_by_rows): a row of len elements of esize
 * bytes is SMALL (0) if len*esize <= 4096, MEDIUM (1) if <= 32768, else
 * LARGE (2).  The thresholds are this library's choice; the paper gives the
 * three kernel names but no thresholds.
 */
#include <math.h>
#include <stdint.h>

/* ---- one row ----------------------------------------------------------- */

static void softmax_row(const double *x, double *y, int64_t n)
{
    double m = -INFINITY;
    for (int64_t j = 0; j < n; ++j)
        if (x[j] > m)
            m = x[j];
    double s = 0.0;
    for (int64_t j = 0; j < n; ++j)
        s += exp(x[j] - m);
    for (int64_t j = 0; j < n; ++j)
        y[j] = exp(x[j] - m) / s;
}

static void logsoftmax_row(const double *x, double *y, int64_t n)
{
    double m = -INFINITY;
    for (int64_t j = 0; j < n; ++j)
        if (x[j] > m)
            m = x[j];
    double s = 0.0;
    for (int64_t j = 0; j < n; ++j)
        s += exp(x[j] - m);
    const double log_s = log(s);
    for (int64_t j = 0; j < n; ++j)
        y[j] = (x[j] - m) - log_s;
}

static void layernorm_row(const double *x, double *y, const double *gamma,
                          const double *beta, int64_t n, double eps)
{
    double sum = 0.0;
    for (int64_t j = 0; j < n; ++j)
        sum += x[j];
    const double mu = sum / (double)n;
    double sq = 0.0;
    for (int64_t j = 0; j < n; ++j)
        sq += (x[j] - mu) * (x[j] - mu);
    const double var = sq / (double)n;
    const double den = sqrt(var + eps);
    for (int64_t j = 0; j < n; ++j)
        y[j] = (x[j] - mu) / den * gamma[j] + beta[j];
}

static void rmsnorm_row(const double *x, double *y, const double *gamma,
                        int64_t n, double eps)
{
    double sq = 0.0;
    for (int64_t j = 0; j < n; ++j)
        sq += x[j] * x[j];
    const double ms = sq / (double)n;
    const double den = sqrt(ms + eps);
    for (int64_t j = 0; j < n; ++j)
        y[j] = x[j] / den * gamma[j];
}

/* ---- dense rows x cols, contiguous -------------------------------------- */

void oracle_softmax(const double *x, double *y, int64_t rows, int64_t cols,
                    int nthreads)
{
    (void)nthreads;
#pragma omp parallel for schedule(dynamic, 8) num_threads(nthreads)
    for (int64_t r = 0; r < rows; ++r)
        softmax_row(x + r * cols, y + r * cols, cols);
}

void oracle_logsoftmax(const double *x, double *y, int64_t rows, int64_t cols,
                       int nthreads)
{
    (void)nthreads;
#pragma omp parallel for schedule(dynamic, 8) num_threads(nthreads)
    for (int64_t r = 0; r < rows; ++r)
        logsoftmax_row(x + r * cols, y + r * cols, cols);
}

void oracle_layernorm(const double *x, double *y, const double *gamma,
                      const double *beta, int64_t rows, int64_t cols,
                      double eps, int nthreads)
{
    (void)nthreads;
#pragma omp parallel for schedule(dynamic, 8) num_threads(nthreads)
    for (int64_t r = 0; r < rows; ++r)
        layernorm_row(x + r * cols, y + r * cols, gamma, beta, cols, eps);
}

void oracle_rmsnorm(const double *x, double *y, const double *gamma,
                    int64_t rows, int64_t cols, double eps, int nthreads)
{
    (void)nthreads;
#pragma omp parallel for schedule(dynamic, 8) num_threads(nthreads)
    for (int64_t r = 0; r < rows; ++r)
        rmsnorm_row(x + r * cols, y + r * cols, gamma, cols, eps);
}

/* ---- ragged rows: row i = [off[i], off[i+1]) of one packed buffer ------- */

void oracle_softmax_ragged(const double *x, double *y, const int64_t *off,
                           int64_t rows, int nthreads)
{
    (void)nthreads;
#pragma omp parallel for schedule(dynamic, 8) num_threads(nthreads)
    for (int64_t r = 0; r < rows; ++r)
        softmax_row(x + off[r], y + off[r], off[r + 1] - off[r]);
}

void oracle_logsoftmax_ragged(const double *x, double *y, const int64_t *off,
                              int64_t rows, int nthreads)
{
    (void)nthreads;
#pragma omp parallel for schedule(dynamic, 8) num_threads(nthreads)
    for (int64_t r = 0; r < rows; ++r)
        logsoftmax_row(x + off[r], y + off[r], off[r + 1] - off[r]);
}

void oracle_layernorm_ragged(const double *x, double *y, const double *gamma,
                             const double *beta, const int64_t *off,
                             int64_t rows, double eps, int nthreads)
{
    (void)nthreads;
#pragma omp parallel for schedule(dynamic, 8) num_threads(nthreads)
    for (int64_t r = 0; r < rows; ++r)
        layernorm_row(x + off[r], y + off[r], gamma, beta,
                      off[r + 1] - off[r], eps);
}

void oracle_rmsnorm_ragged(const double *x, double *y, const double *gamma,
                           const int64_t *off, int64_t rows, double eps,
                           int nthreads)
{
    (void)nthreads;
#pragma omp parallel for schedule(dynamic, 8) num_threads(nthreads)
    for (int64_t r = 0; r < rows; ++r)
        rmsnorm_row(x + off[r], y + off[r], gamma, off[r + 1] - off[r], eps);
}

/* ---- row-length dispatch rule (launch_by_rows) --------------------------- */

int oracle_bucket(int64_t len, int64_t esize)
{
    const int64_t bytes = len * esize;
    if (bytes <= 4096)
        return 0;
    if (bytes <= 32768)
        return 1;
    return 2;
}
