/*
 * rowop.h -- C ABI of librowop: row-wise reduce-then-normalise operators
 * (softmax, log-softmax, LayerNorm, RMSNorm) on one NVIDIA GB300 (sm_103a).
 *
 * The operator family is the one whose row-length dispatch the paper's
 * running example names (small_row_kernel, medium_row_kernel,
 * large_row_kernel chosen by launch_by_rows, tiled by BLOCK_ROWS; §2.1 "A
 * Running Example").  The paper gives the kernel names only, so the
 * operators follow the textbook / PyTorch definitions:
 *
 *   softmax      y_j = exp(x_j - m) / s,   m = max_j x_j, s = sum_j exp(x_j - m)
 *   log-softmax  y_j = (x_j - m) - log(s)
 *   LayerNorm    y_j = (x_j - mu) / sqrt(var + eps) * gamma_j + beta_j
 *                (mu = mean, var = biased variance of the row)
 *   RMSNorm      y_j = x_j / sqrt(mean_j(x_j^2) + eps) * gamma_j
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 * - All pointers are DEVICE pointers owned by the caller; the library never
 *   allocates device memory on a call and keeps no pointer after it returns.
 * - Element type is rowop_dtype_t: float32, or bfloat16 / float16 with
 *   float32 arithmetic inside and round-to-nearest-even on output.  gamma and beta
 *   have the element type of the data.  gamma == NULL means all ones and
 *   beta == NULL all zeros.
 * - Dense layout: row r starts at element r*ld of `in` and of `out`; ld is in
 *   elements, ld >= cols, and is shared by in and out.  Any element-aligned
 *   pointer and any ld are accepted: 16-byte aligned rows take the vector
 *   path, other rows take per-element loads and stores at the row edges.
 * - Ragged layout: row i is elements [offsets[i], offsets[i+1]) of one packed
 *   buffer (the same offsets index `in` and `out`); offsets is a DEVICE
 *   int64 array of rows+1 non-decreasing entries; gamma_j / beta_j are
 *   indexed by the column j inside the row, so gamma/beta hold max_len
 *   entries.  Rows whose length is negative (decreasing offsets) or larger
 *   than max_len are skipped and flagged (see rowop_check_status).
 * - in == out (exact in-place) is allowed; partial overlap is undefined.
 * - Calls are asynchronous with respect to the host and ordered on `stream`
 *   (NULL = legacy default stream), like cuBLAS.  Argument errors are found
 *   before anything is launched and are returned synchronously.  A launch
 *   failure returns ROWOP_ERR_CUDA.  Device-side conditions (a bounded wait
 *   that ran out, rejected ragged rows) are recorded in a device status word
 *   that rowop_check_status() reads.
 * - rows == 0 is a valid no-op.  Results are deterministic: the same call on
 *   the same data gives bitwise the same output, and a row's result depends
 *   only on its values, its length and its start address modulo 16 bytes
 *   (so a ragged row equals a dense call on the same row at the same
 *   alignment, bit for bit).
 */
#ifndef ROWOP_H
#define ROWOP_H

#include <stddef.h>
#include <stdint.h>

#ifndef __DRIVER_TYPES_H__
typedef struct CUstream_st *cudaStream_t;
#endif

#if defined(__GNUC__)
#define ROWOP_API __attribute__((visibility("default")))
#else
#define ROWOP_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef enum rowop_dtype {
    ROWOP_F32 = 0,  /* float32 in, float32 out                         */
    ROWOP_BF16 = 1, /* bfloat16 in/out, float32 arithmetic, RNE output */
    ROWOP_F16 = 2   /* float16 in/out, float32 arithmetic, RNE output  */
} rowop_dtype_t;

typedef enum rowop_status {
    ROWOP_OK = 0,
    ROWOP_ERR_INVALID_ARG = 1,        /* NULL / misaligned pointer, bad size, ld < cols, eps < 0 */
    ROWOP_ERR_UNSUPPORTED_DTYPE = 2,  /* dtype is not ROWOP_F32, ROWOP_BF16 or ROWOP_F16 */
    ROWOP_ERR_WORKSPACE = 3,          /* ragged workspace NULL, misaligned or too small */
    ROWOP_ERR_CUDA = 4,               /* a CUDA runtime call or launch failed */
    ROWOP_ERR_TIMEOUT = 5,            /* a bounded device wait ran out (see rowop_check_status) */
    ROWOP_ERR_BAD_OFFSETS = 6,        /* ragged rows were skipped: decreasing offsets or len > max_len */
    ROWOP_ERR_TOO_LONG = 7            /* row longer than rowop_max_row_len() */
} rowop_status_t;

/* Row-length buckets of launch_by_rows (§2.1): the kernel design a row goes to. */
typedef enum rowop_bucket {
    ROWOP_SMALL = 0,   /* row bytes <= 4096: a group of <= 32 lanes per row, registers   */
    ROWOP_MEDIUM = 1,  /* row bytes <= 32768: one CTA per row, row staged by TMA bulk copy */
    ROWOP_LARGE = 2    /* longer: a thread-block cluster splits the row, partials via DSMEM */
} rowop_bucket_t;

/* ---- dense rows x cols ---------------------------------------------------
 * in    : rows x cols elements of dtype, row stride ld (elements)
 * out   : same layout and ld as in; written in full for every row
 * Returns ROWOP_OK or an error code; nothing is launched on error.        */

/* Softmax along each row. */
ROWOP_API int rowop_softmax(const void *in, void *out, int64_t rows, int64_t cols,
                  int64_t ld, rowop_dtype_t dtype, cudaStream_t stream);

/* Log-softmax along each row, computed as (x - max) - log(sum). */
ROWOP_API int rowop_logsoftmax(const void *in, void *out, int64_t rows, int64_t cols,
                     int64_t ld, rowop_dtype_t dtype, cudaStream_t stream);

/* LayerNorm along each row (biased variance, eps inside the square root);
 * gamma/beta: cols elements each, or NULL.  eps >= 0. */
ROWOP_API int rowop_layernorm(const void *in, void *out, const void *gamma,
                    const void *beta, int64_t rows, int64_t cols, int64_t ld,
                    rowop_dtype_t dtype, float eps, cudaStream_t stream);

/* RMSNorm along each row (no mean subtraction, no beta); gamma: cols
 * elements, or NULL.  eps >= 0. */
ROWOP_API int rowop_rmsnorm(const void *in, void *out, const void *gamma, int64_t rows,
                  int64_t cols, int64_t ld, rowop_dtype_t dtype, float eps,
                  cudaStream_t stream);

/* ---- fused residual add + norm (dense) ------------------------------------
 * sum_out = x + r (rounded to dtype: the updated residual stream), then
 * y = LayerNorm(sum_out) or RMSNorm(sum_out) of the sum as stored -- the two
 * steps of a pre-norm transformer block in one pass over HBM (read x and r,
 * write sum_out and y).  x, r, sum_out and y share the rows x cols layout and
 * ld; gamma/beta as above.  sum_out may be x or r itself (the residual stream
 * updated in place); y must not overlap x, r or sum_out.                    */
ROWOP_API int rowop_add_layernorm(const void *x, const void *r, void *sum_out, void *y,
                                  const void *gamma, const void *beta, int64_t rows,
                                  int64_t cols, int64_t ld, rowop_dtype_t dtype, float eps,
                                  cudaStream_t stream);

ROWOP_API int rowop_add_rmsnorm(const void *x, const void *r, void *sum_out, void *y,
                                const void *gamma, int64_t rows, int64_t cols, int64_t ld,
                                rowop_dtype_t dtype, float eps, cudaStream_t stream);

/* ---- backward passes (dense) ----------------------------------------------
 * The paper states only the forward operators of this family (§2.1); the
 * backward passes are their derivatives (chain rule) for an upstream
 * gradient dy of the output:
 *
 *   softmax      dx_j = y_j (dy_j - s),        s = sum_j dy_j y_j
 *   log-softmax  dx_j = dy_j - exp(y_j) s,     s = sum_j dy_j
 *   LayerNorm    xhat_j = (x_j - mu) rstd, rstd = 1/sqrt(var + eps), g_j = dy_j gamma_j,
 *                dx_j = rstd (g_j - mean(g) - xhat_j mean(g xhat)),
 *                dgamma_j = sum over rows of dy_j xhat_j,  dbeta_j = sum over rows of dy_j
 *   RMSNorm      xhat_j = x_j rstd, rstd = 1/sqrt(mean(x^2) + eps), g_j = dy_j gamma_j,
 *                dx_j = rstd (g_j - xhat_j mean(g xhat)),
 *                dgamma_j = sum over rows of dy_j xhat_j
 *
 * The softmax family takes the forward OUTPUT y; the norms take the forward
 * INPUT x and recompute mu / rstd exactly as the forward defines them (no
 * saved statistics are needed).  y or x, dy and dx share the rows x cols
 * layout and ld (ld >= cols); dx may be dy itself, or x / y itself (exact
 * in-place); partial overlap is undefined.  gamma: cols elements or NULL
 * (ones).  dgamma / dbeta: cols elements of dtype, or NULL when not wanted;
 * they are sums over ALL rows, and rows == 0 sets them to zero.  Rows that
 * are 16-byte congruent across y/x, dy and dx (and ld*esize a multiple of 16)
 * take 16-byte loads and stores, other rows element accesses.
 *
 * Norm workspace: when dgamma or dbeta is requested, `ws` (device, 16-byte
 * aligned, ws_bytes >= rowop_{layernorm,rmsnorm}_backward_workspace_size(cols)
 * on the current device) receives one float32 partial row per CTA; the
 * partials are then added in index order, so the result is reproducible bit
 * for bit on one device (the number of partials follows its SM count).  ws
 * may be NULL when neither is requested.  The workspace must not be shared
 * by calls that can run concurrently.
 *
 * Rows up to ROWOP_BWD_MAX_COLS_SOFTMAX (softmax family) or
 * ROWOP_BWD_MAX_COLS_NORM (norms) elements; longer rows return
 * ROWOP_ERR_TOO_LONG.  Errors: ROWOP_ERR_INVALID_ARG (NULL or misaligned
 * pointer, cols <= 0 with work to do, ld < cols, eps < 0),
 * ROWOP_ERR_WORKSPACE, ROWOP_ERR_UNSUPPORTED_DTYPE, ROWOP_ERR_CUDA.        */
#define ROWOP_BWD_MAX_COLS_SOFTMAX 262144
#define ROWOP_BWD_MAX_COLS_NORM 262144
#define ROWOP_BWD_MAX_COLS_NORM_RAGGED 131072

ROWOP_API int rowop_softmax_backward(const void *y, const void *dy, void *dx, int64_t rows,
                                     int64_t cols, int64_t ld, rowop_dtype_t dtype,
                                     cudaStream_t stream);

ROWOP_API int rowop_logsoftmax_backward(const void *y, const void *dy, void *dx, int64_t rows,
                                        int64_t cols, int64_t ld, rowop_dtype_t dtype,
                                        cudaStream_t stream);

ROWOP_API int rowop_layernorm_backward(const void *x, const void *dy, const void *gamma,
                                       void *dx, void *dgamma, void *dbeta, int64_t rows,
                                       int64_t cols, int64_t ld, rowop_dtype_t dtype, float eps,
                                       void *ws, size_t ws_bytes, cudaStream_t stream);

ROWOP_API int rowop_rmsnorm_backward(const void *x, const void *dy, const void *gamma,
                                     void *dx, void *dgamma, int64_t rows, int64_t cols,
                                     int64_t ld, rowop_dtype_t dtype, float eps, void *ws,
                                     size_t ws_bytes, cudaStream_t stream);

/* Softmax / log-softmax backward over ragged rows: row i is elements
 * [offsets[i], offsets[i+1]) of y, dy and dx alike (the ragged layout
 * above), dx as the dense backward defines it.  ws is a ragged workspace of
 * at least rowop_ragged_workspace_size(rows) bytes: the call runs the
 * classify pass into it, then one launch per row bucket.  max_len <=
 * ROWOP_BWD_MAX_COLS_SOFTMAX; rows longer than max_len or with decreasing
 * offsets are skipped and flagged as in the forward ragged calls.  dx may be
 * dy or y itself; partial overlap is undefined. */
ROWOP_API int rowop_softmax_backward_ragged(const void *y, const void *dy, void *dx,
                                            const int64_t *offsets, int64_t rows,
                                            int64_t max_len, rowop_dtype_t dtype, void *ws,
                                            size_t ws_bytes, cudaStream_t stream);

ROWOP_API int rowop_logsoftmax_backward_ragged(const void *y, const void *dy, void *dx,
                                               const int64_t *offsets, int64_t rows,
                                               int64_t max_len, rowop_dtype_t dtype, void *ws,
                                               size_t ws_bytes, cudaStream_t stream);

/* LayerNorm / RMSNorm backward over ragged rows (§2.1's row-wise norms on
 * the ragged layout above): row i is elements [offsets[i], offsets[i+1]) of
 * x, dy and dx alike, and column j of every row uses gamma[j] (max_len
 * elements, or NULL = ones).  dx of each row is the dense backward's, for a
 * row of that length.  dgamma[j] (and, for LayerNorm, dbeta[j]) for
 * j < max_len sums dy_j xhat_j (dy_j) over the rows longer than j: max_len
 * elements of dtype each, or NULL when not wanted; rows == 0 sets them to
 * zero.  Rows may start at any element.
 *
 * Two designs, chosen per call (each with its own summation order):
 *   * x, dy and dx at the same offset past a 16-byte boundary and
 *     max_len >= 2048: column stripes.  A first kernel writes each row's
 *     statistics over each stripe of 512 16-byte chunks (4096 bf16 / fp16
 *     or 2048 fp32 elements, counted from the 16-byte boundary at or
 *     before the row's first element).
 *     A second adds them into the row statistics, writes dx and sums
 *     dgamma / dbeta into one float32 partial row per group of rows; a
 *     finalize adds the groups in index order.  x and dy are read twice.
 *   * otherwise: the forward's classify plan, one launch per row bucket,
 *     and one float32 partial row per CTA for each bucket, added in index
 *     order, the buckets in order (SMALL, MEDIUM, LARGE).
 * Either way nothing is atomic: the result is reproducible bit for bit on
 * one device.
 *
 * ws: device, 256-byte aligned, at least
 * rowop_{layernorm,rmsnorm}_backward_ragged_workspace_size(rows, max_len,
 * dtype) bytes on the current device (enough for either design).  The
 * workspace must not be shared by concurrent calls.
 *
 * max_len <= ROWOP_BWD_MAX_COLS_NORM_RAGGED (else ROWOP_ERR_TOO_LONG); rows longer
 * than max_len or with decreasing offsets are skipped and flagged as in the
 * forward ragged calls.  dx may be dy or x itself; partial overlap is
 * undefined.  Errors: ROWOP_ERR_INVALID_ARG (NULL or misaligned pointer,
 * rows < 0, max_len < 0, eps < 0), ROWOP_ERR_WORKSPACE,
 * ROWOP_ERR_UNSUPPORTED_DTYPE, ROWOP_ERR_CUDA. */
ROWOP_API int rowop_layernorm_backward_ragged(const void *x, const void *dy, const void *gamma,
                                              void *dx, void *dgamma, void *dbeta,
                                              const int64_t *offsets, int64_t rows,
                                              int64_t max_len, rowop_dtype_t dtype, float eps,
                                              void *ws, size_t ws_bytes, cudaStream_t stream);

ROWOP_API int rowop_rmsnorm_backward_ragged(const void *x, const void *dy, const void *gamma,
                                            void *dx, void *dgamma, const int64_t *offsets,
                                            int64_t rows, int64_t max_len, rowop_dtype_t dtype,
                                            float eps, void *ws, size_t ws_bytes,
                                            cudaStream_t stream);

/* Workspace bytes of a ragged norm backward call of `rows` rows up to
 * max_len elements of dtype on the current device; 0 if an argument is
 * invalid or the device cannot be queried. */
ROWOP_API size_t rowop_layernorm_backward_ragged_workspace_size(int64_t rows, int64_t max_len,
                                                                rowop_dtype_t dtype);
ROWOP_API size_t rowop_rmsnorm_backward_ragged_workspace_size(int64_t rows, int64_t max_len,
                                                              rowop_dtype_t dtype);

/* Workspace bytes for dgamma (and dbeta) of rows of `cols` elements on the
 * current device; 0 if cols <= 0 or the device cannot be queried. */
ROWOP_API size_t rowop_layernorm_backward_workspace_size(int64_t cols);
ROWOP_API size_t rowop_rmsnorm_backward_workspace_size(int64_t cols);

/* ---- ragged rows (int64 CSR offsets into one packed buffer) ---------------
 * offsets : device int64[rows + 1], non-decreasing
 * max_len : an upper bound on every row's length (>= 0); sizes the on-chip
 *           staging and bounds gamma/beta, which hold max_len elements
 * ws      : device workspace of at least rowop_ragged_workspace_size(rows)
 *           bytes, 256-byte aligned, owned by the caller.  It must not be
 *           used by another call that may run at the same time.  After the
 *           call (once the stream reaches it) byte ws[256 + i] holds the
 *           bucket row i was dispatched to (255 = row rejected), and the
 *           uint32 at ws[0] holds this call's device status bits.
 * All buckets are handled in one pass over the rows (a classify launch, then
 * one fused launch that serves all three buckets).                         */

ROWOP_API size_t rowop_ragged_workspace_size(int64_t rows);

ROWOP_API int rowop_softmax_ragged(const void *in, void *out, const int64_t *offsets,
                         int64_t rows, int64_t max_len, rowop_dtype_t dtype,
                         void *ws, size_t ws_bytes, cudaStream_t stream);

ROWOP_API int rowop_logsoftmax_ragged(const void *in, void *out,
                            const int64_t *offsets, int64_t rows,
                            int64_t max_len, rowop_dtype_t dtype, void *ws,
                            size_t ws_bytes, cudaStream_t stream);

ROWOP_API int rowop_layernorm_ragged(const void *in, void *out, const void *gamma,
                           const void *beta, const int64_t *offsets,
                           int64_t rows, int64_t max_len, rowop_dtype_t dtype,
                           float eps, void *ws, size_t ws_bytes,
                           cudaStream_t stream);

ROWOP_API int rowop_rmsnorm_ragged(const void *in, void *out, const void *gamma,
                         const int64_t *offsets, int64_t rows,
                         int64_t max_len, rowop_dtype_t dtype, float eps,
                         void *ws, size_t ws_bytes, cudaStream_t stream);

/* ---- ragged plans: classify once, run many operators ---------------------
 * rowop_ragged_plan runs only the classify pass of launch_by_rows (bucket per
 * row and the three row lists) into ws.  A *_ragged_planned call then skips
 * that pass and reuses the plan: it must get the same offsets (unchanged
 * contents), rows, max_len, dtype and ws as the plan, on the same stream or
 * after it.  Each planned call leaves the plan reusable for the next one.
 * The plain *_ragged calls above are plan + planned call in one.          */

ROWOP_API int rowop_ragged_plan(const int64_t *offsets, int64_t rows,
                                int64_t max_len, rowop_dtype_t dtype, void *ws,
                                size_t ws_bytes, cudaStream_t stream);

ROWOP_API int rowop_softmax_ragged_planned(const void *in, void *out,
                                           const int64_t *offsets, int64_t rows,
                                           int64_t max_len, rowop_dtype_t dtype,
                                           void *ws, size_t ws_bytes,
                                           cudaStream_t stream);

ROWOP_API int rowop_logsoftmax_ragged_planned(const void *in, void *out,
                                              const int64_t *offsets,
                                              int64_t rows, int64_t max_len,
                                              rowop_dtype_t dtype, void *ws,
                                              size_t ws_bytes,
                                              cudaStream_t stream);

ROWOP_API int rowop_layernorm_ragged_planned(const void *in, void *out,
                                             const void *gamma, const void *beta,
                                             const int64_t *offsets, int64_t rows,
                                             int64_t max_len, rowop_dtype_t dtype,
                                             float eps, void *ws, size_t ws_bytes,
                                             cudaStream_t stream);

ROWOP_API int rowop_rmsnorm_ragged_planned(const void *in, void *out,
                                           const void *gamma,
                                           const int64_t *offsets, int64_t rows,
                                           int64_t max_len, rowop_dtype_t dtype,
                                           float eps, void *ws, size_t ws_bytes,
                                           cudaStream_t stream);

/* ---- ragged LayerNorm without a caller workspace ---------------------------
 * The paper has no counterpart: this is a library convenience.  Some callers
 * cannot provide the workspace: a kernel plugin inside another runtime (an
 * inference engine, a framework's custom-op slot) is handed only its input
 * and output buffers and has no allocator of its own to ask; and code on a
 * latency-critical path often may not call cudaMalloc / cudaFree, which can
 * synchronise the device and stall every stream.  For them this is
 * rowop_layernorm_ragged with the same arguments minus ws / ws_bytes: the
 * workspace is a fixed array in the library's device memory, sized for
 * ROWOP_STATIC_MAX_ROWS rows (about 3.2 MB), one per device, held by every
 * GPU that loads the library until the process exits.  Nothing is
 * allocated or freed by the call.  Results equal those of
 * rowop_layernorm_ragged bit for bit.
 *   rows > ROWOP_STATIC_MAX_ROWS  -> ROWOP_ERR_WORKSPACE, nothing launched.
 * The first call on a device looks the array's address up (a CUDA runtime
 * query, made with that device current); make it before capturing the stream
 * into a graph.  Every call starts with the classify pass, which rewrites the
 * per-call state the fused kernel needs zeroed (bucket counts, work counters,
 * status) before that kernel reads it, so nothing carries over from a
 * previous call.  All calls on one device share the one array: calls that
 * may run at the same time (on different streams, or from different host
 * threads without ordering) race on it and give undefined results.  The
 * bucket bytes described for ws above are not exposed. */
#define ROWOP_STATIC_MAX_ROWS 65536

ROWOP_API int rowop_layernorm_ragged_static(const void *in, void *out,
                                            const void *gamma, const void *beta,
                                            const int64_t *offsets, int64_t rows,
                                            int64_t max_len, rowop_dtype_t dtype,
                                            float eps, cudaStream_t stream);

/* ---- Hyena FFT-size padding (§6, "Representative cross-layer trace") -------
 * out[r][c] = scale * in[r][c] for 0 <= c < seqlen and 0 for
 * seqlen <= c < fft_size, for every row r < rows: the zero-padded, scaled
 * input of an FFT convolution.
 * in    : rows x seqlen elements of dtype, row stride ld_in >= seqlen (may be
 *         NULL when seqlen == 0)
 * out   : rows x fft_size elements of dtype, row stride ld_out >= fft_size;
 *         written in full for every row (columns past fft_size untouched)
 * fft_size >= seqlen >= 0; scale finite.  bf16: the product is formed in
 * fp32 and rounded to nearest even.  in and out must not overlap.          */
ROWOP_API int rowop_pad_scale(const void *in, void *out, int64_t rows, int64_t seqlen,
                              int64_t fft_size, int64_t ld_in, int64_t ld_out,
                              float scale, rowop_dtype_t dtype, cudaStream_t stream);

/* ---- MoE group score (§2.1, "A Running Example") --------------------------
 * For every token t and every group g of 32 consecutive experts:
 *   out[t][g] = max over i != j of (s[t][32g+i] + s[t][32g+j]),
 * the sum of the group's two largest scores, a tied maximum counting twice.
 * Computed by value only (no index is ever produced), in fp32.
 * scores : tokens x experts of dtype, row stride ld >= experts; experts a
 *          positive multiple of 32; scores finite or -inf
 * out    : tokens x (experts / 32) float32, contiguous                     */
ROWOP_API int rowop_moe_group_top2(const void *scores, float *out, int64_t tokens,
                                   int64_t experts, int64_t ld, rowop_dtype_t dtype,
                                   cudaStream_t stream);

/* ---- dispatch rule, limits, status ---------------------------------------- */

/* launch_by_rows (§2.1): the bucket for a row of len elements (len >= 0):
 * SMALL if len*esize <= 4096, MEDIUM if <= 32768, else LARGE.
 * Returns -1 for len < 0 or an unknown dtype.  Pure host function. */
ROWOP_API int rowop_select_bucket(int64_t len, rowop_dtype_t dtype);

/* Longest row (elements) the library accepts for dtype, dense or ragged. */
ROWOP_API int64_t rowop_max_row_len(rowop_dtype_t dtype);

/* The library's dispatch thresholds and limits, as this build uses them.
 * None of them depends on the device or on the environment.  The bucket
 * rule (launch_by_rows, §2.1) is: SMALL if len * esize <= small_max_bytes,
 * MEDIUM if <= medium_max_bytes, else LARGE. */
typedef struct rowop_config {
    uint32_t size;                  /* bytes of this struct the library filled */
    uint32_t chunk_bytes;           /* 16: the unit of every vector load / store */
    uint32_t tile_bytes;            /* 1024: a warp's unit of a MEDIUM / LARGE row */
    uint32_t max_cluster;           /* largest thread-block cluster a row is split over */
    int64_t small_max_bytes;        /* 4096 */
    int64_t medium_max_bytes;       /* 32768 */
    int64_t max_row_len[3];         /* rowop_max_row_len() per rowop_dtype_t */
    int64_t resident_max_tiles[2];  /* longest row portion (tiles) a CTA holds in
                                       registers: [0] float32, [1] 16-bit types */
    int64_t staged_max_tiles;       /* longest portion a CTA holds staged in shared memory */
    int64_t stage_budget_bytes[2];  /* shared memory for stages per CTA: [0] resident
                                       design at two CTAs an SM, [1] staged (three) */
    int64_t wait_limit_ns;          /* a bounded device wait gives up after this long */
    int64_t static_max_rows;        /* ROWOP_STATIC_MAX_ROWS */
} rowop_config_t;

/* Fills *cfg (which must not be NULL; ROWOP_ERR_INVALID_ARG otherwise) and
 * returns ROWOP_OK.  Pure host function. */
ROWOP_API int rowop_get_config(rowop_config_t *cfg);

/* Human-readable name of a status code (static storage, never NULL). */
ROWOP_API const char *rowop_status_string(int status);

/* The CUDA runtime's description of the last CUDA error that made a call of
 * this thread return ROWOP_ERR_CUDA ("no error" if none has; static storage,
 * never NULL).  Pure host function. */
ROWOP_API const char *rowop_last_cuda_error(void);

/* Synchronises `stream` (the host waits until all work queued on it has
 * finished), then reads and clears the device status word of the current
 * device: returns ROWOP_OK, ROWOP_ERR_TIMEOUT if any bounded device wait ran
 * out, ROWOP_ERR_BAD_OFFSETS if ragged rows were rejected (timeout wins when
 * both are set), or ROWOP_ERR_CUDA if the synchronisation failed.
 * The status word belongs to the device, not to a call or a stream: every
 * call on the device, on any stream (rowop_layernorm_ragged_static
 * included), sets its bits, and the first rowop_check_status to run reads
 * and clears them.  Work still running on other streams may set bits after
 * the read.  To attribute a condition to one call, run it alone on its
 * stream, or synchronise the other streams first. */
ROWOP_API int rowop_check_status(cudaStream_t stream);

/* Test hook for the bounded-wait path, launching one tiny kernel that waits
 * on an on-chip barrier nothing will complete, for at most limit_ns
 * nanoseconds (1 .. 10^9), then records a timeout in the status word and
 * returns.  No memory traffic is in flight while it waits.  Returns
 * ROWOP_ERR_INVALID_ARG for an out-of-range limit. */
ROWOP_API int rowop_debug_wait_timeout(int64_t limit_ns, cudaStream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* ROWOP_H */
