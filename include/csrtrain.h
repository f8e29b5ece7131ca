/*
 * csrtrain.h -- C ABI of the GB300 (sm_103a) CSR-weight training step.
 *
 * Method: Lee & Lee, "Compressed Learning of Deep Neural Networks for
 * OpenCL-Capable Embedded Systems", arXiv 1905.07931. A training step over
 * layers whose weight matrices are held in compressed sparse row form
 * (Section 3.1): forward product Y = W X (Section 3.2.1), backward product
 * dX = W^T dY (Section 3.2.2), the dense weight gradient for the l1-proximal
 * phase and the gradient sampled at the stored entries for the debias phase
 * (Section 2.4), the soft-threshold proximal update (Section 2.2, Eq. prox,
 * Section 3.3) followed by re-compaction of the CSR arrays after every update.
 *
 * Conventions shared by every call
 * --------------------------------
 *  - Layout. W is M x K (M = outputs, K = inputs). Dense activations are
 *    feature-major, row-major with the sample index contiguous: X is K x n,
 *    Y and dY are M x n. (The paper's Caffe orientation X_T = X_B W' holds
 *    samples in rows; this is its transpose.) All floating-point data is
 *    IEEE float32; indices are int32; M * K must be below 2^31.
 *  - Memory. Every pointer inside a csrt_csr and every array argument is a
 *    DEVICE pointer unless stated otherwise; the csrt_csr struct itself and
 *    the small out-parameters are HOST memory. The caller owns and allocates
 *    every buffer. The library allocates no memory of its own.
 *  - Streams. `stream` is a cudaStream_t passed as void* (NULL = the legacy
 *    default stream). Every call only enqueues work on that stream; none
 *    synchronises except csrt_get_status. No call reads nnz on the host:
 *    nnz lives on the device in row_ptr[M].
 *  - Workspace. Calls that take `ws` need a device scratch buffer of at least
 *    csrt_workspace_bytes(...) bytes, initialised once with
 *    csrt_workspace_init. Its first 256 bytes hold a device status word that
 *    accumulates data-dependent errors (see CSRT_DEV_*); the next 64 KiB hold
 *    counters that the sparse products use and leave at zero (so the
 *    workspace must start zeroed, as csrt_workspace_init leaves it). A
 *    workspace serves one stream at a time: calls on two streams need two
 *    workspaces.
 *  - Errors. Each call returns CSRT_OK or a CSRT_ERR_* code at once for bad
 *    arguments or a failed launch; no work is enqueued in that case.
 *    Data-dependent errors (capacity overflow, a bounded wait that ran out,
 *    non-finite values) cannot be known on the host without a sync; kernels
 *    OR them into the device status word, read by csrt_get_status.
 *    csrt_last_error() returns a message for the last failing call on the
 *    calling host thread.
 */
#ifndef CSRTRAIN_H
#define CSRTRAIN_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Return codes. */
#define CSRT_OK 0
#define CSRT_ERR_ARG 1        /* invalid argument: nothing enqueued */
#define CSRT_ERR_CUDA 2       /* a CUDA runtime call or launch failed */
#define CSRT_ERR_WORKSPACE 3  /* workspace smaller than required */

/* Device status bits (OR-ed by kernels into the workspace status word). */
#define CSRT_DEV_CAPACITY 1   /* an output CSR needed more entries than its capacity;
                                 the CSR written is truncated but structurally valid
                                 (row_ptr clamped to capacity). required_nnz reports
                                 the count that was needed. */
#define CSRT_DEV_TIMEOUT 2    /* a bounded wait (on another block, or on a bulk copy
                                 into shared memory) gave up; results invalid */
#define CSRT_DEV_NONFINITE 4  /* the prox step met a NaN in w - eta*G (dropped) */
#define CSRT_DEV_INVALID 8    /* csrt_validate_csr found a broken invariant */

/* weight_grad_dense precision. */
#define CSRT_PREC_FP32 0      /* float32 FMA on the CUDA cores */
#define CSRT_PREC_TF32 1      /* tcgen05 tensor cores, kind::tf32, float32 accumulate */

/*
 * A CSR matrix (Section 3.1, Figure "spformats" (iii): row_ptrs, col_indices,
 * elements), plus an optional transposed copy of the same pattern.
 *
 * Section 3.2.2 notes that the backward product reads W column by column,
 * which row-wise CSR storage cannot serve with coalesced loads, and that a
 * second, column-ordered copy of the nonzeros would remove the problem. The
 * t_* arrays are that copy:
 * W^T in CSR form (entries sorted by column, then row) and, for each CSR
 * entry k, its position t_pos[k] in the transposed arrays. They are needed by
 * spmm_bwd_t only; layers whose input gradient is never needed can leave
 * them NULL.
 */
typedef struct csrt_csr {
    int32_t rows;        /* M */
    int32_t cols;        /* K */
    int64_t capacity;    /* allocated entries of col_idx/val (and t_col_idx/t_val/t_pos) */
    int32_t *row_ptr;    /* [rows+1]; row_ptr[0] = 0, row_ptr[rows] = nnz */
    int32_t *col_idx;    /* [capacity]; ascending and unique within a row */
    float *val;          /* [capacity] */
    int32_t *t_row_ptr;  /* [cols+1] or NULL */
    int32_t *t_col_idx;  /* [capacity] or NULL: row index of each transposed entry */
    float *t_val;        /* [capacity] or NULL */
    int32_t *t_pos;      /* [capacity] or NULL: CSR entry k sits at t_*[t_pos[k]] */
} csrt_csr;

/* ------------------------------------------------------------------------ */
/* Workspace and status                                                      */
/* ------------------------------------------------------------------------ */

/* Bytes of workspace needed by every call below for matrices of at most
 * `rows` x `cols` and products with at most `max_n` columns. Host only. */
int csrt_workspace_bytes(int32_t rows, int32_t cols, int32_t max_n, size_t *bytes);

/* csrt_check_bounded_waits -- failure detection, checked without a fault
 * (the paper has no counterpart). Runs the library's two kinds of bounded
 * wait against events that never happen: the decoupled look-back of the
 * compaction kernels waiting on a predecessor tile that never publishes, and
 * an mbarrier wait (as in the TMA / tensor-core pipelines) on a barrier
 * nothing arrives on. Each gives up after its iteration limit (well under a
 * second), sets CSRT_DEV_TIMEOUT in the status word and returns, leaving the
 * context usable. Clear the status afterwards (csrt_clear_status). Uses the
 * first 16 bytes of the workspace scratch. */
int csrt_check_bounded_waits(void *ws, size_t ws_bytes, void *stream);

/* csrt_fma_peak_run -- measurement aid (not part of the training step): a
 * kernel of `blocks` blocks of 512 threads, each thread running 8 independent
 * FP32 fused multiply-add chains for `iters` rounds, then storing one float
 * to out[blocks*512] (device). *flops (host, may be NULL) receives the
 * floating-point operations it performs (2 per FMA). The caller times it
 * (e.g. with events on `stream`) to obtain the GPU's FP32 FMA throughput,
 * the roof of the CUDA-core sparse products. */
int csrt_fma_peak_run(float *out, int32_t blocks, int32_t iters, double *flops, void *stream);

/* Zero the whole workspace (status word included) on `stream`. */
int csrt_workspace_init(void *ws, size_t ws_bytes, void *stream);

/* Synchronise `stream`, then copy the status bits and the largest required
 * nnz reported by a capacity overflow to the host. Either out-pointer may be
 * NULL. Does not clear the status (see csrt_clear_status). */
int csrt_get_status(const void *ws, int32_t *flags, int64_t *required_nnz, void *stream);

/* Clear the status word on `stream`. */
int csrt_clear_status(void *ws, void *stream);

/* csrt_validate_csr -- structural check of a CSR (the paper has no
 * counterpart; the preconditions every call here assumes, Section 3.1's
 * format): row_ptr[0] == 0, 0 <= row_ptr[r] <= row_ptr[r+1] <= capacity,
 * and within each row 0 <= col_idx < cols, strictly ascending. If t_row_ptr
 * is set, the transposed arrays too: the same checks on (t_row_ptr,
 * t_col_idx) with rows and cols swapped, equal entry counts, and for every
 * entry k of row r: t_pos[k] lies in column col_idx[k]'s range, t_col_idx
 * there is r and t_val holds val[k]'s bits. Every index is bounded before it
 * is used, so a corrupted CSR cannot cause an out-of-range read. A broken
 * invariant sets CSRT_DEV_INVALID in the status word (csrt_get_status) and
 * records the first row found (csrt_get_invalid_row). Arrays are device
 * memory of the lengths the csrt_csr comment gives; nothing is written but
 * the status header. */
int csrt_validate_csr(const csrt_csr *w, void *ws, size_t ws_bytes, void *stream);

/* Synchronise `stream`, then report the row where csrt_validate_csr first
 * found a broken invariant: r < rows for the CSR, rows + 1 + c for column c
 * of the transposed copy (rows for unequal entry counts), rows + cols + 1 + r
 * for a transposed position of row r's entries; -1 if none (cleared by
 * csrt_clear_status). */
int csrt_get_invalid_row(const void *ws, int64_t *row, void *stream);

/* Message for the last failing call on this host thread ("" if none). */
const char *csrt_last_error(void);

/* Number of kernels the library launched on the calling host thread since
 * the last reset (an instrument for counting launches inside a timed region). */
int64_t csrt_launch_count(int reset);

/* ------------------------------------------------------------------------ */
/* The training-step calls                                                   */
/* ------------------------------------------------------------------------ */

/* csr_from_dense -- Section 3.1. Compress a dense row-major rows x cols
 * matrix, keeping every entry with value != 0 (+0.0 and -0.0 dropped, NaN
 * and Inf kept) in row-major order. Writes out->row_ptr, col_idx, val; if
 * out->t_row_ptr is not NULL also builds the transposed arrays
 * (csr_transpose). out->rows/cols must equal rows/cols. An output needing
 * more than out->capacity entries sets CSRT_DEV_CAPACITY. */
int csr_from_dense(const float *dense, int32_t rows, int32_t cols, csrt_csr *out,
                   void *ws, size_t ws_bytes, void *stream);

/* csr_transpose -- the column-wise copy of Section 3.2.2. Rebuilds
 * w->t_row_ptr, t_col_idx, t_val and t_pos from w's CSR arrays
 * (deterministic: entries of a column are ordered by row). All four t_*
 * pointers must be set. */
int csr_transpose(csrt_csr *w, void *ws, size_t ws_bytes, void *stream);

/* spmm_fwd -- Section 3.2.1 (dense x compressed', the forward pass).
 * Y[M x n] = W X[K x n]: Y[i, c] = sum over stored k of row i of
 * val[k] * X[col_idx[k], c], float32 accumulation. Y is overwritten.
 * Products with n <= 16 (64 for float4-aligned X and Y) stream col_idx and
 * val through shared memory with bulk copies when both arrays are 16-byte
 * aligned (else a 32-lane kernel runs); a copy that does not complete within
 * the wait's limit sets CSRT_DEV_TIMEOUT. */
int spmm_fwd(const csrt_csr *w, const float *x, int32_t n, float *y,
             void *ws, size_t ws_bytes, void *stream);

/* spmm_bwd_t -- Section 3.2.2 (dense x compressed, the backward pass).
 * dX[K x n] = W^T dY[M x n], through the transposed arrays (which must be
 * current: built by csr_from_dense / csr_transpose / prox_update_compact and
 * kept in step by debias_update). dX is overwritten. */
int spmm_bwd_t(const csrt_csr *w, const float *dy, int32_t n, float *dx,
               void *ws, size_t ws_bytes, void *stream);

/* spmm_fwd with the layer epilogue fused (same arithmetic as spmm_fwd then
 * csrt_bias_act_fwd): Y[i, c] = act(fl32(sum + bias[i])), act = ReLU when
 * relu != 0, identity otherwise. bias (M floats) may be NULL. */
int spmm_fwd_bias_act(const csrt_csr *w, const float *x, int32_t n, const float *bias, int32_t relu,
                      float *y, void *ws, size_t ws_bytes, void *stream);

/* spmm_bwd_t with the ReLU backward of the layer below fused (same result as
 * spmm_bwd_t then csrt_relu_bwd): dX[j, c] = (W^T dY)[j, c] where
 * y_below[j, c] > 0, else 0. y_below is K x n, the output of the layer below. */
int spmm_bwd_t_relu(const csrt_csr *w, const float *dy, int32_t n, const float *y_below, float *dx,
                    void *ws, size_t ws_bytes, void *stream);

/* spmm_fwd_noalloc -- the same product as spmm_fwd for callers that cannot
 * allocate device memory (for example code embedded in a framework that owns
 * every device allocation and forbids direct cudaMalloc, or a serving loop
 * that may not risk an allocation). The paper has no counterpart: it is an
 * interface choice of this library. n may be at most 4096 (larger n is
 * rejected with CSRT_ERR_ARG). The scratch for rows split between work units
 * lives in a fixed device array inside the library (8 MiB of floats + 256 KiB
 * of row slots, held by every GPU that loads the library until the process
 * exits). A call needs (units x n-tiles) x (columns per tile) floats of it,
 * at most (SMs x 32 + n-tiles) x 256, so every n <= 4096 fits on GPUs of up
 * to 255 SMs; a shape that does not fit is rejected with CSRT_ERR_ARG. A
 * bounded wait that gives up sets CSRT_DEV_TIMEOUT in the library's own
 * status word (read it with spmm_fwd_noalloc_status). The first call of
 * either entry point on a device looks the arrays up with
 * cudaGetSymbolAddress (make it before any stream capture). All calls share
 * the array: calls whose kernels overlap on the GPU race and must be
 * serialised by the caller. */
int spmm_fwd_noalloc(const csrt_csr *w, const float *x, int32_t n, float *y, void *stream);

/* spmm_fwd_noalloc_status -- synchronise `stream`, then copy the status word
 * of spmm_fwd_noalloc (its own, not a workspace's: CSRT_DEV_TIMEOUT if a
 * bounded wait of any call since the last clear gave up) to *flags (host).
 * clear != 0 then zeroes it. Allocates nothing. */
int spmm_fwd_noalloc_status(int32_t *flags, int32_t clear, void *stream);

/* weight_grad_dense -- gradient of every weight for the prox phase (the
 * matrix w - eta*G of Section 3.3 needs G at all M x K entries).
 * G[i, j] = sum_c dY[i, c] X[j, c]; dY is m x n, X is k x n, G is m x k,
 * all row-major. No 1/n factor is applied. precision: CSRT_PREC_FP32 or
 * CSRT_PREC_TF32 (operands rounded to TF32, float32 accumulation). */
int weight_grad_dense(const float *dy, const float *x, int32_t m, int32_t k, int32_t n,
                      float *g, int32_t precision, void *ws, size_t ws_bytes, void *stream);

/* weight_grad_sddmm -- gradient at the stored entries only, for the debias
 * phase (Section 2.4: zero weights are not trained).
 * g_nnz[k] = sum_c dY[i_k, c] X[j_k, c] for every stored entry k = (i_k, j_k).
 * g_nnz has at least nnz entries. */
int weight_grad_sddmm(const csrt_csr *w, const float *dy, const float *x, int32_t n,
                      float *g_nnz, void *ws, size_t ws_bytes, void *stream);

/* prox_update_compact -- Eq. prox with the soft threshold of Section 2.2,
 * applied to the dense matrix w - eta*G as in Section 3.3, then compacted
 * back to CSR (Section 4.4: compression after every update).
 * For every (i, j), row-major, with w = the stored value or +0:
 *   thr = fl32(eta*lambda), t = fl32(eta*G[i,j]), z = fl32(w - t) (no FMA),
 *   keep iff |z| > thr, kept value = z - thr (z > 0) or z + thr (z < 0).
 * G is a dense row-major M x K float32 matrix. w_out must be a different CSR
 * with the same shape; capacity M*K can never overflow (zero weights may
 * re-enter). If w_out->t_row_ptr is not NULL the transposed arrays of w_out
 * are rebuilt too. eta and lambda must be finite and >= 0. */
int prox_update_compact(const csrt_csr *w_in, const float *g, float eta, float lambda,
                        csrt_csr *w_out, void *ws, size_t ws_bytes, void *stream);

/* prox_rmsprop_update_compact -- one step of Prox-RMSProp (Algorithm 1):
 * the prox step of prox_update_compact taken along the search direction d
 * instead of G. v (dense row-major M x K float32, the running average of
 * G*G, zero before the first step) is updated in place. Per entry, every
 * operation rounded once to float32 in this order, c = fl32(1 - beta):
 *   v <- fl(fl(beta*v) + fl(c*fl(G*G)));  d = fl(G / fl(fl(sqrt(v)) + eps))
 * then t = fl32(eta*d), z = fl32(w - t) and the threshold fl32(eta*lambda)
 * exactly as in prox_update_compact (the threshold is not scaled by the
 * adaptive denominator). beta in [0, 1), eps finite and > 0; v must not alias
 * G. A non-finite d drops the entry and sets CSRT_DEV_NONFINITE. */
int prox_rmsprop_update_compact(const csrt_csr *w_in, const float *g, float *v, float eta, float lambda,
                                float beta, float eps, csrt_csr *w_out, void *ws, size_t ws_bytes,
                                void *stream);

/* prox_adam_update_compact -- step t (t >= 1, counted by the caller) of
 * Prox-ADAM (Algorithm 2): the prox step along the bias-corrected Adam
 * direction. m and v (dense row-major M x K float32, the first and second
 * moments of G, zero before step 1) are updated in place. Per entry, with
 * c_i = fl32(1 - beta_i) and bc_i = fl32(1 - beta_i^t) (power in float64):
 *   m <- fl(fl(beta1*m) + fl(c1*G));  v <- fl(fl(beta2*v) + fl(c2*fl(G*G)))
 *   d = fl(fl(m/bc1) / fl(fl(sqrt(fl(v/bc2))) + eps))
 * then the prox step of prox_update_compact along d. beta1, beta2 in [0, 1),
 * eps finite and > 0; m, v and G must not alias each other. */
int prox_adam_update_compact(const csrt_csr *w_in, const float *g, float *m, float *v, int32_t t, float eta,
                             float lambda, float beta1, float beta2, float eps, csrt_csr *w_out, void *ws,
                             size_t ws_bytes, void *stream);

/* weight_grad_prox_update -- weight_grad_dense followed by
 * prox_update_compact without writing G: the tensor-core GEMM's epilogue forms
 * z = w - eta*G from the accumulator and applies the soft threshold of Section
 * 2.2 (Eq. prox, Section 3.3). The GEMM runs twice: a count pass writes the
 * keep bitmask and per-row counts, and after the row-pointer scan a write pass
 * recomputes the same accumulator and writes the kept entries of w_out at
 * their final positions (the transposed arrays, when set, are then built from
 * the bitmask). The result is bit-identical to weight_grad_dense(precision) +
 * prox_update_compact.
 * The fused path runs for precision CSRT_PREC_TF32 on tcgen05 GPUs with
 * n % 4 == 0, rows and cols >= 64, cols % 32 == 0, cols <= 16384 and 16-byte
 * aligned dY and X; otherwise the two calls run unfused through g_scratch
 * (M x K floats, may be NULL when the fused path applies). */
int weight_grad_prox_update(const csrt_csr *w_in, const float *dy, const float *x, int32_t n,
                            float eta, float lambda, int32_t precision, float *g_scratch,
                            csrt_csr *w_out, void *ws, size_t ws_bytes, void *stream);

/* debias_update -- the retraining step of Section 2.4 / Section 4.3 (zero
 * weights fixed and not updated): val[k] <- fl32(val[k] - fl32(eta*g_nnz[k]))
 * for every stored entry; row_ptr and col_idx are untouched, and a value
 * reaching 0.0 stays stored. If w->t_val is not NULL the transposed values
 * are updated through t_pos. */
int debias_update(csrt_csr *w, const float *g_nnz, float eta, void *stream);

/* ------------------------------------------------------------------------ */
/* Network glue (Caffe layers the paper uses but does not describe).         */
/* Convolution activations are C x (B*H*W) matrices: channel, then sample,   */
/* then row, then column.                                                    */
/* ------------------------------------------------------------------------ */

/* y[i, c] += bias[i]; then y = max(y, 0) if relu != 0. In place, m x n. */
int csrt_bias_act_fwd(float *y, const float *bias, int32_t m, int32_t n, int32_t relu, void *stream);

/* dy[e] = y[e] > 0 ? dy[e] : 0 for e < count (ReLU backward through its output). */
int csrt_relu_bwd(float *dy, const float *y, int64_t count, void *stream);

/* gb[i] = sum_c dy[i, c]; bias[i] <- fl32(bias[i] - fl32(eta*gb[i])).
 * gb_out (m floats) may be NULL. Plain SGD, no regulariser. */
int csrt_bias_grad_sgd(const float *dy, int32_t m, int32_t n, float *bias, float eta,
                       float *gb_out, void *stream);

/* Mean softmax cross-entropy over the n columns of z (classes x n).
 * `loss` holds n + 1 floats: loss[1 + c] = -log softmax(z[:, c])[labels[c]]
 * and loss[0] = their mean (summed in a fixed order).
 * dz = (softmax(z) - onehot(labels)) / n (the 1/|B| of the minibatch
 * gradient, Section 2.2). labels are int32 in [0, classes). */
int csrt_softmax_xent(const float *z, const int32_t *labels, int32_t classes, int32_t n,
                      float *dz, float *loss, void *stream);

/* Unfold x (c x (b*h*w)) into cols ((c*k*k) x (b*ho*wo)), stride 1, no
 * padding: cols[c*k*k + ky*k + kx][s*ho*wo + oy*wo + ox] = x[c][s][oy+ky][ox+kx]. */
int csrt_im2col(const float *x, int32_t c, int32_t b, int32_t h, int32_t w, int32_t k,
                float *cols, void *stream);

/* Adjoint of csrt_im2col: dx = sum of every column entry onto its pixel. */
int csrt_col2im(const float *dcols, int32_t c, int32_t b, int32_t h, int32_t w, int32_t k,
                float *dx, void *stream);

/* csrt_conv2d_sparse_fwd -- the forward product of a convolution layer with
 * compressed filters (Section 3.2: W x the unfolded input, here without
 * unfolding it): y[m][s*ho*wo + oy*wo + ox] = act(fl32(sum over the stored
 * taps t = (ci*k + ky)*k + kx of row m of W of val * x[ci][s][oy+ky][ox+kx]
 * + bias[m])), float32 accumulation in CSR order. x is c x (b*h*w), y is
 * W->rows x (b*ho*wo), stride 1, no padding; W has c*k*k columns and at most
 * 65535 rows. bias (W->rows floats) may be NULL; act = ReLU when relu != 0.
 * The same product as csrt_im2col then spmm_fwd (up to summation order). */
int csrt_conv2d_sparse_fwd(const csrt_csr *w, const float *x, int32_t c, int32_t b, int32_t h, int32_t wd,
                           int32_t k, const float *bias, int32_t relu, float *y, void *stream);

/* 2x2 max pooling, stride 2 (h, w even): y is c x (b*(h/2)*(w/2)); idx (int8)
 * records the winning window position dy*2+dx, first maximum in scan order. */
int csrt_maxpool2_fwd(const float *x, int32_t c, int32_t b, int32_t h, int32_t w,
                      float *y, int8_t *idx, void *stream);

/* Route pooled gradients back: dx (c x (b*h*w)) is overwritten. */
int csrt_maxpool2_bwd(const float *dy, const int8_t *idx, int32_t c, int32_t b, int32_t h,
                      int32_t w, float *dx, void *stream);

/* (c x (b*hw)) -> ((c*hw) x b): xf[ci*hw + s][bi] = x[ci][bi*hw + s] (Caffe
 * flatten order), and its inverse. */
int csrt_flatten(const float *x, int32_t c, int32_t b, int32_t hw, float *xf, void *stream);
int csrt_unflatten(const float *xf, int32_t c, int32_t b, int32_t hw, float *x, void *stream);

#ifdef __cplusplus
}
#endif

#endif /* CSRTRAIN_H */
