/*
 * realq.h - C ABI of the GB300 (sm_103a) REAL-Q per-layer quantization sweep.
 *
 * The library quantizes one linear module W (m x n, out x in, row-major) to
 * b-bit integer codes with per-group scale and zero point.  The sweep is the
 * per-module part of Algorithm 1 of "REAL-Q: E2E LLM Quantization via Dynamic
 * Gradient Descent":
 *   1. accumulate the input second moment H = sum_t x̂_t x̂_t^T of the perturbed
 *      calibration inputs (Sec. 3.2, "GPTQ Recap");
 *   2. damp H and form the upper Cholesky factor U of H^-1 (Alg. 1, "compute
 *      ... H_g and its inverse");
 *   3. sweep the columns in blocks of B: quantize each column and feed its error
 *      back into the later columns of the block (Eq. gptq_update), then apply
 *      the batched update to all columns after the block (Sec. 3.2);
 *   4. after every block take one Adam step on the columns after the block,
 *      descending the aggregated-Fisher surrogate (Eq. fisher_loss,
 *      Eq. block_gd_update), optionally blended with the next transformer
 *      block's Fisher (Eq. slide_window).
 *
 * Conventions shared by every entry point
 *   - Pointers are DEVICE pointers unless marked (host).  Matrices are dense,
 *     row-major, without padding (leading dimension = number of columns).
 *   - The caller owns every buffer; the library allocates no device memory.
 *     Scratch comes from a caller-provided workspace whose size is returned by
 *     the matching *_workspace_size function (256-byte aligned pointer).
 *   - All work is enqueued on `stream` (a cudaStream_t passed as void*; NULL
 *     is the legacy default stream).  Calls are asynchronous unless stated.
 *   - Argument errors are detected on the host before anything is enqueued and
 *     leave every buffer untouched: REALQ_ERR_INVALID_ARG /
 *     REALQ_ERR_WORKSPACE / REALQ_ERR_UNSUPPORTED.  realq_last_error() gives a
 *     thread-local description of the last failure.
 *   - No exception crosses the ABI.  Besides the thread-local error string
 *     and the optional profiling counters, the library keeps only reusable
 *     helpers: for each (calling thread, caller's stream, its priority) a few
 *     auxiliary streams and events, created on the first call that wants
 *     them (prepare's triangular-inverse work and look-ahead, the sweep's
 *     side product) and kept for the life of the thread.  Work on them forks
 *     from the caller's stream and joins back into it inside the call, so
 *     every call stays ordered on the caller's stream; make one call on a
 *     stream before capturing that stream into a CUDA graph.  While
 *     profiling is on they are not used.
 *   - Device-side conditions (a non-positive pivot, a non-finite weight, a
 *     bounded wait that gave up) are recorded in the workspace's status word
 *     and read by the calls documented to synchronize (realq_hessian_prepare,
 *     realq_prepare_status, realq_workspace_status).
 */
#ifndef REALQ_H
#define REALQ_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef void *realq_stream_t; /* cudaStream_t */

typedef enum {
    REALQ_OK = 0,
    REALQ_ERR_INVALID_ARG = 1, /* null pointer, bad size or bad config value */
    REALQ_ERR_WORKSPACE = 2,   /* workspace missing, too small or misaligned */
    REALQ_ERR_NOT_SPD = 3,     /* damped Hessian not positive definite (prepare) */
    REALQ_ERR_NONFINITE = 4,   /* NaN/Inf met in the weights during the sweep */
    REALQ_ERR_TIMEOUT = 5,     /* a bounded device-side wait gave up */
    REALQ_ERR_CUDA = 6,        /* a CUDA runtime call or launch failed */
    REALQ_ERR_UNSUPPORTED = 7  /* valid but not implemented combination */
} realq_status_t;

typedef enum { REALQ_F32 = 0, REALQ_BF16 = 1 } realq_dtype_t;

/* Quantizer and sweep geometry.
 *   bits        2..4 (codes are stored as 4-bit nibbles).
 *   group_size  columns sharing one (scale, zero) per row; 0 = one group per
 *               row.  Must divide block_size or be a multiple of it.
 *   block_size  column block B of the sweep: 32, 64 or 128 (paper: 128).
 *   symmetric   0: asymmetric min/max grid containing 0 with an integer zero
 *               point; 1: symmetric grid, zero = 2^(bits-1).
 *   damp_frac   lambda = damp_frac * mean(diag(H̄)) is added to the diagonal. */
typedef struct {
    int bits;
    int group_size;
    int block_size;
    int symmetric;
    float damp_frac;
} realq_quant_cfg_t;

enum { REALQ_OPT_ADAM = 0, REALQ_OPT_SGD = 1 };

/* Block-wise gradient descent (Sec. 4.3, App. "Full Setup").
 *   steps_per_block  optimizer steps after each column block (paper: 1; 0
 *                    turns Block-GD off and the sweep is plain GPTQ).
 *   optimizer        REALQ_OPT_ADAM (paper) or REALQ_OPT_SGD.
 *   lr, beta1, beta2, eps   paper: lr per model, 0.9, 0.999, 1e-8.
 *   b_global_start   1-based cumulative column-block index of this module's
 *                    first block within the transformer block (Eq. slide_window).
 *   B_total          column-block steps of the whole transformer block; with
 *                    B_total > 1 and F_next given, the Fisher used after block
 *                    b is alpha F + (1 - alpha) F_next,
 *                    alpha = 1 - (b_global - 1) / (B_total - 1). */
typedef struct {
    int steps_per_block;
    int optimizer;
    float lr;
    float beta1;
    float beta2;
    float eps;
    int b_global_start;
    int B_total;
} realq_bgd_cfg_t;

/* ------------------------------------------------------------------------ */
/* Step 1. Hessian accumulation (Sec. 3.2: H is the second moment of the
 * calibration inputs; REAL-Q uses the perturbed inputs x̂).
 *   H_sum += X̂^T X̂                      (n x n fp32, full symmetric matrix)
 *   D_sum += (X̂ - X)^T X̂   if X_fp != NULL (n x n fp32; D_sum[i][j] =
 *            sum_t (x̂_ti - x_ti) x̂_tj), needed by the surrogate when the
 *            reference output W0 x uses unperturbed inputs.
 * X_hat, X_fp: T_chunk x n, token-major, dtype x_dtype.  T_chunk = 0 is a
 * no-op.  Call once per chunk of calibration tokens; the caller zeroes H_sum
 * (and D_sum) before the first chunk and keeps the token count. Asynchronous.
 * x_dtype = REALQ_BF16: products are exact in fp32, sums are fp32. */
realq_status_t realq_hessian_accumulate(realq_stream_t stream, int64_t n, int64_t T_chunk,
                                        const void *X_hat, const void *X_fp, realq_dtype_t x_dtype,
                                        float *H_sum, float *D_sum, void *ws, size_t ws_bytes);
/* Workspace for one accumulate call: a status word (first 256 bytes) and the
 * token-split partial sums, reduced in a fixed order so results are bitwise
 * repeatable.  ws may be NULL (no split, no status word).  bf16 inputs with
 * n % 8 == 0 and a 16-byte aligned X_hat run on the tensor cores; a tile whose
 * bounded pipeline wait gave up is written as NaN and the status word gets a
 * timeout bit, read with realq_workspace_status(). */
size_t realq_hessian_workspace_size(int64_t n, int64_t T_chunk, realq_dtype_t x_dtype, int has_X_fp);

/* Step 2. Preparation (Alg. 1: Hessian and its inverse; the inverse used by
 * the column step is the Cholesky factorisation of H^-1, whose rows equal the
 * Schur-complement-downdated rows of H^-1 used by Eq. gptq_update).
 *   Hbar_out = H_sum / T_total                       (n x n, undamped)
 *   dead_out[j] = (H_sum[j][j] == 0)                 (n bytes; channel never fires)
 *   Hd = Hbar with Hd[j][j] = 1 on dead channels, plus lambda I,
 *        lambda = damp_frac * mean(diag(Hd before damping))
 *   U_out: upper triangular, Hd^-1 = U^T U           (n x n; strictly lower part = 0)
 * H_sum must be symmetric.  Hbar_out may alias H_sum (in-place).  This call
 * SYNCHRONIZES `stream` once to read the factorisation status: if a pivot is
 * not positive it returns REALQ_ERR_NOT_SPD and *fail_col (host) holds the
 * column, else *fail_col = -1.  Outputs are unspecified after NOT_SPD. */
realq_status_t realq_hessian_prepare(realq_stream_t stream, int64_t n, int64_t T_total, float damp_frac,
                                     const float *H_sum, float *U_out, float *Hbar_out, uint8_t *dead_out,
                                     int64_t *fail_col, void *ws, size_t ws_bytes);
size_t realq_prepare_workspace_size(int64_t n);

/* realq_hessian_prepare without the host synchronisation, for stream
 * capture into a CUDA graph and for callers that check later: the call only
 * enqueues work on `stream` (and on auxiliary streams of the calling thread
 * that fork from and join back into it; make one call on a given stream
 * before capturing it, so that they exist).  Same arguments and results as
 * realq_hessian_prepare; the factorisation status stays in the workspace's
 * first word (-1, or the first column whose pivot was not positive) until
 * the next prepare call on that workspace and is read with
 * realq_prepare_status once the work has completed. */
realq_status_t realq_hessian_prepare_deferred(realq_stream_t stream, int64_t n, int64_t T_total, float damp_frac,
                                              const float *H_sum, float *U_out, float *Hbar_out, uint8_t *dead_out,
                                              void *ws, size_t ws_bytes);
/* Status of the last prepare call on workspace ws (synchronizes `stream`,
 * which must be ordered after that call): REALQ_ERR_NOT_SPD with *fail_col
 * (host) = the column, else REALQ_OK with *fail_col = -1. */
realq_status_t realq_prepare_status(realq_stream_t stream, void *ws, size_t ws_bytes, int64_t *fail_col);

/* Allocation-free variant of realq_hessian_prepare.  The paper has no
 * counterpart: this exists for callers that cannot allocate device memory,
 * e.g. a plugin running inside a host application that owns every device
 * allocation and exposes no allocator through this C interface, or a
 * long-running service that reserves all of its memory up front and must not
 * allocate (or let cudaMalloc / cudaFree synchronize the device) once it runs.
 * Same arguments, results, synchronization and NOT_SPD behaviour as
 * realq_hessian_prepare, without the workspace: its scratch is a file-scope
 * device array of the library sized for n <= REALQ_PREPARE_NOALLOC_MAX_N
 * (about 8.4 MB, held by every GPU that loads the library until the process
 * exits).  Larger n returns REALQ_ERR_INVALID_ARG before any work is queued.
 * The call allocates nothing (no cudaMalloc / cudaFree, no allocating library
 * routine).  Every call looks up the array's device address on the current
 * device; the first call on a device may load the library's device code
 * there, so make that first call before any stream capture.  All calls
 * share the one array, which keeps the last call's
 * contents (the status word is cleared at the start of each call, the rest is
 * overwritten before it is read), so calls that overlap on the GPU race: do
 * not run two of them concurrently on one device. */
#define REALQ_PREPARE_NOALLOC_MAX_N 32768
realq_status_t realq_hessian_prepare_noalloc(realq_stream_t stream, int64_t n, int64_t T_total, float damp_frac,
                                             const float *H_sum, float *U_out, float *Hbar_out, uint8_t *dead_out,
                                             int64_t *fail_col);

/* Token-form mini-batch Block-GD with per-token output clipping (Sec. 4.3,
 * "a calibration mini-batch" per step, 32 sequences in Sec. 5.1; App.
 * "Activation clipping (a_loss_clip) for small Qwen3 models", 0.95 there).
 * The same sweep as realq_quantize_layer_minibatch, but each optimizer step
 * takes its gradient from the mini-batch's tokens:
 *   Δ_t = (Ŵ - W0) x̂_t                       (m, per token of the mini-batch)
 *   q_t = the ceil(a_loss_clip m)-th smallest |Δ_t,i| (a_loss_clip in
 *         double precision, the product and its ceiling in double: for a
 *         percentile written with a few decimals, 0.95 or 0.99, that is the
 *         exact rank, e.g. 0.99 of 8000 values is the 7920th)
 *   kappa_t,i = q_t / |Δ_t,i| if |Δ_t,i| > q_t, else 1   (held constant)
 *   G = (1/T_k) sum_t (kappa_t ⊙ F_eff (kappa_t ⊙ Δ_t)) x̂_tᵀ, free columns
 * and one optimizer step per G.  Mini-batch k holds tokens
 * [k T_mb, min((k+1) T_mb, T)) of X_hat; step s of the block with global
 * index b_global uses k = ((b_global - 1) steps_per_block + s) mod
 * ceil(T / T_mb).  a_loss_clip = 1 scales no channel: the gradient is then
 * the moment form on the mini-batch (F_eff (Ŵ - W0) H̄_k).
 *   X_hat   T x n bf16, token-major, 16-byte aligned, n % 8 == 0; the
 *           calibration tokens whose H gave U and Hbar (unperturbed: the
 *           reference output is W0 x̂).
 *   T_mb    tokens per mini-batch, a multiple of 4, at most 2,097,120.
 * Needs the tensor-core path (m, n multiples of 4, >= 32; block_size > 0).
 * Everything else as realq_quantize_layer.  The products take the token
 * axis on the tensor cores in fp32-level precision (tf32x3); the workspace
 * holds the mini-batch twice in fp32 plus four T_mb x m buffers. */
size_t realq_quantize_tokens_workspace_size(int64_t m, int64_t n, int64_t T_mb, const realq_quant_cfg_t *qcfg,
                                            const realq_bgd_cfg_t *bcfg, int has_F_next);
realq_status_t realq_quantize_layer_tokens(realq_stream_t stream, int64_t m, int64_t n, const void *W0,
                                           realq_dtype_t w_dtype, const float *U, const float *Hbar,
                                           const uint8_t *dead, const void *X_hat, int64_t T, int64_t T_mb,
                                           double a_loss_clip, const realq_quant_cfg_t *qcfg,
                                           const realq_bgd_cfg_t *bcfg, const float *F, const float *F_next,
                                           float *W_work, float *adam_m, float *adam_v, float *bgd_disp,
                                           int64_t *adam_t, uint8_t *codes, float *scale, uint8_t *zero, void *W_deq,
                                           realq_dtype_t deq_dtype, int64_t block_begin, int64_t block_end, void *ws,
                                           size_t ws_bytes);

/* Weight-activation setting (Sec. 5, "Weight-Activation Quantization";
 * W4A4 uses 4 bits and a_clip = 0.9).  Per-token symmetric quantization of
 * the calibration activations X (T x n, row-major, REALQ_BF16 or REALQ_F32):
 * for each token t, xmax = a_clip * max_j |X[t, j]| (1 for a row of zeros),
 * scale[t] = 2 xmax / (2^bits - 1), zero point 2^(bits-1), and
 *   codes[t, j] = clamp(rint(X[t, j] / scale[t]) + 2^(bits-1), 0, 2^bits - 1),
 *   X_q[t, j]   = scale[t] * (codes[t, j] - 2^(bits-1)),
 * formed in fp32 with IEEE-rounded operations and stored in x_dtype (bf16:
 * round to nearest even).  In the activation-aware variant X_q is the x̂ given
 * to realq_hessian_accumulate (with X as X_fp, so that the surrogate keeps
 * the full-precision reference).
 *   X_q     T x n, x_dtype, may alias X.
 *   codes   NULL, or T x ceil(n/2) bytes for bits <= 4 (two codes per byte,
 *           even column in the low nibble), T x n bytes for bits 5..8.
 *   scale   NULL, or T floats.
 * bits in [2, 8], 0 < a_clip <= 1, inputs finite.  Asynchronous; allocates
 * nothing. */
realq_status_t realq_quantize_activations(realq_stream_t stream, int64_t T, int64_t n, const void *X,
                                          realq_dtype_t x_dtype, int bits, float a_clip, void *X_q, uint8_t *codes,
                                          float *scale);

/* Saliency-weighted Hessians of the coarse stage (Sec. 3.3 Eq.
 * saliency_hessian, used by Alg. 1 for every row group g; N_g = 4 in the
 * paper), and the Hessian-side saliency clipping of the appendix.
 *
 * realq_saliency_clip: S is T x n_groups fp32 (row-major: S[t * n_groups + g]
 * is token t's saliency for row group g, >= 0 and finite).  clip_out[g] is the
 * nearest-rank pct-percentile of column g over the T tokens (the smallest
 * value with at least pct * T values at or below it, i.e. the ceil(pct T)-th
 * smallest: an input value, bit for bit); S_out = min(S, clip_out[g])
 * elementwise (may alias S, may be NULL to get the thresholds only).
 * 0 < pct <= 1, in double precision, the rank ceil(pct T) taken in double
 * (exact for a percentile written with a few decimals: 0.99 of 8000 tokens
 * is the 7920th smallest).  Asynchronous; allocates nothing. */
realq_status_t realq_saliency_clip(realq_stream_t stream, int64_t T, int n_groups, const float *S, double pct,
                                   float *S_out, float *clip_out);

/* H_g += sum_t S[t, g] x̂_t x̂_t^T for every group g (H_g: n_groups x n x n
 * fp32, group g at H_g + g n^2) and wsum[g] += sum_t S[t, g] (fp64), for a
 * chunk of T_chunk bf16 tokens X_hat (T_chunk x n; n a multiple of 8, at
 * least 64).  Each product is formed as x_i (s x_j) with s x_j split into two
 * bf16 parts, within 2^-17 relative of s x_i x_j, and accumulated in fp32 as
 * realq_hessian_accumulate does (both triangles are computed; prepare reads
 * the upper one).  ws: at least
 * realq_hessian_weighted_workspace_size(n, T_chunk) bytes, 256-byte aligned;
 * its first word is the status that realq_workspace_status reads.
 * Asynchronous. */
size_t realq_hessian_weighted_workspace_size(int64_t n, int64_t T_chunk);
realq_status_t realq_hessian_accumulate_weighted(realq_stream_t stream, int64_t n, int64_t T_chunk,
                                                 const void *X_hat, int n_groups, const float *S, float *H_g,
                                                 double *wsum, void *ws, size_t ws_bytes);

/* realq_hessian_prepare with a real normaliser: Hbar = H_sum / norm (for a
 * weighted Hessian, norm = the weight sum; the OBS step does not depend on
 * it).  Everything else as realq_hessian_prepare. */
realq_status_t realq_hessian_prepare_scaled(realq_stream_t stream, int64_t n, double norm, float damp_frac,
                                            const float *H_sum, float *U_out, float *Hbar_out, uint8_t *dead_out,
                                            int64_t *fail_col, void *ws, size_t ws_bytes);

/* Dbar = D_sum / T_total (n x n); may alias D_sum.  Asynchronous. */
realq_status_t realq_scale_moment(realq_stream_t stream, int64_t n, int64_t T_total, const float *D_sum,
                                  float *Dbar);

/* Steps 3-4. The column sweep with Block-GD for one module (Alg. 1, loop over
 * blocks b; Eq. gptq_update inside the block, the lazy batch update after it,
 * Eq. block_gd_update on the remaining columns).
 *   W0        m x n, original weights (w_dtype); also the surrogate's reference.
 *   U         n x n from realq_hessian_prepare; Hbar the undamped H / T.
 *   Dbar      n x n or NULL (X = X̂): the gradient is
 *             F_eff [ (Ŵ - W0) Hbar + W0 Dbar ] restricted to the free columns.
 *   dead      n bytes from prepare, or NULL (no dead channels).
 *   bcfg      NULL or steps_per_block = 0: plain GPTQ sweep (F, adam_* unused).
 *   F         m x m symmetric Fisher of the module-output space; F_next the
 *             next transformer block's (NULL: no sliding window).
 *   W_work    m x n fp32 state.  On a sweep starting at block 0 it is
 *             initialised from W0 (dead channels zeroed); on return its columns
 *             < min(block_end*B, n) hold the dequantized weights.
 *   adam_m, adam_v  m x n fp32 Adam moments (zeroed at block 0); adam_t (host)
 *             step counter in/out (set to 0 at block 0).
 *   bgd_disp  m x n fp32: sum of all optimizer steps applied so far (zeroed
 *             at block 0).  After the lazy batch update the OBS compensation
 *             leaves the free columns at a stationary point of the damped
 *             layer-local quadratic, so the surrogate gradient there is
 *               P_R = (bgd_disp Hbar)_R + lambda (bgd_disp - (W - W0))_R
 *                     (+ (W0 Dbar)_R),  0 on dead channels,
 *             the same value as ((W - W0) Hbar)_R without its cancellation;
 *             G = F_eff P_R.  Both products run on the tensor cores with
 *             fp32-level accuracy: as f16x3 (each operand row scaled by a
 *             power of two and split into fp16 hi / lo planes, three kind::f16
 *             MMAs per step) when m and n are multiples of 8, else as tf32x3
 *             (see realq_set_bgd_products).
 *   codes     m x ceil(n/2) bytes, two codes per byte, even column in the low
 *             nibble.  scale (fp32) and zero (uint8): m x ngroups, ngroups =
 *             ceil(n / group_size) (1 when group_size = 0).
 *   W_deq     optional m x n copy of the dequantized weights in deq_dtype
 *             (written for the processed columns), or NULL.
 *   block_begin, block_end  blocks [block_begin, block_end) of the
 *             ceil(n / B) blocks are processed; a sweep interrupted after block k
 *             resumes with block_begin = k + 1 and the same state buffers.
 * Asynchronous.  A NaN/Inf weight met by the column step is recorded in the
 * workspace status word, read by realq_workspace_status(). */
realq_status_t realq_quantize_layer(realq_stream_t stream, int64_t m, int64_t n,
                                    const void *W0, realq_dtype_t w_dtype,
                                    const float *U, const float *Hbar, const float *Dbar, const uint8_t *dead,
                                    const realq_quant_cfg_t *qcfg, const realq_bgd_cfg_t *bcfg,
                                    const float *F, const float *F_next,
                                    float *W_work, float *adam_m, float *adam_v, float *bgd_disp, int64_t *adam_t,
                                    uint8_t *codes, float *scale, uint8_t *zero,
                                    void *W_deq, realq_dtype_t deq_dtype,
                                    int64_t block_begin, int64_t block_end,
                                    void *ws, size_t ws_bytes);

/* The sweep with a row-grouped OBS (Alg. 1: "for all row-groups g"; the
 * saliency-weighted Hessians of Sec. 3.3 Eq. saliency_hessian): the rows of W
 * form n_row_groups contiguous groups of ceil(m / n_row_groups) rows, and
 * group g runs the OBS step and the lazy update against its own factor
 * (U_g + g n^2, from realq_hessian_prepare_scaled of H_g) with its own dead
 * channels (dead_g + g n).  Block-GD still descends the layer surrogate with
 * the plain Hbar for all rows jointly; it needs Hbar_g (the groups' undamped
 * H̄_g = H_g / weight sum, n_row_groups x n x n) and, with row groups, m and
 * n multiples of 4 and at least 32 (REALQ_ERR_UNSUPPORTED otherwise).
 * Everything else (outputs, state, workspace rules, resume) as
 * realq_quantize_layer; the workspace comes from
 * realq_quantize_grouped_workspace_size. */
size_t realq_quantize_grouped_workspace_size(int64_t m, int64_t n, int n_row_groups, const realq_quant_cfg_t *qcfg,
                                             const realq_bgd_cfg_t *bcfg, int has_F_next, int has_Dbar);
realq_status_t realq_quantize_layer_grouped(realq_stream_t stream, int64_t m, int64_t n, const void *W0,
                                            realq_dtype_t w_dtype, int n_row_groups, const float *U_g,
                                            const float *Hbar_g, const uint8_t *dead_g, const float *Hbar,
                                            const float *Dbar, const realq_quant_cfg_t *qcfg,
                                            const realq_bgd_cfg_t *bcfg, const float *F, const float *F_next,
                                            float *W_work, float *adam_m, float *adam_v, float *bgd_disp,
                                            int64_t *adam_t, uint8_t *codes, float *scale, uint8_t *zero,
                                            void *W_deq, realq_dtype_t deq_dtype, int64_t block_begin,
                                            int64_t block_end, void *ws, size_t ws_bytes);

/* The sweep with mini-batch Block-GD (Sec. 4.3: each Block-GD step evaluates
 * the surrogate on a calibration mini-batch; Sec. 5.1: 32 sequences per
 * step).  Hbar_mb holds n_minibatch second moments H̄_k = X̂_kᵀX̂_k / T_k
 * (n_minibatch x n x n, one per mini-batch of the calibration set, e.g. from
 * realq_hessian_accumulate and realq_scale_moment on each mini-batch).  Step
 * s (0-based) of block b takes mini-batch ((b_global - 1) steps_per_block + s)
 * mod n_minibatch, with b_global = bcfg->b_global_start + b, so the steps of a
 * transformer block rotate through the calibration set; its gradient is
 * F_eff ((Ŵ - W0) H̄_k) on the free columns.  The OBS part still uses U and
 * the full Hbar.  Needs Block-GD on the tensor-core path (m, n multiples of
 * 4, at least 32) and unperturbed inputs (no Dbar).  Everything else as
 * realq_quantize_layer; the workspace comes from
 * realq_quantize_minibatch_workspace_size. */
size_t realq_quantize_minibatch_workspace_size(int64_t m, int64_t n, int n_minibatch, const realq_quant_cfg_t *qcfg,
                                               const realq_bgd_cfg_t *bcfg, int has_F_next);
realq_status_t realq_quantize_layer_minibatch(realq_stream_t stream, int64_t m, int64_t n, const void *W0,
                                              realq_dtype_t w_dtype, const float *U, const float *Hbar,
                                              const uint8_t *dead, int n_minibatch, const float *Hbar_mb,
                                              const realq_quant_cfg_t *qcfg, const realq_bgd_cfg_t *bcfg,
                                              const float *F, const float *F_next, float *W_work, float *adam_m,
                                              float *adam_v, float *bgd_disp, int64_t *adam_t, uint8_t *codes,
                                              float *scale, uint8_t *zero, void *W_deq, realq_dtype_t deq_dtype,
                                              int64_t block_begin, int64_t block_end, void *ws, size_t ws_bytes);
size_t realq_quantize_workspace_size(int64_t m, int64_t n, const realq_quant_cfg_t *qcfg,
                                     const realq_bgd_cfg_t *bcfg, int has_F_next, int has_Dbar);

/* realq_quantize_layer with a trace of the surrogate (Eq. fisher_loss, moment
 * form at the layer level, L = 1/2 tr(F_eff ΔW H̄ ΔWᵀ), ΔW = Ŵ - W0 with the
 * quantized columns dequantized and the rest as they stand): for every block
 * b of the range that takes Block-GD steps (all but the layer's last),
 *   block_loss[2 b]     = L before the block's steps (after its OBS and lazy
 *                         update),
 *   block_loss[2 b + 1] = L after them,
 * with the block's F_eff (the sliding window's blend).  block_loss: device,
 * nb x 2 floats (the last block's pair is not written); trace_ws: device,
 * realq_quantize_trace_workspace_size(m, n) bytes.  Unperturbed inputs only
 * (no Dbar).  Each value is a full surrogate evaluation (about 2 m n^2 +
 * 2 m^2 n flops), and the block's optimizer step completes before the second
 * one, so tracing slows the sweep. */
realq_status_t realq_quantize_layer_traced(realq_stream_t stream, int64_t m, int64_t n, const void *W0,
                                           realq_dtype_t w_dtype, const float *U, const float *Hbar,
                                           const uint8_t *dead, const realq_quant_cfg_t *qcfg,
                                           const realq_bgd_cfg_t *bcfg, const float *F, const float *F_next,
                                           float *W_work, float *adam_m, float *adam_v, float *bgd_disp,
                                           int64_t *adam_t, uint8_t *codes, float *scale, uint8_t *zero, void *W_deq,
                                           realq_dtype_t deq_dtype, int64_t block_begin, int64_t block_end, void *ws,
                                           size_t ws_bytes, float *block_loss, void *trace_ws,
                                           size_t trace_ws_bytes);
size_t realq_quantize_trace_workspace_size(int64_t m, int64_t n);

/* Step 4 alone: bcfg->steps_per_block optimizer steps of Eq. block_gd_update
 * on the columns col_start..n-1 of W (columns < col_start are locked; they
 * hold dequantized values).  alpha blends F and F_next (ignored when F_next is
 * NULL).  adam_t (host) is advanced by the number of steps.  Asynchronous. */
realq_status_t realq_bgd_refine(realq_stream_t stream, int64_t m, int64_t n, int64_t col_start,
                                float *W, const void *W0, realq_dtype_t w_dtype,
                                const float *Hbar, const float *Dbar,
                                const float *F, const float *F_next, float alpha,
                                float *adam_m, float *adam_v, int64_t *adam_t,
                                const realq_bgd_cfg_t *bcfg, void *ws, size_t ws_bytes);
size_t realq_bgd_workspace_size(int64_t m, int64_t n, int has_F_next, int has_Dbar);

/* Surrogate of Eq. fisher_loss at the layer level with X = X̂:
 *   *loss_out (device fp32) = 1/2 tr(F (W_hat - W0) Hbar (W_hat - W0)^T).
 * Asynchronous. */
realq_status_t realq_surrogate_loss(realq_stream_t stream, int64_t m, int64_t n,
                                    const float *W_hat, const void *W0, realq_dtype_t w_dtype,
                                    const float *Hbar, const float *F, float *loss_out,
                                    void *ws, size_t ws_bytes);
size_t realq_surrogate_workspace_size(int64_t m, int64_t n);

/* Synchronizes `stream`, returns the device status word recorded at the start
 * of a Hessian, quantize or block-ops workspace (REALQ_OK, REALQ_ERR_TIMEOUT,
 * REALQ_ERR_NONFINITE) and clears it. */
realq_status_t realq_workspace_status(realq_stream_t stream, void *ws, size_t ws_bytes);

/* Diagnostics. */
const char *realq_status_string(realq_status_t s);
const char *realq_last_error(void);

/* Launch accounting and per-kernel timing.
 * realq_launch_count(): number of kernels this library has launched since load.
 * With profiling on, every launch is bracketed by CUDA events recorded on its
 * own stream, and calls keep all of their work on the caller's stream (no
 * auxiliary streams, same arithmetic), so that with one caller stream each
 * interval is the kernel's own time; realq_profile_collect synchronizes those
 * events, writes up to max_entries per-kernel totals and clears them. */
typedef struct {
    char name[48];
    int64_t launches;
    double total_ms;
} realq_kernel_stat_t;
int64_t realq_launch_count(void);
void realq_profile_enable(int on);
int realq_profile_collect(realq_kernel_stat_t *out, int max_entries);


/* CUDA graphs of whole steps.  A step of many small launches over several
 * streams (the block scheduler's) is recorded once and relaunched whole:
 *   realq_graph_begin(stream)   starts a thread-local stream capture of
 *                               `stream` (not the legacy default stream);
 *                               other streams join it by waiting on events
 *                               recorded in it and must join back before
 *                               the end.  Calls made meanwhile only enqueue.
 *   realq_graph_end(stream, node_priorities, &g)
 *                               ends the capture and instantiates the graph;
 *                               with node_priorities != 0 each kernel keeps
 *                               the priority of the stream it was captured
 *                               from (the critical chain of a step can be
 *                               favoured), else all run at the priority of
 *                               the stream the graph is launched into.
 *                               On failure *g = NULL.
 *   realq_graph_launch(g, s)    launches the graph on s (asynchronous); the
 *                               library's kernels in it count towards
 *                               realq_launch_count().
 *   realq_graph_kernels(g)      how many of this library's kernels g holds.
 *   realq_graph_destroy(g)      frees it (NULL is a no-op). */
typedef struct realq_graph_s *realq_graph_t;
realq_status_t realq_graph_begin(realq_stream_t stream);
realq_status_t realq_graph_end(realq_stream_t stream, int node_priorities, realq_graph_t *graph);
realq_status_t realq_graph_launch(realq_graph_t graph, realq_stream_t stream);
int64_t realq_graph_kernels(realq_graph_t graph);
void realq_graph_destroy(realq_graph_t graph);

/* Tuning: the output tile of the fp32-accurate (tf32x3) tensor-core
 * products of Block-GD and the lazy batch update.  0 (default): chosen per
 * launch from its grid (128 x 256 when its waves on the SMs take less time
 * than 128 x 128's), 1: always 128 x 128, 2: always 128 x 256.  Results do
 * not depend on it beyond the fp32 accumulation order of the tensor pipe.
 * Process-wide; not for use while other threads launch.  REALQ_ERR_INVALID_ARG
 * for other values.  No counterpart in the paper. */
realq_status_t realq_set_tensor_tile(int mode);

/* Tuning: the kernel of the column-serial quantize-and-compensate step.  0
 * (default): the kernel whose warps meet at a block-wide barrier after every
 * 32 columns; 1: warps pipelined through shared-memory progress flags where
 * the group parameters are taken at the block start or before it (more
 * instructions per warp for its polling and chunked updates: slower on
 * GB300, 41 against 31 us per 8192-row block).  Both perform the same
 * operations in the same order (identical results).
 * Process-wide.  REALQ_ERR_INVALID_ARG for other values.  No counterpart in
 * the paper. */
realq_status_t realq_set_quant_kernel(int mode);

/* Tuning: the plain Block-GD products (the gradient factor P and G = F_eff P
 * of realq_quantize_layer and the traced sweep).  1 (default): f16x3 where m
 * and n are multiples of 8 (fp16 planes with power-of-two row scales: the
 * same 22 significant bits per operand as tf32x3 at twice the tensor rate);
 * 0: tf32x3.  The row-grouped, mini-batch and token-form sweeps always take
 * tf32x3.  Results differ by fp32-level rounding.  Process-wide; read when
 * a sweep starts.  REALQ_ERR_INVALID_ARG for other values.  No counterpart
 * in the paper. */
realq_status_t realq_set_bgd_products(int mode);

/* Tuning: the f16x3 G product (G = F_eff P with the fused Adam step) on
 * 128 x 256 tiles.  1 (default): a persistent kernel, one CTA per SM walking
 * the tiles, a TMA warp, an MMA warp and eight epilogue warps, with two TMEM
 * accumulators so that a tile's epilogue overlaps the next tile's main
 * loop; 2: the gradient-factor product P as well; 0: one tile per CTA, the
 * epilogue after the main loop.  The same MMAs in the same order per tile
 * and the same epilogue arithmetic (identical results).  Process-wide.
 * REALQ_ERR_INVALID_ARG for other values.  No counterpart in the paper. */
realq_status_t realq_set_tensor_overlap(int mode);

/* Tuning: the causal attention of the block ops.  1 (default): tiled
 * kernels (64 rows of a CTA against 32-wide tiles streamed through shared
 * memory, online softmax; fp32 on the CUDA cores); 0: one thread per query
 * or key row.  The same arithmetic up to the fp32 summation order.
 * Process-wide.  REALQ_ERR_INVALID_ARG for other values.  No counterpart in
 * the paper. */
realq_status_t realq_set_block_attention(int mode);

/* Tuning: the products of the block ops (realq_block_*, and the window
 * quantization's loss).  0 (default): fp32 CUDA-core tiles for all; 1:
 * tf32x3 tensor-core products where the operands fit the workspace's plane
 * scratch.  tf32x3 keeps 22 significant bits of each operand against fp32's
 * 24, and the window's loss (a difference of two forward passes) magnifies
 * that about tenfold: its gradient moves a few group scales of a window
 * sweep by more than 1e-5, while the projections are under 1 % of the
 * window's time (the attention is the rest).
 * Process-wide.  REALQ_ERR_INVALID_ARG for other values.  No counterpart in
 * the paper. */
realq_status_t realq_set_block_products(int mode);

/* The learning rate of decoder block i (1-based) of L under the paper's
 * reverse-cosine schedule over transformer blocks (App. "Full Setup",
 * Eq. reverse_cosine; the first block's rate is 0.01 of the final one, App.
 * "REAL-Q Learning Rates"):
 *   eta_i = eta_base + (eta_final - eta_base) sin(pi/2 (i - 1) / (L - 1)),
 *   eta_base = 0.01 eta_final;  eta_final when L = 1.
 * Host arithmetic in double; *lr_out (host) receives it.  1 <= i <= L and a
 * finite lr_final required, else REALQ_ERR_INVALID_ARG. */
realq_status_t realq_reverse_cosine_lr(int64_t i, int64_t L, double lr_final, double *lr_out);

/* ---- The next decoder block of the exact two-block sliding window ----
 * Sec. 4.4, Eq. (slide_window): while block l is quantized, the loss blends
 * block l's Fisher loss with block l+1's, and the latter is back-propagated
 * from block l+1's output.  These entry points compute that block: its
 * forward pass, and the next block's Fisher loss
 *   L(l+1) = (1/2T) sum_t dz_t^T F' dz_t,  dz = B(h + dh) - B(h),
 * with its gradient g_h = dL(l+1)/d(dh) (T = S L tokens).
 * The block is the pre-norm LLaMA-3.1 / Qwen3 structure:
 *   a = RMSNorm(x; g1), h = x + Attn(a) Wo^T, b = RMSNorm(h; g2),
 *   y = h + (silu(b Wg^T) * (b Wu^T)) Wd^T,
 * RMSNorm(x; g) = x g / sqrt(mean(x^2) + rms_eps); causal grouped-query
 * attention (query head i reads key/value head i / (n_heads / n_kv)) with
 * rotary embedding on the pairs (j, j + head_dim/2) at angle
 * pos * rope_base^(-2j/head_dim), pos the token's place in its sequence, and
 * scale 1/sqrt(head_dim).
 *   dims      n_heads % n_kv == 0, head_dim even and <= 256.
 *   weights   device fp32, row-major (out x in): Wq (n_heads head_dim) x d,
 *             Wk, Wv (n_kv head_dim) x d, Wo d x (n_heads head_dim),
 *             Wg, Wu ffn x d, Wd d x ffn; gains g1, g2 of length d.
 *   x, y, h_ref, dh, g_h
 *             device fp32, S L x d row-major, token (s, t) at row s L + t
 *             (S sequences of L tokens).
 *   F_next    device fp32 d x d (the next block's Fisher).
 *   loss      device fp32 scalar, or NULL.
 *   ws        device workspace of realq_block_workspace_size(dims, S, L)
 *             bytes, 256-byte aligned; it holds the forward caches.  Its
 *             first int is a status word that each call clears at its start
 *             and that a timed-out bounded wait of a tensor-core product
 *             sets (read it with realq_workspace_status).
 * Computed in fp32 with fp32 accumulation (the loss summed in double); with
 * realq_set_block_products(1) the projections and products whose operands
 * fit the workspace's plane scratch run as tf32x3 tensor-core products.
 * Asynchronous on `stream`; argument errors are returned before any launch.
 * S L is at most 4194240 tokens.  Outputs may not alias inputs. */
typedef struct {
    int64_t d, n_heads, n_kv, head_dim, ffn;
    float rms_eps;    /* 1e-6 */
    float rope_base;  /* 10000 */
} realq_block_dims_t;
typedef struct {
    const float *g1, *Wq, *Wk, *Wv, *Wo, *g2, *Wg, *Wu, *Wd;
} realq_block_weights_t;
size_t realq_block_workspace_size(const realq_block_dims_t *dims, int64_t S, int64_t L);
realq_status_t realq_block_forward(realq_stream_t stream, const realq_block_dims_t *dims,
                                   const realq_block_weights_t *weights, int64_t S, int64_t L, const float *x,
                                   float *y, void *ws, size_t ws_bytes);
realq_status_t realq_block_window(realq_stream_t stream, const realq_block_dims_t *dims,
                                  const realq_block_weights_t *weights, int64_t S, int64_t L, const float *h_ref,
                                  const float *dh, const float *F_next, float *g_h, float *loss, void *ws,
                                  size_t ws_bytes);

/* realq_block_module_inputs: the calibration inputs of one module of the
 * block in a forward pass with `weights` on input x (S L x d), written to
 * X_out (S L x n, n the module's in-dimension): q/k/v read RMSNorm(x; g1),
 * o_proj the attention output (S L x n_heads head_dim), gate/up RMSNorm(h;
 * g2), down_proj the SwiGLU product (S L x ffn).  Their second moment is the
 * module's OBS Hessian (Sec. 3.2; in the sequential pipeline, the current
 * pass's inputs).  module 0..6 as below; ws as realq_block_forward. */
realq_status_t realq_block_module_inputs(realq_stream_t stream, const realq_block_dims_t *dims,
                                         const realq_block_weights_t *weights, int64_t S, int64_t L, const float *x,
                                         int module, float *X_out, void *ws, size_t ws_bytes);

/* Module level (any linear module of block l, Eq. slide_window): block l is
 * run at its reference weights on its reference input (h*, the full-precision
 * model) and as the current block (h: Sec. 4.3 evaluates the surrogate by a
 * forward pass through the current transformer block, on the perturbed
 * inputs that the quantized earlier blocks produce), dh = h - h*, and
 *   loss = alpha (1/2T) sum_t dh_t^T F_this dh_t + (1 - alpha) L(l+1)(h*, dh),
 *   grad = d loss / d W_module, back-propagated through block l's own
 *          backward (grad has W_module's shape).
 *   module    0..6 = q_proj, k_proj, v_proj, o_proj, gate_proj, up_proj,
 *             down_proj; W_module has that weight's shape (out x in).
 *   this_block, next_block
 *             both blocks' weights (same dims), at full precision;
 *             this_block holds the reference weight of the module.
 *   this_block_hat
 *             block l's weights in the current pass (the modules quantized
 *             so far), or NULL (= this_block); the module's own entry is
 *             replaced by W_module either way.
 *   x, x_hat  block l's reference input and its input in the current pass
 *             (the model quantized so far), S L x d; x_hat NULL (= x).
 *   alpha     the window's weight in [0, 1].
 *   ws        realq_block_module_workspace_size(dims, S, L, 0) bytes.
 * The final block (App. "Pre-computation of the aggregated Fisher and
 * last-transformer-block handling") has no next block; its loss is the true
 * KL at the LM head, Eq. (kl_loss):
 *   z = RMSNorm(h; gf) Wh^T (Wh vocab x d, gf length d),
 *   realq_block_head_kl:  loss = (1/T) sum_t KL(softmax z(h*_t) || softmax
 *             z(h*_t + dh_t)) and g_h = d loss / d dh, for given h* and dh
 *             (ws: realq_block_head_workspace_size(d, S, L, vocab) bytes);
 *   realq_block_module_kl: the same loss with h* and dh from block l as
 *             above, and grad = d loss / d W_module
 *             (ws: realq_block_module_workspace_size(dims, S, L, vocab)).
 * Same conventions as above (fp32 device buffers, 256-byte aligned
 * workspace, asynchronous on `stream`, host-side argument checks). */
size_t realq_block_module_workspace_size(const realq_block_dims_t *dims, int64_t S, int64_t L, int64_t vocab);
size_t realq_block_head_workspace_size(int64_t d, int64_t S, int64_t L, int64_t vocab);
realq_status_t realq_block_module_window(realq_stream_t stream, const realq_block_dims_t *dims,
                                         const realq_block_weights_t *this_block,
                                         const realq_block_weights_t *this_block_hat,
                                         const realq_block_weights_t *next_block, int64_t S, int64_t L, const float *x,
                                         const float *x_hat, int module, const float *W_module, float alpha,
                                         const float *F_this, const float *F_next, float *grad, float *loss, void *ws,
                                         size_t ws_bytes);
realq_status_t realq_block_head_kl(realq_stream_t stream, int64_t d, int64_t S, int64_t L, const float *gf,
                                   const float *Wh, int64_t vocab, float rms_eps, const float *h_ref, const float *dh,
                                   float *g_h, float *loss, void *ws, size_t ws_bytes);
realq_status_t realq_block_module_kl(realq_stream_t stream, const realq_block_dims_t *dims,
                                     const realq_block_weights_t *this_block,
                                     const realq_block_weights_t *this_block_hat, int64_t S, int64_t L,
                                     const float *x, const float *x_hat, int module, const float *W_module,
                                     const float *gf, const float *Wh, int64_t vocab, float *grad, float *loss,
                                     void *ws, size_t ws_bytes);

/* ---- The sweep with Block-GD on the block ops' loss ----
 * Alg. 1's column sweep for one linear module of decoder block l (Eq.
 * gptq_update inside each block, the lazy batch update after it) with each
 * Block-GD step (Eq. block_gd_update) descending the exact two-block window
 * of Sec. 4.4, Eq. (slide_window) (next_block given) or, for the last
 * decoder block, the true KL at the LM head of Eq. (kl_loss) (next_block
 * NULL; App. "Pre-computation of the aggregated Fisher and
 * last-transformer-block handling") in place of the layer-level surrogate.
 * After block b (columns < b_end quantized; b_end < n), steps_per_block
 * times: G = d loss / d W at W = W_work (the dequantized columns and the
 * free ones), through block l's own backward (realq_block_module_window with
 * alpha = 1 - (b_global - 1)/(B_total - 1), 1 when B_total = 1, b_global =
 * b_global_start + b; or realq_block_module_kl), then one Adam (or SGD) step
 * on the columns >= b_end of W_work with those columns of G.
 *   dims, this_block, this_block_hat, next_block, S, L, module, F_this,
 *   F_next    as realq_block_module_window.  The module's weight in
 *             this_block (fp32) is both the loss's reference and the sweep's
 *             W0; m x n is its shape (out x in).
 *   n_minibatch, x, x_hat
 *             the calibration mini-batches (Sec. 4.3: each step's forward
 *             pass uses a calibration mini-batch): x and x_hat (NULL: x) hold
 *             n_minibatch S sequences of L tokens (n_minibatch S L x d), and
 *             step s of column block b takes mini-batch
 *             ((b_global - 1) steps_per_block + s) mod n_minibatch, the
 *             sequences k S .. k S + S - 1.  The losses before and after a
 *             block's steps are those of its first and last step's
 *             mini-batch.
 *   head_gf, head_Wh, vocab   the final norm and LM head (next_block NULL);
 *             ignored otherwise.
 *   U, dead   realq_hessian_prepare of the module's input second moment
 *             (its calibration inputs in the current pass).
 *   bcfg      steps_per_block >= 1; optimizer, lr, betas, eps,
 *             b_global_start and B_total as for realq_quantize_layer.
 *   W_work, adam_m, adam_v, adam_t, codes, scale, zero, W_deq, deq_dtype,
 *   block_begin, block_end    as realq_quantize_layer (adam_m, adam_v and
 *             adam_t are zeroed at block 0).
 *   block_loss  NULL, or 2 device floats per column block: the loss before
 *             and after the block's steps (blocks with no free columns after
 *             them are left untouched; asking for them costs one more
 *             evaluation of the loss per block).
 *   ws        realq_quantize_window_workspace_size(dims, S, L, module, vocab,
 *             qcfg) bytes (vocab 0 for the window), 256-byte aligned; its
 *             first word is the sweep's status word (realq_workspace_status).
 * Asynchronous on `stream`; argument errors are returned before any launch. */
size_t realq_quantize_window_workspace_size(const realq_block_dims_t *dims, int64_t S, int64_t L, int module,
                                            int64_t vocab, const realq_quant_cfg_t *qcfg);
realq_status_t realq_quantize_layer_window(realq_stream_t stream, const realq_block_dims_t *dims,
                                           const realq_block_weights_t *this_block,
                                           const realq_block_weights_t *this_block_hat,
                                           const realq_block_weights_t *next_block, int64_t S, int64_t L,
                                           int64_t n_minibatch, const float *x, const float *x_hat, int module,
                                           const float *F_this, const float *F_next,
                                           const float *head_gf, const float *head_Wh, int64_t vocab, const float *U,
                                           const uint8_t *dead, const realq_quant_cfg_t *qcfg,
                                           const realq_bgd_cfg_t *bcfg, float *W_work, float *adam_m, float *adam_v,
                                           int64_t *adam_t, uint8_t *codes, float *scale, uint8_t *zero, void *W_deq,
                                           realq_dtype_t deq_dtype, float *block_loss, int64_t block_begin,
                                           int64_t block_end, void *ws, size_t ws_bytes);

#ifdef __cplusplus
}
#endif
#endif /* REALQ_H */
