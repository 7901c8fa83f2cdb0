// Host-side launchers of the library's kernels (internal interface).
#pragma once

#include <vector>

#include "common.cuh"

namespace realq {

// ------------------------------------------------------------------ GEMM ---
// C[M x N] (ldc) <- epilogue(alpha * A[M x K] * B[K x N]), fp32 FFMA, fp32
// accumulation.  B is row-major (B[k * ldb + j]).  A modes:
enum AMode {
    A_ROW = 0,        // A[i][k] = Af[i * lda + k]
    A_ROW_BF16 = 1,   // A[i][k] = bf16 Ab[i * lda + k]
    A_DIFF_F32 = 2,   // A[i][k] = Af[i * lda + k] - Yf[i * ldy + k]
    A_DIFF_BF16 = 3,  // A[i][k] = Af[i * lda + k] - bf16 Yb[i * ldy + k]
    A_KMAJOR = 4,     // A[i][k] = Af[k * lda + i]
};
enum EpiMode {
    EPI_STORE = 0,    // C = alpha * acc
    EPI_SUB = 1,      // C = C - alpha * acc
    EPI_BIAS = 2,     // C = alpha * acc + R[i * ldr + j]
    // Block-GD gradient after the lazy OBS update (column c = col0 + j):
    // C = alpha * acc + lam * (Ad[i][c] - (Wc[i][c] - W0c[i][c])) (+ R[i * ldr + j]),
    // and C = 0 on dead channels; Ad, Wc, W0c have leading dimension ldw.
    EPI_BGD_P = 3,
};
struct GemmArgs {
    int64_t M, N, K;
    const void *A; int64_t lda;
    const void *Y; int64_t ldy;
    const float *B; int64_t ldb;
    float *C; int64_t ldc;
    const float *R; int64_t ldr;
    float alpha;
    // A_ROW only: A(i, k) = sum over s < nsum of A[s * aplane + i * lda + k]
    int nsum; int64_t aplane;
    // K split over gridDim.z; EPI_STORE writes slice z to C + z * cplane
    int ksplit; int64_t cplane;
    // A(i, k) = 0 for k < i: start each CTA's K range at its first row
    int a_upper;
    // B(k, j) = 0 for k > j: end each CTA's K range at its last column
    int b_upper;
    // B(k, j) = sum over s < nsum_b of B[s * bplane + k * ldb + j]
    int nsum_b; int64_t bplane;
    // EPI_BGD_P operands
    const float *Ad; const float *Wc; const void *W0c; int w0_bf16;
    const uint8_t *dead; const float *lam; int64_t col0; int64_t ldw;
};
realq_status_t gemm_f32(cudaStream_t s, AMode am, EpiMode em, const GemmArgs &g, const char *name);

// ------------------------------------------- tensor-core tf32x3 GEMM ---
enum TcMode { TC_STORE = 0, TC_BGD_P = 1, TC_ADAM = 2, TC_ACCUM = 3, TC_BGD_PG = 4, TC_SYRK = 5 };
struct TcEpi {
    int mode;
    float *C; int64_t ldc;                                   // TC_STORE
    const float *Ad; const float *W; const void *W0; int w0_bf16;  // TC_BGD_P
    const uint8_t *dead; const float *lam; const float *R0; int64_t ldw; int64_t col0;
    float *Pth; float *Ptl; int64_t ldp;
    float *M;                                                // running A H̄ (acc += M, M = acc)
    float *Wm; float *mA; float *vA; float *D; float *Sh; float *Sl;  // TC_ADAM (ldw, col0 shared)
    float lr, b1, b2, eps, bc1, bc2; int sgd;
    int64_t czs;                                             // TC_STORE with a K split: C of split z at C + z czs
    int b_tri;   // B(j, k) = 0 for k > j (K range relative to the output column): a CTA's K ends at its last column
    // TC_STORE without a K split: C = alpha_s acc + R (R nullable, row stride ldr) when affine is set
    int affine; float alpha_s; const float *R; int64_t ldr;
    // f16x3 maps: the accumulator is in units of the operands' power-of-two
    // row scales; output (i, j) is acc ainv[i] binv[j] (both null otherwise).
    // With them, TC_BGD_P writes P^T in fp32 to Pth (Ptl null) and TC_ADAM
    // the step's negation in fp32 to Sh (Sl null), to be split afterwards.
    const float *ainv; const float *binv;
};
// The operand maps of one product, for both tile shapes of the kernel
// (128 x 128 outputs with 32-wide K slices, 128 x 256 with 16-wide slices).
struct TcMaps {
    alignas(64) unsigned char storage[8 * 128];
    int f16 = 0;   // fp16 planes (f16x3) instead of tf32 planes
};
bool tc_gemm_eligible(int64_t m, int64_t n);
// Tile shape of the tf32x3 products: 0 chosen per launch by its grid, 1 always
// 128 x 128, 2 always 128 x 256 (process-wide).
void tc_set_tile_mode(int mode);
// 1 (default): the wide-tile f16x3 G product (fused Adam epilogue) runs as a
// persistent kernel that overlaps each tile's epilogue with the next tile's
// main loop; 2: the gradient-factor product too; 0: one tile per CTA
// (process-wide).
void tc_set_overlap(int mode);
// The column-serial quantizer: 0 the barrier-phased kernel everywhere
// (default), 1 the pipelined kernel where the group parameters come at the
// block start or before it (process-wide).
void quant_set_kernel(int mode);
// hi / lo planes of the transpose of the rows x cols block at src (row stride
// lds): dst[c * ldd + r] for r < rows, c < cols.
realq_status_t tc_trans_planes(cudaStream_t s, int64_t rows, int64_t cols, const float *src, int64_t lds,
                               float *dh, float *dl, int64_t ldd);
// hi / lo planes of the rows x cols block at src (row stride lds), written
// to hi / lo with row stride ldd: columns 0..pad-1 of each row, those from
// cols on zero (pad >= cols, ldd >= pad).
realq_status_t tc_split_rows(cudaStream_t s, int64_t rows, int64_t cols, const float *src, int64_t lds, float *hi,
                             float *lo, int64_t ldd, int64_t pad);
// The operands of the lazy batch update W[:, be:] -= E_b U[bs:be, be:] as
// K-major tf32 planes: Eh/El = hi/lo of -E_b (m x B, from Et, kb x m with
// leading dimension ldet; skipped when Et is NULL), Ph/Pl = hi/lo of
// U[bs + k, be + j] (r x B, r = n - be).  kb a multiple of 32, <= B.
realq_status_t tc_trail_planes(cudaStream_t s, int64_t m, const float *Et, int64_t ldet, int64_t n, const float *U,
                               int64_t bs, int64_t be, int kb, int B, float *Eh, float *El, float *Ph, float *Pl);
realq_status_t tc_split(cudaStream_t s, int64_t count, const float *x, const float *y, float alpha, float *hi,
                        float *lo);
// The maps of an f16x3 product: fp16 hi / lo planes, K-major, row strides
// lda / ldb (multiples of 8 elements, 16-byte aligned bases).
realq_status_t tc_make_maps_f16(TcMaps *out, const __half *a_hi, const __half *a_lo, int64_t a_rows, int64_t a_k,
                                int64_t lda, const __half *b_hi, const __half *b_lo, int64_t b_rows, int64_t b_k,
                                int64_t ldb);
// fp16 hi / lo planes of rows of x (or of alpha x + (1 - alpha) y), columns
// c0 .. c1 - 1 (row stride lds), written at the same columns of hi / lo (row
// stride ldd), each row scaled by a power of two s_r that puts its largest
// magnitude in [2^14, 2^15): hi = fp16(s_r v), lo = fp16(s_r v - hi);
// inv[r] = 1 / s_r.
realq_status_t tc_split_f16_rows(cudaStream_t s, int64_t rows, int64_t c0, int64_t c1, const float *x, const float *y,
                                 float alpha, int64_t lds, __half *hi, __half *lo, int64_t ldd, float *inv);
// Precision of the plain Block-GD products (process-wide): 1 f16x3 where the
// shapes allow (default), 0 tf32x3 everywhere.
void bgd_set_products(int mode);
int bgd_products();
realq_status_t tc_make_maps(TcMaps *out, const float *a_hi, const float *a_lo, int64_t a_rows, int64_t a_k,
                            int64_t lda, const float *b_hi, const float *b_lo, int64_t b_rows, int64_t b_k,
                            int64_t ldb);
realq_status_t tc_gemm_x3(cudaStream_t s, const TcMaps &maps, int64_t M, int64_t N, int64_t K, int k_off,
                              int b_row0, const TcEpi &e, int *err, const char *name, int a_row0 = 0, int kchunk = 0,
                              int exact = 0);   // exact & 1: A exact in tf32 (no low plane), & 2: B
// g = sum_z part[z] (fixed order) and one optimizer step on the m x N block at
// column e.col0 (the TC_ADAM epilogue as a separate pass)
realq_status_t tc_gsum_adam(cudaStream_t s, int64_t m, int64_t N, int nz, const float *part, const TcEpi &e);
template <typename TY>
realq_status_t tc_split_diff(cudaStream_t s, int64_t count, const float *x, const TY *y, float *hi, float *lo);

// ------------------------------------------------- activation quantizer ---
realq_status_t act_quant(cudaStream_t s, int64_t T, int64_t n, const void *X, realq_dtype_t dt, int bits, float a_clip,
                         void *Xq, uint8_t *codes, float *scale);

// ------------------------------------------- saliency-weighted Hessians ---
size_t saliency_clip_ws_bytes();
realq_status_t saliency_clip(cudaStream_t s, int64_t T, int ng, const float *S, double pct, float *S_out,
                             float *clip_out);
size_t weighted_ws_bytes(int64_t n, int64_t T);
realq_status_t hessian_weighted(cudaStream_t s, int64_t n, int64_t T, const void *X, int ng, const float *S,
                                float *Hg, double *wsum, void *ws, size_t ws_bytes);

// --------------------------------------------------------------- Hessian ---
int hessian_splits(int64_t n, int64_t T, int num_sms);
int num_sms();
size_t hessian_ws_bytes(int64_t n, int64_t T, int has_xfp);
realq_status_t hessian_accumulate(cudaStream_t s, int64_t n, int64_t T, const void *X, const void *Xfp,
                                  realq_dtype_t dt, float *H, float *D, void *ws, size_t ws_bytes);
realq_status_t hessian_reduce(cudaStream_t s, int64_t n, int splits, const float *part, float *out, int mode);
bool hessian_tc_eligible(int64_t n, int64_t T, const void *X);
realq_status_t hessian_syrk_tc(cudaStream_t s, int64_t n, int64_t T, const void *X, float *H, int *err, void *ws,
                               size_t ws_bytes, int sms, float *H2 = nullptr);
// out += sign X_Aᵀ X_B.  chunk_stages: 64-token stages per TMEM accumulator
// pass before promotion (0: default).  symmetric: the product is known to be
// symmetric (X_B = diag(s) X_A up to rounding): lower tiles only, mirrored.
realq_status_t hessian_cross_tc(cudaStream_t s, int64_t n, int64_t T, const void *XA, const void *XB, float *out,
                                float sign, int *err, void *ws, size_t ws_bytes, int sms, int chunk_stages = 0,
                                bool symmetric = false);
int hessian_splits_tiles(int64_t tiles, int64_t T, int sms);

// --------------------------------------------------------------- prepare ---
size_t prepare_ws_bytes(int64_t n);
realq_status_t prepare(cudaStream_t s, int64_t n, double norm, float damp, const float *H, float *U, float *Hbar,
                       uint8_t *dead, int64_t *fail_col, void *ws, size_t ws_bytes);
realq_status_t prepare_deferred(cudaStream_t s, int64_t n, double norm, float damp, const float *H, float *U,
                                float *Hbar, uint8_t *dead, void *ws, size_t ws_bytes);
realq_status_t scale_copy(cudaStream_t s, int64_t count, float mul, const float *in, float *out);
// Host-side checks of the block ops' arguments for one module (the exact
// window when next_block is given, else the final block's KL at the LM head
// gf, Wh of vocab rows; this_block_hat may be NULL): the module's weight
// shape m x n and the block ops' workspace bytes.  Launches nothing.
realq_status_t block_loss_check(const realq_block_dims_t *dims, const realq_block_weights_t *this_block,
                                const realq_block_weights_t *this_block_hat, const realq_block_weights_t *next_block,
                                int64_t S, int64_t L, const float *x, int module, const float *F_this,
                                const float *F_next, const float *gf, const float *Wh, int64_t vocab, const char *who,
                                int64_t *m, int64_t *n, size_t *ws_bytes);
// One Adam (or SGD) step of Eq. block_gd_update on the columns c0.. of the
// m x n weights W with a full-width m x n gradient G (the block ops' module
// gradient): PyTorch-form Adam with bias corrections for step t >= 1.
// The block ops' causal attention, tiled (attention.cu): the forward (o and
// lse), the query gradient and the key / value gradients.
realq_status_t attn_fwd_tiled(cudaStream_t st, int64_t S, int64_t L, int64_t H, int64_t Hkv, int64_t dh,
                              const float *q, const float *k, const float *v, float *o, float *lse, const char *name);
realq_status_t attn_bwd_q_tiled(cudaStream_t st, int64_t S, int64_t L, int64_t H, int64_t Hkv, int64_t dh,
                                const float *q, const float *k, const float *v, const float *go, const float *lse,
                                const float *D, float *gq, const char *name);
realq_status_t attn_bwd_kv_tiled(cudaStream_t st, int64_t S, int64_t L, int64_t H, int64_t Hkv, int64_t dh,
                                 const float *q, const float *k, const float *v, const float *go, const float *lse,
                                 const float *D, float *gk, float *gv, const char *name);
// While one lives, the block ops called on this thread record a timed-out
// wait of their tensor-core products in *status (the caller's status word)
// instead of the status word at the start of their own workspace.
struct BlockStatusScope {
    explicit BlockStatusScope(int *status);
    ~BlockStatusScope();
    int *prev;
};
realq_status_t adam_cols(cudaStream_t s, int64_t m, int64_t n, int64_t c0, const float *G, float *W, float *mA,
                         float *vA, float lr, float b1, float b2, float eps, int64_t t, int sgd);
realq_status_t prepare_noalloc(cudaStream_t s, int64_t n, int64_t T, float damp, const float *H, float *U, float *Hbar,
                               uint8_t *dead, int64_t *fail_col);

// ----------------------------------------------------------------- sweep ---
struct SweepPlan {
    int64_t m, n;
    const void *W0; realq_dtype_t w_dtype;
    const float *U, *Hbar, *Dbar;
    const uint8_t *dead;
    int bits, group, block, sym;           // group = effective group size (n when per-row)
    int ngroups;
    // Block-GD
    int bgd_steps, optimizer;
    float lr, beta1, beta2, eps;
    int b_global_start, B_total;
    const float *F, *F_next;
    float damp;
    float *W, *adam_m, *adam_v, *disp;
    int64_t *adam_t;
    uint8_t *codes; float *scale; uint8_t *zero;
    void *W_deq; realq_dtype_t deq_dtype;
    // workspace pieces
    int *status;
    float *lam;
    float *Et, *P, *G, *Feff, *R0;
    // the lazy batch update on the tensor cores (tf32x3): planes of -E_b
    // (m x block) and of the block's U panel transposed (n x block)
    int trail_tc = 0, trail_maps = 0;
    float *Eh = nullptr, *El = nullptr, *UPh = nullptr, *UPl = nullptr;
    TcMaps mapsTr;
    // tensor-core path: hi / lo planes and tensor maps
    int tc;
    float *Sh, *Sl, *Hh, *Hl, *Fh, *Fl, *Pth, *Ptl;
    // f16x3 (the plain Block-GD products): the step and P^T in fp32 in Sh /
    // Pth, the fp16 hi / lo planes of the step, P^T, H̄ and F_eff in Sl, Ptl,
    // Hh and Fh, and their row scales' inverses
    int f16;
    float *scS, *scF, *scH, *scP;
    float *M;        // M = A H̄ (per row group: A H̄_g), kept current for the free columns
    int64_t step_c;  // first column of the last optimizer step not yet in M (n: none)
    TcMaps mapsP, mapsG;
    // row-grouped OBS (Alg. 1 "for all row-groups g"): rgroups contiguous row
    // groups of rg_rows rows, group g quantized against U_g; rgroups == 1
    // means U, Hbar and dead for every row
    int rgroups;
    int grouped;     // OBS of the row groups on their own H̄_g (the grouped entry point)
    int64_t rg_rows;
    const float *Ug, *Hbar_g;
    const uint8_t *dead_g;
    float *lam_g;                               // lambda_g per group (workspace)
    float *HGh, *HGl, *GGh, *GGl, *DWh, *DWl;   // tf32 planes of H̄_g, H̄_g - H̄, W - W0
    std::vector<TcMaps> mapsMg, mapsQg;
    // mini-batch Block-GD: step s of block b draws mini-batch
    // ((b_global - 1) steps + s) mod nmb, with moment H̄_mb (nmb x n x n)
    int nmb;
    const float *Hbar_mb;
    float *MBh, *MBl;                           // tf32 planes of H̄ - H̄_mb,k
    std::vector<TcMaps> mapsMB;
    int f_split_alpha_valid;
    float f_split_alpha;
    // token-form mini-batch Block-GD with per-token output clipping: the
    // calibration tokens X̂ (T_tok x n bf16) form ntok mini-batches of tmb
    // tokens; rank_q = the 0-based rank of the clip threshold among m
    // channels (m - 1: no channel scaled)
    const void *Xtok = nullptr;
    int64_t Ttok = 0, tmb = 0, rank_q = 0;
    int ntok = 0;
    float *Xf = nullptr, *XfT = nullptr, *Dk = nullptr, *Yh = nullptr, *Yl = nullptr,
          *Zk = nullptr, *Gc = nullptr;
    std::vector<TcMaps> mapsT1, mapsT2, mapsT3;
    // The optimizer step's G product is split: the next block's columns on
    // the sweep's stream (the next OBS block needs only those), the other
    // free columns on a side stream, joined before anything else reads or
    // writes them.  wide == nullptr: everything on the sweep's stream.
    float *Gpart = nullptr;                  // K-split partials of the next block's G (8 x m x B)
    // tracing: the surrogate with the block's F_eff before and after its
    // Block-GD steps, into block_loss[2 b], block_loss[2 b + 1] (device)
    float *block_loss = nullptr;
    void *trace_ws = nullptr;
    cudaStream_t wide = nullptr;
    cudaEvent_t wide_fork = nullptr, wide_done = nullptr;
    int wide_pending = 0;
};
realq_status_t sweep_side_stream(cudaStream_t s, SweepPlan &p);
bool profiling();   // per-launch event profiling on (work then stays on the caller's stream)
realq_status_t sweep_join_wide(cudaStream_t s, SweepPlan &p);
size_t sweep_ws_bytes(int64_t m, int64_t n, int block, int has_bgd, int has_fnext, int has_dbar, int rgroups = 0,
                      int nmb = 0, int64_t tmb = 0);
realq_status_t tok_xconv(cudaStream_t s, int64_t T, int64_t n, const void *X, float *Xf, float *XfT, int64_t ldT);
realq_status_t tok_clip(cudaStream_t s, int64_t T, int64_t m, float *D, int64_t k, float *Yh, float *Yl);
realq_status_t tok_gt(cudaStream_t s, int64_t T, int64_t m, const float *kap, const float *Z, float inv_T, float *gTh,
                      float *gTl, int64_t ldT);
void sweep_carve(SweepPlan &p, void *ws, int has_bgd, int has_fnext, int has_dbar);
realq_status_t sweep_init(cudaStream_t s, SweepPlan &p);
realq_status_t sweep_block(cudaStream_t s, SweepPlan &p, int64_t b);
realq_status_t sweep_prologue_r0(cudaStream_t s, SweepPlan &p, bool fresh);
realq_status_t bgd_step(cudaStream_t s, SweepPlan &p, int64_t col_start, float alpha);
realq_status_t surrogate(cudaStream_t s, int64_t m, int64_t n, const float *What, const void *W0,
                         realq_dtype_t w_dtype, const float *Hbar, const float *F, float *loss, void *ws);
size_t surrogate_ws_bytes(int64_t m, int64_t n);

}  // namespace realq
