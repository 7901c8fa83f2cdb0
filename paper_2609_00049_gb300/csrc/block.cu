// The decoder block of the exact two-block sliding window on the GPU: the
// launch executor of block_ops.cuh (one thread per flat index, the fp32 SIMT
// GEMM for the projections) and the C ABI entry points realq_block_* of
// include/realq.h (the block's forward, the next block's window, the
// module-level window, the final block's KL head), and the optimizer step of
// the sweep whose Block-GD gradient comes from those ops.
#include "kernels.cuh"
#include "block_ops.cuh"

namespace realq {
namespace {

template <class Fn>
__global__ void __launch_bounds__(256) map_kernel(int64_t count, Fn fn) {
    const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (i < count) fn(i);
}

int g_attn_tiled = 1;   // realq_set_block_attention

// Each step returns nonzero once a launch has failed; the first failure's
// status is kept and nothing more is launched.  With plane scratch (planes:
// four buffers of cap floats) the projections whose shapes the tensor-core
// path takes run as tf32x3 products on tcgen05: the operands are split into
// K-major tf32 hi / lo planes (transposed where stored the other way) and
// C = alpha A B + R is formed in the product's epilogue; the others, and
// every product without scratch, run on the fp32 CUDA-core tiles.
struct DevExec {
    cudaStream_t s;
    float *planes = nullptr;
    size_t cap = 0;
    int *err = nullptr;   // status word of the products' bounded waits
    realq_status_t st = REALQ_OK;

    bool tc_ok(const blk::Gemm &g) const {
        return planes && g.M >= 32 && g.N >= 32 && g.M % 4 == 0 && g.N % 4 == 0 && g.K >= 32 && g.K % 4 == 0 &&
               (size_t)g.M * g.K <= cap && (size_t)g.N * g.K <= cap && g.M < (1ll << 31) && g.N < (1ll << 31) &&
               g.K < (1ll << 31);
    }

    template <class Fn>
    int map(int64_t count, const Fn &fn, const char *name) {
        if (st != REALQ_OK) return 1;
        if (count <= 0) return 0;
        {
            Launch L(name, s);
            map_kernel<<<(unsigned)ceil_div(count, 256), 256, 0, s>>>(count, fn);
        }
        st = check_launch(name);
        return st != REALQ_OK;
    }

    // The attention passes run as tiled kernels (attention.cu) unless the
    // per-row bodies are selected (realq_set_block_attention).
    int map(int64_t count, const blk::AttnFwd &f, const char *name) {
        if (!g_attn_tiled) return map<blk::AttnFwd>(count, f, name);
        if (st != REALQ_OK) return 1;
        if (count <= 0) return 0;
        st = attn_fwd_tiled(s, count / (f.a.H * f.a.L), f.a.L, f.a.H, f.a.Hkv, f.a.dh, f.q, f.k, f.v, f.o, f.lse,
                            name);
        return st != REALQ_OK;
    }
    int map(int64_t count, const blk::AttnBwdQ &f, const char *name) {
        if (!g_attn_tiled) return map<blk::AttnBwdQ>(count, f, name);
        if (st != REALQ_OK) return 1;
        if (count <= 0) return 0;
        st = attn_bwd_q_tiled(s, count / (f.a.H * f.a.L), f.a.L, f.a.H, f.a.Hkv, f.a.dh, f.q, f.k, f.v, f.go, f.lse,
                              f.D, f.gq, name);
        return st != REALQ_OK;
    }
    int map(int64_t count, const blk::AttnBwdKV &f, const char *name) {
        if (!g_attn_tiled) return map<blk::AttnBwdKV>(count, f, name);
        if (st != REALQ_OK) return 1;
        if (count <= 0) return 0;
        st = attn_bwd_kv_tiled(s, count / (f.a.Hkv * f.a.L), f.a.L, f.a.H, f.a.Hkv, f.a.dh, f.q, f.k, f.v, f.go,
                               f.lse, f.D, f.gk, f.gv, name);
        return st != REALQ_OK;
    }

    int gemm(const blk::Gemm &g, const char *name) {
        if (st != REALQ_OK) return 1;
        if (tc_ok(g)) {
            float *Ah = planes, *Al = planes + cap, *Bh = planes + 2 * cap, *Bl = planes + 3 * cap;
            // A (M x K): rows of A, or A stored K x M (column i of the stored matrix)
            st = g.a_kmajor ? tc_trans_planes(s, g.K, g.M, g.A, g.lda, Ah, Al, g.K)
                            : tc_split_rows(s, g.M, g.K, g.A, g.lda, Ah, Al, g.K, g.K);
            // B (K x N, row-major): its columns as rows of K
            if (st == REALQ_OK) st = tc_trans_planes(s, g.K, g.N, g.B, g.ldb, Bh, Bl, g.K);
            TcMaps maps;
            if (st == REALQ_OK) st = tc_make_maps(&maps, Ah, Al, g.M, g.K, g.K, Bh, Bl, g.N, g.K, g.K);
            if (st == REALQ_OK) {
                TcEpi e{};
                e.mode = TC_STORE;
                e.C = g.C;
                e.ldc = g.ldc;
                e.affine = 1;
                e.alpha_s = g.alpha;
                e.R = g.R;
                e.ldr = g.ldr;
                st = tc_gemm_x3(s, maps, g.M, g.N, g.K, 0, 0, e, err, name);
            }
            return st != REALQ_OK;
        }
        GemmArgs a{};
        a.M = g.M; a.N = g.N; a.K = g.K;
        a.A = g.A; a.lda = g.lda;
        a.B = g.B; a.ldb = g.ldb;
        a.C = g.C; a.ldc = g.ldc;
        a.R = g.R; a.ldr = g.ldr;
        a.alpha = g.alpha;
        a.nsum = 1; a.nsum_b = 1; a.ksplit = 1;
        st = gemm_f32(s, g.a_kmajor ? A_KMAJOR : A_ROW, g.R ? EPI_BIAS : EPI_STORE, a, name);
        return st != REALQ_OK;
    }
};

__global__ void __launch_bounds__(256) adam_cols_kernel(int64_t m, int64_t r, int64_t n, int64_t c0, const float *G,
                                                        float *W, float *mA, float *vA, float lr, float b1, float b2,
                                                        float eps, float bc1, float bc2, int sgd) {
    const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= m * r) return;
    const int64_t w = (idx / r) * n + c0 + idx % r;
    const float g = G[w];
    float step;
    if (sgd) {
        step = lr * g;
    } else {
        const float mv = b1 * mA[w] + (1.f - b1) * g;
        const float vv = b2 * vA[w] + (1.f - b2) * g * g;
        mA[w] = mv;
        vA[w] = vv;
        step = lr * (mv / bc1) / (sqrtf(vv / bc2) + eps);
    }
    W[w] -= step;
}

realq_status_t check_block(const realq_block_dims_t *dims, const realq_block_weights_t *w, int64_t S, int64_t L,
                           const char *who, blk::Dims *out) {
    if (!dims || !w) return fail(REALQ_ERR_INVALID_ARG, "%s: NULL dims or weights", who);
    if (S <= 0 || L <= 0) return fail(REALQ_ERR_INVALID_ARG, "%s: S, L > 0 required", who);
    if (dims->d <= 0 || dims->n_heads <= 0 || dims->n_kv <= 0 || dims->head_dim <= 0 || dims->ffn <= 0)
        return fail(REALQ_ERR_INVALID_ARG, "%s: d, n_heads, n_kv, head_dim, ffn > 0 required", who);
    if (dims->n_heads % dims->n_kv != 0) return fail(REALQ_ERR_INVALID_ARG, "%s: n_heads %% n_kv != 0", who);
    if (dims->head_dim % 2 != 0 || dims->head_dim > blk::kMaxHeadDim)
        return fail(REALQ_ERR_INVALID_ARG, "%s: head_dim must be even and <= %d", who, blk::kMaxHeadDim);
    if (!(dims->rms_eps > 0.f) || !std::isfinite(dims->rms_eps))
        return fail(REALQ_ERR_INVALID_ARG, "%s: rms_eps > 0 required", who);
    if (!(dims->rope_base > 1.f) || !std::isfinite(dims->rope_base))
        return fail(REALQ_ERR_INVALID_ARG, "%s: rope_base > 1 required", who);
    if (!w->g1 || !w->Wq || !w->Wk || !w->Wv || !w->Wo || !w->g2 || !w->Wg || !w->Wu || !w->Wd)
        return fail(REALQ_ERR_INVALID_ARG, "%s: NULL weight", who);
    const int64_t big = (int64_t)1 << 38;
    if (S * L > 64LL * 65535LL || dims->d > big / (S * L) || dims->ffn > big / (S * L) ||
        dims->n_heads * dims->head_dim > big / (S * L))
        return fail(REALQ_ERR_UNSUPPORTED, "%s: S L <= 4194240 tokens and under 2^38 elements per buffer", who);
    *out = blk::Dims{S, L, dims->d, dims->n_heads, dims->n_kv, dims->head_dim, dims->ffn, dims->rms_eps,
                     dims->rope_base};
    return REALQ_OK;
}

blk::Weights weights_of(const realq_block_weights_t *w) {
    return blk::Weights{w->g1, w->Wq, w->Wk, w->Wv, w->Wo, w->g2, w->Wg, w->Wu, w->Wd};
}

realq_status_t check_ws_block(void *ws, size_t have, size_t need, const char *who) {
    if (!ws || have < need || reinterpret_cast<uintptr_t>(ws) % kAlign)
        return fail(REALQ_ERR_WORKSPACE, "%s: workspace of %zu bytes (%zu-byte aligned) required", who, need, kAlign);
    return REALQ_OK;
}

realq_status_t check_module(int module, const float *Wm, const float *grad, const char *who) {
    if (module < blk::M_Q || module > blk::M_DOWN)
        return fail(REALQ_ERR_INVALID_ARG, "%s: module must be 0..6 (q, k, v, o, gate, up, down)", who);
    if (!Wm || !grad) return fail(REALQ_ERR_INVALID_ARG, "%s: NULL module weight or gradient", who);
    return REALQ_OK;
}

realq_status_t check_head(const float *gf, const float *Wh, int64_t vocab, const blk::Dims &dm, const char *who) {
    if (!gf || !Wh) return fail(REALQ_ERR_INVALID_ARG, "%s: NULL head gain or weight", who);
    if (vocab <= 0 || vocab > ((int64_t)1 << 38) / dm.T())
        return fail(REALQ_ERR_INVALID_ARG, "%s: 0 < vocab and S L vocab < 2^38 required", who);
    return REALQ_OK;
}

// Every block workspace starts with the tensor-core scratch: a status word
// (its first int; kAlign bytes) and four operand planes of tc_cap floats,
// enough for every projection of the block (M K and N K at most
// max(T, d) max(d, H dh, f)) and, with a head, for the logits product
// (max(T, V) d).  Products with a larger operand run on the CUDA cores.
size_t tc_cap(const blk::Dims &dm, int64_t vocab) {
    const size_t T = (size_t)dm.T(), d = (size_t)dm.d;
    const size_t wide = std::max(d, std::max((size_t)dm.qw(), (size_t)dm.f));
    size_t cap = std::max(T, d) * wide;
    if (vocab > 0) cap = std::max(cap, std::max(T, (size_t)vocab) * d);
    return (cap + 63) / 64 * 64;   // each plane 256-byte aligned
}

size_t tc_scratch(const blk::Dims &dm, int64_t vocab) { return kAlign + 4 * blk::rnd(tc_cap(dm, vocab) * 4); }

size_t module_ws(const blk::Dims &dm, int64_t vocab) {
    if (vocab > 0)
        return tc_scratch(dm, vocab) + blk::carve(dm, nullptr, nullptr) + blk::carve_module(dm, nullptr, nullptr) +
               blk::carve_head(dm, vocab, nullptr, nullptr);
    return tc_scratch(dm, 0) + 2 * blk::carve(dm, nullptr, nullptr) + blk::carve_module(dm, nullptr, nullptr);
}

size_t block_ws(const blk::Dims &dm) { return tc_scratch(dm, 0) + blk::carve(dm, nullptr, nullptr); }

size_t head_ws(const blk::Dims &dm, int64_t vocab) {
    return tc_scratch(dm, vocab) + blk::carve_head(dm, vocab, nullptr, nullptr);
}

// the status word recorded by the block ops' products; the window
// quantization driver points it at its sweep's own status word for the
// calls it makes
thread_local int *g_status_override = nullptr;

int g_block_tc = 0;   // realq_set_block_products

// An executor on the scratch at the start of ws; returns the rest of ws.
// The status word is cleared at the start of the call unless overridden.
char *exec_at(DevExec *X, void *ws, const blk::Dims &dm, int64_t vocab) {
    char *p = static_cast<char *>(ws);
    X->cap = tc_cap(dm, vocab);
    X->planes = g_block_tc ? reinterpret_cast<float *>(p + kAlign) : nullptr;
    if (g_status_override) {
        X->err = g_status_override;
    } else {
        X->err = reinterpret_cast<int *>(p);
        const cudaError_t r = cudaMemsetAsync(p, 0, sizeof(int), X->s);
        if (r != cudaSuccess) X->st = fail(REALQ_ERR_CUDA, "block ops: %s", cudaGetErrorString(r));
    }
    return p + tc_scratch(dm, vocab);
}

}  // namespace

realq_status_t block_loss_check(const realq_block_dims_t *dims, const realq_block_weights_t *this_block,
                                const realq_block_weights_t *this_block_hat, const realq_block_weights_t *next_block,
                                int64_t S, int64_t L, const float *x, int module, const float *F_this,
                                const float *F_next, const float *gf, const float *Wh, int64_t vocab, const char *who,
                                int64_t *m, int64_t *n, size_t *ws_bytes) {
    blk::Dims dm{};
    REALQ_TRY(check_block(dims, this_block, S, L, who, &dm));
    if (this_block_hat) REALQ_TRY(check_block(dims, this_block_hat, S, L, who, &dm));
    if (module < blk::M_Q || module > blk::M_DOWN)
        return fail(REALQ_ERR_INVALID_ARG, "%s: module must be 0..6 (q, k, v, o, gate, up, down)", who);
    if (!x) return fail(REALQ_ERR_INVALID_ARG, "%s: NULL x", who);
    if (next_block) {
        REALQ_TRY(check_block(dims, next_block, S, L, who, &dm));
        if (!F_this || !F_next) return fail(REALQ_ERR_INVALID_ARG, "%s: NULL F_this or F_next", who);
        *ws_bytes = module_ws(dm, 0);
    } else {
        REALQ_TRY(check_head(gf, Wh, vocab, dm, who));
        *ws_bytes = module_ws(dm, vocab);
    }
    const int64_t qw = dm.qw(), kw = dm.kw();
    switch (module) {
        case blk::M_Q: *m = qw; *n = dm.d; break;
        case blk::M_K: case blk::M_V: *m = kw; *n = dm.d; break;
        case blk::M_O: *m = dm.d; *n = qw; break;
        case blk::M_GATE: case blk::M_UP: *m = dm.f; *n = dm.d; break;
        default: *m = dm.d; *n = dm.f; break;
    }
    return REALQ_OK;
}

BlockStatusScope::BlockStatusScope(int *status) : prev(g_status_override) { g_status_override = status; }
BlockStatusScope::~BlockStatusScope() { g_status_override = prev; }

realq_status_t adam_cols(cudaStream_t s, int64_t m, int64_t n, int64_t c0, const float *G, float *W, float *mA,
                         float *vA, float lr, float b1, float b2, float eps, int64_t t, int sgd) {
    const int64_t r = n - c0;
    if (m <= 0 || r <= 0) return REALQ_OK;
    const float bc1 = (float)(1.0 - std::pow((double)b1, (double)t));
    const float bc2 = (float)(1.0 - std::pow((double)b2, (double)t));
    {
        Launch L("window_adam", s);
        adam_cols_kernel<<<(unsigned)ceil_div(m * r, 256), 256, 0, s>>>(m, r, n, c0, G, W, mA, vA, lr, b1, b2, eps,
                                                                        bc1, bc2, sgd);
    }
    return check_launch("window_adam");
}

}  // namespace realq

using namespace realq;

extern "C" {

realq_status_t realq_set_block_attention(int mode) {
    if (mode != 0 && mode != 1) return fail(REALQ_ERR_INVALID_ARG, "set_block_attention: mode must be 0 or 1");
    g_attn_tiled = mode;
    return REALQ_OK;
}

realq_status_t realq_set_block_products(int mode) {
    if (mode != 0 && mode != 1) return fail(REALQ_ERR_INVALID_ARG, "set_block_products: mode must be 0 or 1");
    g_block_tc = mode;
    return REALQ_OK;
}

size_t realq_block_workspace_size(const realq_block_dims_t *dims, int64_t S, int64_t L) {
    if (!dims || S <= 0 || L <= 0 || dims->head_dim <= 0) return 0;
    const blk::Dims dm{S, L, dims->d, dims->n_heads, dims->n_kv, dims->head_dim, dims->ffn, dims->rms_eps,
                       dims->rope_base};
    return block_ws(dm);
}

realq_status_t realq_block_forward(realq_stream_t stream, const realq_block_dims_t *dims,
                                   const realq_block_weights_t *weights, int64_t S, int64_t L, const float *x,
                                   float *y, void *ws, size_t ws_bytes) {
    blk::Dims dm{};
    REALQ_TRY(check_block(dims, weights, S, L, "block_forward", &dm));
    if (!x || !y) return fail(REALQ_ERR_INVALID_ARG, "block_forward: NULL x or y");
    REALQ_TRY(check_ws_block(ws, ws_bytes, block_ws(dm), "block_forward"));
    DevExec X{static_cast<cudaStream_t>(stream)};
    blk::Buffers B{};
    blk::carve(dm, exec_at(&X, ws, dm, 0), &B);
    const blk::Weights W = weights_of(weights);
    blk::setup(X, dm, W, B);
    blk::forward(X, dm, W, B, x, y);
    return X.st;
}

realq_status_t realq_block_window(realq_stream_t stream, const realq_block_dims_t *dims,
                                  const realq_block_weights_t *weights, int64_t S, int64_t L, const float *h_ref,
                                  const float *dh, const float *F_next, float *g_h, float *loss, void *ws,
                                  size_t ws_bytes) {
    blk::Dims dm{};
    REALQ_TRY(check_block(dims, weights, S, L, "block_window", &dm));
    if (!h_ref || !dh || !F_next || !g_h) return fail(REALQ_ERR_INVALID_ARG, "block_window: NULL argument");
    REALQ_TRY(check_ws_block(ws, ws_bytes, block_ws(dm), "block_window"));
    DevExec X{static_cast<cudaStream_t>(stream)};
    blk::Buffers B{};
    blk::carve(dm, exec_at(&X, ws, dm, 0), &B);
    const blk::Weights W = weights_of(weights);
    blk::setup(X, dm, W, B);
    blk::window(X, dm, W, B, h_ref, dh, F_next, g_h, loss);
    return X.st;
}

realq_status_t realq_block_module_inputs(realq_stream_t stream, const realq_block_dims_t *dims,
                                         const realq_block_weights_t *weights, int64_t S, int64_t L, const float *x,
                                         int module, float *X_out, void *ws, size_t ws_bytes) {
    const char *who = "block_module_inputs";
    blk::Dims dm{};
    REALQ_TRY(check_block(dims, weights, S, L, who, &dm));
    if (module < blk::M_Q || module > blk::M_DOWN)
        return fail(REALQ_ERR_INVALID_ARG, "%s: module must be 0..6 (q, k, v, o, gate, up, down)", who);
    if (!x || !X_out) return fail(REALQ_ERR_INVALID_ARG, "%s: NULL x or X_out", who);
    REALQ_TRY(check_ws_block(ws, ws_bytes, block_ws(dm), who));
    DevExec X{static_cast<cudaStream_t>(stream)};
    blk::Buffers B{};
    blk::carve(dm, exec_at(&X, ws, dm, 0), &B);
    blk::module_input(X, dm, weights_of(weights), B, x, module, X_out);
    return X.st;
}

size_t realq_block_module_workspace_size(const realq_block_dims_t *dims, int64_t S, int64_t L, int64_t vocab) {
    if (!dims || S <= 0 || L <= 0 || dims->head_dim <= 0 || vocab < 0) return 0;
    const blk::Dims dm{S, L, dims->d, dims->n_heads, dims->n_kv, dims->head_dim, dims->ffn, dims->rms_eps,
                       dims->rope_base};
    return module_ws(dm, vocab);
}

size_t realq_block_head_workspace_size(int64_t d, int64_t S, int64_t L, int64_t vocab) {
    if (d <= 0 || S <= 0 || L <= 0 || vocab <= 0) return 0;
    const blk::Dims dm{S, L, d, 1, 1, 2, 1, 1e-6f, 10000.f};
    return head_ws(dm, vocab);
}

realq_status_t realq_block_module_window(realq_stream_t stream, const realq_block_dims_t *dims,
                                         const realq_block_weights_t *this_block,
                                         const realq_block_weights_t *this_block_hat,
                                         const realq_block_weights_t *next_block, int64_t S, int64_t L, const float *x,
                                         const float *x_hat, int module, const float *W_module, float alpha,
                                         const float *F_this, const float *F_next, float *grad, float *loss, void *ws,
                                         size_t ws_bytes) {
    const char *who = "block_module_window";
    blk::Dims dm{};
    REALQ_TRY(check_block(dims, this_block, S, L, who, &dm));
    if (this_block_hat) REALQ_TRY(check_block(dims, this_block_hat, S, L, who, &dm));
    REALQ_TRY(check_block(dims, next_block, S, L, who, &dm));
    REALQ_TRY(check_module(module, W_module, grad, who));
    if (!x || !F_this || !F_next) return fail(REALQ_ERR_INVALID_ARG, "%s: NULL x, F_this or F_next", who);
    if (!(alpha >= 0.f && alpha <= 1.f)) return fail(REALQ_ERR_INVALID_ARG, "%s: alpha must be in [0, 1]", who);
    REALQ_TRY(check_ws_block(ws, ws_bytes, module_ws(dm, 0), who));
    DevExec X{static_cast<cudaStream_t>(stream)};
    blk::Buffers Bl{}, Bn{};
    blk::ModuleBuffers M{};
    char *p = exec_at(&X, ws, dm, 0);
    p += blk::carve(dm, p, &Bl);
    p += blk::carve(dm, p, &Bn);
    blk::carve_module(dm, p, &M);
    const blk::Weights Wref = weights_of(this_block);
    const blk::Weights Wcur = weights_of(this_block_hat ? this_block_hat : this_block);
    blk::module_window(X, dm, Wref, blk::with_module(Wcur, module, W_module), weights_of(next_block), Bl, Bn, M, x,
                       x_hat ? x_hat : x, module, alpha, F_this, F_next, grad, loss);
    return X.st;
}

realq_status_t realq_block_head_kl(realq_stream_t stream, int64_t d, int64_t S, int64_t L, const float *gf,
                                   const float *Wh, int64_t vocab, float rms_eps, const float *h_ref, const float *dh,
                                   float *g_h, float *loss, void *ws, size_t ws_bytes) {
    const char *who = "block_head_kl";
    if (d <= 0 || S <= 0 || L <= 0 || S * L > 64LL * 65535LL || d > ((int64_t)1 << 38) / (S * L))
        return fail(REALQ_ERR_INVALID_ARG, "%s: d, S, L > 0 and S L <= 4194240 required", who);
    if (!(rms_eps > 0.f) || !std::isfinite(rms_eps)) return fail(REALQ_ERR_INVALID_ARG, "%s: rms_eps > 0", who);
    const blk::Dims dm{S, L, d, 1, 1, 2, 1, rms_eps, 10000.f};
    REALQ_TRY(check_head(gf, Wh, vocab, dm, who));
    if (!h_ref || !dh || !g_h) return fail(REALQ_ERR_INVALID_ARG, "%s: NULL h_ref, dh or g_h", who);
    REALQ_TRY(check_ws_block(ws, ws_bytes, head_ws(dm, vocab), who));
    DevExec X{static_cast<cudaStream_t>(stream)};
    blk::HeadBuffers H{};
    blk::carve_head(dm, vocab, exec_at(&X, ws, dm, vocab), &H);
    blk::kl_head(X, dm, blk::Head{gf, Wh, vocab}, H, h_ref, dh, g_h, loss);
    return X.st;
}

realq_status_t realq_block_module_kl(realq_stream_t stream, const realq_block_dims_t *dims,
                                     const realq_block_weights_t *this_block,
                                     const realq_block_weights_t *this_block_hat, int64_t S, int64_t L,
                                     const float *x, const float *x_hat, int module, const float *W_module,
                                     const float *gf, const float *Wh, int64_t vocab, float *grad, float *loss,
                                     void *ws, size_t ws_bytes) {
    const char *who = "block_module_kl";
    blk::Dims dm{};
    REALQ_TRY(check_block(dims, this_block, S, L, who, &dm));
    if (this_block_hat) REALQ_TRY(check_block(dims, this_block_hat, S, L, who, &dm));
    REALQ_TRY(check_module(module, W_module, grad, who));
    REALQ_TRY(check_head(gf, Wh, vocab, dm, who));
    if (!x) return fail(REALQ_ERR_INVALID_ARG, "%s: NULL x", who);
    REALQ_TRY(check_ws_block(ws, ws_bytes, module_ws(dm, vocab), who));
    DevExec X{static_cast<cudaStream_t>(stream)};
    blk::Buffers Bl{};
    blk::ModuleBuffers M{};
    blk::HeadBuffers H{};
    char *p = exec_at(&X, ws, dm, vocab);
    p += blk::carve(dm, p, &Bl);
    p += blk::carve_module(dm, p, &M);
    blk::carve_head(dm, vocab, p, &H);
    const blk::Weights Wref = weights_of(this_block);
    const blk::Weights Wcur = weights_of(this_block_hat ? this_block_hat : this_block);
    blk::module_kl(X, dm, Wref, blk::with_module(Wcur, module, W_module), Bl, M, blk::Head{gf, Wh, vocab}, H, x,
                   x_hat ? x_hat : x, module, grad, loss);
    return X.st;
}

}  // extern "C"
