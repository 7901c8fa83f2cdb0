// The decoder block of the exact two-block sliding window on the GPU: the
// launch executor of block_ops.cuh (one thread per flat index, the fp32 SIMT
// GEMM for the projections) and the C ABI entry points realq_block_forward
// and realq_block_window (include/realq.h).
#include "kernels.cuh"
#include "block_ops.cuh"

namespace realq {
namespace {

template <class Fn>
__global__ void __launch_bounds__(256) map_kernel(int64_t count, Fn fn) {
    const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (i < count) fn(i);
}

// Each step returns nonzero once a launch has failed; the first failure's
// status is kept and nothing more is launched.
struct DevExec {
    cudaStream_t s;
    realq_status_t st = REALQ_OK;

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

    int gemm(const blk::Gemm &g, const char *name) {
        if (st != REALQ_OK) return 1;
        GemmArgs a{};
        a.M = g.M; a.N = g.N; a.K = g.K;
        a.A = g.A; a.lda = g.lda;
        a.B = g.B; a.ldb = g.ldb;
        a.C = g.C; a.ldc = g.ldc;
        a.R = g.R; a.ldr = g.ldr;
        a.alpha = g.alpha;
        a.nsum = 1; a.nsum_b = 1; a.ksplit = 1;
        st = gemm_f32(s, A_ROW, g.R ? EPI_BIAS : EPI_STORE, a, name);
        return st != REALQ_OK;
    }
};

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

}  // namespace
}  // namespace realq

using namespace realq;

extern "C" {

size_t realq_block_workspace_size(const realq_block_dims_t *dims, int64_t S, int64_t L) {
    if (!dims || S <= 0 || L <= 0 || dims->head_dim <= 0) return 0;
    const blk::Dims dm{S, L, dims->d, dims->n_heads, dims->n_kv, dims->head_dim, dims->ffn, dims->rms_eps,
                       dims->rope_base};
    return blk::carve(dm, nullptr, nullptr);
}

realq_status_t realq_block_forward(realq_stream_t stream, const realq_block_dims_t *dims,
                                   const realq_block_weights_t *weights, int64_t S, int64_t L, const float *x,
                                   float *y, void *ws, size_t ws_bytes) {
    blk::Dims dm{};
    REALQ_TRY(check_block(dims, weights, S, L, "block_forward", &dm));
    if (!x || !y) return fail(REALQ_ERR_INVALID_ARG, "block_forward: NULL x or y");
    const size_t need = blk::carve(dm, nullptr, nullptr);
    if (!ws || ws_bytes < need || reinterpret_cast<uintptr_t>(ws) % kAlign)
        return fail(REALQ_ERR_WORKSPACE, "block_forward: workspace of %zu bytes (%zu-byte aligned) required", need,
                    kAlign);
    blk::Buffers B{};
    blk::carve(dm, ws, &B);
    DevExec X{static_cast<cudaStream_t>(stream)};
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
    const size_t need = blk::carve(dm, nullptr, nullptr);
    if (!ws || ws_bytes < need || reinterpret_cast<uintptr_t>(ws) % kAlign)
        return fail(REALQ_ERR_WORKSPACE, "block_window: workspace of %zu bytes (%zu-byte aligned) required", need,
                    kAlign);
    blk::Buffers B{};
    blk::carve(dm, ws, &B);
    DevExec X{static_cast<cudaStream_t>(stream)};
    const blk::Weights W = weights_of(weights);
    blk::setup(X, dm, W, B);
    blk::window(X, dm, W, B, h_ref, dh, F_next, g_h, loss);
    return X.st;
}

}  // extern "C"
