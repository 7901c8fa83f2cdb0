// Host build of the decoder block's launch sequence (block_ops.cuh) for the
// CPU tests: every per-thread body is called for each index of its launch in
// turn, and each GEMM of the sequence is a plain fp32 triple loop with the
// same arguments.  This checks the bodies' index arithmetic and the argument
// of every step against the fp64 oracle without a GPU; it is test code and is
// never part of the library.
#include <cstdlib>
#include <vector>

#include "block_ops.cuh"

namespace {

// 0: each launch's indices in increasing order; 1: in decreasing order.  A
// launch whose result depends on the order has indices that read what
// another index of the same launch writes, which the GPU does not order.
int g_order = 0;

bool overlaps(const void *a, size_t an, const void *b, size_t bn) {
    const char *p = static_cast<const char *>(a), *q = static_cast<const char *>(b);
    return p < q + bn && q < p + an;
}

struct HostExec {
    template <class Fn>
    int map(int64_t count, const Fn &fn, const char *) {
        if (g_order == 0)
            for (int64_t i = 0; i < count; ++i) fn(i);
        else
            for (int64_t i = count - 1; i >= 0; --i) fn(i);
        return 0;
    }
    // The GPU GEMM's CTAs read A and B while others write C, so C may share
    // no byte with A or B; R may be C itself (each element is read by the
    // thread that writes it) but not overlap it otherwise.  Returns 2 when an
    // operand breaks that.
    int gemm(const realq::blk::Gemm &g, const char *) {
        const size_t cb = (size_t)((g.M - 1) * g.ldc + g.N) * sizeof(float);
        const size_t ab = (size_t)(g.a_kmajor ? (g.K - 1) * g.lda + g.M : (g.M - 1) * g.lda + g.K) * sizeof(float);
        const size_t bb = (size_t)((g.K - 1) * g.ldb + g.N) * sizeof(float);
        if (overlaps(g.C, cb, g.A, ab) || overlaps(g.C, cb, g.B, bb)) return 2;
        if (g.R && g.R != g.C && overlaps(g.C, cb, g.R, (size_t)((g.M - 1) * g.ldr + g.N) * sizeof(float))) return 2;
        for (int64_t i = 0; i < g.M; ++i)
            for (int64_t j = 0; j < g.N; ++j) {
                float acc = 0.f;
                for (int64_t k = 0; k < g.K; ++k)
                    acc += (g.a_kmajor ? g.A[k * g.lda + i] : g.A[i * g.lda + k]) * g.B[k * g.ldb + j];
                const float r = g.R ? g.R[i * g.ldr + j] : 0.f;
                g.C[i * g.ldc + j] = g.alpha * acc + r;
            }
        return 0;
    }
};

realq::blk::Dims dims_of(const int64_t *v, const float *fv) {
    return realq::blk::Dims{v[0], v[1], v[2], v[3], v[4], v[5], v[6], fv[0], fv[1]};
}

realq::blk::Weights weights_of(const float *const *w) {
    return realq::blk::Weights{w[0], w[1], w[2], w[3], w[4], w[5], w[6], w[7], w[8]};
}

}  // namespace

extern "C" void emu_set_order(int order) { g_order = order; }

// iv = {S, L, d, H, Hkv, dh, f}, fv = {eps, rope_base},
// w = {g1, Wq, Wk, Wv, Wo, g2, Wg, Wu, Wd}
extern "C" size_t emu_block_workspace(const int64_t *iv, const float *fv) {
    return realq::blk::carve(dims_of(iv, fv), nullptr, nullptr);
}

extern "C" int emu_block_forward(const int64_t *iv, const float *fv, const float *const *w, const float *x,
                                 float *y, void *ws) {
    const realq::blk::Dims dm = dims_of(iv, fv);
    realq::blk::Buffers B{};
    realq::blk::carve(dm, ws, &B);
    HostExec X;
    const realq::blk::Weights W = weights_of(w);
    int e = realq::blk::setup(X, dm, W, B);
    e |= realq::blk::forward(X, dm, W, B, x, y);
    return e;
}

extern "C" int emu_block_window(const int64_t *iv, const float *fv, const float *const *w, const float *h_ref,
                                const float *dh, const float *F_next, float *g, float *loss, void *ws) {
    const realq::blk::Dims dm = dims_of(iv, fv);
    realq::blk::Buffers B{};
    realq::blk::carve(dm, ws, &B);
    HostExec X;
    const realq::blk::Weights W = weights_of(w);
    int e = realq::blk::setup(X, dm, W, B);
    e |= realq::blk::window(X, dm, W, B, h_ref, dh, F_next, g, loss);
    return e;
}

// the input of module (0..6) in a forward pass with weights w on x, into X
extern "C" int emu_module_inputs(const int64_t *iv, const float *fv, const float *const *w, const float *x,
                                 int module, float *X, void *ws) {
    const realq::blk::Dims dm = dims_of(iv, fv);
    realq::blk::Buffers B{};
    realq::blk::carve(dm, ws, &B);
    HostExec E;
    return realq::blk::module_input(E, dm, weights_of(w), B, x, module, X);
}

// the exact window of one module of block l: wl = block l, wh = block l's
// weights in the current pass (NULL: wl), wn = next block, x / x_hat = block
// l's reference and current inputs (x_hat NULL: x), Wm = the module's weight
// (module 0..6 = q, k, v, o, gate, up, down)
extern "C" size_t emu_module_workspace(const int64_t *iv, const float *fv, int64_t V) {
    const realq::blk::Dims dm = dims_of(iv, fv);
    size_t b = 2 * realq::blk::carve(dm, nullptr, nullptr) + realq::blk::carve_module(dm, nullptr, nullptr);
    if (V > 0) b += realq::blk::carve_head(dm, V, nullptr, nullptr);
    return b;
}

extern "C" int emu_module_window(const int64_t *iv, const float *fv, const float *const *wl, const float *const *wh,
                                 const float *const *wn, const float *x, const float *x_hat, int module,
                                 const float *Wm, float alpha, const float *F_this, const float *F_next, float *gW,
                                 float *loss, void *ws) {
    using namespace realq::blk;
    const Dims dm = dims_of(iv, fv);
    Buffers Bl{}, Bn{};
    ModuleBuffers M{};
    char *p = static_cast<char *>(ws);
    p += carve(dm, p, &Bl);
    p += carve(dm, p, &Bn);
    carve_module(dm, p, &M);
    HostExec X;
    const Weights Wref = weights_of(wl);
    return module_window(X, dm, Wref, with_module(weights_of(wh ? wh : wl), module, Wm), weights_of(wn), Bl, Bn, M, x,
                         x_hat ? x_hat : x, module, alpha, F_this, F_next, gW, loss);
}

extern "C" int emu_head_kl(const int64_t *iv, const float *fv, const float *gf, const float *Wh, int64_t V,
                           const float *h_ref, const float *dh, float *g, float *loss, void *ws) {
    using namespace realq::blk;
    const Dims dm = dims_of(iv, fv);
    HeadBuffers H{};
    carve_head(dm, V, ws, &H);
    HostExec X;
    return kl_head(X, dm, Head{gf, Wh, V}, H, h_ref, dh, g, loss);
}

extern "C" int emu_module_kl(const int64_t *iv, const float *fv, const float *const *wl, const float *const *wh,
                             const float *x, const float *x_hat, int module, const float *Wm, const float *gf,
                             const float *Wh, int64_t V, float *gW, float *loss, void *ws) {
    using namespace realq::blk;
    const Dims dm = dims_of(iv, fv);
    Buffers Bl{};
    ModuleBuffers M{};
    HeadBuffers H{};
    char *p = static_cast<char *>(ws);
    p += carve(dm, p, &Bl);
    p += carve_module(dm, p, &M);
    carve_head(dm, V, p, &H);
    HostExec X;
    const Weights Wref = weights_of(wl);
    return module_kl(X, dm, Wref, with_module(weights_of(wh ? wh : wl), module, Wm), Bl, M, Head{gf, Wh, V}, H, x,
                     x_hat ? x_hat : x, module, gW, loss);
}
