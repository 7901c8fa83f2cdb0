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

struct HostExec {
    template <class Fn>
    int map(int64_t count, const Fn &fn, const char *) {
        for (int64_t i = 0; i < count; ++i) fn(i);
        return 0;
    }
    int gemm(const realq::blk::Gemm &g, const char *) {
        for (int64_t i = 0; i < g.M; ++i)
            for (int64_t j = 0; j < g.N; ++j) {
                float acc = 0.f;
                for (int64_t k = 0; k < g.K; ++k) acc += g.A[i * g.lda + k] * g.B[k * g.ldb + j];
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
