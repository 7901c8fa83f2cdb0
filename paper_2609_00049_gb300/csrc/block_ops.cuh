// The decoder block of the exact two-block sliding window (Sec. 4.4,
// Eq. slide_window): its forward pass, its backward pass with respect to the
// block input, and the next block's Fisher loss
//   L(l+1) = (1/2T) sum_t Δz_t^T F' Δz_t,  Δz = B(h + Δh) - B(h),
// with its gradient in Δh.
//
// The block is the pre-norm LLaMA-3.1 / Qwen3 structure:
//   a = RMSNorm(x; g1),  h = x + Attn(a) W_o^T,
//   b = RMSNorm(h; g2),  y = h + (silu(b W_g^T) * (b W_u^T)) W_d^T,
// RMSNorm(x; g) = x g / sqrt(mean(x^2) + eps); grouped-query causal attention
// with H query heads of width dh, H_kv key/value heads (query head i reads
// key/value head i / (H / H_kv)), rotary embedding on the pairs (j, j + dh/2)
// at angle pos * base^(-2j/dh), scale 1/sqrt(dh).
//
// Everything here is plain C++ that the CUDA build and a host build both
// compile: the per-thread bodies are functors called with one flat index,
// and the whole sequence of launches and GEMMs is a template over an
// executor (`X::map(count, functor)`, `X::gemm(Gemm)`).  The library's
// executor launches one thread per index and the fp32 SIMT GEMM; the tests
// build a host executor from the same header to check the index arithmetic
// and the argument of every step before any GPU run.
//
// Layout: tokens are rows, T = S L, token (s, t) at row s L + t.  q, the
// attention output o and their gradients are T x (H dh) with head h at
// columns h dh ..; k, v are T x (H_kv dh).  lse and the softmax row terms
// are (S, H, L).  All fp32.
#pragma once

#include <cmath>
#include <cstddef>
#include <cstdint>

#if defined(__CUDACC__)
#define RQ_HD __host__ __device__ __forceinline__
#else
#define RQ_HD inline
#endif

namespace realq {
namespace blk {

constexpr int kMaxHeadDim = 256;

struct Dims {
    int64_t S, L;            // sequences and tokens per sequence
    int64_t d, H, Hkv, dh, f;
    float eps;               // RMSNorm epsilon
    float rope_base;
    int64_t T() const { return S * L; }
    int64_t qw() const { return H * dh; }
    int64_t kw() const { return Hkv * dh; }
};

struct Weights {             // row-major (out x in), fp32
    const float *g1, *Wq, *Wk, *Wv, *Wo, *g2, *Wg, *Wu, *Wd;
};

// C = alpha A B (+ R): A M x K (lda), B K x N (ldb), C and R M x N (ldc, ldr);
// R may be C itself (each element is read before it is written).  With
// a_kmajor, A(i, k) = A[k * lda + i] (A stored K x M: a weight gradient
// A^T B over the token axis).
struct Gemm {
    int64_t M, N, K;
    const float *A; int64_t lda;
    const float *B; int64_t ldb;
    float *C; int64_t ldc;
    const float *R; int64_t ldr;
    float alpha;
    int a_kmajor;
};

// ------------------------------------------------------------ bodies ---

// out[j * rows + i] = in[i * cols + j]
struct Transpose {
    const float *in; float *out; int64_t rows, cols;
    RQ_HD void operator()(int64_t idx) const {
        const int64_t i = idx / cols, j = idx % cols;
        out[j * rows + i] = in[idx];
    }
};

// out = a + beta b
struct Axpy {
    const float *a; const float *b; float *out; float beta;
    RQ_HD void operator()(int64_t i) const { out[i] = a[i] + beta * b[i]; }
};

// rotary tables: cos / sin of pos * base^(-2j/dh), pos < L, j < dh/2 (the
// angle in double, then rounded to fp32)
struct RopeTable {
    float *cs; float *sn; int64_t half; double base; int64_t dh;
    RQ_HD void operator()(int64_t idx) const {
        const int64_t pos = idx / half, j = idx % half;
        const double ang = (double)pos * pow(base, -2.0 * (double)j / (double)dh);
        cs[idx] = (float)cos(ang);
        sn[idx] = (float)sin(ang);
    }
};

// one token row: y = x g r, r = 1 / sqrt(mean(x^2) + eps)
struct RmsFwd {
    const float *x; const float *g; float *y; float *r; int64_t d; float eps;
    RQ_HD void operator()(int64_t t) const {
        const float *xr = x + t * d;
        float ss = 0.f;
        for (int64_t k = 0; k < d; ++k) ss += xr[k] * xr[k];
        const float rr = 1.f / sqrtf(ss / (float)d + eps);
        r[t] = rr;
        float *yr = y + t * d;
        for (int64_t k = 0; k < d; ++k) yr[k] = xr[k] * rr * g[k];
    }
};

// one token row of the RMSNorm backward:
//   gx = base + gy g r - x r^3 (sum_k gy_k g_k x_k) / d   (base may be null;
//   gx may alias base or gy, not x)
struct RmsBwd {
    const float *x; const float *g; const float *r; const float *gy; const float *base; float *gx; int64_t d;
    RQ_HD void operator()(int64_t t) const {
        const float *xr = x + t * d, *gr = gy + t * d;
        const float rr = r[t];
        float dot = 0.f;
        for (int64_t k = 0; k < d; ++k) dot += gr[k] * g[k] * xr[k];
        const float c = rr * rr * rr * dot / (float)d;
        float *o = gx + t * d;
        const float *br = base ? base + t * d : nullptr;
        for (int64_t k = 0; k < d; ++k) {
            const float v = gr[k] * g[k] * rr - xr[k] * c;
            o[k] = br ? br[k] + v : v;
        }
    }
};

// rotary rotation of one pair (j, j + dh/2) of one head of one token, in
// place; inverse = 1 applies the transpose (the backward)
struct Rope {
    float *v; int64_t ld; int64_t heads, half, dh, L; const float *cs; const float *sn; int inverse;
    RQ_HD void operator()(int64_t idx) const {
        const int64_t j = idx % half;
        const int64_t hh = (idx / half) % heads;
        const int64_t row = idx / (half * heads);
        const int64_t pos = row % L;
        float *p = v + row * ld + hh * dh;
        const float c = cs[pos * half + j], s = sn[pos * half + j];
        const float x1 = p[j], x2 = p[j + half];
        if (!inverse) {
            p[j] = x1 * c - x2 * s;
            p[j + half] = x1 * s + x2 * c;
        } else {
            p[j] = x1 * c + x2 * s;
            p[j + half] = -x1 * s + x2 * c;
        }
    }
};

struct AttnShape {
    int64_t L, H, Hkv, dh;
    RQ_HD int64_t rep() const { return H / Hkv; }
    RQ_HD int64_t qw() const { return H * dh; }
    RQ_HD int64_t kw() const { return Hkv * dh; }
};

// one query row (s, h, t): o = sum_{u <= t} softmax_u(q_t . k_u / sqrt(dh)) v_u
// with a running maximum; lse = the log of the softmax denominator (with the
// maximum added back)
struct AttnFwd {
    const float *q; const float *k; const float *v; float *o; float *lse; AttnShape a;
    RQ_HD void operator()(int64_t idx) const {
        const int64_t t = idx % a.L, h = (idx / a.L) % a.H, s = idx / (a.L * a.H);
        const int64_t kvh = h / a.rep();
        const float *qr = q + (s * a.L + t) * a.qw() + h * a.dh;
        const float scale = 1.f / sqrtf((float)a.dh);
        float acc[kMaxHeadDim];
        for (int64_t e = 0; e < a.dh; ++e) acc[e] = 0.f;
        float mx = -INFINITY, l = 0.f;
        for (int64_t u = 0; u <= t; ++u) {
            const float *kr = k + (s * a.L + u) * a.kw() + kvh * a.dh;
            const float *vr = v + (s * a.L + u) * a.kw() + kvh * a.dh;
            float sc = 0.f;
            for (int64_t e = 0; e < a.dh; ++e) sc += qr[e] * kr[e];
            sc *= scale;
            if (sc > mx) {
                const float c = expf(mx - sc);   // 0 on the first key
                l = l * c + 1.f;
                for (int64_t e = 0; e < a.dh; ++e) acc[e] = acc[e] * c + vr[e];
                mx = sc;
            } else {
                const float p = expf(sc - mx);
                l += p;
                for (int64_t e = 0; e < a.dh; ++e) acc[e] += p * vr[e];
            }
        }
        float *orow = o + (s * a.L + t) * a.qw() + h * a.dh;
        const float inv = 1.f / l;
        for (int64_t e = 0; e < a.dh; ++e) orow[e] = acc[e] * inv;
        lse[idx] = mx + logf(l);
    }
};

// the softmax backward's row term D(s, h, t) = dO_t . O_t
struct AttnRowDot {
    const float *go; const float *o; float *D; AttnShape a;
    RQ_HD void operator()(int64_t idx) const {
        const int64_t t = idx % a.L, h = (idx / a.L) % a.H, s = idx / (a.L * a.H);
        const int64_t off = (s * a.L + t) * a.qw() + h * a.dh;
        float acc = 0.f;
        for (int64_t e = 0; e < a.dh; ++e) acc += go[off + e] * o[off + e];
        D[idx] = acc;
    }
};

// one query row's gradient:
//   dq_t = (1/sqrt(dh)) sum_{u <= t} p_tu (dO_t . v_u - D_t) k_u,
//   p_tu = exp(q_t . k_u / sqrt(dh) - lse_t)
struct AttnBwdQ {
    const float *q; const float *k; const float *v; const float *go; const float *lse; const float *D; float *gq;
    AttnShape a;
    RQ_HD void operator()(int64_t idx) const {
        const int64_t t = idx % a.L, h = (idx / a.L) % a.H, s = idx / (a.L * a.H);
        const int64_t kvh = h / a.rep();
        const int64_t off = (s * a.L + t) * a.qw() + h * a.dh;
        const float *qr = q + off, *gr = go + off;
        const float scale = 1.f / sqrtf((float)a.dh);
        const float ls = lse[idx], Dt = D[idx];
        float acc[kMaxHeadDim];
        for (int64_t e = 0; e < a.dh; ++e) acc[e] = 0.f;
        for (int64_t u = 0; u <= t; ++u) {
            const float *kr = k + (s * a.L + u) * a.kw() + kvh * a.dh;
            const float *vr = v + (s * a.L + u) * a.kw() + kvh * a.dh;
            float sc = 0.f, dp = 0.f;
            for (int64_t e = 0; e < a.dh; ++e) {
                sc += qr[e] * kr[e];
                dp += gr[e] * vr[e];
            }
            const float p = expf(sc * scale - ls);
            const float ds = p * (dp - Dt);
            for (int64_t e = 0; e < a.dh; ++e) acc[e] += ds * kr[e];
        }
        float *out = gq + off;
        for (int64_t e = 0; e < a.dh; ++e) out[e] = acc[e] * scale;
    }
};

// one key/value row (s, kv head, u), summed over the query heads that read it
// and the queries t >= u:
//   dk_u = (1/sqrt(dh)) sum p_tu (dO_t . v_u - D_t) q_t,   dv_u = sum p_tu dO_t
struct AttnBwdKV {
    const float *q; const float *k; const float *v; const float *go; const float *lse; const float *D; float *gk;
    float *gv; AttnShape a;
    RQ_HD void operator()(int64_t idx) const {
        const int64_t u = idx % a.L, kvh = (idx / a.L) % a.Hkv, s = idx / (a.L * a.Hkv);
        const int64_t koff = (s * a.L + u) * a.kw() + kvh * a.dh;
        const float *kr = k + koff, *vr = v + koff;
        const float scale = 1.f / sqrtf((float)a.dh);
        float ak[kMaxHeadDim], av[kMaxHeadDim];
        for (int64_t e = 0; e < a.dh; ++e) ak[e] = av[e] = 0.f;
        for (int64_t h = kvh * a.rep(); h < (kvh + 1) * a.rep(); ++h) {
            for (int64_t t = u; t < a.L; ++t) {
                const int64_t off = (s * a.L + t) * a.qw() + h * a.dh;
                const int64_t ri = (s * a.H + h) * a.L + t;
                const float *qr = q + off, *gr = go + off;
                float sc = 0.f, dp = 0.f;
                for (int64_t e = 0; e < a.dh; ++e) {
                    sc += qr[e] * kr[e];
                    dp += gr[e] * vr[e];
                }
                const float p = expf(sc * scale - lse[ri]);
                const float ds = p * (dp - D[ri]);
                for (int64_t e = 0; e < a.dh; ++e) {
                    ak[e] += ds * qr[e];
                    av[e] += p * gr[e];
                }
            }
        }
        for (int64_t e = 0; e < a.dh; ++e) {
            gk[koff + e] = ak[e] * scale;
            gv[koff + e] = av[e];
        }
    }
};

RQ_HD float sigmoidf_(float z) { return 1.f / (1.f + expf(-z)); }

// m = silu(zg) zu
struct SwigluFwd {
    const float *zg; const float *zu; float *m;
    RQ_HD void operator()(int64_t i) const {
        const float g = zg[i];
        m[i] = g * sigmoidf_(g) * zu[i];
    }
};

// gzg = gm zu silu'(zg), gzu = gm silu(zg), silu'(z) = s (1 + z (1 - s));
// written over zg and zu in place
struct SwigluBwd {
    const float *gm; float *zg; float *zu;
    RQ_HD void operator()(int64_t i) const {
        const float g = zg[i], u = zu[i], c = gm[i];
        const float sg = sigmoidf_(g);
        zg[i] = c * u * (sg * (1.f + g * (1.f - sg)));
        zu[i] = c * g * sg;
    }
};

// per-token w_t . dz_t, and the fixed-order sum of those (one thread)
struct RowDot {
    const float *a; const float *b; float *out; int64_t d;
    RQ_HD void operator()(int64_t t) const {
        float acc = 0.f;
        for (int64_t k = 0; k < d; ++k) acc += a[t * d + k] * b[t * d + k];
        out[t] = acc;
    }
};
// the sum of count values in fixed order: chunk c of kChunk values into
// part[c] (double), then the parts in order, halved, into out
constexpr int64_t kChunk = 1024;
struct ChunkSum {
    const float *rows; double *part; int64_t count;
    RQ_HD void operator()(int64_t c) const {
        double acc = 0.0;
        const int64_t end = (c + 1) * kChunk < count ? (c + 1) * kChunk : count;
        for (int64_t t = c * kChunk; t < end; ++t) acc += (double)rows[t];
        part[c] = acc;
    }
};
struct ScaledSum {
    const double *part; float *out; int64_t nparts; double scale;
    RQ_HD void operator()(int64_t) const {
        double acc = 0.0;
        for (int64_t c = 0; c < nparts; ++c) acc += part[c];
        *out = (float)(scale * acc);
    }
};

// out = alpha a + (1 - alpha) b for two device scalars
struct Blend {
    const float *a; const float *b; float *out; float alpha;
    RQ_HD void operator()(int64_t) const { *out = alpha * *a + (1.f - alpha) * *b; }
};

// The KL head of the final block, one token row of V logits:
//   kl_t = sum_v p_v (log p_v - log q_v),  p = softmax(z0_t), q = softmax(z1_t),
// and z1_t is overwritten by (q - p) / T, the gradient of (1/T) sum_t kl_t.
struct KlRow {
    const float *z0; float *z1; float *kl; int64_t V; float inv_T;
    RQ_HD void operator()(int64_t t) const {
        const float *a = z0 + t * V;
        float *b = z1 + t * V;
        float ma = a[0], mb = b[0];
        for (int64_t v = 1; v < V; ++v) {
            ma = a[v] > ma ? a[v] : ma;
            mb = b[v] > mb ? b[v] : mb;
        }
        float sa = 0.f, sb = 0.f;
        for (int64_t v = 0; v < V; ++v) {
            sa += expf(a[v] - ma);
            sb += expf(b[v] - mb);
        }
        const float la = ma + logf(sa), lb = mb + logf(sb);   // log-partition functions
        float acc = 0.f;
        for (int64_t v = 0; v < V; ++v) {
            const float lp = a[v] - la, lq = b[v] - lb;
            const float p = expf(lp), q = expf(lq);
            acc += p * (lp - lq);
            b[v] = (q - p) * inv_T;
        }
        kl[t] = acc;
    }
};

// --------------------------------------------------------- workspace ---

struct Buffers {
    // transposed weights (in x out) for the forward GEMMs
    float *WqT, *WkT, *WvT, *WoT, *WgT, *WuT, *WdT;
    float *cs, *sn;
    // forward caches of the last forward pass
    float *x, *a, *r1, *q, *k, *v, *o, *lse, *h, *b, *r2, *zg, *zu, *m, *y;
    // the window: the reference output, the upstream gradient, row sums
    float *z0, *w, *rows;
    double *part;
    // backward scratch
    float *go, *D, *gk, *gv;
};

inline size_t rnd(size_t bytes) { return (bytes + 255) / 256 * 256; }

// the bytes of Buffers for dims (each buffer 256-byte aligned), and the
// buffers carved from base when base is not null
inline size_t carve(const Dims &dm, void *base, Buffers *bf) {
    const size_t T = (size_t)dm.T(), d = (size_t)dm.d, f = (size_t)dm.f, qw = (size_t)dm.qw(), kw = (size_t)dm.kw();
    const size_t rows = (size_t)dm.S * (size_t)dm.H * (size_t)dm.L;
    const size_t tab = (size_t)dm.L * (size_t)(dm.dh / 2);
    size_t off = 0;
    char *p = static_cast<char *>(base);
    auto take = [&](size_t count) -> float * {
        float *r = p ? reinterpret_cast<float *>(p + off) : nullptr;
        off += rnd(count * sizeof(float));
        return r;
    };
    Buffers B{};
    B.WqT = take(d * qw); B.WkT = take(d * kw); B.WvT = take(d * kw); B.WoT = take(qw * d);
    B.WgT = take(d * f); B.WuT = take(d * f); B.WdT = take(f * d);
    B.cs = take(tab); B.sn = take(tab);
    B.x = take(T * d); B.a = take(T * d); B.r1 = take(T);
    B.q = take(T * qw); B.k = take(T * kw); B.v = take(T * kw); B.o = take(T * qw); B.lse = take(rows);
    B.h = take(T * d); B.b = take(T * d); B.r2 = take(T);
    B.zg = take(T * f); B.zu = take(T * f); B.m = take(T * f); B.y = take(T * d);
    B.z0 = take(T * d); B.w = take(T * d); B.rows = take(T);
    B.part = reinterpret_cast<double *>(take(2 * ((T + kChunk - 1) / kChunk)));
    B.go = take(T * qw); B.D = take(rows); B.gk = take(T * kw); B.gv = take(T * kw);
    if (bf) *bf = B;
    return off;
}

// ------------------------------------------------------------ passes ---

inline Gemm gemm_rr(int64_t M, int64_t N, int64_t K, const float *A, const float *B, float *C, const float *R = nullptr,
                    float alpha = 1.f) {
    // A M x K, B K x N, C (and R) M x N, all dense row-major
    return Gemm{M, N, K, A, K, B, N, C, N, R, N, alpha, 0};
}

// the weight gradient gW (out x in) = gout^T in over T tokens: gout T x out,
// in T x in, both row-major
inline Gemm gemm_wgrad(int64_t T, int64_t out, int64_t in, const float *gout, const float *xin, float *gW) {
    return Gemm{out, in, T, gout, out, xin, in, gW, in, nullptr, in, 1.f, 1};
}

// the modules of the block, in the paper's order (q, k, v, o, gate, up, down)
enum Module : int { M_Q = 0, M_K = 1, M_V = 2, M_O = 3, M_GATE = 4, M_UP = 5, M_DOWN = 6 };

// the weight transposes and the rotary tables (once per call)
template <class X>
int setup(X &x, const Dims &dm, const Weights &W, const Buffers &B) {
    const int64_t d = dm.d, f = dm.f, qw = dm.qw(), kw = dm.kw();
    int e = 0;
    e |= x.map(qw * d, Transpose{W.Wq, B.WqT, qw, d}, "blk_transpose");
    e |= x.map(kw * d, Transpose{W.Wk, B.WkT, kw, d}, "blk_transpose");
    e |= x.map(kw * d, Transpose{W.Wv, B.WvT, kw, d}, "blk_transpose");
    e |= x.map(d * qw, Transpose{W.Wo, B.WoT, d, qw}, "blk_transpose");
    e |= x.map(f * d, Transpose{W.Wg, B.WgT, f, d}, "blk_transpose");
    e |= x.map(f * d, Transpose{W.Wu, B.WuT, f, d}, "blk_transpose");
    e |= x.map(d * f, Transpose{W.Wd, B.WdT, d, f}, "blk_transpose");
    e |= x.map(dm.L * (dm.dh / 2), RopeTable{B.cs, B.sn, dm.dh / 2, (double)dm.rope_base, dm.dh}, "blk_rope_table");
    return e;
}

// y = block(xin), the caches of the pass left in B (xin is copied to B.x
// unless it is B.x)
template <class X>
int forward(X &x, const Dims &dm, const Weights &W, const Buffers &B, const float *xin, float *y) {
    const int64_t T = dm.T(), d = dm.d, f = dm.f, qw = dm.qw(), kw = dm.kw();
    const AttnShape as{dm.L, dm.H, dm.Hkv, dm.dh};
    int e = 0;
    if (xin != B.x) e |= x.map(T * d, Axpy{xin, xin, B.x, 0.f}, "blk_copy");
    e |= x.map(T, RmsFwd{B.x, W.g1, B.a, B.r1, d, dm.eps}, "blk_rms_fwd");
    e |= x.gemm(gemm_rr(T, qw, d, B.a, B.WqT, B.q), "blk_proj");
    e |= x.gemm(gemm_rr(T, kw, d, B.a, B.WkT, B.k), "blk_proj");
    e |= x.gemm(gemm_rr(T, kw, d, B.a, B.WvT, B.v), "blk_proj");
    e |= x.map(T * dm.H * (dm.dh / 2), Rope{B.q, qw, dm.H, dm.dh / 2, dm.dh, dm.L, B.cs, B.sn, 0}, "blk_rope");
    e |= x.map(T * dm.Hkv * (dm.dh / 2), Rope{B.k, kw, dm.Hkv, dm.dh / 2, dm.dh, dm.L, B.cs, B.sn, 0}, "blk_rope");
    e |= x.map(dm.S * dm.H * dm.L, AttnFwd{B.q, B.k, B.v, B.o, B.lse, as}, "blk_attn_fwd");
    e |= x.gemm(gemm_rr(T, d, qw, B.o, B.WoT, B.h, B.x), "blk_proj");           // h = x + o Wo^T
    e |= x.map(T, RmsFwd{B.h, W.g2, B.b, B.r2, d, dm.eps}, "blk_rms_fwd");
    e |= x.gemm(gemm_rr(T, f, d, B.b, B.WgT, B.zg), "blk_proj");
    e |= x.gemm(gemm_rr(T, f, d, B.b, B.WuT, B.zu), "blk_proj");
    e |= x.map(T * f, SwigluFwd{B.zg, B.zu, B.m}, "blk_swiglu_fwd");
    e |= x.gemm(gemm_rr(T, d, f, B.m, B.WdT, y, B.h), "blk_proj");              // y = h + m Wd^T
    return e;
}

// gx = (d y / d x)^T gy for the caches of the last forward pass, and, for
// module >= 0, that module's weight gradient gW (out x in) = gout^T in,
// taken where both factors are still in the buffers.  gy is read only; gx
// (null: not computed) may not alias any buffer of B except B.y.
template <class X>
int backward(X &x, const Dims &dm, const Weights &W, const Buffers &B, const float *gy, float *gx, int module = -1,
             float *gW = nullptr) {
    const int64_t T = dm.T(), d = dm.d, f = dm.f, qw = dm.qw(), kw = dm.kw();
    const AttnShape as{dm.L, dm.H, dm.Hkv, dm.dh};
    const int64_t rows = dm.S * dm.H * dm.L;
    int e = 0;
    // MLP: W_d's gradient gy^T m, then gm = gy Wd (into m) and the SwiGLU
    // backward over zg / zu
    if (module == M_DOWN) e |= x.gemm(gemm_wgrad(T, d, f, gy, B.m, gW), "blk_wgrad");
    e |= x.gemm(gemm_rr(T, f, d, gy, W.Wd, B.m), "blk_proj_bwd");
    e |= x.map(T * f, SwigluBwd{B.m, B.zg, B.zu}, "blk_swiglu_bwd");
    if (module == M_GATE) e |= x.gemm(gemm_wgrad(T, f, d, B.zg, B.b, gW), "blk_wgrad");
    if (module == M_UP) e |= x.gemm(gemm_wgrad(T, f, d, B.zu, B.b, gW), "blk_wgrad");
    if (module == M_DOWN || module == M_GATE || module == M_UP) return e;
    // gb = gzg Wg + gzu Wu (into b)
    e |= x.gemm(gemm_rr(T, d, f, B.zg, W.Wg, B.b), "blk_proj_bwd");
    e |= x.gemm(gemm_rr(T, d, f, B.zu, W.Wu, B.b, B.b), "blk_proj_bwd");
    // gh = gy + RMSNorm2 backward (into y)
    e |= x.map(T, RmsBwd{B.h, W.g2, B.r2, B.b, gy, B.y, d}, "blk_rms_bwd");
    if (module == M_O) return e | x.gemm(gemm_wgrad(T, d, qw, B.y, B.o, gW), "blk_wgrad");
    // attention: go = gh Wo, the row terms, dq (into o), dk, dv
    e |= x.gemm(gemm_rr(T, qw, d, B.y, W.Wo, B.go), "blk_proj_bwd");
    e |= x.map(rows, AttnRowDot{B.go, B.o, B.D, as}, "blk_attn_rowdot");
    e |= x.map(rows, AttnBwdQ{B.q, B.k, B.v, B.go, B.lse, B.D, B.o, as}, "blk_attn_bwd_q");
    e |= x.map(dm.S * dm.Hkv * dm.L, AttnBwdKV{B.q, B.k, B.v, B.go, B.lse, B.D, B.gk, B.gv, as}, "blk_attn_bwd_kv");
    e |= x.map(T * dm.H * (dm.dh / 2), Rope{B.o, qw, dm.H, dm.dh / 2, dm.dh, dm.L, B.cs, B.sn, 1}, "blk_rope");
    e |= x.map(T * dm.Hkv * (dm.dh / 2), Rope{B.gk, kw, dm.Hkv, dm.dh / 2, dm.dh, dm.L, B.cs, B.sn, 1}, "blk_rope");
    if (module == M_Q) return e | x.gemm(gemm_wgrad(T, qw, d, B.o, B.a, gW), "blk_wgrad");
    if (module == M_K) return e | x.gemm(gemm_wgrad(T, kw, d, B.gk, B.a, gW), "blk_wgrad");
    if (module == M_V) return e | x.gemm(gemm_wgrad(T, kw, d, B.gv, B.a, gW), "blk_wgrad");
    if (!gx) return e;
    // ga = gq Wq + gk Wk + gv Wv (into a)
    e |= x.gemm(gemm_rr(T, d, qw, B.o, W.Wq, B.a), "blk_proj_bwd");
    e |= x.gemm(gemm_rr(T, d, kw, B.gk, W.Wk, B.a, B.a), "blk_proj_bwd");
    e |= x.gemm(gemm_rr(T, d, kw, B.gv, W.Wv, B.a, B.a), "blk_proj_bwd");
    // gx = gh + RMSNorm1 backward
    e |= x.map(T, RmsBwd{B.x, W.g1, B.r1, B.a, B.y, gx, d}, "blk_rms_bwd");
    return e;
}

// the next block's Fisher loss of Eq. slide_window and its gradient in Δh:
//   Δz = B(h + Δh) - B(h),  w = Δz F' / T,  loss = (1/2) sum_t w_t . Δz_t,
//   g = (d B / d x at h + Δh)^T w
template <class X>
int window(X &x, const Dims &dm, const Weights &W, const Buffers &B, const float *h_ref, const float *dh_,
           const float *F_next, float *g, float *loss) {
    const int64_t T = dm.T(), d = dm.d;
    int e = 0;
    e |= forward(x, dm, W, B, h_ref, B.z0);
    e |= x.map(T * d, Axpy{h_ref, dh_, B.x, 1.f}, "blk_axpy");
    e |= forward(x, dm, W, B, B.x, B.y);
    e |= x.map(T * d, Axpy{B.y, B.z0, B.z0, -1.f}, "blk_axpy");                // Δz (into z0)
    e |= x.gemm(gemm_rr(T, d, d, B.z0, F_next, B.w, nullptr, 1.f / (float)T), "blk_fisher");
    if (loss) {
        const int64_t np = (T + kChunk - 1) / kChunk;
        e |= x.map(T, RowDot{B.w, B.z0, B.rows, d}, "blk_rowdot");
        e |= x.map(np, ChunkSum{B.rows, B.part, T}, "blk_chunksum");
        e |= x.map(1, ScaledSum{B.part, loss, np, 0.5}, "blk_sum");
    }
    e |= backward(x, dm, W, B, B.w, g);
    return e;
}

// The input of one module in a forward pass of the block (weights W, input
// xin), copied to Xout (T x n, the module's in-dimension n): q/k/v read the
// attention norm's output a, o_proj the attention output o, gate/up the MLP
// norm's output b, down_proj the SwiGLU product m.  Its second moment is the
// module's OBS Hessian.
template <class X>
int module_input(X &x, const Dims &dm, const Weights &W, const Buffers &B, const float *xin, int module,
                 float *Xout) {
    const int64_t T = dm.T();
    int e = setup(x, dm, W, B);
    e |= forward(x, dm, W, B, xin, B.y);
    const float *src = B.a;
    int64_t n = dm.d;
    if (module == M_O) { src = B.o; n = dm.qw(); }
    else if (module == M_GATE || module == M_UP) { src = B.b; n = dm.d; }
    else if (module == M_DOWN) { src = B.m; n = dm.f; }
    e |= x.map(T * n, Axpy{src, src, Xout, 0.f}, "blk_copy");
    return e;
}

// ------------------------------------------------- module-level losses ---

// block l's side of the module-level losses: the reference and perturbed
// outputs, the upstream gradient, this block's Fisher term, scalars
struct ModuleBuffers {
    float *href, *dh, *gnext, *tmp, *gh, *wthis, *rows;
    double *part;
    float *lthis, *lnext;
};

inline size_t carve_module(const Dims &dm, void *base, ModuleBuffers *mb) {
    const size_t T = (size_t)dm.T(), d = (size_t)dm.d;
    size_t off = 0;
    char *p = static_cast<char *>(base);
    auto take = [&](size_t count) -> float * {
        float *r = p ? reinterpret_cast<float *>(p + off) : nullptr;
        off += rnd(count * sizeof(float));
        return r;
    };
    ModuleBuffers M{};
    M.href = take(T * d); M.dh = take(T * d); M.gnext = take(T * d); M.tmp = take(T * d); M.gh = take(T * d);
    M.wthis = take(T * d); M.rows = take(T);
    M.part = reinterpret_cast<double *>(take(2 * ((T + kChunk - 1) / kChunk)));
    M.lthis = take(1); M.lnext = take(1);
    if (mb) *mb = M;
    return off;
}

// the final norm and LM head: z = RMSNorm(h; gf) Wh^T, Wh V x d
struct Head {
    const float *gf; const float *Wh; int64_t V;
};
struct HeadBuffers {
    float *WhT, *u, *r, *z0, *z1, *x1, *kl, *gu;
    double *part;
};

inline size_t carve_head(const Dims &dm, int64_t V, void *base, HeadBuffers *hb) {
    const size_t T = (size_t)dm.T(), d = (size_t)dm.d, v = (size_t)V;
    size_t off = 0;
    char *p = static_cast<char *>(base);
    auto take = [&](size_t count) -> float * {
        float *r = p ? reinterpret_cast<float *>(p + off) : nullptr;
        off += rnd(count * sizeof(float));
        return r;
    };
    HeadBuffers H{};
    H.WhT = take(d * v); H.u = take(T * d); H.r = take(T); H.z0 = take(T * v); H.z1 = take(T * v);
    H.x1 = take(T * d); H.kl = take(T); H.gu = take(T * d);
    H.part = reinterpret_cast<double *>(take(2 * ((T + kChunk - 1) / kChunk)));
    if (hb) *hb = H;
    return off;
}

// The final block's loss, the true KL at the LM head (Eq. kl_loss):
//   z0 = RMSNorm(h*; gf) Wh^T,  z1 = RMSNorm(h* + Δh; gf) Wh^T,
//   loss = (1/T) sum_t KL(softmax z0_t || softmax z1_t),
//   g = d loss / d Δh = RMSNorm backward of ((softmax z1 - softmax z0) Wh / T)
template <class X>
int kl_head(X &x, const Dims &dm, const Head &hd, const HeadBuffers &H, const float *h_ref, const float *dh_,
            float *g, float *loss) {
    const int64_t T = dm.T(), d = dm.d, V = hd.V;
    int e = 0;
    e |= x.map(V * d, Transpose{hd.Wh, H.WhT, V, d}, "blk_transpose");
    e |= x.map(T, RmsFwd{h_ref, hd.gf, H.u, H.r, d, dm.eps}, "blk_rms_fwd");
    e |= x.gemm(gemm_rr(T, V, d, H.u, H.WhT, H.z0), "blk_head");
    e |= x.map(T * d, Axpy{h_ref, dh_, H.x1, 1.f}, "blk_axpy");
    e |= x.map(T, RmsFwd{H.x1, hd.gf, H.u, H.r, d, dm.eps}, "blk_rms_fwd");
    e |= x.gemm(gemm_rr(T, V, d, H.u, H.WhT, H.z1), "blk_head");
    e |= x.map(T, KlRow{H.z0, H.z1, H.kl, V, 1.f / (float)T}, "blk_kl_row");
    e |= x.gemm(gemm_rr(T, d, V, H.z1, hd.Wh, H.gu), "blk_head_bwd");
    e |= x.map(T, RmsBwd{H.x1, hd.gf, H.r, H.gu, nullptr, g, d}, "blk_rms_bwd");
    if (loss) {
        const int64_t np = (T + kChunk - 1) / kChunk;
        e |= x.map(np, ChunkSum{H.kl, H.part, T}, "blk_chunksum");
        e |= x.map(1, ScaledSum{H.part, loss, np, 1.0 / (double)T}, "blk_sum");
    }
    return e;
}

// block l's reference pass (full-precision weights Wref on the reference
// input xin) and its current pass (Wcur, the weights quantized so far with
// the module's weight replaced, on the perturbed input xhat; Sec. 4.3): h*
// into M.href, Δh = h - h* into M.dh, and the current pass's caches left in
// Bl for the module's backward
template <class X>
int module_delta(X &x, const Dims &dm, const Weights &Wref, const Weights &Wcur, const Buffers &Bl,
                 const ModuleBuffers &M, const float *xin, const float *xhat) {
    const int64_t T = dm.T(), d = dm.d;
    int e = 0;
    e |= setup(x, dm, Wref, Bl);
    e |= forward(x, dm, Wref, Bl, xin, M.href);
    e |= setup(x, dm, Wcur, Bl);
    e |= forward(x, dm, Wcur, Bl, xhat, M.dh);
    e |= x.map(T * d, Axpy{M.dh, M.href, M.dh, -1.f}, "blk_axpy");
    return e;
}

// The exact two-block sliding window of one module of block l (Eq.
// slide_window), its loss and the gradient in the module's weight:
//   loss = alpha (1/2T) sum_t Δh_t^T F Δh_t + (1 - alpha) L(l+1)(h*, Δh),
//   g_h = alpha Δh F / T + (1 - alpha) dL(l+1)/dΔh, back through block l.
// Wcur is the current pass's weights with the module's weight replaced
// (module_delta); Wn the next block's.
template <class X>
int module_window(X &x, const Dims &dm, const Weights &Wref, const Weights &Wcur, const Weights &Wn, const Buffers &Bl,
                  const Buffers &Bn, const ModuleBuffers &M, const float *xin, const float *xhat, int module,
                  float alpha, const float *F_this, const float *F_next, float *gW, float *loss) {
    const int64_t T = dm.T(), d = dm.d;
    const int64_t np = (T + kChunk - 1) / kChunk;
    int e = module_delta(x, dm, Wref, Wcur, Bl, M, xin, xhat);
    e |= setup(x, dm, Wn, Bn);
    e |= window(x, dm, Wn, Bn, M.href, M.dh, F_next, M.gnext, M.lnext);
    e |= x.gemm(gemm_rr(T, d, d, M.dh, F_this, M.wthis, nullptr, 1.f / (float)T), "blk_fisher");
    e |= x.map(T, RowDot{M.wthis, M.dh, M.rows, d}, "blk_rowdot");
    e |= x.map(np, ChunkSum{M.rows, M.part, T}, "blk_chunksum");
    e |= x.map(1, ScaledSum{M.part, M.lthis, np, 0.5}, "blk_sum");
    e |= x.map(T * d, Axpy{M.gnext, M.gnext, M.tmp, -alpha}, "blk_axpy");   // (1 - alpha) g_next
    e |= x.map(T * d, Axpy{M.tmp, M.wthis, M.gh, alpha}, "blk_axpy");       // + alpha Δh F / T
    if (loss) e |= x.map(1, Blend{M.lthis, M.lnext, loss, alpha}, "blk_blend");
    e |= backward(x, dm, Wcur, Bl, M.gh, nullptr, module, gW);
    return e;
}

// The final block's loss of one module: the KL at the LM head between the
// reference output and the current pass's (module_delta), and the gradient
// in the module's weight.
template <class X>
int module_kl(X &x, const Dims &dm, const Weights &Wref, const Weights &Wcur, const Buffers &Bl,
              const ModuleBuffers &M, const Head &hd, const HeadBuffers &H, const float *xin, const float *xhat,
              int module, float *gW, float *loss) {
    int e = module_delta(x, dm, Wref, Wcur, Bl, M, xin, xhat);
    e |= kl_head(x, dm, hd, H, M.href, M.dh, M.gh, loss);
    e |= backward(x, dm, Wcur, Bl, M.gh, nullptr, module, gW);
    return e;
}

// the block weights with one module's weight replaced
inline Weights with_module(Weights w, int module, const float *Wm) {
    switch (module) {
        case M_Q: w.Wq = Wm; break;
        case M_K: w.Wk = Wm; break;
        case M_V: w.Wv = Wm; break;
        case M_O: w.Wo = Wm; break;
        case M_GATE: w.Wg = Wm; break;
        case M_UP: w.Wu = Wm; break;
        default: w.Wd = Wm; break;
    }
    return w;
}

}  // namespace blk
}  // namespace realq
