// Causal grouped-query attention of the decoder block ops (the exact window
// of Sec. 4.4, Eq. slide_window), tiled for the GPU: the same three passes as
// the per-row bodies of block_ops.cuh (AttnFwd, AttnBwdQ, AttnBwdKV), each
// CTA holding a tile of rows in shared memory and streaming the other side
// through it, in fp32 on the CUDA cores (fp32 FFMA accuracy, as the window's
// difference of two forward passes needs).
//
// Layouts (as the bodies'): q, o, gq: (S L) x (H dh), head h at columns
// h dh; k, v, gk, gv: (S L) x (Hkv dh); lse, D: index (s H + h) L + t; query
// head h reads key/value head h / (H / Hkv); scale 1/sqrt(dh).
//
//   attn_fwd     one CTA per (s, h, 64 queries): key tiles of 32 through
//                shared memory, online softmax per row; o and lse
//   attn_bwd_q   one CTA per (s, h, 64 queries): P and dS recomputed per key
//                tile, dq = scale sum dS k
//   attn_bwd_kv  one CTA per (s, kv head, 64 keys): over the group's query
//                heads and the query tiles at or after the keys, dv = sum P^T
//                dO and dk = scale sum dS^T q
// Every output element is written by one thread in a fixed order: the
// passes are deterministic.  256 threads; thread (ty, tx) = (tid / 16, tid %
// 16) owns 4 rows of its CTA's row tile, the key (or query) columns tx and
// tx + 16 of a score tile, and head-dimension columns tx + 16 j.
#include <type_traits>

#include "kernels.cuh"

namespace realq {
namespace {

constexpr int BR = 64;   // rows per CTA (queries, or keys in attn_bwd_kv)
constexpr int BC = 32;   // columns per streamed tile
constexpr int NT = 256;

// shared-memory row pitch for head dimension dh: odd, so that the 16 rows a
// warp's threads read at one column fall in distinct banks
__host__ __device__ inline int pitch_of(int dh) { return dh | 1; }

// s[i][j] = sum_e A[r0 + i][e] B[tx + 16 j][e] over e < dh
__device__ __forceinline__ void dots4x2(const float *A, const float *Bm, int pitch, int dh, int r0, int tx,
                                        float (&s)[4][2]) {
#pragma unroll
    for (int i = 0; i < 4; ++i) s[i][0] = s[i][1] = 0.f;
    const float *a0 = A + r0 * pitch, *b0 = Bm + tx * pitch, *b1 = Bm + (tx + 16) * pitch;
    for (int e = 0; e < dh; ++e) {
        const float x0 = b0[e], x1 = b1[e];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const float a = a0[i * pitch + e];
            s[i][0] = fmaf(a, x0, s[i][0]);
            s[i][1] = fmaf(a, x1, s[i][1]);
        }
    }
}

// rows [row0, row0 + nrows) of a (S L) x ld matrix, columns col0 .. col0 + dh,
// into shared memory (pitch), zero past the sequence end
__device__ __forceinline__ void load_rows(float *dst, int pitch, const float *src, int64_t ld, int64_t base_row,
                                          int64_t first, int nrows, int64_t L, int64_t col0, int dh) {
    for (int idx = threadIdx.x; idx < nrows * dh; idx += NT) {
        const int r = idx / dh, e = idx % dh;
        const int64_t t = first + r;
        dst[r * pitch + e] = t < L ? src[(base_row + t) * ld + col0 + e] : 0.f;
    }
}

template <int MAXD>
__global__ void __launch_bounds__(NT) attn_fwd_kernel(int64_t L, int H, int Hkv, int dh, const float *q,
                                                      const float *k, const float *v, float *o, float *lse,
                                                      int64_t qtiles) {
    extern __shared__ float sm[];
    const int pitch = pitch_of(dh);
    float *Qs = sm, *Ks = Qs + BR * pitch, *Vs = Ks + BC * pitch, *Ps = Vs + BC * pitch;   // Ps: BR x (BC + 1)
    const int64_t bid = blockIdx.x;
    const int64_t qt = bid % qtiles, h = (bid / qtiles) % H, s = bid / (qtiles * H);
    const int64_t kvh = h / (H / Hkv);
    const int64_t qw = (int64_t)H * dh, kw = (int64_t)Hkv * dh;
    const int64_t q0 = qt * BR, base = s * L;
    const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4, r0 = ty * 4;
    const float scale = 1.f / sqrtf((float)dh);
    load_rows(Qs, pitch, q, qw, base, q0, BR, L, h * dh, dh);
    float mx[4], l[4], acc[4][MAXD / 16];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        mx[i] = -INFINITY;
        l[i] = 0.f;
#pragma unroll
        for (int j = 0; j < MAXD / 16; ++j) acc[i][j] = 0.f;
    }
    const int64_t qlast = (q0 + BR < L ? q0 + BR : L) - 1;
    for (int64_t k0 = 0; k0 <= qlast; k0 += BC) {
        __syncthreads();   // the previous tile's readers are done
        load_rows(Ks, pitch, k, kw, base, k0, BC, L, kvh * dh, dh);
        load_rows(Vs, pitch, v, kw, base, k0, BC, L, kvh * dh, dh);
        __syncthreads();
        float sc[4][2];
        dots4x2(Qs, Ks, pitch, dh, r0, tx, sc);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int64_t t = q0 + r0 + i;
            float p0 = -INFINITY, p1 = -INFINITY;
            if (k0 + tx <= t && k0 + tx < L) p0 = sc[i][0] * scale;
            if (k0 + tx + 16 <= t && k0 + tx + 16 < L) p1 = sc[i][1] * scale;
            float m = fmaxf(p0, p1);
#pragma unroll
            for (int o_ = 8; o_ > 0; o_ >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o_));
            const float mnew = fmaxf(mx[i], m);
            // rows with no key yet (mnew = -inf) keep everything at zero
            const float c = mnew == -INFINITY ? 1.f : expf(mx[i] - mnew);
            const float e0 = mnew == -INFINITY ? 0.f : expf(p0 - mnew);
            const float e1 = mnew == -INFINITY ? 0.f : expf(p1 - mnew);
            float rs = e0 + e1;
#pragma unroll
            for (int o_ = 8; o_ > 0; o_ >>= 1) rs += __shfl_xor_sync(0xffffffffu, rs, o_);
            l[i] = l[i] * c + rs;
            mx[i] = mnew;
#pragma unroll
            for (int j = 0; j < MAXD / 16; ++j) acc[i][j] *= c;
            Ps[(r0 + i) * (BC + 1) + tx] = e0;
            Ps[(r0 + i) * (BC + 1) + tx + 16] = e1;
        }
        __syncthreads();
        for (int c = 0; c < BC; ++c) {
            float pr[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) pr[i] = Ps[(r0 + i) * (BC + 1) + c];
            const float *vr = Vs + c * pitch;
#pragma unroll
            for (int j = 0; j < MAXD / 16; ++j) {
                const int d = tx + 16 * j;
                const float x = d < dh ? vr[d] : 0.f;
#pragma unroll
                for (int i = 0; i < 4; ++i) acc[i][j] = fmaf(pr[i], x, acc[i][j]);
            }
        }
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int64_t t = q0 + r0 + i;
        if (t >= L) continue;
        const float inv = 1.f / l[i];
        float *orow = o + (base + t) * qw + h * dh;
#pragma unroll
        for (int j = 0; j < MAXD / 16; ++j) {
            const int d = tx + 16 * j;
            if (d < dh) orow[d] = acc[i][j] * inv;
        }
        if (tx == 0) lse[(s * H + h) * L + t] = mx[i] + logf(l[i]);
    }
}

template <int MAXD>
__global__ void __launch_bounds__(NT) attn_bwd_q_kernel(int64_t L, int H, int Hkv, int dh, const float *q,
                                                        const float *k, const float *v, const float *go,
                                                        const float *lse, const float *D, float *gq,
                                                        int64_t qtiles) {
    extern __shared__ float sm[];
    const int pitch = pitch_of(dh);
    float *Qs = sm, *Gs = Qs + BR * pitch, *Ks = Gs + BR * pitch, *Vs = Ks + BC * pitch;
    float *Ss = Vs + BC * pitch;   // dS: BR x (BC + 1)
    const int64_t bid = blockIdx.x;
    const int64_t qt = bid % qtiles, h = (bid / qtiles) % H, s = bid / (qtiles * H);
    const int64_t kvh = h / (H / Hkv);
    const int64_t qw = (int64_t)H * dh, kw = (int64_t)Hkv * dh;
    const int64_t q0 = qt * BR, base = s * L;
    const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4, r0 = ty * 4;
    const float scale = 1.f / sqrtf((float)dh);
    load_rows(Qs, pitch, q, qw, base, q0, BR, L, h * dh, dh);
    load_rows(Gs, pitch, go, qw, base, q0, BR, L, h * dh, dh);
    float ls[4], Dt[4], acc[4][MAXD / 16];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int64_t t = q0 + r0 + i;
        ls[i] = t < L ? lse[(s * H + h) * L + t] : 0.f;
        Dt[i] = t < L ? D[(s * H + h) * L + t] : 0.f;
#pragma unroll
        for (int j = 0; j < MAXD / 16; ++j) acc[i][j] = 0.f;
    }
    const int64_t qlast = (q0 + BR < L ? q0 + BR : L) - 1;
    for (int64_t k0 = 0; k0 <= qlast; k0 += BC) {
        __syncthreads();
        load_rows(Ks, pitch, k, kw, base, k0, BC, L, kvh * dh, dh);
        load_rows(Vs, pitch, v, kw, base, k0, BC, L, kvh * dh, dh);
        __syncthreads();
        float sc[4][2], dp[4][2];
        dots4x2(Qs, Ks, pitch, dh, r0, tx, sc);
        dots4x2(Gs, Vs, pitch, dh, r0, tx, dp);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int64_t t = q0 + r0 + i;
#pragma unroll
            for (int j = 0; j < 2; ++j) {
                const int64_t u = k0 + tx + 16 * j;
                const float p = (u <= t && u < L && t < L) ? expf(sc[i][j] * scale - ls[i]) : 0.f;
                Ss[(r0 + i) * (BC + 1) + tx + 16 * j] = p * (dp[i][j] - Dt[i]);
            }
        }
        __syncthreads();
        for (int c = 0; c < BC; ++c) {
            float ds[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) ds[i] = Ss[(r0 + i) * (BC + 1) + c];
            const float *kr = Ks + c * pitch;
#pragma unroll
            for (int j = 0; j < MAXD / 16; ++j) {
                const int d = tx + 16 * j;
                const float x = d < dh ? kr[d] : 0.f;
#pragma unroll
                for (int i = 0; i < 4; ++i) acc[i][j] = fmaf(ds[i], x, acc[i][j]);
            }
        }
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int64_t t = q0 + r0 + i;
        if (t >= L) continue;
        float *out = gq + (base + t) * qw + h * dh;
#pragma unroll
        for (int j = 0; j < MAXD / 16; ++j) {
            const int d = tx + 16 * j;
            if (d < dh) out[d] = acc[i][j] * scale;
        }
    }
}

template <int MAXD>
__global__ void __launch_bounds__(NT) attn_bwd_kv_kernel(int64_t L, int H, int Hkv, int dh, const float *q,
                                                         const float *k, const float *v, const float *go,
                                                         const float *lse, const float *D, float *gk, float *gv,
                                                         int64_t ktiles) {
    extern __shared__ float sm[];
    const int pitch = pitch_of(dh);
    float *Ks = sm, *Vs = Ks + BR * pitch, *Qs = Vs + BR * pitch, *Gs = Qs + BC * pitch;
    float *Ps = Gs + BC * pitch;       // P^T: BR (keys) x (BC + 1)
    float *Ss = Ps + BR * (BC + 1);    // dS^T
    __shared__ float lsq[BC], Dq[BC];
    const int64_t bid = blockIdx.x;
    const int64_t kt = bid % ktiles, kvh = (bid / ktiles) % Hkv, s = bid / (ktiles * Hkv);
    const int rep = H / Hkv;
    const int64_t qw = (int64_t)H * dh, kw = (int64_t)Hkv * dh;
    const int64_t u0 = kt * BR, base = s * L;
    const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4, r0 = ty * 4;
    const float scale = 1.f / sqrtf((float)dh);
    load_rows(Ks, pitch, k, kw, base, u0, BR, L, kvh * dh, dh);
    load_rows(Vs, pitch, v, kw, base, u0, BR, L, kvh * dh, dh);
    float ak[4][MAXD / 16], av[4][MAXD / 16];
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < MAXD / 16; ++j) ak[i][j] = av[i][j] = 0.f;
    for (int64_t h = kvh * rep; h < (kvh + 1) * rep; ++h) {
        for (int64_t t0 = u0 - u0 % BC; t0 < L; t0 += BC) {
            __syncthreads();
            load_rows(Qs, pitch, q, qw, base, t0, BC, L, h * dh, dh);
            load_rows(Gs, pitch, go, qw, base, t0, BC, L, h * dh, dh);
            if (threadIdx.x < BC) {
                const int64_t t = t0 + threadIdx.x;
                lsq[threadIdx.x] = t < L ? lse[(s * H + h) * L + t] : 0.f;
                Dq[threadIdx.x] = t < L ? D[(s * H + h) * L + t] : 0.f;
            }
            __syncthreads();
            // scores of key rows r0 + i against query columns tx, tx + 16
            float sc[4][2], dp[4][2];
            dots4x2(Ks, Qs, pitch, dh, r0, tx, sc);
            dots4x2(Vs, Gs, pitch, dh, r0, tx, dp);
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const int64_t u = u0 + r0 + i;
#pragma unroll
                for (int j = 0; j < 2; ++j) {
                    const int c = tx + 16 * j;
                    const int64_t t = t0 + c;
                    const float p = (t >= u && t < L && u < L) ? expf(sc[i][j] * scale - lsq[c]) : 0.f;
                    Ps[(r0 + i) * (BC + 1) + c] = p;
                    Ss[(r0 + i) * (BC + 1) + c] = p * (dp[i][j] - Dq[c]);
                }
            }
            __syncthreads();
            for (int c = 0; c < BC; ++c) {
                float pp[4], ds[4];
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    pp[i] = Ps[(r0 + i) * (BC + 1) + c];
                    ds[i] = Ss[(r0 + i) * (BC + 1) + c];
                }
                const float *qr = Qs + c * pitch, *gr = Gs + c * pitch;
#pragma unroll
                for (int j = 0; j < MAXD / 16; ++j) {
                    const int d = tx + 16 * j;
                    const float xq = d < dh ? qr[d] : 0.f, xg = d < dh ? gr[d] : 0.f;
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        ak[i][j] = fmaf(ds[i], xq, ak[i][j]);
                        av[i][j] = fmaf(pp[i], xg, av[i][j]);
                    }
                }
            }
        }
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int64_t u = u0 + r0 + i;
        if (u >= L) continue;
        const int64_t off = (base + u) * kw + kvh * dh;
#pragma unroll
        for (int j = 0; j < MAXD / 16; ++j) {
            const int d = tx + 16 * j;
            if (d < dh) {
                gk[off + d] = ak[i][j] * scale;
                gv[off + d] = av[i][j];
            }
        }
    }
}

size_t fwd_smem(int dh) { return (size_t)((BR + 2 * BC) * pitch_of(dh) + BR * (BC + 1)) * sizeof(float); }
size_t bwd_q_smem(int dh) { return (size_t)((2 * BR + 2 * BC) * pitch_of(dh) + BR * (BC + 1)) * sizeof(float); }
size_t bwd_kv_smem(int dh) { return (size_t)((2 * BR + 2 * BC) * pitch_of(dh) + 2 * BR * (BC + 1)) * sizeof(float); }

realq_status_t attn_check(int64_t S, int64_t L, int64_t H, int64_t Hkv, int64_t dh, const char *who) {
    if (S <= 0 || L <= 0 || H <= 0 || Hkv <= 0 || H % Hkv != 0 || dh <= 0 || dh > 256)
        return fail(REALQ_ERR_INVALID_ARG, "%s: bad attention shape", who);
    if (S * H * ((L + BR - 1) / BR) > 0x7FFFFFFFll) return fail(REALQ_ERR_UNSUPPORTED, "%s: too many tiles", who);
    return REALQ_OK;
}

template <class F>
realq_status_t by_width(int64_t dh, F f) {
    if (dh <= 32) return f(std::integral_constant<int, 32>());
    if (dh <= 64) return f(std::integral_constant<int, 64>());
    if (dh <= 128) return f(std::integral_constant<int, 128>());
    return f(std::integral_constant<int, 256>());
}

}  // namespace

realq_status_t attn_fwd_tiled(cudaStream_t st, int64_t S, int64_t L, int64_t H, int64_t Hkv, int64_t dh,
                              const float *q, const float *k, const float *v, float *o, float *lse,
                              const char *name) {
    REALQ_TRY(attn_check(S, L, H, Hkv, dh, name));
    const int64_t qt = (L + BR - 1) / BR;
    const size_t smem = fwd_smem((int)dh);
    return by_width(dh, [&](auto w) -> realq_status_t {
        constexpr int MAXD = decltype(w)::value;
        REALQ_TRY(set_smem_limit(reinterpret_cast<const void *>(attn_fwd_kernel<MAXD>), (int)smem));
        {
            Launch Lc(name, st);
            attn_fwd_kernel<MAXD><<<(unsigned)(S * H * qt), NT, smem, st>>>(L, (int)H, (int)Hkv, (int)dh, q, k, v, o,
                                                                            lse, qt);
        }
        return check_launch(name);
    });
}

realq_status_t attn_bwd_q_tiled(cudaStream_t st, int64_t S, int64_t L, int64_t H, int64_t Hkv, int64_t dh,
                                const float *q, const float *k, const float *v, const float *go, const float *lse,
                                const float *D, float *gq, const char *name) {
    REALQ_TRY(attn_check(S, L, H, Hkv, dh, name));
    const int64_t qt = (L + BR - 1) / BR;
    const size_t smem = bwd_q_smem((int)dh);
    return by_width(dh, [&](auto w) -> realq_status_t {
        constexpr int MAXD = decltype(w)::value;
        REALQ_TRY(set_smem_limit(reinterpret_cast<const void *>(attn_bwd_q_kernel<MAXD>), (int)smem));
        {
            Launch Lc(name, st);
            attn_bwd_q_kernel<MAXD><<<(unsigned)(S * H * qt), NT, smem, st>>>(L, (int)H, (int)Hkv, (int)dh, q, k, v,
                                                                              go, lse, D, gq, qt);
        }
        return check_launch(name);
    });
}

realq_status_t attn_bwd_kv_tiled(cudaStream_t st, int64_t S, int64_t L, int64_t H, int64_t Hkv, int64_t dh,
                                 const float *q, const float *k, const float *v, const float *go, const float *lse,
                                 const float *D, float *gk, float *gv, const char *name) {
    REALQ_TRY(attn_check(S, L, H, Hkv, dh, name));
    const int64_t kt = (L + BR - 1) / BR;
    const size_t smem = bwd_kv_smem((int)dh);
    return by_width(dh, [&](auto w) -> realq_status_t {
        constexpr int MAXD = decltype(w)::value;
        REALQ_TRY(set_smem_limit(reinterpret_cast<const void *>(attn_bwd_kv_kernel<MAXD>), (int)smem));
        {
            Launch Lc(name, st);
            attn_bwd_kv_kernel<MAXD><<<(unsigned)(S * Hkv * kt), NT, smem, st>>>(L, (int)H, (int)Hkv, (int)dh, q, k,
                                                                                 v, go, lse, D, gk, gv, kt);
        }
        return check_launch(name);
    });
}

}  // namespace realq
