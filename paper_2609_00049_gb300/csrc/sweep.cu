// Steps a4-a8 of the sweep for one module (Alg. 1, loop over column blocks):
//   quantize the B columns of block b with OBS error feedback inside the block
//   (Eq. gptq_update, written with rows of U: err_j = (w_j - deq_j) / U_jj,
//   W[:, k] -= err_j U_jk), the lazy batch update of all later columns
//   (Sec. 3.2: W[:, rest] -= E_b U[b, rest]), then Block-GD on the later columns
//   (Eq. block_gd_update) with the layer-level Fisher surrogate, optionally
//   blended with the next block's Fisher (Eq. slide_window).
#include "kernels.cuh"

#include <cmath>

namespace realq {
namespace {


// quant(.) grid of one group from its min / max (the reading fixed by the
// oracle: the grid contains 0; degenerate groups get [-1, 1]).  fp32, IEEE
// division, round-half-to-even.
__device__ __forceinline__ void grid_params(float mn, float mx, int bits, int sym, float &sc, float &zr) {
    const float maxq = (float)((1 << bits) - 1);
    float xmin = fminf(mn, 0.f), xmax = fmaxf(mx, 0.f);
    if (sym) {
        xmax = fmaxf(-xmin, xmax);
        xmin = -xmax;
    }
    if (xmin == 0.f && xmax == 0.f) {
        xmin = -1.f;
        xmax = 1.f;
    }
    sc = (xmax - xmin) / maxq;
    zr = sym ? (float)(1 << (bits - 1)) : rintf(-xmin / sc);
}

template <typename TW>
__global__ void init_work_kernel(int64_t m, int64_t n, const TW *W0, const uint8_t *dead, float *W) {
    const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= m * n) return;
    const int64_t j = idx % n;
    W[idx] = (dead && dead[j]) ? 0.f : load_as_float(W0, idx);
}

// one warp per row: min / max of W[i, c0:c1) -> (scale, zero) of group gi
__global__ void group_params_kernel(int64_t m, int64_t n, const float *W, int64_t c0, int64_t c1, int gi,
                                    int ngroups, int bits, int sym, float *scale, uint8_t *zero) {
    const int64_t i = (int64_t)blockIdx.x * (blockDim.x / 32) + threadIdx.x / 32;
    const int lane = threadIdx.x & 31;
    if (i >= m) return;
    float mn = 0.f, mx = 0.f;
    for (int64_t c = c0 + lane; c < c1; c += 32) {
        const float w = W[i * n + c];
        mn = fminf(mn, w);
        mx = fmaxf(mx, w);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        mn = fminf(mn, __shfl_xor_sync(0xffffffffu, mn, o));
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    }
    if (lane == 0) {
        float sc, zr;
        grid_params(mn, mx, bits, sym, sc, zr);
        scale[i * ngroups + gi] = sc;
        zero[i * ngroups + gi] = (uint8_t)zr;
    }
}

struct QArgs {
    int64_t m, n, bs;
    int kb;
    float *W;
    const float *U;
    int g, ngroups, bits, sym;
    float *scale;
    uint8_t *zero;
    uint8_t *codes;
    int64_t ncb;
    float *Et;
    int64_t ldet;          // leading dimension of Et (all rows of the layer)
    int *status;
};

// Column-serial quantize + in-block OBS propagation for block [bs, bs + kb).
// A CTA takes QB_ROWS rows and B/32 warps: warp w keeps columns
// [32w, 32w + 32) of the CTA's rows in registers (lane = row).  Phase s: warp
// s quantizes its 32 columns one after the other, feeding each column's error
// to its later columns at once, and publishes the 32 errors of every row;
// then every warp w > s applies them to its columns, column by column in
// order, so each weight sees exactly the updates of the plain column loop.
// U's B x B diagonal block is staged once in shared memory (rows padded to
// keep float4 reads aligned).  G > 0: group parameters are computed at every
// G-th column (a multiple of 32) from the current weights, with the min / max
// of the group's sub-blocks gathered through shared memory; G = 0: they were
// computed before the block.
constexpr int QB_ROWS = 32;
}  // namespace
constexpr int kGSplit = 8;   // K slices of the next block's G product
namespace {

template <int B, int G>
__global__ void __launch_bounds__(B) quant_block_kernel(const QArgs a) {
    constexpr int NW = B / 32;            // warps = sub-blocks
    constexpr int UP = B + 4;             // U row pitch (floats)
    extern __shared__ __align__(16) float qsm[];
    float *Us = qsm;                      // B x UP: U[j][k] for j < k, else 0
    float *invd = Us + B * UP;            // B
    float *Es = invd + B;                 // QB_ROWS x 33: errors of the current sub-block
    float *mm = Es + QB_ROWS * 33;        // 2 x NW x QB_ROWS: group min / max partials
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int kb = a.kb;
    if ((a.n & 3) == 0 && kb == B) {
        // (unrolled so that several loads are in flight per thread)
#pragma unroll 8
        for (int idx = threadIdx.x; idx < B * B / 4; idx += blockDim.x) {
            const int j = (idx * 4) / B, k = (idx * 4) % B;
            const float4 v = *reinterpret_cast<const float4 *>(a.U + (a.bs + j) * a.n + a.bs + k);
            float *d = Us + j * UP + k;
            d[0] = (k + 0 > j) ? v.x : 0.f;
            d[1] = (k + 1 > j) ? v.y : 0.f;
            d[2] = (k + 2 > j) ? v.z : 0.f;
            d[3] = (k + 3 > j) ? v.w : 0.f;
        }
    } else {
        for (int idx = threadIdx.x; idx < B * B; idx += blockDim.x) {
            const int j = idx / B, k = idx % B;
            Us[j * UP + k] = (j < kb && k < kb && k > j) ? a.U[(a.bs + j) * a.n + a.bs + k] : 0.f;
        }
    }
    for (int j = threadIdx.x; j < B; j += blockDim.x)
        invd[j] = (j < kb) ? 1.f / a.U[(a.bs + j) * a.n + a.bs + j] : 0.f;

    const int64_t i = (int64_t)blockIdx.x * QB_ROWS + lane;   // this lane's row
    const bool live = i < a.m;
    const int c0 = warp * 32;                                   // this warp's first column
    float r[32];
    {
        const float *wrow = a.W + (live ? i : 0) * a.n + a.bs + c0;
        if ((a.n & 3) == 0 && c0 + 32 <= kb) {
#pragma unroll
            for (int c = 0; c < 32; c += 4) {
                const float4 v = live ? *reinterpret_cast<const float4 *>(wrow + c) : make_float4(0.f, 0.f, 0.f, 0.f);
                r[c] = v.x; r[c + 1] = v.y; r[c + 2] = v.z; r[c + 3] = v.w;
            }
        } else {
#pragma unroll
            for (int c = 0; c < 32; ++c) r[c] = (live && c0 + c < kb) ? wrow[c] : 0.f;
        }
    }
    float sc = 1.f, zr = 0.f;
    if (G == 0 && live) {
        const int gi = (int)(a.bs / a.g);
        sc = a.scale[i * a.ngroups + gi];
        zr = (float)a.zero[i * a.ngroups + gi];
    }
    __syncthreads();

    const float maxq = (float)((1 << a.bits) - 1);
    bool bad = false;
#pragma unroll 1
    for (int s = 0; s < NW && s * 32 < kb; ++s) {
        if (G > 0 && ((s * 32) % (G > 0 ? G : 1)) == 0) {
            // min / max of the group's columns (sub-blocks s .. s + G/32 - 1)
            constexpr int GS = (G > 0 ? G : 32) / 32;
            if (warp >= s && warp < s + GS) {
                float mn = 0.f, mx = 0.f;
#pragma unroll
                for (int c = 0; c < 32; ++c)
                    if (c0 + c < kb) {
                        mn = fminf(mn, r[c]);
                        mx = fmaxf(mx, r[c]);
                    }
                mm[warp * QB_ROWS + lane] = mn;
                mm[(NW + warp) * QB_ROWS + lane] = mx;
            }
            __syncthreads();
            if (warp == s) {
                float mn = 0.f, mx = 0.f;
                for (int w = s; w < s + GS && w < NW; ++w) {
                    mn = fminf(mn, mm[w * QB_ROWS + lane]);
                    mx = fmaxf(mx, mm[(NW + w) * QB_ROWS + lane]);
                }
                grid_params(mn, mx, a.bits, a.sym, sc, zr);
                if (live) {
                    const int gi = (int)((a.bs + s * 32) / a.g);
                    a.scale[i * a.ngroups + gi] = sc;
                    a.zero[i * a.ngroups + gi] = (uint8_t)zr;
                }
                // the next sub-blocks of the same group quantize with these parameters
                mm[lane] = sc;
                mm[QB_ROWS + lane] = zr;
            }
            __syncthreads();
            if (warp > s && warp < s + GS) {
                sc = mm[lane];
                zr = mm[QB_ROWS + lane];
            }
        }
        if (warp == s) {
            uint32_t packed[4] = {0u, 0u, 0u, 0u};
            // rint(w / sc) through the reciprocal: x = w * rn(1/sc) is within
            // 3 * 2^-24 |w / sc| of the quotient and of its IEEE rounding, so
            // where x is farther than 4 * 2^-24 |x| from every half-integer
            // both round to the same integer; nearer (and for non-finite
            // values) the IEEE division decides, so the code is the one of
            // rint(w / sc) in every case and the chain from one column's
            // error to the next column's code avoids the division
            const float rcp = __frcp_rn(sc);
#pragma unroll
            for (int jj = 0; jj < 32; ++jj) {
                const int j = c0 + jj;
                float err = 0.f;
                uint32_t qi = 0;
                if (j < kb) {
                    const float w = r[jj];
                    bad |= !isfinite(w);
                    const float x = __fmul_rn(w, rcp);
                    float qx = rintf(x);
                    const float gap = 0.5f - fabsf(x - qx);
                    if (!(gap > 2.4e-7f * fabsf(x) + 1e-30f)) qx = rintf(w / sc);
                    float q = qx + zr;
                    q = fminf(fmaxf(q, 0.f), maxq);
                    const float dq = sc * (q - zr);
                    err = (w - dq) * invd[j];
                    r[jj] = dq;
                    qi = (uint32_t)q;
#pragma unroll
                    for (int kk = jj + 1; kk < 32; ++kk) r[kk] = fmaf(-err, Us[j * UP + c0 + kk], r[kk]);
                }
                Es[lane * 33 + jj] = err;
                if (live && j < kb) a.Et[(int64_t)j * a.ldet + i] = err;
                packed[jj >> 3] |= (qi & 15u) << ((jj & 7) * 4);
            }
            if (live) {
                uint8_t *crow = a.codes + i * a.ncb + (a.bs + c0) / 2;
                if (c0 + 32 <= kb && (((uintptr_t)crow) & 15) == 0) {
                    *reinterpret_cast<uint4 *>(crow) = make_uint4(packed[0], packed[1], packed[2], packed[3]);
                } else {
                    for (int jj = 0; jj < 32 && c0 + jj < kb; jj += 2)
                        crow[jj / 2] = (uint8_t)((packed[jj >> 3] >> ((jj & 7) * 4)) & 0xFFu);
                }
            }
        }
        __syncthreads();
        if (warp > s) {
            // the 32 errors of sub-block s, column by column in order (the
            // column loop stays rolled: the kernel's code then fits the
            // instruction cache)
#pragma unroll 1
            for (int jj = 0; jj < 32; ++jj) {
                const float ej = Es[lane * 33 + jj];
                const float *urow = Us + (s * 32 + jj) * UP + c0;
#pragma unroll
                for (int c = 0; c < 32; c += 4) {
                    const float4 u = *reinterpret_cast<const float4 *>(urow + c);
                    r[c] = fmaf(-ej, u.x, r[c]);
                    r[c + 1] = fmaf(-ej, u.y, r[c + 1]);
                    r[c + 2] = fmaf(-ej, u.z, r[c + 2]);
                    r[c + 3] = fmaf(-ej, u.w, r[c + 3]);
                }
            }
        }
        __syncthreads();
    }
    if (live) {
        float *wout = a.W + i * a.n + a.bs + c0;
        if ((a.n & 3) == 0 && c0 + 32 <= kb) {
#pragma unroll
            for (int c = 0; c < 32; c += 4) *reinterpret_cast<float4 *>(wout + c) = make_float4(r[c], r[c + 1], r[c + 2], r[c + 3]);
        } else {
#pragma unroll
            for (int c = 0; c < 32; ++c)
                if (c0 + c < kb) wout[c] = r[c];
        }
    }
    if (bad) atomicOr(a.status, ST_NONFINITE);
}

// The same column-serial quantize + in-block OBS as quant_block_kernel, with
// the phases pipelined: warp w applies sub-block s's errors in chunks of 8
// columns as soon as warp s has published them (a per-warp progress flag in
// shared memory) and starts its own chain right after, instead of every warp
// waiting at a CTA barrier for the slowest one after every phase.  Each
// weight still receives exactly the updates of the plain column loop in the
// same order (sub-blocks in order, columns in order), so the results are the
// kernel's above bit for bit.  U's diagonal block is staged as its 32 x 32
// blocks on or above the diagonal only (row pitch 36 keeps float4 reads
// aligned), which leaves room for three CTAs per SM beside the error
// buffers.  Group parameters at the block start (G = B) or before it (G = 0).
template <int B>
struct QPipe {
    static constexpr int NW = B / 32;
    static constexpr int NSLOT = NW * (NW + 1) / 2;
    static constexpr int P = 36;
    static constexpr int NBUF = NW > 1 ? NW - 1 : 1;
    static constexpr size_t floats = (size_t)NSLOT * 32 * P + B + (size_t)NBUF * QB_ROWS * 33 + 2 * NW * QB_ROWS + NW;
};

// slot of the 32 x 32 block (s, w), s <= w, in row-major order of the upper triangle
__device__ __forceinline__ int qslot(int s, int w, int nw) { return s * nw - s * (s - 1) / 2 + (w - s); }

template <int B, int G>
__global__ void __launch_bounds__(B) quant_block_pipe_kernel(const QArgs a) {
    static_assert(G == 0 || G == B, "group parameters at the block start or before it");
    using QP = QPipe<B>;
    constexpr int NW = QP::NW, P = QP::P;
    extern __shared__ __align__(16) float qsm[];
    float *Ut = qsm;                                   // NSLOT x 32 x P
    float *invd = Ut + QP::NSLOT * 32 * P;             // B
    float *Es = invd + B;                              // NBUF x QB_ROWS x 33
    float *mm = Es + QP::NBUF * QB_ROWS * 33;          // 2 x NW x QB_ROWS
    volatile int *flags = reinterpret_cast<volatile int *>(mm + 2 * NW * QB_ROWS);   // NW
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int kb = a.kb;
    if (threadIdx.x < NW) flags[threadIdx.x] = 0;
    // U's blocks on or above the diagonal: slot (s, w) row jj col c holds
    // U[bs + 32 s + jj][bs + 32 w + c] where that lies strictly above the
    // diagonal of the block, else 0
    for (int idx = threadIdx.x; idx < QP::NSLOT * 32 * 8; idx += blockDim.x) {
        const int slot = idx / 256, rr = (idx / 8) % 32, c4 = (idx % 8) * 4;
        int s = 0, w = 0;
        for (int t = 0, k = 0; t < NW; ++t)
            for (int u = t; u < NW; ++u, ++k)
                if (k == slot) { s = t; w = u; }
        const int j = s * 32 + rr;
        float v[4];
        if ((a.n & 3) == 0 && kb == B) {
            const float4 q = *reinterpret_cast<const float4 *>(a.U + (a.bs + j) * a.n + a.bs + w * 32 + c4);
            v[0] = q.x; v[1] = q.y; v[2] = q.z; v[3] = q.w;
        } else {
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const int k = w * 32 + c4 + e;
                v[e] = (j < kb && k < kb) ? a.U[(a.bs + j) * a.n + a.bs + k] : 0.f;
            }
        }
        float *d = Ut + slot * 32 * P + rr * P + c4;
#pragma unroll
        for (int e = 0; e < 4; ++e) d[e] = (s < w || c4 + e > rr) ? v[e] : 0.f;
    }
    for (int j = threadIdx.x; j < B; j += blockDim.x)
        invd[j] = (j < kb) ? 1.f / a.U[(a.bs + j) * a.n + a.bs + j] : 0.f;

    const int64_t i = (int64_t)blockIdx.x * QB_ROWS + lane;   // this lane's row
    const bool live = i < a.m;
    const int c0 = warp * 32;                                   // this warp's first column
    float r[32];
    {
        const float *wrow = a.W + (live ? i : 0) * a.n + a.bs + c0;
        if ((a.n & 3) == 0 && c0 + 32 <= kb) {
#pragma unroll
            for (int c = 0; c < 32; c += 4) {
                const float4 v = live ? *reinterpret_cast<const float4 *>(wrow + c) : make_float4(0.f, 0.f, 0.f, 0.f);
                r[c] = v.x; r[c + 1] = v.y; r[c + 2] = v.z; r[c + 3] = v.w;
            }
        } else {
#pragma unroll
            for (int c = 0; c < 32; ++c) r[c] = (live && c0 + c < kb) ? wrow[c] : 0.f;
        }
    }
    float sc = 1.f, zr = 0.f;
    if (G == 0 && live) {
        const int gi = (int)(a.bs / a.g);
        sc = a.scale[i * a.ngroups + gi];
        zr = (float)a.zero[i * a.ngroups + gi];
    }
    if (G == B) {
        // one group: min / max over the block's columns from every warp
        float mn = 0.f, mx = 0.f;
#pragma unroll
        for (int c = 0; c < 32; ++c)
            if (c0 + c < kb) {
                mn = fminf(mn, r[c]);
                mx = fmaxf(mx, r[c]);
            }
        mm[warp * QB_ROWS + lane] = mn;
        mm[(NW + warp) * QB_ROWS + lane] = mx;
    }
    __syncthreads();
    if (G == B) {
        if (warp == 0) {
            float mn = 0.f, mx = 0.f;
            for (int w = 0; w < NW; ++w) {
                mn = fminf(mn, mm[w * QB_ROWS + lane]);
                mx = fmaxf(mx, mm[(NW + w) * QB_ROWS + lane]);
            }
            grid_params(mn, mx, a.bits, a.sym, sc, zr);
            if (live) {
                const int gi = (int)(a.bs / a.g);
                a.scale[i * a.ngroups + gi] = sc;
                a.zero[i * a.ngroups + gi] = (uint8_t)zr;
            }
            // (each lane overwrites only partials it has already read)
            mm[lane] = sc;
            mm[QB_ROWS + lane] = zr;
        }
        __syncthreads();
        sc = mm[lane];
        zr = mm[QB_ROWS + lane];
    }

    const float maxq = (float)((1 << a.bits) - 1);
    bool bad = false, late = false;
    if (c0 < kb) {
        // the errors of every earlier sub-block, chunk by chunk as published
#pragma unroll 1
        for (int s = 0; s < warp; ++s) {
            const float *E = Es + s * QB_ROWS * 33;
#pragma unroll 1
            for (int ch = 0; ch < 4; ++ch) {
                if (lane == 0) {
                    uint32_t it = 0;
                    while (flags[s] < ch + 1) {
                        if (++it > (1u << 22)) {
                            late = true;
                            break;
                        }
                        __nanosleep(32);
                    }
                }
                __syncwarp();
                __threadfence_block();
#pragma unroll 1
                for (int jj = ch * 8; jj < ch * 8 + 8; ++jj) {
                    const float ej = E[lane * 33 + jj];
                    const float *urow = Ut + qslot(s, warp, NW) * 32 * P + jj * P;
#pragma unroll
                    for (int c = 0; c < 32; c += 4) {
                        const float4 u = *reinterpret_cast<const float4 *>(urow + c);
                        r[c] = fmaf(-ej, u.x, r[c]);
                        r[c + 1] = fmaf(-ej, u.y, r[c + 1]);
                        r[c + 2] = fmaf(-ej, u.z, r[c + 2]);
                        r[c + 3] = fmaf(-ej, u.w, r[c + 3]);
                    }
                }
            }
        }
        // this warp's own columns, one after the other
        const bool publish = c0 + 32 < kb && warp < NW - 1;
        float *Eo = Es + (warp < QP::NBUF ? warp : 0) * QB_ROWS * 33;
        const float *ud = Ut + qslot(warp, warp, NW) * 32 * P;
        uint32_t packed[4] = {0u, 0u, 0u, 0u};
        // rint(w / sc) through the reciprocal, as in quant_block_kernel
        const float rcp = __frcp_rn(sc);
#pragma unroll
        for (int jj = 0; jj < 32; ++jj) {
            const int j = c0 + jj;
            float err = 0.f;
            uint32_t qi = 0;
            if (j < kb) {
                const float w = r[jj];
                bad |= !isfinite(w);
                const float x = __fmul_rn(w, rcp);
                float qx = rintf(x);
                const float gap = 0.5f - fabsf(x - qx);
                if (!(gap > 2.4e-7f * fabsf(x) + 1e-30f)) qx = rintf(w / sc);
                float q = qx + zr;
                q = fminf(fmaxf(q, 0.f), maxq);
                const float dq = sc * (q - zr);
                err = (w - dq) * invd[j];
                r[jj] = dq;
                qi = (uint32_t)q;
#pragma unroll
                for (int kk = jj + 1; kk < 32; ++kk) r[kk] = fmaf(-err, ud[jj * P + kk], r[kk]);
            }
            if (publish) Eo[lane * 33 + jj] = err;
            if (live && j < kb) a.Et[(int64_t)j * a.ldet + i] = err;
            packed[jj >> 3] |= (qi & 15u) << ((jj & 7) * 4);
            if (publish && (jj & 7) == 7) {
                __syncwarp();
                if (lane == 0) {
                    __threadfence_block();
                    flags[warp] = (jj >> 3) + 1;
                }
            }
        }
        if (live) {
            uint8_t *crow = a.codes + i * a.ncb + (a.bs + c0) / 2;
            if (c0 + 32 <= kb && (((uintptr_t)crow) & 15) == 0) {
                *reinterpret_cast<uint4 *>(crow) = make_uint4(packed[0], packed[1], packed[2], packed[3]);
            } else {
                for (int jj = 0; jj < 32 && c0 + jj < kb; jj += 2)
                    crow[jj / 2] = (uint8_t)((packed[jj >> 3] >> ((jj & 7) * 4)) & 0xFFu);
            }
        }
        if (live) {
            float *wout = a.W + i * a.n + a.bs + c0;
            if ((a.n & 3) == 0 && c0 + 32 <= kb) {
#pragma unroll
                for (int c = 0; c < 32; c += 4)
                    *reinterpret_cast<float4 *>(wout + c) = make_float4(r[c], r[c + 1], r[c + 2], r[c + 3]);
            } else {
#pragma unroll
                for (int c = 0; c < 32; ++c)
                    if (c0 + c < kb) wout[c] = r[c];
            }
        }
    }
    late = __shfl_sync(0xffffffffu, late ? 1 : 0, 0) != 0;
    if (bad) atomicOr(a.status, ST_NONFINITE);
    if (late && lane == 0) atomicOr(a.status, ST_TIMEOUT);
}

// One optimizer step on the free columns c0..n-1; the applied step is also
// accumulated into D (the optimizer displacement) when D is given.
__global__ void adam_kernel(int64_t m, int64_t r, int64_t n, int64_t c0, const float *G, float *W, float *mA,
                            float *vA, float *D, float lr, float b1, float b2, float eps, float bc1, float bc2,
                            int sgd) {
    const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= m * r) return;
    const int64_t i = idx / r, c = idx % r;
    const int64_t w = i * n + c0 + c;
    const float g = G[idx];
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
    if (D) D[w] -= step;
}

// lambda = damp * mean(diag(Hbar) with dead channels counted as 1), the same
// fixed-order fp64 reduction as the preparation step.
__global__ void lambda_kernel(int64_t n, const float *Hbar, const uint8_t *dead, float damp, float *lam_out) {
    __shared__ double red[1024];
    double s = 0.0;
    for (int64_t j = threadIdx.x; j < n; j += blockDim.x)
        s += (dead && dead[j]) ? 1.0 : (double)Hbar[j * n + j];
    red[threadIdx.x] = s;
    __syncthreads();
    for (int w = blockDim.x / 2; w > 0; w >>= 1) {
        if ((int)threadIdx.x < w) red[threadIdx.x] += red[threadIdx.x + w];
        __syncthreads();
    }
    if (threadIdx.x == 0) *lam_out = (float)((double)damp * (red[0] / (double)n));
}

__global__ void feff_kernel(int64_t count, const float *F, const float *Fn, float alpha, float *out) {
    const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (idx < count) out[idx] = alpha * F[idx] + (1.f - alpha) * Fn[idx];
}

template <typename TO>
__global__ void copy_cols_kernel(int64_t m, int64_t n, int64_t c0, int64_t c1, const float *W, TO *out) {
    const int64_t w = c1 - c0;
    const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= m * w) return;
    const int64_t i = idx / w, c = c0 + idx % w;
    if constexpr (sizeof(TO) == 2) out[i * n + c] = __float2bfloat16_rn(W[i * n + c]);
    else out[i * n + c] = W[i * n + c];
}

template <typename TW>
__global__ void diff_kernel(int64_t count, const float *A, const TW *W0, float *out) {
    const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (idx < count) out[idx] = A[idx] - load_as_float(W0, idx);
}

// 1/2 sum X1 .* X2 in fp64, two fixed-order stages
constexpr int RED_BLOCKS = 512;
__global__ void dot_partial_kernel(int64_t count, const float *X1, const float *X2, double *part) {
    __shared__ double red[256];
    double s = 0.0;
    for (int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; idx < count; idx += (int64_t)gridDim.x * blockDim.x)
        s += (double)X1[idx] * (double)X2[idx];
    red[threadIdx.x] = s;
    __syncthreads();
    for (int w = 128; w > 0; w >>= 1) {
        if ((int)threadIdx.x < w) red[threadIdx.x] += red[threadIdx.x + w];
        __syncthreads();
    }
    if (threadIdx.x == 0) part[blockIdx.x] = red[0];
}
__global__ void dot_final_kernel(const double *part, int nparts, float *out) {
    __shared__ double red[RED_BLOCKS];
    red[threadIdx.x] = threadIdx.x < nparts ? part[threadIdx.x] : 0.0;
    __syncthreads();
    for (int w = RED_BLOCKS / 2; w > 0; w >>= 1) {
        if ((int)threadIdx.x < w) red[threadIdx.x] += red[threadIdx.x + w];
        __syncthreads();
    }
    if (threadIdx.x == 0) *out = (float)(0.5 * red[0]);
}

inline unsigned blocks_for(int64_t count, int threads = 256) { return (unsigned)((count + threads - 1) / threads); }

template <int B, int G>
realq_status_t launch_qb(cudaStream_t s, const QArgs &qa) {
    const size_t smem = (size_t)(B * (B + 4) + B + QB_ROWS * 33 + 2 * (B / 32) * QB_ROWS) * sizeof(float);
    REALQ_TRY(set_smem_limit(reinterpret_cast<const void *>(quant_block_kernel<B, G>), (int)smem));
    {
        Launch L("quant_block", s);
        quant_block_kernel<B, G><<<ceil_div(qa.m, QB_ROWS), B, smem, s>>>(qa);
    }
    return check_launch("quant_block");
}

int g_quant_kernel = 0;   // 0: the barrier-phased quantizer (default), 1: the pipelined one where it applies
}  // namespace

void quant_set_kernel(int mode) { g_quant_kernel = mode; }

namespace {

template <int B, int G>
realq_status_t launch_qb_pipe(cudaStream_t s, const QArgs &qa) {
    const size_t smem = QPipe<B>::floats * sizeof(float);
    REALQ_TRY(set_smem_limit(reinterpret_cast<const void *>(quant_block_pipe_kernel<B, G>), (int)smem));
    {
        Launch L("quant_block", s);
        quant_block_pipe_kernel<B, G><<<ceil_div(qa.m, QB_ROWS), B, smem, s>>>(qa);
    }
    return check_launch("quant_block");
}

template <int B>
realq_status_t launch_qb_g(cudaStream_t s, const QArgs &qa, int Gk) {
    if (g_quant_kernel == 1 && Gk == 0) return launch_qb_pipe<B, 0>(s, qa);
    if (g_quant_kernel == 1 && Gk == B) return launch_qb_pipe<B, B>(s, qa);
    if (Gk == 0) return launch_qb<B, 0>(s, qa);
    if (Gk == B) return launch_qb<B, B>(s, qa);
    if (B >= 64 && Gk == B / 2) return launch_qb<B, (B >= 64 ? B / 2 : B)>(s, qa);
    if (B >= 128 && Gk == B / 4) return launch_qb<B, (B >= 128 ? B / 4 : B)>(s, qa);
    return fail(REALQ_ERR_UNSUPPORTED, "group size %d inside block %d", Gk, B);
}

}  // namespace

// Workspace of a sweep.  With Block-GD on shapes the tensor-core path can
// address (m, n multiples of 4), the gradient GEMMs run as tf32x3 on tcgen05
// and need hi / lo planes of the displacement, H̄, F and P^T; otherwise the
// fp32 SIMT path needs P, G (and F_eff).  block = 0: Block-GD only (literal
// gradient form, SIMT).
// The lazy batch update runs on the tensor cores (tf32x3) when both GEMM
// operands take the tensor-core path's shapes and the block is a whole
// number of 32-wide K slices.
static bool trail_tc_eligible(int64_t m, int64_t n, int block) {
    return (block == 32 || block == 64 || block == 128) && tc_gemm_eligible(m, n);
}

size_t sweep_ws_bytes(int64_t m, int64_t n, int block, int has_bgd, int has_fnext, int has_dbar, int rgroups,
                      int nmb, int64_t tmb) {
    const size_t mn = align_up((size_t)m * n * sizeof(float));
    const size_t nn = align_up((size_t)n * n * sizeof(float));
    size_t b = align_up(sizeof(int)) + align_up(sizeof(float)) + align_up((size_t)block * m * sizeof(float));
    if (trail_tc_eligible(m, n, block))
        b += 2 * align_up((size_t)block * m * sizeof(float)) + 2 * align_up((size_t)block * n * sizeof(float));
    if (rgroups > 0) b += align_up((size_t)rgroups * sizeof(float));
    if (has_bgd) {
        if (block > 0 && tc_gemm_eligible(m, n)) {
            b += 5 * mn + 2 * nn + 2 * align_up((size_t)m * m * sizeof(float));
            b += align_up((size_t)kGSplit * m * block * sizeof(float));
            b += align_up((size_t)(2 * m + 2 * n) * sizeof(float));   // row scales of the f16 planes
            if (rgroups > 0) b += 2 * mn + 4 * (size_t)rgroups * nn;
            if (nmb > 0) b += (rgroups > 0 ? 0 : 2 * mn) + 2 * (size_t)nmb * nn;
            if (tmb > 0) {
                // ΔW planes, the mini-batch in fp32 both ways (exact in tf32:
                // no low plane), Δ (then kappa), the clipped residual's planes
                // (then the gradient factor's), Z and the gradient
                const size_t tn = align_up((size_t)tmb * n * sizeof(float));
                const size_t tm = align_up((size_t)tmb * m * sizeof(float));
                b += 3 * mn + 2 * tn + 4 * tm;
            }
        } else {
            b += 2 * mn;
            if (has_fnext) b += align_up((size_t)m * m * sizeof(float));
        }
        if (has_dbar) b += mn;
    }
    return b;
}

void sweep_carve(SweepPlan &p, void *ws, int has_bgd, int has_fnext, int has_dbar) {
    Carve cv(ws);
    const size_t mn = (size_t)p.m * p.n;
    p.status = cv.take<int>(1);
    p.lam = cv.take<float>(1);
    p.Et = cv.take<float>((size_t)p.block * p.m);
    p.trail_tc = trail_tc_eligible(p.m, p.n, p.block) ? 1 : 0;
    p.trail_maps = 0;
    p.Eh = p.El = p.UPh = p.UPl = nullptr;
    if (p.trail_tc) {
        p.Eh = cv.take<float>((size_t)p.block * p.m);
        p.El = cv.take<float>((size_t)p.block * p.m);
        p.UPh = cv.take<float>((size_t)p.block * p.n);
        p.UPl = cv.take<float>((size_t)p.block * p.n);
    }
    p.P = p.G = p.Feff = p.R0 = nullptr;
    p.Sh = p.Sl = p.Hh = p.Hl = p.Fh = p.Fl = p.Pth = p.Ptl = p.M = nullptr;
    p.f16 = 0;
    p.scS = p.scF = p.scH = p.scP = nullptr;
    p.HGh = p.HGl = p.GGh = p.GGl = p.DWh = p.DWl = p.MBh = p.MBl = nullptr;
    p.lam_g = p.grouped ? cv.take<float>((size_t)p.rgroups) : nullptr;
    p.step_c = p.n;
    p.tc = 0;
    if (has_bgd) {
        if (p.block > 0 && tc_gemm_eligible(p.m, p.n)) {
            p.tc = 1;
            p.Sh = cv.take<float>(mn);
            p.Sl = cv.take<float>(mn);
            p.M = cv.take<float>(mn);
            p.Pth = cv.take<float>(mn);
            p.Ptl = cv.take<float>(mn);
            p.Hh = cv.take<float>((size_t)p.n * p.n);
            p.Hl = cv.take<float>((size_t)p.n * p.n);
            p.Fh = cv.take<float>((size_t)p.m * p.m);
            p.Fl = cv.take<float>((size_t)p.m * p.m);
            p.Gpart = cv.take<float>((size_t)kGSplit * p.m * p.block);
            float *scl = cv.take<float>((size_t)(2 * p.m + 2 * p.n));
            // the plain Block-GD products as f16x3 (fp16 planes with row
            // scales): twice the tf32 rate at the same accuracy; the
            // row-grouped, mini-batch and token forms keep tf32 planes
            p.f16 = bgd_products() == 1 && !p.grouped && p.nmb == 0 && p.tmb == 0 && p.m % 8 == 0 && p.n % 8 == 0 &&
                    p.block % 8 == 0;
            p.scS = scl;
            p.scF = scl + p.m;
            p.scH = scl + 2 * p.m;
            p.scP = scl + 2 * p.m + p.n;
            if (p.nmb > 0) {
                p.MBh = cv.take<float>((size_t)p.nmb * p.n * p.n);
                p.MBl = cv.take<float>((size_t)p.nmb * p.n * p.n);
                if (!p.grouped) {
                    p.DWh = cv.take<float>(mn);
                    p.DWl = cv.take<float>(mn);
                }
            }
            if (p.tmb > 0) {
                p.DWh = cv.take<float>(mn);
                p.DWl = cv.take<float>(mn);
                p.Gc = cv.take<float>(mn);
                p.Xf = cv.take<float>((size_t)p.tmb * p.n);
                p.XfT = cv.take<float>((size_t)p.tmb * p.n);
                p.Dk = cv.take<float>((size_t)p.tmb * p.m);
                p.Yh = cv.take<float>((size_t)p.tmb * p.m);
                p.Yl = cv.take<float>((size_t)p.tmb * p.m);
                p.Zk = cv.take<float>((size_t)p.tmb * p.m);
            }
            if (p.grouped) {
                p.DWh = cv.take<float>(mn);
                p.DWl = cv.take<float>(mn);
                const size_t gnn = (size_t)p.rgroups * p.n * p.n;
                p.HGh = cv.take<float>(gnn);
                p.HGl = cv.take<float>(gnn);
                p.GGh = cv.take<float>(gnn);
                p.GGl = cv.take<float>(gnn);
            }
        } else {
            p.P = cv.take<float>(mn);
            p.G = cv.take<float>(mn);
            if (has_fnext) p.Feff = cv.take<float>((size_t)p.m * p.m);
        }
        if (has_dbar) p.R0 = cv.take<float>(mn);
    }
}

realq_status_t sweep_init(cudaStream_t s, SweepPlan &p) {
    const int64_t mn = p.m * p.n;
    // per row group: the group's dead channels (one group: dead)
    for (int gr = 0; gr < p.rgroups; ++gr) {
        const int64_t row0 = gr * p.rg_rows, rows = std::min<int64_t>(p.rg_rows, p.m - row0);
        if (rows <= 0) break;
        const uint8_t *dd = p.grouped ? p.dead_g + (size_t)gr * p.n : p.dead;
        const int64_t cnt = rows * p.n;
        Launch L("init_work", s);
        if (p.w_dtype == REALQ_BF16)
            init_work_kernel<<<blocks_for(cnt), 256, 0, s>>>(
                rows, p.n, static_cast<const __nv_bfloat16 *>(p.W0) + row0 * p.n, dd, p.W + row0 * p.n);
        else
            init_work_kernel<<<blocks_for(cnt), 256, 0, s>>>(rows, p.n, static_cast<const float *>(p.W0) + row0 * p.n,
                                                             dd, p.W + row0 * p.n);
    }
    REALQ_TRY(check_launch("init_work"));
    if (p.bgd_steps > 0) {
        if (p.optimizer == REALQ_OPT_ADAM) {
            REALQ_CUDA_TRY(cudaMemsetAsync(p.adam_m, 0, (size_t)mn * sizeof(float), s));
            REALQ_CUDA_TRY(cudaMemsetAsync(p.adam_v, 0, (size_t)mn * sizeof(float), s));
        }
        if (p.disp) REALQ_CUDA_TRY(cudaMemsetAsync(p.disp, 0, (size_t)mn * sizeof(float), s));
        *p.adam_t = 0;
    }
    return REALQ_OK;
}

static realq_status_t compute_r0(cudaStream_t s, SweepPlan &p) {
    GemmArgs g{};
    g.M = p.m; g.N = p.n; g.K = p.n;
    g.A = p.W0; g.lda = p.n;
    g.B = p.Dbar; g.ldb = p.n;
    g.C = p.R0; g.ldc = p.n;
    g.alpha = 1.f;
    return gemm_f32(s, p.w_dtype == REALQ_BF16 ? A_ROW_BF16 : A_ROW, EPI_STORE, g, "bgd_r0_gemm");
}

static realq_status_t fisher_for(cudaStream_t s, SweepPlan &p, float alpha, const float **Fuse) {
    *Fuse = p.F;
    if (p.F_next == nullptr || alpha == 1.f) return REALQ_OK;
    if (alpha == 0.f) {
        *Fuse = p.F_next;
        return REALQ_OK;
    }
    {
        Launch L("fisher_blend", s);
        feff_kernel<<<blocks_for(p.m * p.m), 256, 0, s>>>(p.m * p.m, p.F, p.F_next, alpha, p.Feff);
    }
    *Fuse = p.Feff;
    return check_launch("fisher_blend");
}

// One Block-GD step on columns c0..n-1.  identity = 1 (inside the sweep, right
// after the lazy batch update): P from the optimizer displacement through the
// OBS stationarity identity; identity = 0: P = (W - W0) Hbar (+ W0 Dbar).
static realq_status_t bgd_one(cudaStream_t s, SweepPlan &p, int64_t c0, const float *Fuse, int identity) {
    const int64_t r = p.n - c0;
    GemmArgs g{};
    g.M = p.m; g.N = r;
    g.C = p.P; g.ldc = r;
    g.R = p.R0 ? p.R0 + c0 : nullptr; g.ldr = p.n;
    g.alpha = 1.f;
    if (identity) {
        // columns of the first block never received a step: skip them in K
        const int64_t k0 = std::min<int64_t>(p.block, c0);
        g.K = p.n - k0;
        g.A = p.disp + k0; g.lda = p.n;
        g.B = p.Hbar + k0 * p.n + c0; g.ldb = p.n;
        g.Ad = p.disp; g.Wc = p.W; g.W0c = p.W0; g.w0_bf16 = p.w_dtype == REALQ_BF16;
        g.dead = p.dead; g.lam = p.lam; g.col0 = c0; g.ldw = p.n;
        REALQ_TRY(gemm_f32(s, A_ROW, EPI_BGD_P, g, "bgd_p_gemm"));
    } else {
        g.K = p.n;
        g.A = p.W; g.lda = p.n;
        g.Y = p.W0; g.ldy = p.n;
        g.B = p.Hbar + c0; g.ldb = p.n;
        REALQ_TRY(gemm_f32(s, p.w_dtype == REALQ_BF16 ? A_DIFF_BF16 : A_DIFF_F32, p.R0 ? EPI_BIAS : EPI_STORE, g,
                           "bgd_p_gemm"));
    }
    GemmArgs h{};
    h.M = p.m; h.N = r; h.K = p.m;
    h.A = Fuse; h.lda = p.m;
    h.B = p.P; h.ldb = r;
    h.C = p.G; h.ldc = r;
    h.alpha = 1.f;
    REALQ_TRY(gemm_f32(s, A_ROW, EPI_STORE, h, "bgd_g_gemm"));
    const int64_t t = ++(*p.adam_t);
    const double bc1 = 1.0 - std::pow((double)p.beta1, (double)t);
    const double bc2 = 1.0 - std::pow((double)p.beta2, (double)t);
    {
        Launch L("bgd_adam", s);
        adam_kernel<<<blocks_for(p.m * r), 256, 0, s>>>(p.m, r, p.n, c0, p.G, p.W, p.adam_m, p.adam_v, p.disp, p.lr,
                                                         p.beta1, p.beta2, p.eps, (float)bc1, (float)bc2,
                                                         p.optimizer == REALQ_OPT_SGD);
    }
    return check_launch("bgd_adam");
}

// The fp16 planes of the f16x3 products, in the regions of the tf32 ones
// (each region holds m n, n n or m m floats: room for both fp16 planes).
static __half *h16(float *region) { return reinterpret_cast<__half *>(region); }
static __half *S16h(const SweepPlan &p) { return h16(p.Sl); }
static __half *S16l(const SweepPlan &p) { return h16(p.Sl) + (size_t)p.m * p.n; }
static __half *P16h(const SweepPlan &p) { return h16(p.Ptl); }
static __half *P16l(const SweepPlan &p) { return h16(p.Ptl) + (size_t)p.m * p.n; }
static __half *H16h(const SweepPlan &p) { return h16(p.Hh); }
static __half *H16l(const SweepPlan &p) { return h16(p.Hh) + (size_t)p.n * p.n; }
static __half *F16h(const SweepPlan &p) { return h16(p.Fh); }
static __half *F16l(const SweepPlan &p) { return h16(p.Fh) + (size_t)p.m * p.m; }

// G = F_eff P on the free columns c0.. and one Adam step on them.  On the
// last step of a block the next block's columns (c0 .. c0 + B) run first, K
// split into slices whose fixed-order sum takes the step, and the rest (fused
// Adam epilogue) on the side stream when there is one: the next OBS block
// waits only for its own columns, and sweep_join_wide orders the rest before
// the next trailing update (the next reader or writer of those columns).
static realq_status_t g_adam(cudaStream_t s, SweepPlan &p, int64_t c0, bool last) {
    const int64_t r = p.n - c0;
    const int64_t t = ++(*p.adam_t);
    TcEpi g{};
    g.mode = TC_ADAM;
    g.ldw = p.n; g.col0 = c0;
    g.Wm = p.W; g.mA = p.adam_m; g.vA = p.adam_v; g.D = p.disp; g.Sh = p.Sh; g.Sl = p.f16 ? nullptr : p.Sl;
    if (p.f16) {
        g.ainv = p.scF;
        g.binv = p.scP;
    }
    g.lr = p.lr; g.b1 = p.beta1; g.b2 = p.beta2; g.eps = p.eps;
    g.bc1 = (float)(1.0 - std::pow((double)p.beta1, (double)t));
    g.bc2 = (float)(1.0 - std::pow((double)p.beta2, (double)t));
    g.sgd = p.optimizer == REALQ_OPT_SGD;
    const int64_t nb = std::min<int64_t>(p.block, r);
    if (!last) return tc_gemm_x3(s, p.mapsG, p.m, r, p.m, 0, 0, g, p.status, "bgd_g_gemm_adam");
    // (the split below is the same arithmetic with or without the side
    // stream, so a sweep resumed at any block gives the same bits)
    cudaStream_t ws = (p.wide && r > nb) ? p.wide : s;
    if (ws != s) {
        REALQ_CUDA_TRY(cudaEventRecord(p.wide_fork, s));
        REALQ_CUDA_TRY(cudaStreamWaitEvent(p.wide, p.wide_fork, 0));
    }
    // the next block's columns: few tiles with K = m, so K is split into
    // kGSplit slices (more CTAs, shorter chains), summed in a fixed order by
    // the pass that takes the optimizer step
    const int ks = p.f16 ? 64 : 32;
    const int kchunk = (int)((ceil_div(p.m, kGSplit) + ks - 1) / ks * ks);
    const int nz = ceil_div(p.m, kchunk);
    TcEpi st{};
    st.mode = TC_STORE;
    st.C = p.Gpart; st.ldc = nb; st.czs = p.m * nb;
    st.ainv = g.ainv; st.binv = g.binv;
    REALQ_TRY(tc_gemm_x3(s, p.mapsG, p.m, nb, p.m, 0, 0, st, p.status, "bgd_g_gemm_adam", 0, kchunk));
    REALQ_TRY(tc_gsum_adam(s, p.m, nb, nz, p.Gpart, g));
    if (r <= nb) return REALQ_OK;
    TcEpi gw = g;
    gw.col0 = c0 + nb;
    if (p.f16) gw.binv = p.scP + nb;
    REALQ_TRY(tc_gemm_x3(ws, p.mapsG, p.m, r - nb, p.m, 0, (int)nb, gw, p.status, "bgd_g_gemm_adam"));
    if (ws != s) {
        REALQ_CUDA_TRY(cudaEventRecord(p.wide_done, p.wide));
        p.wide_pending = 1;
    }
    return REALQ_OK;
}

realq_status_t sweep_join_wide(cudaStream_t s, SweepPlan &p) {
    if (!p.wide_pending) return REALQ_OK;
    REALQ_CUDA_TRY(cudaStreamWaitEvent(s, p.wide_done, 0));
    p.wide_pending = 0;
    return REALQ_OK;
}

// Side stream of the calling thread for the split G product, one per
// (device, caller's stream, its priority), created on first use and kept for
// the life of the thread.
namespace {
struct SideStream {
    int device = -1, priority = 0;
    cudaStream_t caller = nullptr, stream = nullptr;
    cudaEvent_t fork = nullptr, done = nullptr;
};
thread_local std::vector<SideStream> g_side;
}  // namespace

realq_status_t sweep_side_stream(cudaStream_t s, SweepPlan &p) {
    int dev = 0, prio = 0;
    REALQ_CUDA_TRY(cudaGetDevice(&dev));
    REALQ_CUDA_TRY(cudaStreamGetPriority(s, &prio));
    SideStream *f = nullptr;
    for (SideStream &x : g_side)
        if (x.device == dev && x.priority == prio && x.caller == s) f = &x;
    if (!f) {
        // one step below the caller's priority: when the side product's CTAs
        // hold the SMs, the next OBS block's CTAs are placed first as they free
        int least = 0, greatest = 0;
        REALQ_CUDA_TRY(cudaDeviceGetStreamPriorityRange(&least, &greatest));
        SideStream a;
        REALQ_CUDA_TRY(cudaStreamCreateWithPriority(&a.stream, cudaStreamNonBlocking, std::min(prio + 1, least)));
        REALQ_CUDA_TRY(cudaEventCreateWithFlags(&a.fork, cudaEventDisableTiming));
        REALQ_CUDA_TRY(cudaEventCreateWithFlags(&a.done, cudaEventDisableTiming));
        a.device = dev;
        a.priority = prio;
        a.caller = s;
        g_side.push_back(a);
        f = &g_side.back();
    }
    p.wide = f->stream;
    p.wide_fork = f->fork;
    p.wide_done = f->done;
    p.wide_pending = 0;
    return REALQ_OK;
}

// One Block-GD step on the free columns [c0, n) on the tensor cores
// (identity form).  The first product brings M = A H̄ up to date for them:
// the last step moved A only in its own free columns [step_c, n), so
// M[:, c0:] += step[:, step_c:] H̄[step_c:, c0:] (K = n - step_c instead of
// n), and its epilogue forms P from M and writes Pᵀ's tf32 planes; then
// G = F_eff P with the optimizer step (g_adam).
static realq_status_t bgd_one_tc(cudaStream_t s, SweepPlan &p, int64_t c0, bool last) {
    const int64_t r = p.n - c0;
    const int64_t k0 = p.step_c;
    TcEpi e{};
    e.mode = TC_BGD_P;
    e.Ad = p.disp; e.W = p.W; e.W0 = p.W0; e.w0_bf16 = p.w_dtype == REALQ_BF16;
    e.dead = p.dead; e.lam = p.lam; e.R0 = p.R0; e.ldw = p.n; e.col0 = c0;
    e.Pth = p.Pth; e.Ptl = p.Ptl; e.ldp = p.m; e.M = p.M;
    if (p.f16) {
        // the last step's fp16 planes over its columns [k0, n) (K of this
        // product); P^T comes out in fp32 and is split for the G product
        REALQ_TRY(tc_split_f16_rows(s, p.m, k0, p.n, p.Sh, nullptr, 1.f, p.n, S16h(p), S16l(p), p.n, p.scS));
        e.Ptl = nullptr;
        e.ainv = p.scS;
        e.binv = p.scH + c0;
    }
    REALQ_TRY(tc_gemm_x3(s, p.mapsP, p.m, r, p.n - k0, (int)k0, (int)c0, e, p.status, "bgd_p_gemm"));
    if (p.f16) REALQ_TRY(tc_split_f16_rows(s, r, 0, p.m, p.Pth, nullptr, 1.f, p.m, P16h(p), P16l(p), p.m, p.scP));
    REALQ_TRY(g_adam(s, p, c0, last));
    p.step_c = c0;
    return REALQ_OK;
}

// One optimizer step with a row-grouped OBS.  Rows of group g were swept
// against H_g,d = H̄_g + lambda_g I, so the stationarity identity holds for
// H_g,d, and P_R = ((Ŵ - W0) H̄)_R for those rows is
//   M_g + lambda_g (A - ΔW) - ΔW (H̄_g - H̄),   M_g = A H̄_g  (rows of g),
// which is the one-Hessian form when H̄_g = H̄.  M_g is kept current like M;
// ΔW (H̄_g - H̄) takes the full K = n.  Then G = F_eff P and Adam for all rows.
static realq_status_t bgd_one_tc_grouped(cudaStream_t s, SweepPlan &p, int64_t c0, bool last) {
    const int64_t r = p.n - c0;
    const int64_t k0 = p.step_c;
    if (p.w_dtype == REALQ_BF16)
        REALQ_TRY(tc_split_diff(s, p.m * p.n, p.W, static_cast<const __nv_bfloat16 *>(p.W0), p.DWh, p.DWl));
    else
        REALQ_TRY(tc_split_diff(s, p.m * p.n, p.W, static_cast<const float *>(p.W0), p.DWh, p.DWl));
    const size_t w0sz = p.w_dtype == REALQ_BF16 ? 2 : 4;
    for (int gr = 0; gr < p.rgroups; ++gr) {
        const int64_t row0 = gr * p.rg_rows, rows = std::min<int64_t>(p.rg_rows, p.m - row0);
        if (rows <= 0) break;
        if (k0 < p.n) {
            TcEpi e{};
            e.mode = TC_ACCUM;
            e.M = p.M + row0 * p.n; e.ldw = p.n; e.col0 = c0;
            REALQ_TRY(tc_gemm_x3(s, p.mapsMg[gr], rows, r, p.n - k0, (int)k0, (int)c0, e, p.status, "bgd_m_gemm",
                                     (int)row0));
        }
        TcEpi q{};
        q.mode = TC_BGD_PG;
        q.Ad = p.disp + row0 * p.n; q.W = p.W + row0 * p.n;
        q.W0 = static_cast<const char *>(p.W0) + (size_t)row0 * p.n * w0sz; q.w0_bf16 = p.w_dtype == REALQ_BF16;
        q.dead = p.dead_g + (size_t)gr * p.n; q.lam = p.lam_g + gr; q.R0 = p.R0 ? p.R0 + row0 * p.n : nullptr;
        q.ldw = p.n; q.col0 = c0; q.M = p.M + row0 * p.n;
        q.Pth = p.Pth + row0; q.Ptl = p.Ptl + row0; q.ldp = p.m;
        REALQ_TRY(tc_gemm_x3(s, p.mapsQg[gr], rows, r, p.n, 0, (int)c0, q, p.status, "bgd_p_gemm", (int)row0));
    }
    REALQ_TRY(g_adam(s, p, c0, last));
    p.step_c = c0;
    return REALQ_OK;
}

// One optimizer step on a calibration mini-batch: the gradient factor is
// ((Ŵ - W0) H̄_mb)_R = (stationarity form with H̄)_R + (ΔW (H̄_mb - H̄))_R,
// i.e. M + lambda (A - ΔW) - ΔW (H̄ - H̄_mb,k), with M = A H̄ kept current.
static realq_status_t bgd_one_tc_mb(cudaStream_t s, SweepPlan &p, int64_t c0, int kmb, bool last) {
    const int64_t r = p.n - c0;
    const int64_t k0 = p.step_c;
    if (p.w_dtype == REALQ_BF16)
        REALQ_TRY(tc_split_diff(s, p.m * p.n, p.W, static_cast<const __nv_bfloat16 *>(p.W0), p.DWh, p.DWl));
    else
        REALQ_TRY(tc_split_diff(s, p.m * p.n, p.W, static_cast<const float *>(p.W0), p.DWh, p.DWl));
    if (k0 < p.n) {
        TcEpi e{};
        e.mode = TC_ACCUM;
        e.M = p.M; e.ldw = p.n; e.col0 = c0;
        REALQ_TRY(tc_gemm_x3(s, p.mapsP, p.m, r, p.n - k0, (int)k0, (int)c0, e, p.status, "bgd_m_gemm"));
    }
    TcEpi q{};
    q.mode = TC_BGD_PG;
    q.Ad = p.disp; q.W = p.W; q.W0 = p.W0; q.w0_bf16 = p.w_dtype == REALQ_BF16;
    q.dead = p.dead; q.lam = p.lam; q.R0 = nullptr;
    q.ldw = p.n; q.col0 = c0; q.M = p.M;
    q.Pth = p.Pth; q.Ptl = p.Ptl; q.ldp = p.m;
    REALQ_TRY(tc_gemm_x3(s, p.mapsMB[kmb], p.m, r, p.n, 0, (int)c0, q, p.status, "bgd_p_gemm"));
    REALQ_TRY(g_adam(s, p, c0, last));
    p.step_c = c0;
    return REALQ_OK;
}

// One optimizer step on mini-batch kmb in token form, with the per-token
// output clipping (rank_q = m - 1 scales nothing):
//   Δ = X̂_k (Ŵ - W0)ᵀ, kappa from the per-token threshold, Y = kappa ⊙ Δ,
//   Z = Y F_eff, g = kappa ⊙ Z / T_k, G = gᵀ X̂_k[:, c0:], then Adam.
// The token axis of the last product is taken in fixed-order chunks of 8192
// (each accumulated into G in turn), so the accumulation is deterministic
// and each chunk's tensor-core sum stays short.
static realq_status_t bgd_one_tokens(cudaStream_t s, SweepPlan &p, int64_t c0, int kmb) {
    const int64_t r = p.n - c0;
    const int64_t Tk = std::min<int64_t>(p.tmb, p.Ttok - (int64_t)kmb * p.tmb);
    const void *Xk = static_cast<const __nv_bfloat16 *>(p.Xtok) + (size_t)kmb * p.tmb * p.n;
    REALQ_TRY(tok_xconv(s, Tk, p.n, Xk, p.Xf, p.XfT, p.tmb));
    if (p.w_dtype == REALQ_BF16)
        REALQ_TRY(tc_split_diff(s, p.m * p.n, p.W, static_cast<const __nv_bfloat16 *>(p.W0), p.DWh, p.DWl));
    else
        REALQ_TRY(tc_split_diff(s, p.m * p.n, p.W, static_cast<const float *>(p.W0), p.DWh, p.DWl));
    TcEpi e1{};
    e1.mode = TC_STORE;
    e1.C = p.Dk; e1.ldc = p.m;
    REALQ_TRY(tc_gemm_x3(s, p.mapsT1[kmb], Tk, p.m, p.n, 0, 0, e1, p.status, "tok_residual_gemm", 0, 0, 1));
    REALQ_TRY(tok_clip(s, Tk, p.m, p.Dk, p.rank_q, p.Yh, p.Yl));
    TcEpi e2{};
    e2.mode = TC_STORE;
    e2.C = p.Zk; e2.ldc = p.m;
    REALQ_TRY(tc_gemm_x3(s, p.mapsT2[kmb], Tk, p.m, p.m, 0, 0, e2, p.status, "tok_fisher_gemm"));
    REALQ_TRY(tok_gt(s, Tk, p.m, p.Dk, p.Zk, (float)(1.0 / (double)Tk), p.Yh, p.Yl, p.tmb));
    REALQ_CUDA_TRY(cudaMemsetAsync(p.Gc, 0, (size_t)p.m * r * sizeof(float), s));
    TcEpi e3{};
    e3.mode = TC_ACCUM;
    e3.M = p.Gc; e3.ldw = r; e3.col0 = 0;
    constexpr int64_t kChunk = 8192;
    for (int64_t k0 = 0; k0 < Tk; k0 += kChunk)
        REALQ_TRY(tc_gemm_x3(s, p.mapsT3[kmb], p.m, r, std::min<int64_t>(kChunk, Tk - k0), (int)k0, (int)c0, e3,
                                 p.status, "tok_grad_gemm", 0, 0, 2));
    const int64_t t = ++(*p.adam_t);
    const double bc1 = 1.0 - std::pow((double)p.beta1, (double)t);
    const double bc2 = 1.0 - std::pow((double)p.beta2, (double)t);
    {
        Launch L("bgd_adam", s);
        adam_kernel<<<blocks_for(p.m * r), 256, 0, s>>>(p.m, r, p.n, c0, p.Gc, p.W, p.adam_m, p.adam_v, p.disp, p.lr,
                                                         p.beta1, p.beta2, p.eps, (float)bc1, (float)bc2,
                                                         p.optimizer == REALQ_OPT_SGD);
    }
    REALQ_TRY(check_launch("bgd_adam"));
    p.step_c = c0;
    return REALQ_OK;
}

realq_status_t bgd_step(cudaStream_t s, SweepPlan &p, int64_t col_start, float alpha) {
    if (col_start >= p.n) return REALQ_OK;
    if (p.Dbar) REALQ_TRY(compute_r0(s, p));
    const float *Fuse = nullptr;
    REALQ_TRY(fisher_for(s, p, alpha, &Fuse));
    for (int k = 0; k < p.bgd_steps; ++k) REALQ_TRY(bgd_one(s, p, col_start, Fuse, 0));
    return REALQ_OK;
}

namespace {
__global__ void blend_kernel(float alpha, const float *a, const float *b, float *out) {
    out[0] = alpha * a[0] + (1.f - alpha) * b[0];
}
}  // namespace

// The surrogate of the current weights (quantized columns dequantized, the
// rest as they stand) with F_eff = alpha F + (1 - alpha) F_next, which is
// linear in F: alpha L(F) + (1 - alpha) L(F_next).
static realq_status_t trace_loss(cudaStream_t s, SweepPlan &p, float alpha, float *out) {
    const size_t sb = surrogate_ws_bytes(p.m, p.n);
    float *tmp = reinterpret_cast<float *>(static_cast<char *>(p.trace_ws) + sb);
    REALQ_TRY(surrogate(s, p.m, p.n, p.W, p.W0, p.w_dtype, p.Hbar, p.F, p.F_next ? tmp : out, p.trace_ws));
    if (!p.F_next) return REALQ_OK;
    REALQ_TRY(surrogate(s, p.m, p.n, p.W, p.W0, p.w_dtype, p.Hbar, p.F_next, tmp + 1, p.trace_ws));
    {
        Launch L("trace_blend", s);
        blend_kernel<<<1, 1, 0, s>>>(alpha, tmp, tmp + 1, out);
    }
    return check_launch("trace_blend");
}

realq_status_t sweep_block(cudaStream_t s, SweepPlan &p, int64_t b) {
    const int B = p.block;
    const int64_t bs = b * B;
    const int64_t be = std::min<int64_t>(bs + B, p.n);
    const int kb = (int)(be - bs);
    // a single group no wider than a block is handled inside the block kernel
    const int params_here = p.group <= B || (p.group >= p.n && p.n <= B);
    if (!params_here && bs % p.group == 0) {
        // a group wider than the block reads columns beyond it
        REALQ_TRY(sweep_join_wide(s, p));
        Launch L("group_params", s);
        group_params_kernel<<<ceil_div(p.m, 8), 256, 0, s>>>(p.m, p.n, p.W, bs, std::min<int64_t>(bs + p.group, p.n),
                                                              (int)(bs / p.group), p.ngroups, p.bits, p.sym, p.scale,
                                                              p.zero);
    }
    if (!params_here) REALQ_TRY(check_launch("group_params"));
    const int Gk = !params_here ? 0 : (p.group >= p.n ? B : p.group);
    for (int gr = 0; gr < p.rgroups; ++gr) {
        // row group gr against its own U (one group: all rows, U)
        const int64_t row0 = gr * p.rg_rows, rows = std::min<int64_t>(p.rg_rows, p.m - row0);
        if (rows <= 0) break;
        const int64_t ncb = (p.n + 1) / 2;
        QArgs qa{};
        qa.m = rows; qa.n = p.n; qa.bs = bs; qa.kb = kb;
        qa.W = p.W + row0 * p.n; qa.U = p.Ug + (size_t)gr * p.n * p.n;
        qa.g = p.group; qa.ngroups = p.ngroups; qa.bits = p.bits; qa.sym = p.sym;
        qa.scale = p.scale + row0 * p.ngroups; qa.zero = p.zero + row0 * p.ngroups; qa.codes = p.codes + row0 * ncb;
        qa.ncb = ncb;
        qa.Et = p.Et + row0; qa.ldet = p.m; qa.status = p.status;
        if (B == 128) REALQ_TRY(launch_qb_g<128>(s, qa, Gk));
        else if (B == 64) REALQ_TRY(launch_qb_g<64>(s, qa, Gk));
        else REALQ_TRY(launch_qb_g<32>(s, qa, Gk));
    }
    if (p.W_deq) {
        Launch L("copy_deq", s);
        if (p.deq_dtype == REALQ_BF16)
            copy_cols_kernel<<<blocks_for(p.m * kb), 256, 0, s>>>(p.m, p.n, bs, be, p.W, static_cast<__nv_bfloat16 *>(p.W_deq));
        else
            copy_cols_kernel<<<blocks_for(p.m * kb), 256, 0, s>>>(p.m, p.n, bs, be, p.W, static_cast<float *>(p.W_deq));
    }
    if (p.W_deq) REALQ_TRY(check_launch("copy_deq"));
    REALQ_TRY(sweep_join_wide(s, p));
    if (be >= p.n) return REALQ_OK;
    // lazy batch update of every later column: W[:, be:] -= E_b U[bs:be, be:]
    // (per row group with its own U).  On the tensor cores: the planes of -E_b
    // and of the U panel, then W[:, be:] += (-E_b) U[bs:be, be:] as a tf32x3
    // product accumulated into W.
    if (p.trail_tc) {
        if (!p.trail_maps) {
            REALQ_TRY(tc_make_maps(&p.mapsTr, p.Eh, p.El, p.m, B, B, p.UPh, p.UPl, p.n, B, B));
            p.trail_maps = 1;
        }
        for (int gr = 0; gr < p.rgroups; ++gr) {
            const int64_t row0 = gr * p.rg_rows, rows = std::min<int64_t>(p.rg_rows, p.m - row0);
            if (rows <= 0) break;
            REALQ_TRY(tc_trail_planes(s, p.m, gr == 0 ? p.Et : nullptr, p.m, p.n, p.Ug + (size_t)gr * p.n * p.n, bs,
                                      be, kb, B, p.Eh, p.El, p.UPh, p.UPl));
            TcEpi e{};
            e.mode = TC_ACCUM;
            e.M = p.W + row0 * p.n;
            e.ldw = p.n;
            e.col0 = be;
            REALQ_TRY(tc_gemm_x3(s, p.mapsTr, rows, p.n - be, kb, 0, 0, e, p.status, "trailing_update",
                                     (int)row0));
        }
    }
    for (int gr = 0; gr < p.rgroups && !p.trail_tc; ++gr) {
        const int64_t row0 = gr * p.rg_rows, rows = std::min<int64_t>(p.rg_rows, p.m - row0);
        if (rows <= 0) break;
        GemmArgs g{};
        g.M = rows; g.N = p.n - be; g.K = kb;
        g.A = p.Et + row0; g.lda = p.m;
        g.B = p.Ug + (size_t)gr * p.n * p.n + bs * p.n + be; g.ldb = p.n;
        g.C = p.W + row0 * p.n + be; g.ldc = p.n;
        g.alpha = 1.f;
        REALQ_TRY(gemm_f32(s, A_KMAJOR, EPI_SUB, g, "trailing_update"));
    }
    if (p.bgd_steps <= 0) return REALQ_OK;
    const int64_t b_global = p.b_global_start + b;
    float alpha = 1.f;
    if (p.B_total > 1) alpha = (float)(1.0 - (double)(b_global - 1) / (double)(p.B_total - 1));
    if (p.tc) {
        // F_eff planes: split once for a plain F, per block under the sliding window
        const float a_eff = p.F_next ? alpha : 1.f;
        if (!p.f_split_alpha_valid || p.f_split_alpha != a_eff) {
            const float *Fn = (p.F_next && a_eff != 1.f) ? p.F_next : nullptr;
            if (p.f16)
                REALQ_TRY(tc_split_f16_rows(s, p.m, 0, p.m, p.F, Fn, a_eff, p.m, F16h(p), F16l(p), p.m, p.scF));
            else
                REALQ_TRY(tc_split(s, p.m * p.m, p.F, Fn, a_eff, p.Fh, p.Fl));
            p.f_split_alpha_valid = 1;
            p.f_split_alpha = a_eff;
        }
        if (p.block_loss) REALQ_TRY(trace_loss(s, p, p.F_next ? alpha : 1.f, p.block_loss + 2 * b));
        for (int k = 0; k < p.bgd_steps; ++k) {
            const bool last = k == p.bgd_steps - 1;
            if (p.tmb > 0)
                REALQ_TRY(bgd_one_tokens(s, p, be, (int)(((b_global - 1) * p.bgd_steps + k) % p.ntok)));
            else if (p.nmb > 0)
                REALQ_TRY(bgd_one_tc_mb(s, p, be, (int)(((b_global - 1) * p.bgd_steps + k) % p.nmb), last));
            else
                REALQ_TRY(p.grouped ? bgd_one_tc_grouped(s, p, be, last) : bgd_one_tc(s, p, be, last));
        }
        if (p.block_loss) {
            REALQ_TRY(sweep_join_wide(s, p));
            REALQ_TRY(trace_loss(s, p, p.F_next ? alpha : 1.f, p.block_loss + 2 * b + 1));
        }
        return REALQ_OK;
    }
    const float *Fuse = nullptr;
    REALQ_TRY(fisher_for(s, p, alpha, &Fuse));
    if (p.block_loss) REALQ_TRY(trace_loss(s, p, p.F_next ? alpha : 1.f, p.block_loss + 2 * b));
    for (int k = 0; k < p.bgd_steps; ++k) REALQ_TRY(bgd_one(s, p, be, Fuse, 1));
    if (p.block_loss) REALQ_TRY(trace_loss(s, p, p.F_next ? alpha : 1.f, p.block_loss + 2 * b + 1));
    return REALQ_OK;
}

realq_status_t sweep_prologue_r0(cudaStream_t s, SweepPlan &p, bool fresh) {
    if (p.bgd_steps <= 0) return REALQ_OK;
    {
        Launch L("bgd_lambda", s);
        lambda_kernel<<<1, 1024, 0, s>>>(p.n, p.Hbar, p.dead, p.damp, p.lam);
    }
    REALQ_TRY(check_launch("bgd_lambda"));
    if (p.Dbar) REALQ_TRY(compute_r0(s, p));
    if (p.tc) {
        // planes of H̄ and the tensor maps of both GEMMs; M = A H̄ from the
        // caller's displacement (zero on a fresh sweep; a resumed sweep takes
        // nothing from an earlier workspace)
        if (p.f16) {
            // (H̄ is symmetric: row j of its planes is column j of H̄)
            REALQ_TRY(tc_split_f16_rows(s, p.n, 0, p.n, p.Hbar, nullptr, 1.f, p.n, H16h(p), H16l(p), p.n, p.scH));
            REALQ_TRY(tc_make_maps_f16(&p.mapsP, S16h(p), S16l(p), p.m, p.n, p.n, H16h(p), H16l(p), p.n, p.n, p.n));
            REALQ_TRY(tc_make_maps_f16(&p.mapsG, F16h(p), F16l(p), p.m, p.m, p.m, P16h(p), P16l(p), p.n, p.m, p.m));
        } else {
            REALQ_TRY(tc_split(s, p.n * p.n, p.Hbar, nullptr, 1.f, p.Hh, p.Hl));
            REALQ_TRY(tc_make_maps(&p.mapsP, p.Sh, p.Sl, p.m, p.n, p.n, p.Hh, p.Hl, p.n, p.n, p.n));
            REALQ_TRY(tc_make_maps(&p.mapsG, p.Fh, p.Fl, p.m, p.m, p.m, p.Pth, p.Ptl, p.n, p.m, p.m));
        }
        p.f_split_alpha_valid = 0;
        p.step_c = p.n;
        if (p.grouped) {
            // per row group: lambda_g, planes of H̄_g and H̄_g - H̄, the maps of
            // the M_g update and of the correction product
            const size_t nn = (size_t)p.n * p.n;
            p.mapsMg.assign(p.rgroups, TcMaps{});
            p.mapsQg.assign(p.rgroups, TcMaps{});
            for (int gr = 0; gr < p.rgroups; ++gr) {
                {
                    Launch L("bgd_lambda", s);
                    lambda_kernel<<<1, 1024, 0, s>>>(p.n, p.Hbar_g + gr * nn, p.dead_g + (size_t)gr * p.n, p.damp,
                                                     p.lam_g + gr);
                }
                REALQ_TRY(check_launch("bgd_lambda"));
                REALQ_TRY(tc_split(s, (int64_t)nn, p.Hbar_g + gr * nn, nullptr, 1.f, p.HGh + gr * nn, p.HGl + gr * nn));
                REALQ_TRY(tc_split_diff(s, (int64_t)nn, p.Hbar_g + gr * nn, p.Hbar, p.GGh + gr * nn, p.GGl + gr * nn));
                REALQ_TRY(tc_make_maps(&p.mapsMg[gr], p.Sh, p.Sl, p.m, p.n, p.n, p.HGh + gr * nn, p.HGl + gr * nn, p.n,
                                       p.n, p.n));
                REALQ_TRY(tc_make_maps(&p.mapsQg[gr], p.DWh, p.DWl, p.m, p.n, p.n, p.GGh + gr * nn, p.GGl + gr * nn,
                                       p.n, p.n, p.n));
            }
        }
        if (p.nmb > 0) {
            // planes of H̄ - H̄_mb,k and the maps of the correction product
            const size_t nn = (size_t)p.n * p.n;
            p.mapsMB.assign(p.nmb, TcMaps{});
            for (int k = 0; k < p.nmb; ++k) {
                REALQ_TRY(tc_split_diff(s, (int64_t)nn, p.Hbar, p.Hbar_mb + k * nn, p.MBh + k * nn, p.MBl + k * nn));
                REALQ_TRY(tc_make_maps(&p.mapsMB[k], p.DWh, p.DWl, p.m, p.n, p.n, p.MBh + k * nn, p.MBl + k * nn,
                                       p.n, p.n, p.n));
            }
        }
        if (p.tmb > 0) {
            // per mini-batch (the last may be short, and the products must
            // see zeros past its tokens): Δ = X̂_k ΔWᵀ, Z = Y F_eff and
            // G = gᵀ X̂_k with the token axis as K (X̂_k is exact in tf32: its
            // low plane is never loaded, the map's second plane is a stand-in)
            p.mapsT1.assign(p.ntok, TcMaps{});
            p.mapsT2.assign(p.ntok, TcMaps{});
            p.mapsT3.assign(p.ntok, TcMaps{});
            for (int k = 0; k < p.ntok; ++k) {
                const int64_t Tk = std::min<int64_t>(p.tmb, p.Ttok - (int64_t)k * p.tmb);
                REALQ_TRY(tc_make_maps(&p.mapsT1[k], p.Xf, p.Xf, Tk, p.n, p.n, p.DWh, p.DWl, p.m, p.n, p.n));
                REALQ_TRY(tc_make_maps(&p.mapsT2[k], p.Yh, p.Yl, Tk, p.m, p.m, p.Fh, p.Fl, p.m, p.m, p.m));
                REALQ_TRY(tc_make_maps(&p.mapsT3[k], p.Yh, p.Yl, p.m, Tk, p.tmb, p.XfT, p.XfT, p.n, Tk, p.tmb));
            }
        }
        if (fresh) {
            REALQ_CUDA_TRY(cudaMemsetAsync(p.M, 0, (size_t)p.m * p.n * sizeof(float), s));
        } else {
            if (p.f16)
                REALQ_TRY(tc_split_f16_rows(s, p.m, 0, p.n, p.disp, nullptr, 1.f, p.n, S16h(p), S16l(p), p.n, p.scS));
            else
                REALQ_TRY(tc_split(s, p.m * p.n, p.disp, nullptr, 1.f, p.Sh, p.Sl));
            if (p.grouped) {
                for (int gr = 0; gr < p.rgroups; ++gr) {
                    const int64_t row0 = gr * p.rg_rows, rows = std::min<int64_t>(p.rg_rows, p.m - row0);
                    if (rows <= 0) break;
                    TcEpi e{};
                    e.mode = TC_STORE;
                    e.C = p.M + row0 * p.n; e.ldc = p.n;
                    REALQ_TRY(tc_gemm_x3(s, p.mapsMg[gr], rows, p.n, p.n, 0, 0, e, p.status, "bgd_m_gemm",
                                             (int)row0));
                }
            } else {
                TcEpi e{};
                e.mode = TC_STORE;
                e.C = p.M; e.ldc = p.n;
                if (p.f16) {
                    e.ainv = p.scS;
                    e.binv = p.scH;
                }
                REALQ_TRY(tc_gemm_x3(s, p.mapsP, p.m, p.n, p.n, 0, 0, e, p.status, "bgd_m_gemm"));
            }
        }
    }
    return REALQ_OK;
}

size_t surrogate_ws_bytes(int64_t m, int64_t n) {
    return 3 * align_up((size_t)m * n * sizeof(float)) + align_up(RED_BLOCKS * sizeof(double));
}

realq_status_t surrogate(cudaStream_t s, int64_t m, int64_t n, const float *What, const void *W0,
                         realq_dtype_t w_dtype, const float *Hbar, const float *F, float *loss, void *ws) {
    Carve cv(ws);
    float *dW = cv.take<float>((size_t)m * n);
    float *X1 = cv.take<float>((size_t)m * n);
    float *X2 = cv.take<float>((size_t)m * n);
    double *part = cv.take<double>(RED_BLOCKS);
    {
        Launch L("surrogate_diff", s);
        if (w_dtype == REALQ_BF16)
            diff_kernel<<<blocks_for(m * n), 256, 0, s>>>(m * n, What, static_cast<const __nv_bfloat16 *>(W0), dW);
        else
            diff_kernel<<<blocks_for(m * n), 256, 0, s>>>(m * n, What, static_cast<const float *>(W0), dW);
    }
    REALQ_TRY(check_launch("surrogate_diff"));
    GemmArgs g{};
    g.M = m; g.N = n; g.K = n;
    g.A = dW; g.lda = n; g.B = Hbar; g.ldb = n; g.C = X1; g.ldc = n; g.alpha = 1.f;
    REALQ_TRY(gemm_f32(s, A_ROW, EPI_STORE, g, "surrogate_gemm"));
    GemmArgs h{};
    h.M = m; h.N = n; h.K = m;
    h.A = F; h.lda = m; h.B = dW; h.ldb = n; h.C = X2; h.ldc = n; h.alpha = 1.f;
    REALQ_TRY(gemm_f32(s, A_ROW, EPI_STORE, h, "surrogate_gemm"));
    {
        Launch L("surrogate_reduce", s);
        dot_partial_kernel<<<RED_BLOCKS, 256, 0, s>>>(m * n, X1, X2, part);
    }
    REALQ_TRY(check_launch("surrogate_reduce"));
    {
        Launch L("surrogate_reduce", s);
        dot_final_kernel<<<1, RED_BLOCKS, 0, s>>>(part, RED_BLOCKS, loss);
    }
    return check_launch("surrogate_reduce");
}

}  // namespace realq
