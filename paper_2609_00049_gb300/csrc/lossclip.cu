// Token-form Block-GD gradient on a calibration mini-batch with the per-token
// output clipping of the small-model runs (App. "Activation clipping
// (a_loss_clip) for small Qwen3 models", a_loss_clip = 0.95):
//   Δ = X̂_k ΔWᵀ                      (T_k x m, tensor cores, tf32x3)
//   q_t = the ceil(pct m)-th smallest |Δ_t,i| of token t (an exact order
//         statistic: radix select over the bit patterns of |Δ|)
//   κ_t,i = q_t / |Δ_t,i| where |Δ_t,i| > q_t, else 1 (detached)
//   Z = (κ ⊙ Δ) F_eff                 (T_k x m, tensor cores)
//   G = (κ ⊙ Z)ᵀ X̂_k / T_k            (m x r, tensor cores, K = T_k in
//                                       fixed-order chunks)
// These kernels are the elementwise and layout steps between the products:
// the conversion of the bf16 mini-batch to fp32 (token-major for the first
// product, channel-major for the last), the per-token select that forms the
// clipped residual's tf32 planes, and the transposed, scaled gradient factor.
#include "kernels.cuh"
#include "tc.cuh"

namespace realq {
namespace {

constexpr int TILE = 32;

// Xf = X (T x n, token-major, fp32) and XfT = Xᵀ (n x T, leading dimension ldT)
__global__ void __launch_bounds__(256) xconv_kernel(int64_t T, int64_t n, const __nv_bfloat16 *X, float *Xf,
                                                    float *XfT, int64_t ldT) {
    __shared__ float tile[TILE][TILE + 1];
    const int64_t j0 = (int64_t)blockIdx.x * TILE, t0 = (int64_t)blockIdx.y * TILE;
    const int tx = threadIdx.x, ty = threadIdx.y;
    for (int r = ty; r < TILE; r += 8) {
        const int64_t t = t0 + r, j = j0 + tx;
        float v = 0.f;
        if (t < T && j < n) {
            v = __bfloat162float(X[t * n + j]);
            Xf[t * n + j] = v;
        }
        tile[r][tx] = v;
    }
    __syncthreads();
    for (int r = ty; r < TILE; r += 8) {
        const int64_t j = j0 + r, t = t0 + tx;
        if (j < n && t < T) XfT[j * ldT + t] = tile[tx][r];
    }
}

// One warp per token: q = the (k+1)-th smallest |D[t, :]| (k 0-based), then
// kappa into D and the tf32 planes of kappa * D into Yh / Yl.  With STAGE the
// token's row is read from global memory once and kept in shared memory for
// the four select passes and the final one (CLIP_WARPS rows per CTA).
constexpr int CLIP_WARPS = 4;

template <bool STAGE>
__global__ void __launch_bounds__(CLIP_WARPS * 32) clip_kernel(int64_t T, int64_t m, float *D, int64_t k, float *Yh,
                                                               float *Yl) {
    __shared__ unsigned int hist[CLIP_WARPS][256];
    extern __shared__ float rowbuf[];
    const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t t = (int64_t)blockIdx.x * CLIP_WARPS + w;
    if (t >= T) return;
    float *grow = D + t * m;
    float *row = grow;
    if (STAGE) {
        row = rowbuf + (int64_t)w * m;
        for (int64_t i = lane; i < m; i += 32) row[i] = grow[i];
        __syncwarp();
    }
    unsigned int *h = hist[w];
    uint32_t prefix = 0u, mask = 0u;
    int64_t kr = k;
    for (int shift = 24; shift >= 0; shift -= 8) {
#pragma unroll
        for (int b = 0; b < 8; ++b) h[lane * 8 + b] = 0u;
        __syncwarp();
        for (int64_t i = lane; i < m; i += 32) {
            const uint32_t key = __float_as_uint(row[i]) & 0x7FFFFFFFu;
            if ((key & mask) == prefix) atomicAdd(&h[(key >> shift) & 255u], 1u);
        }
        __syncwarp();
        // lane l owns bins 8l .. 8l + 7; an inclusive scan of the lane sums
        // finds the lane whose bins hold rank kr
        unsigned int own = 0u;
#pragma unroll
        for (int b = 0; b < 8; ++b) own += h[lane * 8 + b];
        unsigned int incl = own;
#pragma unroll
        for (int d = 1; d < 32; d <<= 1) {
            const unsigned int u = __shfl_up_sync(0xFFFFFFFFu, incl, d);
            if (lane >= d) incl += u;
        }
        const unsigned int excl = incl - own;
        const bool mine = (int64_t)excl <= kr && kr < (int64_t)incl;
        const unsigned int who = __ballot_sync(0xFFFFFFFFu, mine);
        int bucket = 0;
        int64_t rest = 0;
        if (mine) {
            int64_t c = excl;
            int b = lane * 8;
            while (b < lane * 8 + 7 && kr >= c + (int64_t)h[b]) c += h[b++];
            bucket = b;
            rest = kr - c;
        }
        const int src = who ? __ffs(who) - 1 : 31;
        bucket = __shfl_sync(0xFFFFFFFFu, bucket, src);
        rest = __shfl_sync(0xFFFFFFFFu, rest, src);
        kr = rest;
        prefix |= (uint32_t)bucket << shift;
        mask |= 255u << shift;
        __syncwarp();
    }
    const float q = __uint_as_float(prefix);
    for (int64_t i = lane; i < m; i += 32) {
        const float d = row[i];
        const float a = fabsf(d);
        const float kap = a > q ? __fdiv_rn(q, a) : 1.f;
        const float y = __fmul_rn(kap, d);
        const float hi = tc::tf32_hi(y);
        Yh[t * m + i] = hi;
        Yl[t * m + i] = y - hi;
        grow[i] = kap;
    }
}

// gT[i, t] = kappa[t, i] Z[t, i] / T as tf32 planes, transposed (m x T, ldT)
__global__ void __launch_bounds__(256) gt_kernel(int64_t T, int64_t m, const float *kap, const float *Z, float inv_T,
                                                 float *gTh, float *gTl, int64_t ldT) {
    __shared__ float tile[TILE][TILE + 1];
    const int64_t i0 = (int64_t)blockIdx.x * TILE, t0 = (int64_t)blockIdx.y * TILE;
    const int tx = threadIdx.x, ty = threadIdx.y;
    for (int r = ty; r < TILE; r += 8) {
        const int64_t t = t0 + r, i = i0 + tx;
        tile[r][tx] = (t < T && i < m) ? __fmul_rn(__fmul_rn(kap[t * m + i], Z[t * m + i]), inv_T) : 0.f;
    }
    __syncthreads();
    for (int r = ty; r < TILE; r += 8) {
        const int64_t i = i0 + r, t = t0 + tx;
        if (i < m && t < T) {
            const float v = tile[tx][r];
            const float hi = tc::tf32_hi(v);
            gTh[i * ldT + t] = hi;
            gTl[i * ldT + t] = v - hi;
        }
    }
}

}  // namespace

realq_status_t tok_xconv(cudaStream_t s, int64_t T, int64_t n, const void *X, float *Xf, float *XfT, int64_t ldT) {
    if (T <= 0) return REALQ_OK;
    {
        Launch L("tok_xconv", s);
        xconv_kernel<<<dim3((unsigned)ceil_div(n, TILE), (unsigned)ceil_div(T, TILE)), dim3(TILE, 8), 0, s>>>(
            T, n, static_cast<const __nv_bfloat16 *>(X), Xf, XfT, ldT);
    }
    return check_launch("tok_xconv");
}

realq_status_t tok_clip(cudaStream_t s, int64_t T, int64_t m, float *D, int64_t k, float *Yh, float *Yl) {
    if (T <= 0) return REALQ_OK;
    const size_t stage = (size_t)CLIP_WARPS * m * sizeof(float);
    constexpr size_t kMaxStage = 160 * 1024;
    REALQ_TRY(set_smem_limit(reinterpret_cast<const void *>(clip_kernel<true>), (int)kMaxStage));
    {
        Launch L("tok_clip", s);
        if (stage <= kMaxStage)
            clip_kernel<true><<<(unsigned)ceil_div(T, CLIP_WARPS), CLIP_WARPS * 32, stage, s>>>(T, m, D, k, Yh, Yl);
        else
            clip_kernel<false><<<(unsigned)ceil_div(T, CLIP_WARPS), CLIP_WARPS * 32, 0, s>>>(T, m, D, k, Yh, Yl);
    }
    return check_launch("tok_clip");
}

realq_status_t tok_gt(cudaStream_t s, int64_t T, int64_t m, const float *kap, const float *Z, float inv_T, float *gTh,
                      float *gTl, int64_t ldT) {
    if (T <= 0) return REALQ_OK;
    {
        Launch L("tok_grad_t", s);
        gt_kernel<<<dim3((unsigned)ceil_div(m, TILE), (unsigned)ceil_div(T, TILE)), dim3(TILE, 8), 0, s>>>(
            T, m, kap, Z, inv_T, gTh, gTl, ldT);
    }
    return check_launch("tok_grad_t");
}

}  // namespace realq
