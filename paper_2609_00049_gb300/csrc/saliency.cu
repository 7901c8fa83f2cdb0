// Saliency-weighted Hessians of the coarse stage (Sec. 3.3, Eq.
// saliency_hessian; Alg. 1 "for all row-groups g"; the appendix's
// Hessian-side saliency clipping):
//   H_g = sum_t s'[t, g] x̂_t x̂_t^T,   s'[t, g] = min(s[t, g], c_g),
// c_g the nearest-rank 99th percentile of group g's saliencies over the
// tokens.
//
// The percentile is an exact order statistic: one CTA per group runs a radix
// select over the bit patterns of the (non-negative) saliencies, 8 bits per
// pass from the top, so the threshold is one of the inputs, bit for bit.
// The weighted product runs on the bf16 tensor cores as H_g = X̂ᵀ (s' X̂):
// the scaled rows y_t = s'_t x̂_t of one group are split into two bf16 parts,
// y = y_hi + y_lo (16 significant bits together), and accumulated by two
// full-tile cross passes X̂ᵀ y_hi + X̂ᵀ y_lo; x̂ is exact in bf16, so each
// product is within 2^-17 relative of s' x_i x_j, and the accumulation is
// promoted to fp32 registers every 128 tokens.  The sum is symmetric up to
// that rounding, so only tiles on or below the diagonal are formed, then
// mirrored.  A single bf16 rounding
// (2^-9) is not enough: with heavy-tailed saliency a few dozen tokens carry
// most of the weight and the rounding does not average out.  The weight sums
// are fixed-order fp64 reductions.
#include "kernels.cuh"

namespace realq {
namespace {

constexpr int SEL_THREADS = 1024;
// Saliency spreads token magnitudes over decades, so a TMEM accumulator loses
// the low bits of small terms against a running sum dominated by a few large
// ones; promote to fp32 registers every 2 stages (128 tokens) instead of 16.
constexpr int kPromoteStages = 2;

__device__ __forceinline__ uint32_t key_of(float v) { return __float_as_uint(fmaxf(v, 0.f)); }

__global__ void __launch_bounds__(SEL_THREADS) select_kernel(int64_t T, int ng, const float *S, int64_t k,
                                                             float *clip_out) {
    __shared__ unsigned int hist[256];
    __shared__ uint32_t s_prefix;
    __shared__ int64_t s_k;
    const int g = blockIdx.x;
    if (threadIdx.x == 0) {
        s_prefix = 0u;
        s_k = k;
    }
    uint32_t mask = 0u;
    for (int shift = 24; shift >= 0; shift -= 8) {
        for (int i = threadIdx.x; i < 256; i += SEL_THREADS) hist[i] = 0u;
        __syncthreads();
        const uint32_t prefix = s_prefix;
        for (int64_t t = threadIdx.x; t < T; t += SEL_THREADS) {
            const uint32_t key = key_of(S[t * ng + g]);
            if ((key & mask) == prefix) atomicAdd(&hist[(key >> shift) & 255u], 1u);
        }
        __syncthreads();
        if (threadIdx.x == 0) {
            int64_t kr = s_k;
            int b = 0;
            for (; b < 255; ++b) {
                if (kr < (int64_t)hist[b]) break;
                kr -= hist[b];
            }
            s_prefix = prefix | ((uint32_t)b << shift);
            s_k = kr;
        }
        mask |= 255u << shift;
        __syncthreads();
    }
    if (threadIdx.x == 0) clip_out[g] = __uint_as_float(s_prefix);
}

__global__ void clip_kernel(int64_t count, int ng, const float *S, const float *c, float *out) {
    const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (i < count) out[i] = fminf(S[i], c[i % ng]);
}

// y = s[t, g] x[t, :] (fp32, one rounding), split into bf16 parts; 8 elements
// (16 bytes) per thread, n a multiple of 8
__global__ void wscale_kernel(int64_t T, int64_t n, const __nv_bfloat16 *X, const float *S, int g, int ng,
                              __nv_bfloat16 *Yhi, __nv_bfloat16 *Ylo) {
    const int64_t v = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (v >= T * n / 8) return;
    const int64_t i = v * 8;
    const float w = fmaxf(S[(i / n) * ng + g], 0.f);
    const uint4 xv = *reinterpret_cast<const uint4 *>(X + i);
    const __nv_bfloat16 *xe = reinterpret_cast<const __nv_bfloat16 *>(&xv);
    uint4 hv, lv;
    __nv_bfloat16 *he = reinterpret_cast<__nv_bfloat16 *>(&hv);
    __nv_bfloat16 *le = reinterpret_cast<__nv_bfloat16 *>(&lv);
#pragma unroll
    for (int k = 0; k < 8; ++k) {
        const float y = w * __bfloat162float(xe[k]);
        he[k] = __float2bfloat16_rn(y);
        le[k] = __float2bfloat16_rn(y - __bfloat162float(he[k]));
    }
    *reinterpret_cast<uint4 *>(Yhi + i) = hv;
    *reinterpret_cast<uint4 *>(Ylo + i) = lv;
}

// wsum[g] += sum_t s[t, g] in fp64, one CTA per group, fixed order
__global__ void __launch_bounds__(1024) wsum_kernel(int64_t T, int ng, const float *S, double *wsum) {
    __shared__ double red[1024];
    const int g = blockIdx.x;
    double a = 0.0;
    for (int64_t t = threadIdx.x; t < T; t += 1024) a += (double)S[t * ng + g];
    red[threadIdx.x] = a;
    __syncthreads();
    for (int w = 512; w > 0; w >>= 1) {
        if ((int)threadIdx.x < w) red[threadIdx.x] += red[threadIdx.x + w];
        __syncthreads();
    }
    if (threadIdx.x == 0) wsum[g] += red[0];
}

}  // namespace

size_t saliency_clip_ws_bytes() { return 0; }

realq_status_t saliency_clip(cudaStream_t s, int64_t T, int ng, const float *S, double pct, float *S_out,
                             float *clip_out) {
    if (T <= 0) return REALQ_OK;
    int64_t k = (int64_t)std::ceil(pct * (double)T) - 1;
    if (k < 0) k = 0;
    if (k > T - 1) k = T - 1;
    {
        Launch L("saliency_select", s);
        select_kernel<<<ng, SEL_THREADS, 0, s>>>(T, ng, S, k, clip_out);
    }
    REALQ_TRY(check_launch("saliency_select"));
    if (S_out) {
        const int64_t count = T * ng;
        Launch L("saliency_clip", s);
        clip_kernel<<<(unsigned)((count + 255) / 256), 256, 0, s>>>(count, ng, S, clip_out, S_out);
    }
    return S_out ? check_launch("saliency_clip") : REALQ_OK;
}

size_t weighted_ws_bytes(int64_t n, int64_t T) {
    return align_up(hessian_ws_bytes(n, T, 0)) + 2 * align_up((size_t)T * n * sizeof(__nv_bfloat16));
}

realq_status_t hessian_weighted(cudaStream_t s, int64_t n, int64_t T, const void *X, int ng, const float *S,
                                float *Hg, double *wsum, void *ws, size_t ws_bytes) {
    if (T == 0) return REALQ_OK;
    // [Hessian workspace: status word, token-split partials][y_hi][y_lo] of one group
    const size_t hbytes = hessian_ws_bytes(n, T, 0);
    char *base = static_cast<char *>(ws);
    int *err = reinterpret_cast<int *>(base);
    void *part = base + align_up(sizeof(int));
    const size_t pbytes = hbytes - align_up(sizeof(int));
    __nv_bfloat16 *Yhi = reinterpret_cast<__nv_bfloat16 *>(base + align_up(hbytes));
    __nv_bfloat16 *Ylo = Yhi + align_up((size_t)T * n * sizeof(__nv_bfloat16)) / sizeof(__nv_bfloat16);
    const bool tc = hessian_tc_eligible(n, T, X) && hessian_tc_eligible(n, T, Yhi) && hessian_tc_eligible(n, T, Ylo);
    if (!tc) return fail(REALQ_ERR_UNSUPPORTED, "weighted Hessian: n must be a multiple of 8 and >= 64");
    for (int g = 0; g < ng; ++g) {
        {
            Launch L("saliency_scale", s);
            wscale_kernel<<<(unsigned)((T * n / 8 + 255) / 256), 256, 0, s>>>(
                T, n, static_cast<const __nv_bfloat16 *>(X), S, g, ng, Yhi, Ylo);
        }
        REALQ_TRY(check_launch("saliency_scale"));
        float *Hout = Hg + (size_t)g * n * n;
        REALQ_TRY(hessian_cross_tc(s, n, T, X, Yhi, Hout, 1.f, err, part, pbytes, num_sms(), kPromoteStages, true));
        REALQ_TRY(hessian_cross_tc(s, n, T, X, Ylo, Hout, 1.f, err, part, pbytes, num_sms(), kPromoteStages, true));
    }
    {
        Launch L("saliency_wsum", s);
        wsum_kernel<<<ng, 1024, 0, s>>>(T, ng, S, wsum);
    }
    return check_launch("saliency_wsum");
}

}  // namespace realq
