// Weight-activation setting (Sec. 5, "Weight-Activation Quantization"):
// per-token symmetric b-bit quantization of calibration activations with a
// clipping ratio.  In the activation-aware variant the weights are then
// quantized against these activations: they become the x̂ of the Hessian, and
// the full-precision activations stay the reference of the surrogate (the
// cross moment D).
//
// One warp per token row.  Pass 1 reduces max |x| over the row; pass 2
// quantizes on the grid of quant(.)'s symmetric mode over the clipped range
// [-a_clip max|x|, a_clip max|x|]: scale = 2 xmax / (2^b - 1), zero point
// 2^(b-1), q = clamp(rint(x / scale) + zero, 0, 2^b - 1), x_q = scale (q - zero)
// formed in fp32 and stored in the input's format.  Every operation that
// decides an integer is an explicitly rounded fp32 operation (no contraction),
// so the codes are reproducible bit for bit.  A row of zeros gets the range
// [-1, 1].
#include "kernels.cuh"

namespace realq {
namespace {

constexpr unsigned FULL = 0xFFFFFFFFu;

__device__ __forceinline__ float to_f(float v) { return v; }
__device__ __forceinline__ float to_f(__nv_bfloat16 v) { return __bfloat162float(v); }
__device__ __forceinline__ void store(float *p, float v) { *p = v; }
__device__ __forceinline__ void store(__nv_bfloat16 *p, float v) { *p = __float2bfloat16_rn(v); }

template <typename TX>
__global__ void __launch_bounds__(256) act_quant_kernel(int64_t T, int64_t n, const TX *X, TX *Xq, uint8_t *codes,
                                                        float *scale_out, int bits, float a_clip) {
    const int lane = threadIdx.x & 31;
    const int64_t t = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    if (t >= T) return;
    const TX *x = X + t * n;
    float amax = 0.f;
    for (int64_t c = lane; c < n; c += 32) amax = fmaxf(amax, fabsf(to_f(x[c])));
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) amax = fmaxf(amax, __shfl_xor_sync(FULL, amax, o));
    const int maxq = (1 << bits) - 1, zero = 1 << (bits - 1);
    float xmax = __fmul_rn(a_clip, amax);
    if (xmax == 0.f) xmax = 1.f;
    const float scale = __fdiv_rn(__fadd_rn(xmax, xmax), (float)maxq);
    if (lane == 0 && scale_out) scale_out[t] = scale;
    TX *xq = Xq + t * n;
    const bool packed = bits <= 4;
    const int64_t ldc = packed ? (n + 1) / 2 : n;
    for (int64_t c0 = 0; c0 < n; c0 += 32) {
        const int64_t c = c0 + lane;
        int q = 0;
        if (c < n) {
            float r = rintf(__fdiv_rn(to_f(x[c]), scale));
            r = fminf(fmaxf(r, (float)(-zero - 1)), (float)(maxq - zero + 1));
            q = min(max((int)r + zero, 0), maxq);
            store(xq + c, __fmul_rn(scale, (float)(q - zero)));
        }
        if (codes) {
            if (packed) {
                const int hi = __shfl_down_sync(FULL, q, 1);
                if (c < n && (lane & 1) == 0) codes[t * ldc + c / 2] = (uint8_t)(q | ((c + 1 < n ? hi : 0) << 4));
            } else if (c < n) {
                codes[t * ldc + c] = (uint8_t)q;
            }
        }
    }
}

}  // namespace

realq_status_t act_quant(cudaStream_t s, int64_t T, int64_t n, const void *X, realq_dtype_t dt, int bits, float a_clip,
                         void *Xq, uint8_t *codes, float *scale) {
    if (T == 0) return REALQ_OK;
    const int64_t warps = T;
    const unsigned blocks = (unsigned)((warps * 32 + 255) / 256);
    {
        Launch L("act_quant", s);
        if (dt == REALQ_BF16)
            act_quant_kernel<<<blocks, 256, 0, s>>>(T, n, static_cast<const __nv_bfloat16 *>(X),
                                                    static_cast<__nv_bfloat16 *>(Xq), codes, scale, bits, a_clip);
        else
            act_quant_kernel<<<blocks, 256, 0, s>>>(T, n, static_cast<const float *>(X), static_cast<float *>(Xq),
                                                    codes, scale, bits, a_clip);
    }
    return check_launch("act_quant");
}

}  // namespace realq
