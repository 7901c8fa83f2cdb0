// fp32 SIMT GEMM used where the sweep needs fp32-faithful contractions:
// the Block-GD gradient (Eq. block_gd_update: P = (Ŵ - W0) H̄, G = F P), the
// lazy batch update of Sec. 3.2 (W_rest -= E U[b, rest]) and the updates of
// the blocked Cholesky / triangular inverse.  128 x 128 output tile per CTA,
// 8 x 8 outputs per thread, K staged 8 at a time through shared memory.
#include "kernels.cuh"

namespace realq {
namespace {

constexpr int BM = 128, BN = 128, BK = 8, THREADS = 256;

template <int AM>
__device__ __forceinline__ float load_a(const GemmArgs &g, int64_t i, int64_t k) {
    if (AM == A_ROW) return static_cast<const float *>(g.A)[i * g.lda + k];
    if (AM == A_ROW_BF16) return __bfloat162float(static_cast<const __nv_bfloat16 *>(g.A)[i * g.lda + k]);
    if (AM == A_DIFF_F32)
        return static_cast<const float *>(g.A)[i * g.lda + k] - static_cast<const float *>(g.Y)[i * g.ldy + k];
    if (AM == A_DIFF_BF16)
        return static_cast<const float *>(g.A)[i * g.lda + k] -
               __bfloat162float(static_cast<const __nv_bfloat16 *>(g.Y)[i * g.ldy + k]);
    return static_cast<const float *>(g.A)[k * g.lda + i];  // A_KMAJOR
}

template <int AM, int EM>
__global__ void __launch_bounds__(THREADS) sgemm_kernel(const GemmArgs g) {
    __shared__ __align__(16) float As[BK][BM + 4];
    __shared__ __align__(16) float Bs[BK][BN + 4];
    const int tid = threadIdx.x;
    const int tx = tid & 15, ty = tid >> 4;
    const int64_t m0 = (int64_t)blockIdx.y * BM, n0 = (int64_t)blockIdx.x * BN;
    float acc[8][8];
#pragma unroll
    for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int j = 0; j < 8; ++j) acc[i][j] = 0.f;

    for (int64_t k0 = 0; k0 < g.K; k0 += BK) {
#pragma unroll
        for (int r = 0; r < (BM * BK) / THREADS; ++r) {
            const int idx = tid + r * THREADS;
            int ii, kk;
            if (AM == A_KMAJOR) { kk = idx / BM; ii = idx % BM; }
            else { ii = idx / BK; kk = idx % BK; }
            const int64_t gi = m0 + ii, gk = k0 + kk;
            As[kk][ii] = (gi < g.M && gk < g.K) ? load_a<AM>(g, gi, gk) : 0.f;
        }
#pragma unroll
        for (int r = 0; r < (BN * BK) / THREADS; ++r) {
            const int idx = tid + r * THREADS;
            const int kk = idx / BN, jj = idx % BN;
            const int64_t gk = k0 + kk, gj = n0 + jj;
            Bs[kk][jj] = (gk < g.K && gj < g.N) ? g.B[gk * g.ldb + gj] : 0.f;
        }
        __syncthreads();
#pragma unroll
        for (int kk = 0; kk < BK; ++kk) {
            float a[8], b[8];
            const float4 a0 = *reinterpret_cast<const float4 *>(&As[kk][ty * 4]);
            const float4 a1 = *reinterpret_cast<const float4 *>(&As[kk][64 + ty * 4]);
            const float4 b0 = *reinterpret_cast<const float4 *>(&Bs[kk][tx * 4]);
            const float4 b1 = *reinterpret_cast<const float4 *>(&Bs[kk][64 + tx * 4]);
            a[0] = a0.x; a[1] = a0.y; a[2] = a0.z; a[3] = a0.w;
            a[4] = a1.x; a[5] = a1.y; a[6] = a1.z; a[7] = a1.w;
            b[0] = b0.x; b[1] = b0.y; b[2] = b0.z; b[3] = b0.w;
            b[4] = b1.x; b[5] = b1.y; b[6] = b1.z; b[7] = b1.w;
#pragma unroll
            for (int i = 0; i < 8; ++i)
#pragma unroll
                for (int j = 0; j < 8; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
        }
        __syncthreads();
    }
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        const int64_t gi = m0 + (i < 4 ? ty * 4 + i : 64 + ty * 4 + (i - 4));
        if (gi >= g.M) continue;
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            const int64_t gj = n0 + (j < 4 ? tx * 4 + j : 64 + tx * 4 + (j - 4));
            if (gj >= g.N) continue;
            float *c = g.C + gi * g.ldc + gj;
            const float v = g.alpha * acc[i][j];
            if (EM == EPI_STORE) *c = v;
            else if (EM == EPI_SUB) *c = *c - v;
            else if (EM == EPI_BIAS) *c = v + g.R[gi * g.ldr + gj];
            else {
                const int64_t col = g.col0 + gj;
                const int64_t w = gi * g.ldw + col;
                const float w0 = g.w0_bf16 ? __bfloat162float(static_cast<const __nv_bfloat16 *>(g.W0c)[w])
                                           : static_cast<const float *>(g.W0c)[w];
                float p = v + (*g.lam) * (g.Ad[w] - (g.Wc[w] - w0));
                if (g.R) p += g.R[gi * g.ldr + gj];
                if (g.dead && g.dead[col]) p = 0.f;
                *c = p;
            }
        }
    }
}

template <int AM>
realq_status_t dispatch_epi(cudaStream_t s, EpiMode em, const GemmArgs &g, const char *name) {
    dim3 grid(ceil_div(g.N, BN), ceil_div(g.M, BM));
    {
        Launch L(name, s);
        if (em == EPI_STORE) sgemm_kernel<AM, EPI_STORE><<<grid, THREADS, 0, s>>>(g);
        else if (em == EPI_SUB) sgemm_kernel<AM, EPI_SUB><<<grid, THREADS, 0, s>>>(g);
        else if (em == EPI_BIAS) sgemm_kernel<AM, EPI_BIAS><<<grid, THREADS, 0, s>>>(g);
        else sgemm_kernel<AM, EPI_BGD_P><<<grid, THREADS, 0, s>>>(g);
    }
    return check_launch(name);
}

}  // namespace

realq_status_t gemm_f32(cudaStream_t s, AMode am, EpiMode em, const GemmArgs &g, const char *name) {
    if (g.M <= 0 || g.N <= 0) return REALQ_OK;
    if (g.N > (int64_t)BN * 2147483647LL || g.M > (int64_t)BM * 65535LL)
        return fail(REALQ_ERR_UNSUPPORTED, "%s: GEMM too large (%lld x %lld)", name, (long long)g.M, (long long)g.N);
    switch (am) {
        case A_ROW: return dispatch_epi<A_ROW>(s, em, g, name);
        case A_ROW_BF16: return dispatch_epi<A_ROW_BF16>(s, em, g, name);
        case A_DIFF_F32: return dispatch_epi<A_DIFF_F32>(s, em, g, name);
        case A_DIFF_BF16: return dispatch_epi<A_DIFF_BF16>(s, em, g, name);
        default: return dispatch_epi<A_KMAJOR>(s, em, g, name);
    }
}

}  // namespace realq
