// fp32 SIMT GEMM used where the sweep needs fp32-faithful contractions:
// the Block-GD gradient (Eq. block_gd_update: P = (Ŵ - W0) H̄ or its identity
// form, G = F P), the lazy batch update of Sec. 3.2 (W_rest -= E U[b, rest])
// and the updates of the blocked Cholesky / triangular inverse.
//
// C tile BM x BN per CTA (128 x 128, or 64 x 64 when the 128-tile grid would
// leave most SMs idle), 256 threads, K staged 16 at a time through two
// shared-memory buffers: the next K slice is loaded into registers while the
// current one is multiplied, so global latency overlaps the FFMA work.
#include "kernels.cuh"

namespace realq {
namespace {

constexpr int BK = 16, THREADS = 256;

template <int AM>
__device__ __forceinline__ float load_a(const GemmArgs &g, int64_t i, int64_t k) {
    if (AM == A_ROW) {
        const float *a = static_cast<const float *>(g.A) + i * g.lda + k;
        float v = a[0];
        for (int s = 1; s < g.nsum; ++s) v += a[s * g.aplane];
        return v;
    }
    if (AM == A_ROW_BF16) return __bfloat162float(static_cast<const __nv_bfloat16 *>(g.A)[i * g.lda + k]);
    if (AM == A_DIFF_F32)
        return static_cast<const float *>(g.A)[i * g.lda + k] - static_cast<const float *>(g.Y)[i * g.ldy + k];
    if (AM == A_DIFF_BF16)
        return static_cast<const float *>(g.A)[i * g.lda + k] -
               __bfloat162float(static_cast<const __nv_bfloat16 *>(g.Y)[i * g.ldy + k]);
    return static_cast<const float *>(g.A)[k * g.lda + i];  // A_KMAJOR
}

template <int EM>
__device__ __forceinline__ void epilogue(const GemmArgs &g, int64_t gi, int64_t gj, float acc) {
    float *c = g.C + (int64_t)blockIdx.z * g.cplane + gi * g.ldc + gj;
    const float v = g.alpha * acc;
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

// TM x TN outputs per thread: rows ty*4..ty*4+3 (and BM/2 + ty*4.. when
// TM = 8), columns likewise, so every shared-memory read is an aligned float4.
template <int BM, int BN, int AM, int EM>
__global__ void __launch_bounds__(THREADS) sgemm_kernel(const GemmArgs g) {
    constexpr int TM = BM / 16, TN = BN / 16;  // 8x8 or 4x4 per thread
    constexpr int A_PER = BM * BK / THREADS, B_PER = BN * BK / THREADS;
    __shared__ __align__(16) float As[2][BK][BM + 4];
    __shared__ __align__(16) float Bs[2][BK][BN + 4];
    const int tid = threadIdx.x;
    const int tx = tid & 15, ty = tid >> 4;
    const int64_t m0 = (int64_t)blockIdx.y * BM, n0 = (int64_t)blockIdx.x * BN;
    const int64_t kz = (g.K + gridDim.z - 1) / gridDim.z;
    int64_t kbeg = (int64_t)blockIdx.z * kz;
    int64_t kend = min(g.K, kbeg + kz);
    if (g.a_upper && kbeg < m0) kbeg = m0;
    if (g.b_upper && kend > n0 + BN) kend = n0 + BN;

    float acc[TM][TN];
#pragma unroll
    for (int i = 0; i < TM; ++i)
#pragma unroll
        for (int j = 0; j < TN; ++j) acc[i][j] = 0.f;

    float ra[A_PER], rb[B_PER];
    auto fetch = [&](int64_t k0) {
#pragma unroll
        for (int r = 0; r < A_PER; ++r) {
            const int idx = tid + r * THREADS;
            int ii, kk;
            if (AM == A_KMAJOR) { kk = idx / BM; ii = idx % BM; }
            else { ii = idx / BK; kk = idx % BK; }
            const int64_t gi = m0 + ii, gk = k0 + kk;
            ra[r] = (gi < g.M && gk < kend) ? load_a<AM>(g, gi, gk) : 0.f;
        }
#pragma unroll
        for (int r = 0; r < B_PER; ++r) {
            const int idx = tid + r * THREADS;
            const int kk = idx / BN, jj = idx % BN;
            const int64_t gk = k0 + kk, gj = n0 + jj;
            float bv = 0.f;
            if (gk < kend && gj < g.N) {
                const float *bp = g.B + gk * g.ldb + gj;
                bv = bp[0];
                for (int s2 = 1; s2 < g.nsum_b; ++s2) bv += bp[s2 * g.bplane];
            }
            rb[r] = bv;
        }
    };
    auto stash = [&](int buf) {
#pragma unroll
        for (int r = 0; r < A_PER; ++r) {
            const int idx = tid + r * THREADS;
            int ii, kk;
            if (AM == A_KMAJOR) { kk = idx / BM; ii = idx % BM; }
            else { ii = idx / BK; kk = idx % BK; }
            As[buf][kk][ii] = ra[r];
        }
#pragma unroll
        for (int r = 0; r < B_PER; ++r) {
            const int idx = tid + r * THREADS;
            Bs[buf][idx / BN][idx % BN] = rb[r];
        }
    };

    if (kbeg < kend) {
        fetch(kbeg);
        stash(0);
        __syncthreads();
        int buf = 0;
        for (int64_t k0 = kbeg; k0 < kend; k0 += BK) {
            const bool more = k0 + BK < kend;
            if (more) fetch(k0 + BK);
#pragma unroll
            for (int kk = 0; kk < BK; ++kk) {
                float a[TM], b[TN];
                {
                    const float4 lo = *reinterpret_cast<const float4 *>(&As[buf][kk][ty * 4]);
                    a[0] = lo.x; a[1] = lo.y; a[2] = lo.z; a[3] = lo.w;
                    if (TM == 8) {
                        const float4 hi = *reinterpret_cast<const float4 *>(&As[buf][kk][BM / 2 + ty * 4]);
                        a[TM - 4] = hi.x; a[TM - 3] = hi.y; a[TM - 2] = hi.z; a[TM - 1] = hi.w;
                    }
                }
                {
                    const float4 lo = *reinterpret_cast<const float4 *>(&Bs[buf][kk][tx * 4]);
                    b[0] = lo.x; b[1] = lo.y; b[2] = lo.z; b[3] = lo.w;
                    if (TN == 8) {
                        const float4 hi = *reinterpret_cast<const float4 *>(&Bs[buf][kk][BN / 2 + tx * 4]);
                        b[TN - 4] = hi.x; b[TN - 3] = hi.y; b[TN - 2] = hi.z; b[TN - 1] = hi.w;
                    }
                }
#pragma unroll
                for (int i = 0; i < TM; ++i)
#pragma unroll
                    for (int j = 0; j < TN; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
            }
            if (more) {
                stash(buf ^ 1);
                __syncthreads();
                buf ^= 1;
            }
        }
    }
#pragma unroll
    for (int i = 0; i < TM; ++i) {
        const int64_t gi = m0 + (i < 4 ? ty * 4 + i : BM / 2 + ty * 4 + (i - 4));
        if (gi >= g.M) continue;
#pragma unroll
        for (int j = 0; j < TN; ++j) {
            const int64_t gj = n0 + (j < 4 ? tx * 4 + j : BN / 2 + tx * 4 + (j - 4));
            if (gj >= g.N) continue;
            epilogue<EM>(g, gi, gj, acc[i][j]);
        }
    }
}

template <int BM, int BN, int AM>
void launch_epi(cudaStream_t s, EpiMode em, const GemmArgs &g, dim3 grid) {
    if (em == EPI_STORE) sgemm_kernel<BM, BN, AM, EPI_STORE><<<grid, THREADS, 0, s>>>(g);
    else if (em == EPI_SUB) sgemm_kernel<BM, BN, AM, EPI_SUB><<<grid, THREADS, 0, s>>>(g);
    else if (em == EPI_BIAS) sgemm_kernel<BM, BN, AM, EPI_BIAS><<<grid, THREADS, 0, s>>>(g);
    else sgemm_kernel<BM, BN, AM, EPI_BGD_P><<<grid, THREADS, 0, s>>>(g);
}

template <int AM>
realq_status_t dispatch(cudaStream_t s, EpiMode em, const GemmArgs &g, const char *name) {
    const int64_t big_tiles = (int64_t)ceil_div(g.N, 128) * ceil_div(g.M, 128);
    const bool small = big_tiles < num_sms();
    {
        Launch L(name, s);
        const unsigned z = g.ksplit > 1 ? (unsigned)g.ksplit : 1u;
        if (small) launch_epi<64, 64, AM>(s, em, g, dim3(ceil_div(g.N, 64), ceil_div(g.M, 64), z));
        else launch_epi<128, 128, AM>(s, em, g, dim3(ceil_div(g.N, 128), ceil_div(g.M, 128), z));
    }
    return check_launch(name);
}

}  // namespace

realq_status_t gemm_f32(cudaStream_t s, AMode am, EpiMode em, const GemmArgs &g0, const char *name) {
    GemmArgs g = g0;
    if (g.nsum < 1) g.nsum = 1;
    if (g.nsum_b < 1) g.nsum_b = 1;
    if (g.ksplit > 1 && em != EPI_STORE) return fail(REALQ_ERR_UNSUPPORTED, "%s: split K needs a plain store", name);
    if (g.M <= 0 || g.N <= 0) return REALQ_OK;
    if (g.M > 64LL * 65535LL) return fail(REALQ_ERR_UNSUPPORTED, "%s: GEMM M too large (%lld)", name, (long long)g.M);
    switch (am) {
        case A_ROW: return dispatch<A_ROW>(s, em, g, name);
        case A_ROW_BF16: return dispatch<A_ROW_BF16>(s, em, g, name);
        case A_DIFF_F32: return dispatch<A_DIFF_F32>(s, em, g, name);
        case A_DIFF_BF16: return dispatch<A_DIFF_BF16>(s, em, g, name);
        default: return dispatch<A_KMAJOR>(s, em, g, name);
    }
}

}  // namespace realq
