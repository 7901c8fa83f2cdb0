// Step a2 (Sec. 3.2): H_sum += X̂^T X̂ and D_sum += (X̂ - X)^T X̂ over one chunk
// of calibration tokens, CUDA-core fp32 version.  Only tile pairs on or below
// the diagonal of H are computed; each result is added to its tile and to the
// mirrored tile.  When there are too few tiles to fill the GPU the tokens are
// split over `splits` CTAs per tile whose partial sums go to the workspace and
// are reduced in a fixed order (bitwise repeatable).
#include "kernels.cuh"

#include <cmath>

namespace realq {
namespace {

constexpr int TB = 128, TK = 8, THREADS = 256;

__device__ __forceinline__ float ldx(const float *p, int64_t i) { return p[i]; }
__device__ __forceinline__ float ldx(const __nv_bfloat16 *p, int64_t i) { return __bfloat162float(p[i]); }

__device__ __forceinline__ void tile_of(int64_t idx, int lower_only, int nt, int &ti, int &tj) {
    if (lower_only) {
        int r = (int)((sqrt(8.0 * (double)idx + 1.0) - 1.0) * 0.5);
        while ((int64_t)(r + 1) * (r + 2) / 2 <= idx) ++r;
        while ((int64_t)r * (r + 1) / 2 > idx) --r;
        ti = r;
        tj = (int)(idx - (int64_t)r * (r + 1) / 2);
    } else {
        ti = (int)(idx / nt);
        tj = (int)(idx % nt);
    }
}

// mode 0: out += X̂^T X̂ (symmetric, lower tiles + mirror)
// mode 1: out += (X̂ - X)^T X̂ (all tiles)
// direct = 1: accumulate into out; else store partial sums to part + split * n * n
template <typename TX, int MODE>
__global__ void __launch_bounds__(THREADS) hess_kernel(int64_t n, int64_t T, const TX *Xh, const TX *Xf, float *out,
                                                       float *part, int64_t tper, int direct) {
    __shared__ __align__(16) float As[TK][TB + 4];
    __shared__ __align__(16) float Bs[TK][TB + 4];
    const int nt = (int)((n + TB - 1) / TB);
    int ti, tj;
    tile_of(blockIdx.x, MODE == 0, nt, ti, tj);
    const int64_t i0 = (int64_t)ti * TB, j0 = (int64_t)tj * TB;
    const int64_t t_begin = (int64_t)blockIdx.y * tper;
    const int64_t t_end = min(T, t_begin + tper);
    const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
    float acc[8][8];
#pragma unroll
    for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int j = 0; j < 8; ++j) acc[i][j] = 0.f;

    for (int64_t t0 = t_begin; t0 < t_end; t0 += TK) {
#pragma unroll
        for (int r = 0; r < (TB * TK) / THREADS; ++r) {
            const int idx = tid + r * THREADS;
            const int kk = idx / TB, cc = idx % TB;
            const int64_t t = t0 + kk;
            const bool tin = t < t_end;
            const int64_t gi = i0 + cc, gj = j0 + cc;
            float a = 0.f, b = 0.f;
            if (tin && gi < n) {
                a = ldx(Xh, t * n + gi);
                if (MODE == 1) a -= ldx(Xf, t * n + gi);
            }
            if (tin && gj < n) b = ldx(Xh, t * n + gj);
            As[kk][cc] = a;
            Bs[kk][cc] = b;
        }
        __syncthreads();
#pragma unroll
        for (int kk = 0; kk < TK; ++kk) {
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
    float *dst = direct ? out : part + (int64_t)blockIdx.y * n * n;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        const int64_t gi = i0 + (i < 4 ? ty * 4 + i : 64 + ty * 4 + (i - 4));
        if (gi >= n) continue;
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            const int64_t gj = j0 + (j < 4 ? tx * 4 + j : 64 + tx * 4 + (j - 4));
            if (gj >= n) continue;
            if (direct) {
                dst[gi * n + gj] += acc[i][j];
                if (MODE == 0 && ti != tj) dst[gj * n + gi] += acc[i][j];
            } else {
                dst[gi * n + gj] = acc[i][j];
            }
        }
    }
}

// out[i][j] += sum_s part[s][i][j] in split order; mirrored for mode 0
template <int MODE>
__global__ void hess_reduce_kernel(int64_t n, int splits, const float *part, float *out) {
    const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= n * n) return;
    const int64_t i = idx / n, j = idx % n;
    const int64_t ti = i / TB, tj = j / TB;
    if (MODE == 0 && ti < tj) return;
    float s = 0.f;
    for (int k = 0; k < splits; ++k) s += part[(int64_t)k * n * n + idx];
    out[idx] += s;
    if (MODE == 0 && ti > tj) out[j * n + i] += s;
}

template <typename TX>
realq_status_t run(cudaStream_t s, int64_t n, int64_t T, const TX *X, const TX *Xf, float *H, float *D, void *ws,
                   size_t ws_bytes) {
    const int nt = ceil_div(n, TB);
    const int64_t lower = (int64_t)nt * (nt + 1) / 2;
    int splits = hessian_splits(n, T, num_sms());
    const size_t per = (size_t)n * n * sizeof(float) * (Xf ? 2 : 1);
    if (splits > 1 && (ws == nullptr || ws_bytes < per * 2)) splits = 1;
    if (splits > 1 && (size_t)splits * per > ws_bytes) splits = (int)(ws_bytes / per);
    const int64_t tper = (T + splits - 1) / splits;
    float *partH = static_cast<float *>(ws);
    float *partD = partH + (size_t)splits * n * n;
    const int direct = splits == 1;
    if (H) {
        {
            Launch L("hessian_syrk_simt", s);
            hess_kernel<TX, 0><<<dim3((unsigned)lower, splits), THREADS, 0, s>>>(n, T, X, nullptr, H, partH, tper,
                                                                                 direct);
        }
        REALQ_TRY(check_launch("hessian_syrk_simt"));
        if (!direct) REALQ_TRY(hessian_reduce(s, n, splits, partH, H, 0));
    }
    if (Xf) {
        {
            Launch L("hessian_cross_simt", s);
            hess_kernel<TX, 1><<<dim3((unsigned)((int64_t)nt * nt), splits), THREADS, 0, s>>>(n, T, X, Xf, D, partD,
                                                                                             tper, direct);
        }
        REALQ_TRY(check_launch("hessian_cross_simt"));
        if (!direct) REALQ_TRY(hessian_reduce(s, n, splits, partD, D, 1));
    }
    return REALQ_OK;
}

}  // namespace

int num_sms() {
    static int v = 0;
    if (v == 0) {
        int dev = 0, c = 0;
        if (cudaGetDevice(&dev) == cudaSuccess &&
            cudaDeviceGetAttribute(&c, cudaDevAttrMultiProcessorCount, dev) == cudaSuccess && c > 0)
            v = c;
        else
            v = 152;
    }
    return v;
}

realq_status_t hessian_reduce(cudaStream_t s, int64_t n, int splits, const float *part, float *out, int mode) {
    const unsigned blocks = (unsigned)((n * n + 255) / 256);
    {
        Launch L("hessian_reduce", s);
        if (mode == 0) hess_reduce_kernel<0><<<blocks, 256, 0, s>>>(n, splits, part, out);
        else hess_reduce_kernel<1><<<blocks, 256, 0, s>>>(n, splits, part, out);
    }
    return check_launch("hessian_reduce");
}

int hessian_splits(int64_t n, int64_t T, int sms) {
    // tiles of the tensor-core symmetric product: 128-channel row blocks by
    // 256-channel column blocks reaching the diagonal
    const int nti = ceil_div(n, 128);
    int64_t tiles = 0;
    for (int r = 0; r < nti; ++r) tiles += r / 2 + 1;
    return hessian_splits_tiles(tiles, T, sms);
}

// Token splits of a tile grid: the count that minimises the rounds of waves
// per unit of work, ceil(tiles s / sms) / s, plus a small cost per split for
// the partial sums and their reduction; at least 4096 tokens per split and at
// most 16 splits.
int hessian_splits_tiles(int64_t tiles, int64_t T, int sms) {
    int64_t max_s = T / 4096;
    if (max_s > 16) max_s = 16;
    if (max_s < 1) max_s = 1;
    double best = 1e300;
    int bs = 1;
    for (int s2 = 1; s2 <= max_s; ++s2) {
        const int64_t rounds = (tiles * s2 + sms - 1) / sms;
        const double cost = (double)rounds / s2 + 0.01 * s2;
        if (cost < best - 1e-12) {
            best = cost;
            bs = s2;
        }
    }
    return bs;
}

size_t hessian_ws_bytes(int64_t n, int64_t T, int has_xfp) {
    size_t b = align_up(sizeof(int));
    const int splits = hessian_splits(n, T, 152);
    if (splits > 1) b += (size_t)splits * n * n * sizeof(float) * (has_xfp ? 2 : 1);
    return b;
}

realq_status_t hessian_accumulate(cudaStream_t s, int64_t n, int64_t T, const void *X, const void *Xfp,
                                  realq_dtype_t dt, float *H, float *D, void *ws, size_t ws_bytes) {
    if (T == 0) return REALQ_OK;
    int *err = nullptr;
    char *pw = nullptr;
    size_t pbytes = 0;
    if (ws && ws_bytes >= align_up(sizeof(int))) {
        err = static_cast<int *>(ws);
        pw = static_cast<char *>(ws) + align_up(sizeof(int));
        pbytes = ws_bytes - align_up(sizeof(int));
    }
    const bool tc_path = dt == REALQ_BF16 && hessian_tc_eligible(n, T, X);
    const bool tc_cross = tc_path && Xfp && hessian_tc_eligible(n, T, Xfp);
    // tensor cores: H += X̂ᵀX̂ (and D += X̂ᵀX̂ from the same pass), D -= XᵀX̂
    if (tc_path) REALQ_TRY(hessian_syrk_tc(s, n, T, X, H, err, pw, pbytes, num_sms(), tc_cross ? D : nullptr));
    if (tc_cross) REALQ_TRY(hessian_cross_tc(s, n, T, Xfp, X, D, -1.f, err, pw, pbytes, num_sms()));
    float *Hs = tc_path ? nullptr : H;
    if (tc_cross) {
        Xfp = nullptr;
        D = nullptr;
    }
    if (dt == REALQ_BF16)
        return run<__nv_bfloat16>(s, n, T, static_cast<const __nv_bfloat16 *>(X),
                                  static_cast<const __nv_bfloat16 *>(Xfp), Hs, D, pw, pbytes);
    return run<float>(s, n, T, static_cast<const float *>(X), static_cast<const float *>(Xfp), Hs, D, pw, pbytes);
}

}  // namespace realq
