// Step a2 (Sec. 3.2) on the 5th-generation tensor cores: H_sum += X̂^T X̂ for
// bf16 calibration activations.
//
// One CTA owns one 128 x 256 tile (128 channels i by 256 channels j, on or
// below the diagonal at 128-channel granularity) of H and a contiguous range
// of tokens.  X̂ is token-major (T x n), so both MMA operands are read
// MN-major straight from the activation rows: a TMA box of 64 tokens x 64
// channels (128-byte rows, 128-byte swizzle) is one canonical MN-major atom
// stack; two boxes make the 128-channel A operand and four the 256-channel B
// operand (LBO = 8 KB between boxes, SBO = 1 KB between 8-token groups), and
// one tcgen05.mma of M = 128, N = 256, K = 16 covers a 16-token step.  The
// wide tile halves the A traffic per flop and lets a 4-stage, 192 KB ring
// cover twice the MMA time of a 128 x 128 tile's.
//
// Precision: the tensor core's fp32 accumulation loses about one unit in the
// last place per accumulated MMA, in one direction, so a TMEM accumulator that
// takes all 2^18 tokens of a calibration set (2^14 MMAs) drifts by ~1e-3 of
// the entry.  The accumulation is therefore promoted: TMEM holds two 128 x 256
// accumulators, the MMA issuer switches between them every 1024 tokens, and
// the eight drain warps add each finished chunk into fp32 registers (IEEE
// adds) while the other accumulator fills.
//
// Roles (320 threads): warp 8 lane 0 issues TMA into a STAGES-deep ring,
// warp 9 lane 0 issues the MMAs and frees stages with tcgen05.commit; warps
// 0-7 drain the accumulators (warp w owns TMEM lanes 32 (w % 4).. and columns
// 128 (w / 4)..) and finally add their piece to H (mirrored below the
// diagonal block), or store it as a partial sum when tokens are split.
// The cross mode computes the full (non-symmetric) product X_Aᵀ X_B of two
// token-major inputs over all tiles, scaled by a sign and added to the output
// without mirroring: the cross moment of the perturbed-input surrogate is
// D = X̂ᵀX̂ - XᵀX̂, the symmetric pass (also added into D) minus this one.
// Every wait is bounded; on a timeout the tile is written as NaN (so the
// factorisation of H reports a non-finite pivot), the workspace status word
// gets ST_TIMEOUT, and the kernel still frees TMEM and returns.
#include "kernels.cuh"
#include "tc.cuh"

#include <mutex>

namespace realq {
namespace {

constexpr int TM = 128;                          // tile rows (channels i)
constexpr int TN = 256;                          // tile columns (channels j)
constexpr int KSTAGE = 64;                       // tokens per pipeline stage
constexpr int STAGES = 4;
constexpr int CHUNK_STAGES = 16;                 // default: 1024 tokens per TMEM accumulator pass
constexpr int DRAIN_WARPS = 8;                   // two per TMEM lane quarter, 128 columns each
constexpr int THREADS = (DRAIN_WARPS + 2) * 32;  // + the TMA warp and the MMA warp
constexpr int BOX_BYTES = 64 * KSTAGE * 2;       // one TMA box (64 channels x 64 tokens)
constexpr int A_BYTES = TM * KSTAGE * 2;         // 2 boxes
constexpr int B_BYTES = TN * KSTAGE * 2;         // 4 boxes
constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
constexpr int SMEM_BYTES = STAGES * STAGE_BYTES + 1024 + 256;
constexpr uint32_t IDESC = tc::idesc_bf16_f32(TM, TN, 1, 1);
constexpr unsigned FULL = 0xFFFFFFFFu;

// Tiles of the symmetric product: row block ti (128 channels) with every
// 256-wide column block tj that reaches the diagonal (256 tj <= 128 ti).
__host__ __device__ inline int64_t lower_tiles(int nti) {
    int64_t c = 0;
    for (int r = 0; r < nti; ++r) c += r / 2 + 1;
    return c;
}

// The lower tiles in groups of 8 row blocks: a group's tiles column by
// column (within a column, its rows that reach it), so that the CTAs resident
// at one time cover a compact block of the product and share their channel
// blocks through L2.  A bijection onto {(ti, tj): tj <= ti / 2, ti < nti}.
__device__ __forceinline__ void lower_tile(int64_t idx, int nti, int &ti, int &tj) {
    constexpr int G = 8;
    int r0 = 0;
    for (;; r0 += G) {
        const int r1 = min(r0 + G, nti);
        int64_t c = 0;
        for (int r = r0; r < r1; ++r) c += r / 2 + 1;
        if (idx < c || r1 >= nti) break;
        idx -= c;
    }
    const int r1 = min(r0 + G, nti);
    for (int j = 0;; ++j) {
        const int lo = max(r0, 2 * j);
        const int cnt = r1 > lo ? r1 - lo : 0;
        if (cnt == 0) {   // (not reached for idx < lower_tiles(nti))
            ti = r1 - 1;
            tj = 0;
            return;
        }
        if (idx < cnt) {
            ti = lo + (int)idx;
            tj = j;
            return;
        }
        idx -= cnt;
    }
}

__global__ void __launch_bounds__(THREADS, 1)
    hess_tc_kernel(const __grid_constant__ CUtensorMap tmap, const __grid_constant__ CUtensorMap tmapB, int64_t n,
                   int64_t T, int64_t tper, float *H, float *H2, float *part, int direct, int cross, int two_maps,
                   float sign, int chunk_stages, int *err) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint64_t *full = reinterpret_cast<uint64_t *>(smem + STAGES * STAGE_BYTES);
    uint64_t *empty = full + STAGES;
    uint64_t *accf = empty + STAGES;             // [2] accumulator b holds a finished chunk
    uint64_t *acce = accf + 2;                   // [2] accumulator b has been drained
    uint32_t *tslot = reinterpret_cast<uint32_t *>(acce + 2);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(tslot + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nti = (int)((n + TM - 1) / TM), ntj = (int)((n + TN - 1) / TN);
    int ti, tj;
    if (cross) {
        ti = (int)(blockIdx.x / ntj);
        tj = (int)(blockIdx.x % ntj);
    } else {
        lower_tile(blockIdx.x, nti, ti, tj);
    }
    const int i0 = ti * TM, j0 = tj * TN;
    const int64_t t_begin = (int64_t)blockIdx.y * tper;
    const int64_t t_end = min(T, t_begin + tper);
    const int nk = t_end > t_begin ? (int)((t_end - t_begin + KSTAGE - 1) / KSTAGE) : 0;
    const int nch = (nk + chunk_stages - 1) / chunk_stages;

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            tc::mbar_init(tc::smem_u32(&full[s]), 1);
            tc::mbar_init(tc::smem_u32(&empty[s]), 1);
        }
        for (int b = 0; b < 2; ++b) {
            tc::mbar_init(tc::smem_u32(&accf[b]), 1);
            tc::mbar_init(tc::smem_u32(&acce[b]), DRAIN_WARPS);
        }
        *abort_flag = 0;
        tc::fence_barrier_init();
        tc::prefetch_tmap(&tmap);
        if (two_maps) tc::prefetch_tmap(&tmapB);
    }
    if (warp == 0) tc::tmem_alloc(tc::smem_u32(tslot), 2 * TN);
    tc::fence_before_sync();
    __syncthreads();
    tc::fence_after_sync();
    const uint32_t tmem = *tslot;

    float acc[128];
#pragma unroll
    for (int c = 0; c < 128; ++c) acc[c] = 0.f;
    bool good = true;

    if (warp == DRAIN_WARPS) {
        if (lane == 0) {
            // ---------------- TMA producer ----------------
            const CUtensorMap *mb = two_maps ? &tmapB : &tmap;
            int it = 0;
            for (; it < nk; ++it) {
                const int s = it % STAGES;
                const uint32_t r = (uint32_t)(it / STAGES);
                if (!tc::mbar_wait(tc::smem_u32(&empty[s]), (r & 1u) ^ 1u, abort_flag)) {
                    *abort_flag = 1;
                    break;
                }
                const uint32_t fb = tc::smem_u32(&full[s]);
                tc::mbar_arrive_expect_tx(fb, STAGE_BYTES);
                const int y = (int)(t_begin + (int64_t)it * KSTAGE);
                const uint32_t a = tc::smem_u32(smem + s * STAGE_BYTES);
                tc::tma_load_2d(a, &tmap, fb, i0, y);
                tc::tma_load_2d(a + BOX_BYTES, &tmap, fb, i0 + 64, y);
#pragma unroll
                for (int q = 0; q < 4; ++q) tc::tma_load_2d(a + A_BYTES + q * BOX_BYTES, mb, fb, j0 + 64 * q, y);
            }
            // on abort, let the copies already issued land before the CTA exits
            if (*abort_flag) {
                int never = 0;
                for (int k = (it > STAGES ? it - STAGES : 0); k < it; ++k)
                    tc::mbar_wait(tc::smem_u32(&full[k % STAGES]), (uint32_t)(k / STAGES) & 1u, &never,
                                  100000000ull);
            }
        }
    } else if (warp == DRAIN_WARPS + 1) {
        if (lane == 0) {
            // ---------------- MMA issuer ----------------
            for (int c = 0; c < nch && !*abort_flag; ++c) {
                const int b = c & 1;
                if (c >= 2 && !tc::mbar_wait(tc::smem_u32(&acce[b]), (uint32_t)((c >> 1) - 1) & 1u, abort_flag)) {
                    *abort_flag = 1;
                    break;
                }
                tc::fence_after_sync();
                const uint32_t d = tmem + (uint32_t)(b * TN);
                const int it_end = min(nk, (c + 1) * chunk_stages);
                for (int it = c * chunk_stages; it < it_end; ++it) {
                    const int s = it % STAGES;
                    const uint32_t r = (uint32_t)(it / STAGES);
                    if (!tc::mbar_wait(tc::smem_u32(&full[s]), r & 1u, abort_flag)) {
                        *abort_flag = 1;
                        break;
                    }
                    tc::fence_after_sync();
                    const uint32_t a = tc::smem_u32(smem + s * STAGE_BYTES);
                    const uint32_t bop = a + A_BYTES;
                    const bool first = it == c * chunk_stages;
#pragma unroll
                    for (int k = 0; k < KSTAGE / 16; ++k) {
                        const uint64_t da = tc::smem_desc(a + k * 2048, BOX_BYTES, 1024, tc::SW_128B);
                        const uint64_t db = tc::smem_desc(bop + k * 2048, BOX_BYTES, 1024, tc::SW_128B);
                        tc::mma_bf16_ss(d, da, db, IDESC, (first && k == 0) ? 0u : 1u);
                    }
                    tc::mma_commit(tc::smem_u32(&empty[s]));
                }
                tc::mma_commit(tc::smem_u32(&accf[b]));
            }
        }
    } else {
        // ------- drain warps: TMEM chunk -> fp32 registers (lane quarter, column half) -------
        const uint32_t lane_base = (uint32_t)((warp & 3) * 32) << 16;
        const uint32_t col_base = (uint32_t)((warp >> 2) * 128);
        for (int c = 0; c < nch; ++c) {
            const int b = c & 1;
            const bool ok = tc::mbar_wait(tc::smem_u32(&accf[b]), (uint32_t)(c >> 1) & 1u, abort_flag);
            if (!__all_sync(FULL, ok)) {
                good = false;
                break;
            }
            tc::fence_after_sync();
#pragma unroll
            for (int c0 = 0; c0 < 128; c0 += 32) {
                uint32_t v[32];
                tc::tmem_ld_32x32b_x32(tmem + lane_base + (uint32_t)(b * TN) + col_base + (uint32_t)c0, v);
#pragma unroll
                for (int q = 0; q < 32; ++q) acc[c0 + q] += __uint_as_float(v[q]);
            }
            tc::fence_before_sync();
            __syncwarp();
            if (lane == 0) tc::mbar_arrive(tc::smem_u32(&acce[b]));
        }
    }
    __syncwarp();
    const bool all_good = __syncthreads_and(good && !*abort_flag) != 0;

    // ---------------- epilogue: registers -> global (drain warps) ----------------
    // Each drain warp owns a 32-row x 128-column piece, in 128-column block
    // jb of the matrix.  Symmetric product: jb < ti is added and mirrored,
    // jb == ti (the diagonal block) is added in full, jb > ti lies above the
    // diagonal and is left to the tile that holds its mirror image.
    if (warp < DRAIN_WARPS) {
        const int jb = 2 * tj + (warp >> 2);
        const bool write = cross || jb <= ti;
        const bool mirror = !cross && jb < ti;
        const int64_t gi = i0 + (warp & 3) * 32 + lane;
        const int64_t gj0 = (int64_t)jb * 128;
        if (write && gi < n) {
            if (!all_good) {
                // poison: the factorisation of H then reports a non-finite pivot
                for (int q = 0; q < 128 && gj0 + q < n; ++q) {
                    const int64_t gj = gj0 + q;
                    if (direct) {
                        H[gi * n + gj] = __int_as_float(0x7fc00000);
                        if (mirror) H[gj * n + gi] = __int_as_float(0x7fc00000);
                        if (H2) {
                            H2[gi * n + gj] = __int_as_float(0x7fc00000);
                            if (mirror) H2[gj * n + gi] = __int_as_float(0x7fc00000);
                        }
                    } else {
                        part[(int64_t)blockIdx.y * n * n + gi * n + gj] = __int_as_float(0x7fc00000);
                    }
                }
            } else if (nk > 0) {
#pragma unroll
                for (int q = 0; q < 128; ++q) {
                    const int64_t gj = gj0 + q;
                    if (gj < n) {
                        const float v = sign * acc[q];
                        if (direct) {
                            H[gi * n + gj] += v;
                            if (mirror) H[gj * n + gi] += v;
                            if (H2) {
                                H2[gi * n + gj] += v;
                                if (mirror) H2[gj * n + gi] += v;
                            }
                        } else {
                            part[(int64_t)blockIdx.y * n * n + gi * n + gj] = v;
                        }
                    }
                }
            }
        }
    }
    if (!all_good && threadIdx.x == 0 && err) atomicOr(err, ST_TIMEOUT);
    tc::fence_before_sync();
    __syncthreads();
    if (warp == 0) tc::tmem_dealloc(tmem, 2 * TN);
}

using EncodeFn = CUresult (*)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                              const cuuint64_t *, const cuuint32_t *, const cuuint32_t *, CUtensorMapInterleave,
                              CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
EncodeFn g_encode = nullptr;
std::once_flag g_encode_once;

}  // namespace

static CUresult encode_tmap_2d(CUtensorMapDataType dt, CUtensorMap *map, const void *base, uint64_t inner,
                               uint64_t outer, uint64_t row_stride_bytes, uint32_t box_inner, uint32_t box_outer,
                               int swizzle128);

CUresult encode_tmap_2d_bf16(CUtensorMap *map, const void *base, uint64_t inner, uint64_t outer,
                             uint64_t row_stride_bytes, uint32_t box_inner, uint32_t box_outer, int swizzle128) {
    return encode_tmap_2d(CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, map, base, inner, outer, row_stride_bytes, box_inner,
                          box_outer, swizzle128);
}

CUresult encode_tmap_2d_f32(CUtensorMap *map, const void *base, uint64_t inner, uint64_t outer,
                            uint64_t row_stride_bytes, uint32_t box_inner, uint32_t box_outer, int swizzle128) {
    return encode_tmap_2d(CU_TENSOR_MAP_DATA_TYPE_FLOAT32, map, base, inner, outer, row_stride_bytes, box_inner,
                          box_outer, swizzle128);
}

static CUresult encode_tmap_2d(CUtensorMapDataType dt, CUtensorMap *map, const void *base, uint64_t inner,
                               uint64_t outer, uint64_t row_stride_bytes, uint32_t box_inner, uint32_t box_outer,
                               int swizzle128) {
    std::call_once(g_encode_once, [] {
        void *fn = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            g_encode = reinterpret_cast<EncodeFn>(fn);
    });
    if (!g_encode) return CUDA_ERROR_NOT_FOUND;
    cuuint64_t dims[2] = {inner, outer};
    cuuint64_t strides[1] = {row_stride_bytes};
    cuuint32_t box[2] = {box_inner, box_outer};
    cuuint32_t estr[2] = {1, 1};
    return g_encode(map, dt, 2, const_cast<void *>(base), dims, strides, box, estr,
                    CU_TENSOR_MAP_INTERLEAVE_NONE,
                    swizzle128 == 2 ? CU_TENSOR_MAP_SWIZZLE_64B
                                    : (swizzle128 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_NONE),
                    CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
}

CUresult encode_tmap_2d_f16(CUtensorMap *map, const void *base, uint64_t inner, uint64_t outer,
                            uint64_t row_stride_bytes, uint32_t box_inner, uint32_t box_outer, int swizzle) {
    return encode_tmap_2d(CU_TENSOR_MAP_DATA_TYPE_FLOAT16, map, base, inner, outer, row_stride_bytes, box_inner,
                          box_outer, swizzle);
}

bool hessian_tc_eligible(int64_t n, int64_t T, const void *X) {
    return n >= 64 && n % 8 == 0 && (reinterpret_cast<uintptr_t>(X) & 15) == 0 && T > 0 && T < (1ll << 31) &&
           n < (1ll << 31);
}

// out (+= sign X_Aᵀ X_B); symmetric (X_B null): lower tiles mirrored, and
// out2 (if given) receives the same sum.  Token splits go through the
// workspace partials and a fixed-order reduction.
static realq_status_t hess_tc_launch(cudaStream_t s, int64_t n, int64_t T, const void *XA, const void *XB, float *out,
                                     float *out2, float sign, int *err, void *ws, size_t ws_bytes, int sms,
                                     const char *name, int chunk_stages = CHUNK_STAGES, bool sym_pair = false) {
    CUtensorMap mapA, mapB;
    CUresult cr = encode_tmap_2d_bf16(&mapA, XA, (uint64_t)n, (uint64_t)T, (uint64_t)n * 2, 64, KSTAGE, 1);
    if (cr == CUDA_SUCCESS && XB)
        cr = encode_tmap_2d_bf16(&mapB, XB, (uint64_t)n, (uint64_t)T, (uint64_t)n * 2, 64, KSTAGE, 1);
    if (cr != CUDA_SUCCESS) return fail(REALQ_ERR_CUDA, "cuTensorMapEncodeTiled failed (%d)", (int)cr);
    if (!XB) mapB = mapA;
    const int two_maps = XB != nullptr;
    const int cross = two_maps && !sym_pair;
    const int nti = ceil_div(n, TM), ntj = ceil_div(n, TN);
    const int64_t tiles = cross ? (int64_t)nti * ntj : lower_tiles(nti);
    int splits = hessian_splits_tiles(tiles, T, sms);
    const size_t per = (size_t)n * n * sizeof(float);
    if (splits > 1 && (ws == nullptr || ws_bytes < 2 * per)) splits = 1;
    if (splits > 1 && (size_t)splits * per > ws_bytes) splits = (int)(ws_bytes / per);
    int64_t tper = (T + splits - 1) / splits;
    tper = (tper + KSTAGE - 1) / KSTAGE * KSTAGE;
    splits = (int)((T + tper - 1) / tper);
    REALQ_TRY(set_smem_limit(reinterpret_cast<const void *>(hess_tc_kernel), SMEM_BYTES));
    float *part = static_cast<float *>(ws);
    {
        Launch L(name, s);
        hess_tc_kernel<<<dim3((unsigned)tiles, (unsigned)splits), THREADS, SMEM_BYTES, s>>>(
            mapA, mapB, n, T, tper, out, out2, part, splits == 1, cross, two_maps, sign, chunk_stages, err);
    }
    REALQ_TRY(check_launch(name));
    if (splits > 1) {
        REALQ_TRY(hessian_reduce(s, n, splits, part, out, cross ? 1 : 0));
        if (out2) REALQ_TRY(hessian_reduce(s, n, splits, part, out2, cross ? 1 : 0));
    }
    return REALQ_OK;
}

realq_status_t hessian_syrk_tc(cudaStream_t s, int64_t n, int64_t T, const void *X, float *H, int *err, void *ws,
                               size_t ws_bytes, int sms, float *H2) {
    return hess_tc_launch(s, n, T, X, nullptr, H, H2, 1.f, err, ws, ws_bytes, sms, "hessian_syrk_tc");
}

realq_status_t hessian_cross_tc(cudaStream_t s, int64_t n, int64_t T, const void *XA, const void *XB, float *out,
                                float sign, int *err, void *ws, size_t ws_bytes, int sms, int chunk_stages,
                                bool symmetric) {
    return hess_tc_launch(s, n, T, XA, XB, out, nullptr, sign, err, ws, ws_bytes, sms,
                          symmetric ? "hessian_weighted_tc" : "hessian_cross_tc",
                          chunk_stages > 0 ? chunk_stages : CHUNK_STAGES, symmetric);
}

}  // namespace realq
