// Block-GD contractions (Eq. block_gd_update) on the 5th-generation tensor
// cores with fp32-level accuracy: three tf32 products per term,
//   a b ~= a_hi b_hi + a_hi b_lo + a_lo b_hi,
// where a_hi keeps a's top 11 significand bits (exact in tf32) and
// a_lo = a - a_hi.  The dropped a_lo b_lo and the tf32 rounding of the lo
// parts leave ~2^-20 relative error per product, below the fp32 rounding of
// the K-long accumulation itself; the gradient's sign, which Adam's first
// step depends on, is then as reliable as with fp32 FFMA.
//
// C[M x N] = A[M x K] B[N x K]^T with both operands K-major in global memory
// (rows of A, rows of B), each as a hi and a lo plane.  One CTA computes a
// 128 x 128 tile: TMA loads 32-wide K slices of the four planes (128-byte
// rows, 128-byte swizzle) into a 3-stage ring, one thread issues
// 3 x 4 tcgen05.mma (kind::tf32, K = 8) per stage into a TMEM accumulator,
// and eight warps drain it through one of the epilogues (the epilogues are
// bound by the latency of their global loads, so every warp of the CTA
// takes part):
//   TC_STORE  C = acc
//   TC_BGD_P  the Block-GD gradient factor after the lazy OBS update: the
//             running product M = A_disp H̄ takes the latest step (acc),
//             M += acc, and p = M + lambda (A_disp - (W - W0)) (+ W0 Dbar),
//             0 on dead channels, written transposed and split (P^T hi / lo)
//   TC_ADAM   g = acc: one Adam (or SGD) step on W[:, col0 + j], updating the
//             moments and the displacement, and writing the step's hi / lo
//             planes for the next M update
//   TC_ACCUM  M += acc (the running product of one row group)
//   TC_SYRK   M[i][j] -= acc for j >= i only (a symmetric rank-K update of
//             the upper triangle of M; tiles wholly below the diagonal exit
//             at once)
//   TC_BGD_PG the gradient factor of a row group whose OBS used its own
//             H̄_g:  p = M + lambda_g (A_disp - (W - W0)) - acc (+ W0 Dbar),
//             acc = ΔW (H̄_g - H̄); written like TC_BGD_P
// The A operand starts at row a_row0 of its planes (a row group), and the
// epilogue pointers are offset to that row by the caller.  The epilogue is a
// template parameter (one kernel per mode).  With TC_STORE, K may be split
// over grid z (slice z writes its partial tile at C + z czs; a separate
// pass sums the slices in order), and an operand exact in tf32 (a bf16 input
// widened to fp32) skips its low plane: neither loaded nor multiplied.
#include "kernels.cuh"
#include "tc.cuh"

namespace realq {
namespace {

constexpr int TB = 128;                       // tile rows (M)
constexpr int THREADS = 256;                  // 8 warps; warp 0 lane 0 loads, warp 1 lane 0 issues MMAs

// Two tile shapes.  Each tcgen05.mma reads both operands from shared memory,
// and the three products of a K step read A twice and B twice; with the TMA
// writes of the ring that is about 190 bytes of shared-memory traffic per
// cycle for a 128 x 128 tile at the tensor pipe's tf32 rate, above the
// 128 bytes per cycle an SM serves, so that tile tops out near two thirds of
// the pipe.  A 128 x 256 tile reuses each A row for twice the columns
// (about 145 bytes per cycle): it takes 16-wide K slices (64-byte rows,
// 64-byte swizzle) so that a 4-deep ring of both planes still fits.
//
// With fp16 planes (F16) a slice row holds twice the elements in the same
// bytes, each MMA (kind::f16, K = 16) advances 32 bytes as a tf32 MMA (K = 8)
// does, and the f16 rate is twice the tf32 rate: the same kernel at twice the
// flops per byte of shared memory.
template <int TN, bool F16 = false>
struct Tile {
    static constexpr int KB = TN == 256 ? 64 : 128;            // bytes per row of a K slice
    static constexpr int KS = KB / (F16 ? 2 : 4);              // elements per K slice
    static constexpr int STAGES = TN == 256 ? 4 : 3;
    static constexpr uint32_t SWZ = TN == 256 ? tc::SW_64B : tc::SW_128B;
    static constexpr uint32_t SBO = TN == 256 ? 512 : 1024;   // 8 rows of one swizzle atom
    static constexpr int PLANE_A = TB * KB;
    static constexpr int PLANE_B = TN * KB;
    static constexpr int STAGE_BYTES = 2 * PLANE_A + 2 * PLANE_B;   // A hi, A lo, B hi, B lo
    static constexpr int SMEM = STAGES * STAGE_BYTES + 1024 + 256;
    static constexpr uint32_t IDESC = F16 ? tc::idesc_f16_f32(TB, TN) : tc::idesc_tf32_f32(TB, TN);
    static_assert(STAGES * STAGE_BYTES >= TB * (TN + 1) * 4, "epilogue tile must fit the ring");
};

struct Maps {
    CUtensorMap a_hi, a_lo, b_hi, b_lo;
};
// (narrow: the 128 x 128 tile's boxes; wide: the 128 x 256 tile's)
struct MapPair {
    Maps narrow, wide;
};

// M += acc; p = M + lambda (A_disp - (W - W0)) (+ W0 Dbar), 0 on dead channels
__device__ __forceinline__ float bgd_p_value(const TcEpi &e, int64_t i, int64_t j, float v) {
    const int64_t col = e.col0 + j;
    const int64_t w = i * e.ldw + col;
    const float w0 = e.w0_bf16 ? __bfloat162float(static_cast<const __nv_bfloat16 *>(e.W0)[w])
                               : static_cast<const float *>(e.W0)[w];
    v += e.M[w];
    e.M[w] = v;
    float p = v + (*e.lam) * (e.Ad[w] - (e.W[w] - w0));
    if (e.R0) p += e.R0[w];
    if (e.dead && e.dead[col]) p = 0.f;
    return p;
}

// TC_BGD_PG: p = M + lambda (A_disp - (W - W0)) - acc (+ W0 Dbar), 0 on dead channels
__device__ __forceinline__ float bgd_pg_value(const TcEpi &e, int64_t i, int64_t j, float v) {
    const int64_t col = e.col0 + j;
    const int64_t w = i * e.ldw + col;
    const float w0 = e.w0_bf16 ? __bfloat162float(static_cast<const __nv_bfloat16 *>(e.W0)[w])
                               : static_cast<const float *>(e.W0)[w];
    float p = e.M[w] - v + (*e.lam) * (e.Ad[w] - (e.W[w] - w0));
    if (e.R0) p += e.R0[w];
    if (e.dead && e.dead[col]) p = 0.f;
    return p;
}

__device__ __forceinline__ float4 ld4(const float *p) { return *reinterpret_cast<const float4 *>(p); }
__device__ __forceinline__ void st4(float *p, float4 v) { *reinterpret_cast<float4 *>(p) = v; }
__device__ __forceinline__ float4 ld4_w0(const TcEpi &e, int64_t w) {
    if (e.w0_bf16) {
        const uint2 u = *reinterpret_cast<const uint2 *>(static_cast<const __nv_bfloat16 *>(e.W0) + w);
        return make_float4(__uint_as_float(u.x << 16), __uint_as_float(u.x & 0xFFFF0000u),
                           __uint_as_float(u.y << 16), __uint_as_float(u.y & 0xFFFF0000u));
    }
    return ld4(static_cast<const float *>(e.W0) + w);
}

// Gradient factor for 4 rows x 4 columns (rows gi0..gi0+3 and columns
// gj..gj+3 all inside the output); t points at the tile entry of row 0,
// column 0 of the 4x4 patch, pitch tp.  All loads are issued first.
__device__ __forceinline__ void bgd_p_rows4(const TcEpi &e, int64_t gi0, int64_t M, int64_t gj, float *t, int tp) {
    const int64_t col = e.col0 + gj;
    float4 a[4], w[4], w0[4], r0[4], mp[4];
    uchar4 dd = make_uchar4(0, 0, 0, 0);
    if (e.dead) dd = *reinterpret_cast<const uchar4 *>(e.dead + col);
#pragma unroll
    for (int u = 0; u < 4; ++u) {
        const int64_t wi = (gi0 + u) * e.ldw + col;
        mp[u] = ld4(e.M + wi);
        a[u] = ld4(e.Ad + wi);
        w[u] = ld4(e.W + wi);
        w0[u] = ld4_w0(e, wi);
        r0[u] = e.R0 ? ld4(e.R0 + wi) : make_float4(0.f, 0.f, 0.f, 0.f);
    }
    const float lam = *e.lam;
#pragma unroll
    for (int u = 0; u < 4; ++u) {
        float *tr = t + u * tp;
        const float4 mn = make_float4(tr[0] + mp[u].x, tr[1] + mp[u].y, tr[2] + mp[u].z, tr[3] + mp[u].w);
        st4(e.M + (gi0 + u) * e.ldw + col, mn);
        tr[0] = mn.x; tr[1] = mn.y; tr[2] = mn.z; tr[3] = mn.w;
        tr[0] = dd.x ? 0.f : tr[0] + lam * (a[u].x - (w[u].x - w0[u].x)) + r0[u].x;
        tr[1] = dd.y ? 0.f : tr[1] + lam * (a[u].y - (w[u].y - w0[u].y)) + r0[u].y;
        tr[2] = dd.z ? 0.f : tr[2] + lam * (a[u].z - (w[u].z - w0[u].z)) + r0[u].z;
        tr[3] = dd.w ? 0.f : tr[3] + lam * (a[u].w - (w[u].w - w0[u].w)) + r0[u].w;
    }
}

// TC_BGD_PG for 4 rows x 4 columns (same shape rules as bgd_p_rows4).
__device__ __forceinline__ void bgd_pg_rows4(const TcEpi &e, int64_t gi0, int64_t gj, float *t, int tp) {
    const int64_t col = e.col0 + gj;
    float4 a[4], w[4], w0[4], r0[4], mp[4];
    uchar4 dd = make_uchar4(0, 0, 0, 0);
    if (e.dead) dd = *reinterpret_cast<const uchar4 *>(e.dead + col);
#pragma unroll
    for (int u = 0; u < 4; ++u) {
        const int64_t wi = (gi0 + u) * e.ldw + col;
        mp[u] = ld4(e.M + wi);
        a[u] = ld4(e.Ad + wi);
        w[u] = ld4(e.W + wi);
        w0[u] = ld4_w0(e, wi);
        r0[u] = e.R0 ? ld4(e.R0 + wi) : make_float4(0.f, 0.f, 0.f, 0.f);
    }
    const float lam = *e.lam;
#pragma unroll
    for (int u = 0; u < 4; ++u) {
        float *tr = t + u * tp;
        tr[0] = dd.x ? 0.f : mp[u].x - tr[0] + lam * (a[u].x - (w[u].x - w0[u].x)) + r0[u].x;
        tr[1] = dd.y ? 0.f : mp[u].y - tr[1] + lam * (a[u].y - (w[u].y - w0[u].y)) + r0[u].y;
        tr[2] = dd.z ? 0.f : mp[u].z - tr[2] + lam * (a[u].z - (w[u].z - w0[u].z)) + r0[u].z;
        tr[3] = dd.w ? 0.f : mp[u].w - tr[3] + lam * (a[u].w - (w[u].w - w0[u].w)) + r0[u].w;
    }
}

// TC_ACCUM for 4 rows x 4 columns: M += acc
__device__ __forceinline__ void accum_rows4(const TcEpi &e, int64_t gi0, int64_t gj, const float *t, int tp) {
    const int64_t col = e.col0 + gj;
    float4 mp[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) mp[u] = ld4(e.M + (gi0 + u) * e.ldw + col);
#pragma unroll
    for (int u = 0; u < 4; ++u) {
        const float *tr = t + u * tp;
        st4(e.M + (gi0 + u) * e.ldw + col,
            make_float4(mp[u].x + tr[0], mp[u].y + tr[1], mp[u].z + tr[2], mp[u].w + tr[3]));
    }
}

// TC_SYRK for 4 rows x 4 columns: M -= acc on and above the diagonal
__device__ __forceinline__ void syrk_rows4(const TcEpi &e, int64_t gi0, int64_t gj, const float *t, int tp) {
    float4 mp[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) mp[u] = ld4(e.M + (gi0 + u) * e.ldw + gj);
#pragma unroll
    for (int u = 0; u < 4; ++u) {
        const float *tr = t + u * tp;
        const int64_t gi = gi0 + u;
        st4(e.M + gi * e.ldw + gj,
            make_float4(gj + 0 >= gi ? mp[u].x - tr[0] : mp[u].x, gj + 1 >= gi ? mp[u].y - tr[1] : mp[u].y,
                        gj + 2 >= gi ? mp[u].z - tr[2] : mp[u].z, gj + 3 >= gi ? mp[u].w - tr[3] : mp[u].w));
    }
}

__device__ __forceinline__ float adam_step(const TcEpi &e, float g, float &m, float &v) {
    if (e.sgd) return e.lr * g;
    m = e.b1 * m + (1.f - e.b1) * g;
    v = e.b2 * v + (1.f - e.b2) * g * g;
    return e.lr * (m / e.bc1) / (sqrtf(v / e.bc2) + e.eps);
}

// Optimizer step for 4 rows x 4 columns of the free block (same shape rules).
__device__ __forceinline__ void adam_rows4(const TcEpi &e, int64_t gi0, int64_t M, int64_t gj, const float *t, int tp) {
    const int64_t col = e.col0 + gj;
    float4 m[4], v[4], w[4], d[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
        const int64_t wi = (gi0 + u) * e.ldw + col;
        if (!e.sgd) {
            m[u] = ld4(e.mA + wi);
            v[u] = ld4(e.vA + wi);
        }
        w[u] = ld4(e.Wm + wi);
        d[u] = ld4(e.D + wi);
    }
#pragma unroll
    for (int u = 0; u < 4; ++u) {
        const int64_t wi = (gi0 + u) * e.ldw + col;
        const float *tr = t + u * tp;
        float4 st;
        st.x = adam_step(e, tr[0], m[u].x, v[u].x);
        st.y = adam_step(e, tr[1], m[u].y, v[u].y);
        st.z = adam_step(e, tr[2], m[u].z, v[u].z);
        st.w = adam_step(e, tr[3], m[u].w, v[u].w);
        if (!e.sgd) {
            st4(e.mA + wi, m[u]);
            st4(e.vA + wi, v[u]);
        }
        st4(e.Wm + wi, make_float4(w[u].x - st.x, w[u].y - st.y, w[u].z - st.z, w[u].w - st.w));
        st4(e.D + wi, make_float4(d[u].x - st.x, d[u].y - st.y, d[u].z - st.z, d[u].w - st.w));
        // the displacement moved by -st: its planes (or, for f16 planes, -st
        // itself, split later) feed the next M update
        if (!e.Sl) {
            st4(e.Sh + wi, make_float4(-st.x, -st.y, -st.z, -st.w));
            continue;
        }
        const float4 sh = make_float4(tc::tf32_hi(-st.x), tc::tf32_hi(-st.y), tc::tf32_hi(-st.z), tc::tf32_hi(-st.w));
        st4(e.Sh + wi, sh);
        st4(e.Sl + wi, make_float4(-st.x - sh.x, -st.y - sh.y, -st.z - sh.z, -st.w - sh.w));
    }
}

__device__ __forceinline__ void epi_apply(const TcEpi &e, int64_t i, int64_t j, float v) {
    if (e.mode == TC_STORE) {
        e.C[i * e.ldc + j] = v;
        return;
    }
    if (e.mode == TC_ACCUM) {
        e.M[i * e.ldw + e.col0 + j] += v;
        return;
    }
    if (e.mode == TC_SYRK) {
        if (j >= i) e.M[i * e.ldw + j] -= v;
        return;
    }
    const int64_t col = e.col0 + j;
    const int64_t w = i * e.ldw + col;
    // TC_ADAM
    float step;
    if (e.sgd) {
        step = e.lr * v;
    } else {
        const float mv = e.b1 * e.mA[w] + (1.f - e.b1) * v;
        const float vv = e.b2 * e.vA[w] + (1.f - e.b2) * v * v;
        e.mA[w] = mv;
        e.vA[w] = vv;
        step = e.lr * (mv / e.bc1) / (sqrtf(vv / e.bc2) + e.eps);
    }
    e.Wm[w] -= step;
    e.D[w] -= step;
    if (!e.Sl) {
        e.Sh[w] = -step;
        return;
    }
    const float sh = tc::tf32_hi(-step);
    e.Sh[w] = sh;
    e.Sl[w] = -step - sh;
}

// MODE = e.mode, fixed at compile time: one kernel per epilogue (and so one
// name per role in a profiler's launch list); TN = the tile's width; F16 =
// fp16 planes with row scales (f16x3) instead of tf32 planes.
template <int MODE, int TN, bool F16>
__global__ void __launch_bounds__(THREADS, 1)
    gemm_x3_kernel(const __grid_constant__ Maps maps, int64_t M, int64_t N, int64_t K, int k_off, int b_row0,
                       int a_row0, const TcEpi e, int *err, int kchunk, int exact) {
    using TL = Tile<TN, F16>;
    constexpr int KS = TL::KS, STAGES = TL::STAGES, PLANE_A = TL::PLANE_A, PLANE_B = TL::PLANE_B;
    constexpr int STAGE_BYTES = TL::STAGE_BYTES;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint64_t *full = reinterpret_cast<uint64_t *>(smem + STAGES * STAGE_BYTES);
    uint64_t *empty = full + STAGES;
    uint64_t *accb = empty + STAGES;
    uint32_t *tslot = reinterpret_cast<uint32_t *>(accb + 1);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(tslot + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    // Tiles in groups of up to 8 row tiles: consecutive CTAs walk down a
    // group's rows before moving right, so that the CTAs resident at one time
    // cover a compact block of the output and share their A rows and B rows
    // through L2 (row-major order had each wave stream every B row of the
    // product from DRAM again).  A bijection of the tiles: every tile is
    // computed exactly as before.
    int64_t ti, tj;
    {
        const int64_t nx = gridDim.x, ny = gridDim.y;
        const int64_t pid = (int64_t)blockIdx.y * nx + blockIdx.x;
        constexpr int64_t GROUP = 8;
        const int64_t per = GROUP * nx, first = (pid / per) * GROUP;
        const int64_t gm = (ny - first) < GROUP ? (ny - first) : GROUP;
        ti = first + (pid % per) % gm;
        tj = (pid % per) / gm;
    }
    const int64_t i0 = ti * TB, j0 = tj * TN;
    // a symmetric update touches the upper triangle only: a tile wholly
    // below the diagonal has nothing to do (uniform over the CTA, before any
    // barrier or allocation)
    if (MODE == TC_SYRK && j0 + TN <= i0) return;
    // K split over blockIdx.z: this CTA takes K range [kz0, kz0 + Kz)
    const int64_t kz0 = kchunk > 0 ? (int64_t)blockIdx.z * kchunk : 0;
    int64_t Kz = kchunk > 0 ? ((K - kz0) < kchunk ? (K - kz0) : kchunk) : K;
    // a triangular B (zero beyond the output column): this tile's K range
    // ends at its last column (the wrapper takes no K split with it)
    if (e.b_tri && Kz > j0 + TN) Kz = j0 + TN;
    const int nk = (int)((Kz + KS - 1) / KS);

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            tc::mbar_init(tc::smem_u32(&full[s]), 1);
            tc::mbar_init(tc::smem_u32(&empty[s]), 1);
        }
        tc::mbar_init(tc::smem_u32(accb), 1);
        *abort_flag = 0;
        tc::fence_barrier_init();
        tc::prefetch_tmap(&maps.a_hi);
        tc::prefetch_tmap(&maps.a_lo);
        tc::prefetch_tmap(&maps.b_hi);
        tc::prefetch_tmap(&maps.b_lo);
    }
    if (warp == 0) tc::tmem_alloc(tc::smem_u32(tslot), TN);
    tc::fence_before_sync();
    __syncthreads();
    tc::fence_after_sync();
    const uint32_t tmem = *tslot;

    if (warp == 0 && lane == 0) {
        // ---------------- TMA producer ----------------
        int it = 0;
        for (; it < nk; ++it) {
            const int s = it % STAGES;
            const uint32_t r = (uint32_t)(it / STAGES);
            if (!tc::mbar_wait(tc::smem_u32(&empty[s]), (r & 1u) ^ 1u, abort_flag)) {
                *abort_flag = 1;
                break;
            }
            const uint32_t fb = tc::smem_u32(&full[s]);
            // an operand exact in tf32 (exact & 1: A, exact & 2: B) has no
            // low plane to load or multiply
            tc::mbar_arrive_expect_tx(fb, STAGE_BYTES - ((exact & 1) ? PLANE_A : 0) - ((exact & 2) ? PLANE_B : 0));
            const int x = k_off + (int)kz0 + it * KS;
            const uint32_t base = tc::smem_u32(smem + s * STAGE_BYTES);
            tc::tma_load_2d(base, &maps.a_hi, fb, x, a_row0 + (int)i0);
            if (!(exact & 1)) tc::tma_load_2d(base + PLANE_A, &maps.a_lo, fb, x, a_row0 + (int)i0);
            tc::tma_load_2d(base + 2 * PLANE_A, &maps.b_hi, fb, x, b_row0 + (int)j0);
            if (!(exact & 2)) tc::tma_load_2d(base + 2 * PLANE_A + PLANE_B, &maps.b_lo, fb, x, b_row0 + (int)j0);
        }
        if (*abort_flag) {
            int never = 0;
            for (int k = (it > STAGES ? it - STAGES : 0); k < it; ++k)
                tc::mbar_wait(tc::smem_u32(&full[k % STAGES]), (uint32_t)(k / STAGES) & 1u, &never, 100000000ull);
        }
    } else if (warp == 1 && lane == 0 && nk > 0) {
        // ---------------- MMA issuer ----------------
        for (int it = 0; it < nk; ++it) {
            const int s = it % STAGES;
            const uint32_t r = (uint32_t)(it / STAGES);
            if (!tc::mbar_wait(tc::smem_u32(&full[s]), r & 1u, abort_flag)) {
                *abort_flag = 1;
                break;
            }
            tc::fence_after_sync();
            const uint32_t base = tc::smem_u32(smem + s * STAGE_BYTES);
#pragma unroll
            for (int k = 0; k < TL::KB / 32; ++k) {
                // K step k: 32 bytes (8 fp32 or 16 fp16) into every row of the swizzle atom
                const uint64_t ah = tc::smem_desc(base + k * 32, 16, TL::SBO, TL::SWZ);
                const uint64_t al = tc::smem_desc(base + PLANE_A + k * 32, 16, TL::SBO, TL::SWZ);
                const uint64_t bh = tc::smem_desc(base + 2 * PLANE_A + k * 32, 16, TL::SBO, TL::SWZ);
                const uint64_t bl = tc::smem_desc(base + 2 * PLANE_A + PLANE_B + k * 32, 16, TL::SBO, TL::SWZ);
                if constexpr (F16) {
                    tc::mma_f16_ss(tmem, ah, bh, TL::IDESC, (it > 0 || k > 0) ? 1u : 0u);
                    if (!(exact & 2)) tc::mma_f16_ss(tmem, ah, bl, TL::IDESC, 1u);
                    if (!(exact & 1)) tc::mma_f16_ss(tmem, al, bh, TL::IDESC, 1u);
                } else {
                    tc::mma_tf32_ss(tmem, ah, bh, TL::IDESC, (it > 0 || k > 0) ? 1u : 0u);
                    if (!(exact & 2)) tc::mma_tf32_ss(tmem, ah, bl, TL::IDESC, 1u);
                    if (!(exact & 1)) tc::mma_tf32_ss(tmem, al, bh, TL::IDESC, 1u);
                }
            }
            tc::mma_commit(tc::smem_u32(&empty[s]));
        }
        tc::mma_commit(tc::smem_u32(accb));
    }
    __syncwarp();

    // ---------------- epilogue ----------------
    // The accumulator tile goes TMEM -> registers -> shared memory (the
    // pipeline buffers are free once the last MMA committed), so that global
    // reads and writes walk rows (or, for P^T, columns) with consecutive lanes.
    // (K = 0: nothing was issued and the accumulator is zero)
    const bool ok = nk == 0 || tc::mbar_wait(tc::smem_u32(accb), 0, abort_flag);
    tc::fence_after_sync();
    const bool good = __syncthreads_and(ok && !*abort_flag) != 0;
    constexpr int TP = TN + 1;
    float *T = reinterpret_cast<float *>(smem);
    if (good) {
        // warp w reads TMEM lanes 32 (w % 4) .. (its lane quarter), columns
        // TN/2 (w / 4) ..
        const int quarter = warp & 3, half = warp >> 2;
        const int row = quarter * 32 + lane;
#pragma unroll 1
        for (int c0 = half * (TN / 2); c0 < (half + 1) * (TN / 2); c0 += 32) {
            uint32_t v[32];
            if (nk > 0) {
                tc::tmem_ld_32x32b_x32(tmem + ((uint32_t)(quarter * 32) << 16) + (uint32_t)c0, v);
            } else {
#pragma unroll
                for (int q = 0; q < 32; ++q) v[q] = 0u;
            }
            if (F16 && e.ainv && nk > 0) {
                // back from the operands' row scales (powers of two: exact)
                const float sa = i0 + row < M ? e.ainv[i0 + row] : 0.f;
#pragma unroll
                for (int q = 0; q < 32; ++q) {
                    const int64_t gj = j0 + c0 + q;
                    T[row * TP + c0 + q] = gj < N ? __uint_as_float(v[q]) * (sa * e.binv[gj]) : 0.f;
                }
            } else {
#pragma unroll
                for (int q = 0; q < 32; ++q) T[row * TP + c0 + q] = __uint_as_float(v[q]);
            }
        }
    }
    __syncthreads();
    if (good) {
        // rows of the tile, each lane on 4 consecutive columns of a 128-wide
        // column half; the loads of 4 rows are issued before any store so
        // they overlap
        constexpr int RPW = TB / (THREADS / 32);   // tile rows per warp
#pragma unroll 1
        for (int ch = 0; ch < TN; ch += 128) {
            const int cc = ch + lane * 4;
            const int64_t gj = j0 + cc;
            const bool vec = MODE != TC_STORE && gj + 3 < N;
            for (int rb = warp * RPW; rb < warp * RPW + RPW; rb += 4) {
                if (i0 + rb >= M) break;
                // a batch of 4 rows runs vectorized when all 4 exist (M need
                // not be a multiple of 4 for a row group)
                if (vec && i0 + rb + 3 < M) {
                    if (MODE == TC_ADAM) adam_rows4(e, i0 + rb, M, gj, T + rb * TP + cc, TP);
                    else if (MODE == TC_BGD_P) bgd_p_rows4(e, i0 + rb, M, gj, T + rb * TP + cc, TP);
                    else if (MODE == TC_BGD_PG) bgd_pg_rows4(e, i0 + rb, gj, T + rb * TP + cc, TP);
                    else if (MODE == TC_SYRK) syrk_rows4(e, i0 + rb, gj, T + rb * TP + cc, TP);
                    else accum_rows4(e, i0 + rb, gj, T + rb * TP + cc, TP);
                } else {
                    for (int u = 0; u < 4; ++u) {
                        const int rr = rb + u;
                        const int64_t gi = i0 + rr;
                        if (gi >= M) break;
                        for (int q = 0; q < 4; ++q) {
                            if (gj + q >= N) break;
                            float &t = T[rr * TP + cc + q];
                            if (MODE == TC_STORE)
                                e.C[(int64_t)blockIdx.z * e.czs + gi * e.ldc + gj + q] =
                                    e.affine ? e.alpha_s * t + (e.R ? e.R[gi * e.ldr + gj + q] : 0.f) : t;
                            else if (MODE == TC_BGD_P) t = bgd_p_value(e, gi, gj + q, t);
                            else if (MODE == TC_BGD_PG) t = bgd_pg_value(e, gi, gj + q, t);
                            else epi_apply(e, gi, gj + q, t);
                        }
                    }
                }
            }
        }
    }
    __syncthreads();
    if (good && (MODE == TC_BGD_P || MODE == TC_BGD_PG)) {
        // columns of the tile, lanes over rows: P^T rows are contiguous
        constexpr int CPW = TN / (THREADS / 32);   // tile columns per warp
        for (int cc = warp * CPW; cc < warp * CPW + CPW; ++cc) {
            const int64_t gj = j0 + cc;
            if (gj >= N) break;
            for (int rr = lane; rr < TB; rr += 32) {
                const int64_t gi = i0 + rr;
                if (gi >= M) break;
                const float pv = T[rr * TP + cc];
                if (!e.Ptl) {
                    e.Pth[gj * e.ldp + gi] = pv;   // split into f16 planes afterwards
                    continue;
                }
                const float hi = tc::tf32_hi(pv);
                e.Pth[gj * e.ldp + gi] = hi;
                e.Ptl[gj * e.ldp + gi] = pv - hi;
            }
        }
    }
    if (!good && threadIdx.x == 0 && err) atomicOr(err, ST_TIMEOUT);
    tc::fence_before_sync();
    __syncthreads();
    if (warp == 0) tc::tmem_dealloc(tmem, TN);
}

// ---------------------------------------------------------------------------
// Persistent f16x3 products with the epilogue overlapped (the plain Block-GD
// G product; the gradient factor P with realq_set_tensor_overlap(2)).  One CTA
// per SM walks the tiles (t = blockIdx.x, + gridDim.x, ... in the grouped
// order above, K-split slices last) with three roles: warp 0 issues the TMA
// loads of the ring, warp 1 the MMAs, and warps 2..9 run the epilogue.  The
// accumulator is double-buffered in TMEM (2 x 256 columns): while the
// epilogue warps drain tile t's accumulator, the MMAs of tile t + 1 fill the
// other one, so the tensor pipe does not wait for the epilogue's global
// traffic.  The epilogue reads TMEM straight into registers, one output row
// per thread and 32 consecutive columns per load, and applies the same
// per-element operations as the tile kernel (the products' bits are the
// same; the order of the MMAs of a tile is unchanged).  Every wait is
// bounded; a wait that gives up raises the CTA's abort flag, the roles
// leave their loops, the MMAs already issued are drained and TMEM is freed.
constexpr int PTHREADS = 320;
constexpr int PEPI_WARPS = 8;

__device__ __forceinline__ void persistent_tile(int64_t t, int tiles_m, int tiles_n, int &z, int64_t &i0,
                                                int64_t &j0) {
    const int64_t per = (int64_t)tiles_m * tiles_n;
    z = (int)(t / per);
    const int64_t pid = t % per;
    constexpr int64_t GROUP = 8;
    const int64_t pg = GROUP * tiles_n, first = (pid / pg) * GROUP;
    const int64_t gm = (tiles_m - first) < GROUP ? (tiles_m - first) : GROUP;
    i0 = (first + (pid % pg) % gm) * TB;
    j0 = ((pid % pg) / gm) * 256;
}

constexpr int PSTAGES = 4;             // ring stages (the rest of shared memory stages the epilogue)
constexpr int PSTAGE_PITCH = 33;       // a warp's 32 x 32 staging block, padded

// One 32 x 32 block of the output (rows gi0 .., columns gj0 ..), staged in
// st[r * 33 + c] (row r, column c) by the warp that drained it from TMEM:
// the lanes walk columns, so that the global accesses of a row coalesce.
// Rows at or past M and columns at or past N are skipped.
template <int MODE>
__device__ __forceinline__ void persistent_block(const TcEpi &e, int z, int64_t gi0, int64_t gj0, int64_t M,
                                                 int64_t N, float *st, int lane) {
    static_assert(MODE == TC_ADAM || MODE == TC_BGD_P, "persistent epilogues: Adam and the gradient factor");
    const int64_t gj = gj0 + lane;
    const bool col_ok = gj < N;
    (void)z;
    if (MODE == TC_ADAM) {
        // four rows at a time: their loads are issued before any store
        for (int r0 = 0; r0 < 32; r0 += 4) {
            float mv[4], vv[4], wv[4], dv[4];
            int64_t w[4];
            bool ok[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int64_t gi = gi0 + r0 + u;
                ok[u] = gi < M && col_ok;
                w[u] = gi * e.ldw + e.col0 + gj;
                mv[u] = vv[u] = wv[u] = dv[u] = 0.f;
                if (ok[u]) {
                    if (!e.sgd) {
                        mv[u] = e.mA[w[u]];
                        vv[u] = e.vA[w[u]];
                    }
                    wv[u] = e.Wm[w[u]];
                    dv[u] = e.D[w[u]];
                }
            }
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                if (!ok[u]) continue;
                const float stp = adam_step(e, st[(r0 + u) * PSTAGE_PITCH + lane], mv[u], vv[u]);
                if (!e.sgd) {
                    e.mA[w[u]] = mv[u];
                    e.vA[w[u]] = vv[u];
                }
                e.Wm[w[u]] = wv[u] - stp;
                e.D[w[u]] = dv[u] - stp;
                e.Sh[w[u]] = -stp;
            }
        }
        return;
    }
    // TC_BGD_P: the gradient factor per element (lanes over columns), put
    // back into the staging block, then written transposed with the lanes
    // over rows (consecutive rows of P^T's column are consecutive in memory)
#pragma unroll 4
    for (int r = 0; r < 32; ++r) {
        const int64_t gi = gi0 + r;
        if (gi < M && col_ok) st[r * PSTAGE_PITCH + lane] = bgd_p_value(e, gi, gj, st[r * PSTAGE_PITCH + lane]);
    }
    __syncwarp();
    const int64_t gi = gi0 + lane;
    if (gi < M) {
#pragma unroll 4
        for (int c = 0; c < 32; ++c)
            if (gj0 + c < N) e.Pth[(gj0 + c) * e.ldp + gi] = st[lane * PSTAGE_PITCH + c];
    }
}

template <int MODE>
__global__ void __launch_bounds__(PTHREADS, 1)
    gemm_f16x3_persistent_kernel(const __grid_constant__ Maps maps, int64_t M, int64_t N, int64_t K, int k_off,
                                 int b_row0, int a_row0, const TcEpi e, int *err, int kchunk, int tiles_m,
                                 int tiles_n, int nz) {
    using TL = Tile<256, true>;
    constexpr int KS = TL::KS, STAGES = PSTAGES, PLANE_A = TL::PLANE_A, PLANE_B = TL::PLANE_B;
    constexpr int STAGE_BYTES = TL::STAGE_BYTES;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    float *stage_all = reinterpret_cast<float *>(smem + STAGES * STAGE_BYTES);   // 8 warps x 32 x 33
    uint64_t *full = reinterpret_cast<uint64_t *>(stage_all + PEPI_WARPS * 32 * PSTAGE_PITCH);
    uint64_t *empty = full + STAGES;
    uint64_t *tfull = empty + STAGES;     // [2]: MMAs of an accumulator done
    uint64_t *tempty = tfull + 2;         // [2]: the epilogue has read an accumulator
    uint64_t *drain = tempty + 2;         // the MMA thread's last commit
    uint32_t *tslot = reinterpret_cast<uint32_t *>(drain + 1);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(tslot + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t ntiles = (int64_t)tiles_m * tiles_n * nz;
    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            tc::mbar_init(tc::smem_u32(&full[s]), 1);
            tc::mbar_init(tc::smem_u32(&empty[s]), 1);
        }
        for (int a = 0; a < 2; ++a) {
            tc::mbar_init(tc::smem_u32(&tfull[a]), 1);
            tc::mbar_init(tc::smem_u32(&tempty[a]), PEPI_WARPS);
        }
        tc::mbar_init(tc::smem_u32(drain), 1);
        *abort_flag = 0;
        tc::fence_barrier_init();
        tc::prefetch_tmap(&maps.a_hi);
        tc::prefetch_tmap(&maps.a_lo);
        tc::prefetch_tmap(&maps.b_hi);
        tc::prefetch_tmap(&maps.b_lo);
    }
    if (warp == 0) tc::tmem_alloc(tc::smem_u32(tslot), 512);
    tc::fence_before_sync();
    __syncthreads();
    tc::fence_after_sync();
    const uint32_t tmem = *tslot;

    if (warp == 0) {
        if (lane == 0) {
            // ---------------- TMA producer ----------------
            uint32_t it = 0;
            for (int64_t t = blockIdx.x; t < ntiles && !*abort_flag; t += gridDim.x) {
                int z;
                int64_t i0, j0;
                persistent_tile(t, tiles_m, tiles_n, z, i0, j0);
                const int64_t kz0 = kchunk > 0 ? (int64_t)z * kchunk : 0;
                const int64_t Kz = kchunk > 0 ? ((K - kz0) < kchunk ? (K - kz0) : kchunk) : K;
                const int nk = (int)((Kz + KS - 1) / KS);
                for (int kk = 0; kk < nk; ++kk, ++it) {
                    const int s = (int)(it % STAGES);
                    const uint32_t r = it / STAGES;
                    if (!tc::mbar_wait(tc::smem_u32(&empty[s]), (r & 1u) ^ 1u, abort_flag)) {
                        *abort_flag = 1;
                        break;
                    }
                    const uint32_t fb = tc::smem_u32(&full[s]);
                    tc::mbar_arrive_expect_tx(fb, STAGE_BYTES);
                    const int x = k_off + (int)kz0 + kk * KS;
                    const uint32_t base = tc::smem_u32(smem + s * STAGE_BYTES);
                    tc::tma_load_2d(base, &maps.a_hi, fb, x, a_row0 + (int)i0);
                    tc::tma_load_2d(base + PLANE_A, &maps.a_lo, fb, x, a_row0 + (int)i0);
                    tc::tma_load_2d(base + 2 * PLANE_A, &maps.b_hi, fb, x, b_row0 + (int)j0);
                    tc::tma_load_2d(base + 2 * PLANE_A + PLANE_B, &maps.b_lo, fb, x, b_row0 + (int)j0);
                }
            }
            if (*abort_flag) {
                // let the copies in flight land before the CTA leaves
                int never = 0;
                for (uint32_t k = (it > (uint32_t)STAGES ? it - STAGES : 0u); k < it; ++k)
                    tc::mbar_wait(tc::smem_u32(&full[k % STAGES]), (k / STAGES) & 1u, &never, 100000000ull);
            }
        }
    } else if (warp == 1) {
        if (lane == 0) {
            // ---------------- MMA issuer ----------------
            uint32_t it = 0;
            int lt = 0;
            for (int64_t t = blockIdx.x; t < ntiles && !*abort_flag; t += gridDim.x, ++lt) {
                int z;
                int64_t i0, j0;
                persistent_tile(t, tiles_m, tiles_n, z, i0, j0);
                const int64_t kz0 = kchunk > 0 ? (int64_t)z * kchunk : 0;
                const int64_t Kz = kchunk > 0 ? ((K - kz0) < kchunk ? (K - kz0) : kchunk) : K;
                const int nk = (int)((Kz + KS - 1) / KS);
                const int acc = lt & 1;
                // the epilogue has read this accumulator's previous tile
                if (!tc::mbar_wait(tc::smem_u32(&tempty[acc]), (((uint32_t)lt >> 1) & 1u) ^ 1u, abort_flag)) {
                    *abort_flag = 1;
                    break;
                }
                tc::fence_after_sync();
                const uint32_t td = tmem + (uint32_t)(acc * 256);
                bool ok = true;
                for (int kk = 0; kk < nk; ++kk, ++it) {
                    const int s = (int)(it % STAGES);
                    const uint32_t r = it / STAGES;
                    if (!tc::mbar_wait(tc::smem_u32(&full[s]), r & 1u, abort_flag)) {
                        ok = false;
                        break;
                    }
                    tc::fence_after_sync();
                    const uint32_t base = tc::smem_u32(smem + s * STAGE_BYTES);
#pragma unroll
                    for (int k = 0; k < TL::KB / 32; ++k) {
                        const uint64_t ah = tc::smem_desc(base + k * 32, 16, TL::SBO, TL::SWZ);
                        const uint64_t al = tc::smem_desc(base + PLANE_A + k * 32, 16, TL::SBO, TL::SWZ);
                        const uint64_t bh = tc::smem_desc(base + 2 * PLANE_A + k * 32, 16, TL::SBO, TL::SWZ);
                        const uint64_t bl = tc::smem_desc(base + 2 * PLANE_A + PLANE_B + k * 32, 16, TL::SBO, TL::SWZ);
                        tc::mma_f16_ss(td, ah, bh, TL::IDESC, (kk > 0 || k > 0) ? 1u : 0u);
                        tc::mma_f16_ss(td, ah, bl, TL::IDESC, 1u);
                        tc::mma_f16_ss(td, al, bh, TL::IDESC, 1u);
                    }
                    tc::mma_commit(tc::smem_u32(&empty[s]));
                }
                if (!ok) {
                    *abort_flag = 1;
                    break;
                }
                // (K = 0: no MMA; the epilogue reads zeros for nk = 0)
                if (nk > 0) tc::mma_commit(tc::smem_u32(&tfull[acc]));
                else tc::mbar_arrive(tc::smem_u32(&tfull[acc]));
            }
            // every MMA issued has retired before TMEM is freed
            tc::mma_commit(tc::smem_u32(drain));
            int never = 0;
            tc::mbar_wait(tc::smem_u32(drain), 0u, &never, 100000000ull);
        }
    } else {
        // ---------------- epilogue (warps 2..9) ----------------
        const int quarter = warp & 3, half = (warp - 2) >> 2;
        const int row = quarter * 32 + lane;
        int lt = 0;
        for (int64_t t = blockIdx.x; t < ntiles; t += gridDim.x, ++lt) {
            int z;
            int64_t i0, j0;
            persistent_tile(t, tiles_m, tiles_n, z, i0, j0);
            const int64_t kz0 = kchunk > 0 ? (int64_t)z * kchunk : 0;
            const int64_t Kz = kchunk > 0 ? ((K - kz0) < kchunk ? (K - kz0) : kchunk) : K;
            const int acc = lt & 1;
            // (the warp agrees on the outcome: its TMEM loads are warp-wide)
            const bool got = tc::mbar_wait(tc::smem_u32(&tfull[acc]), ((uint32_t)lt >> 1) & 1u, abort_flag);
            if (!__all_sync(0xffffffffu, got)) {
                *abort_flag = 1;
                break;
            }
            tc::fence_after_sync();
            const int64_t gi = i0 + row;
            // (K = 0: nothing was issued into the accumulator; the products are 0)
            const bool none = Kz <= 0;
            const float sa = (gi < M && !none) ? e.ainv[gi] : 0.f;
            float *st = stage_all + (warp - 2) * 32 * PSTAGE_PITCH;
#pragma unroll 1
            for (int c0 = half * 128; c0 < half * 128 + 128; c0 += 32) {
                uint32_t v[32];
                tc::tmem_ld_32x32b_x32(tmem + ((uint32_t)(quarter * 32) << 16) + (uint32_t)(acc * 256 + c0), v);
                if (c0 == half * 128 + 96) {
                    // this warp's last read of the accumulator: hand it back
                    tc::fence_before_sync();
                    __syncwarp();
                    if (lane == 0) tc::mbar_arrive(tc::smem_u32(&tempty[acc]));
                }
                if (j0 + c0 >= N) continue;
                // this lane's row of the 32 x 32 block, unscaled, into the
                // staging block; then the block with the lanes over columns
#pragma unroll
                for (int q = 0; q < 32; ++q) {
                    const int64_t gj = j0 + c0 + q;
                    st[lane * PSTAGE_PITCH + q] =
                        (gj < N && !none) ? __uint_as_float(v[q]) * (sa * e.binv[gj]) : 0.f;
                }
                __syncwarp();
                persistent_block<MODE>(e, z, i0 + quarter * 32, j0 + c0, M, N, st, lane);
                __syncwarp();
            }
        }
    }
    __syncwarp();
    tc::fence_before_sync();
    __syncthreads();
    if (threadIdx.x == 0 && *abort_flag && err) atomicOr(err, ST_TIMEOUT);
    if (warp == 0) tc::tmem_dealloc(tmem, 512);
}

// g = sum over the K splits (z = 0, 1, ... in order), then the TC_ADAM
// epilogue on element (i, j) of the m x N block at column e.col0
__global__ void gsum_adam_kernel(int64_t m, int64_t N, int nz, const float *part, const TcEpi e) {
    const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= m * N) return;
    const int64_t i = idx / N, j = idx % N;
    float g = 0.f;
    for (int z = 0; z < nz; ++z) g += part[(int64_t)z * m * N + idx];
    const int64_t w = i * e.ldw + e.col0 + j;
    float mv = e.sgd ? 0.f : e.mA[w], vv = e.sgd ? 0.f : e.vA[w];
    const float st = adam_step(e, g, mv, vv);
    if (!e.sgd) {
        e.mA[w] = mv;
        e.vA[w] = vv;
    }
    e.Wm[w] -= st;
    e.D[w] -= st;
    if (!e.Sl) {
        e.Sh[w] = -st;
        return;
    }
    const float sh = tc::tf32_hi(-st);
    e.Sh[w] = sh;
    e.Sl[w] = -st - sh;
}

// hi / lo planes of x (or of alpha x + (1 - alpha) y when y is given)
__global__ void split_kernel(int64_t count, const float *x, const float *y, float alpha, float *hi, float *lo) {
    const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= count) return;
    const float v = y ? alpha * x[i] + (1.f - alpha) * y[i] : x[i];
    const float h = tc::tf32_hi(v);
    hi[i] = h;
    lo[i] = v - h;
}

// The lazy batch update's operands as K-major planes (tc_trail_planes): tile
// t < te of a 32 x 32 tiling transposes E (Et[k][i] -> -E[i][k]), the others
// the U panel (U[bs + k][be + j] -> P[j][k]); kt = kb / 32 tiles along k.
__global__ void trail_planes_kernel(int64_t m, int64_t ldet, const float *Et, int64_t n, const float *U, int64_t bs,
                                    int64_t be, int kt, int B, int64_t te, float *Eh, float *El, float *Ph,
                                    float *Pl) {
    __shared__ float tile[32][33];
    const int tx = threadIdx.x, ty = threadIdx.y;
    int64_t t = blockIdx.x;
    if (t < te) {
        const int64_t ti = t / kt;
        const int tk = (int)(t % kt);
        const int64_t i = ti * 32 + tx;
#pragma unroll
        for (int q = 0; q < 32; q += 8) tile[ty + q][tx] = i < m ? Et[(int64_t)(tk * 32 + ty + q) * ldet + i] : 0.f;
        __syncthreads();
#pragma unroll
        for (int q = 0; q < 32; q += 8) {
            const int64_t r = ti * 32 + ty + q;
            if (r < m) {
                const float v = -tile[tx][ty + q];
                const float h = tc::tf32_hi(v);
                Eh[r * B + tk * 32 + tx] = h;
                El[r * B + tk * 32 + tx] = v - h;
            }
        }
        return;
    }
    t -= te;
    const int64_t rcols = n - be;
    const int64_t tj = t / kt;
    const int tk = (int)(t % kt);
    const int64_t j = tj * 32 + tx;
#pragma unroll
    for (int q = 0; q < 32; q += 8)
        tile[ty + q][tx] = j < rcols ? U[(bs + tk * 32 + ty + q) * n + be + j] : 0.f;
    __syncthreads();
#pragma unroll
    for (int q = 0; q < 32; q += 8) {
        const int64_t c = tj * 32 + ty + q;
        if (c < rcols) {
            const float v = tile[tx][ty + q];
            const float h = tc::tf32_hi(v);
            Ph[c * B + tk * 32 + tx] = h;
            Pl[c * B + tk * 32 + tx] = v - h;
        }
    }
}

// hi / lo planes of x - y (y fp32 or bf16)
template <typename TY>
__global__ void split_diff_kernel(int64_t count, const float *x, const TY *y, float *hi, float *lo) {
    const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= count) return;
    const float v = x[i] - load_as_float(y, i);
    const float h = tc::tf32_hi(v);
    hi[i] = h;
    lo[i] = v - h;
}

}  // namespace

template <typename TY>
realq_status_t tc_split_diff(cudaStream_t s, int64_t count, const float *x, const TY *y, float *hi, float *lo) {
    if (count <= 0) return REALQ_OK;
    {
        Launch L("tf32_split", s);
        split_diff_kernel<<<(unsigned)((count + 255) / 256), 256, 0, s>>>(count, x, y, hi, lo);
    }
    return check_launch("tf32_split");
}
template realq_status_t tc_split_diff<float>(cudaStream_t, int64_t, const float *, const float *, float *, float *);
template realq_status_t tc_split_diff<__nv_bfloat16>(cudaStream_t, int64_t, const float *, const __nv_bfloat16 *,
                                                     float *, float *);

bool tc_gemm_eligible(int64_t m, int64_t n) {
    return m % 4 == 0 && n % 4 == 0 && m >= 32 && n >= 32 && m < (1ll << 31) && n < (1ll << 31);
}

realq_status_t tc_split(cudaStream_t s, int64_t count, const float *x, const float *y, float alpha, float *hi,
                        float *lo) {
    if (count <= 0) return REALQ_OK;
    {
        Launch L("tf32_split", s);
        split_kernel<<<(unsigned)((count + 255) / 256), 256, 0, s>>>(count, x, y, alpha, hi, lo);
    }
    return check_launch("tf32_split");
}

namespace {
// dst[c * ldd + r] = planes of src[r * lds + c], 32 x 32 tiles through shared memory
__global__ void trans_planes_kernel(int64_t rows, int64_t cols, const float *src, int64_t lds, float *dh, float *dl,
                                    int64_t ldd, int64_t tiles_c) {
    __shared__ float tile[32][33];
    const int tx = threadIdx.x, ty = threadIdx.y;
    const int64_t tr = blockIdx.x / tiles_c, tcol = blockIdx.x % tiles_c;
    const int64_t c = tcol * 32 + tx;
#pragma unroll
    for (int q = 0; q < 32; q += 8) {
        const int64_t r = tr * 32 + ty + q;
        tile[ty + q][tx] = (r < rows && c < cols) ? src[r * lds + c] : 0.f;
    }
    __syncthreads();
    const int64_t r = tr * 32 + tx;
#pragma unroll
    for (int q = 0; q < 32; q += 8) {
        const int64_t cc = tcol * 32 + ty + q;
        if (cc < cols && r < rows) {
            const float v = tile[tx][ty + q];
            const float h = tc::tf32_hi(v);
            dh[cc * ldd + r] = h;
            dl[cc * ldd + r] = v - h;
        }
    }
}

__global__ void split_rows_kernel(int64_t rows, int64_t cols, const float *src, int64_t lds, float *hi, float *lo,
                                  int64_t ldd, int64_t pad) {
    const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= rows * pad) return;
    const int64_t r = i / pad, c = i % pad;
    const float v = c < cols ? src[r * lds + c] : 0.f;
    const float h = tc::tf32_hi(v);
    hi[r * ldd + c] = h;
    lo[r * ldd + c] = v - h;
}
}  // namespace

realq_status_t tc_trans_planes(cudaStream_t s, int64_t rows, int64_t cols, const float *src, int64_t lds,
                               float *dh, float *dl, int64_t ldd) {
    if (rows <= 0 || cols <= 0) return REALQ_OK;
    const int64_t tr = ceil_div(rows, 32), tcn = ceil_div(cols, 32);
    {
        Launch L("tf32_split", s);
        trans_planes_kernel<<<(unsigned)(tr * tcn), dim3(32, 8), 0, s>>>(rows, cols, src, lds, dh, dl, ldd, tcn);
    }
    return check_launch("tf32_split");
}

realq_status_t tc_split_rows(cudaStream_t s, int64_t rows, int64_t cols, const float *src, int64_t lds, float *hi,
                             float *lo, int64_t ldd, int64_t pad) {
    if (rows <= 0 || cols <= 0) return REALQ_OK;
    if (cols > pad || pad > ldd)
        return fail(REALQ_ERR_INVALID_ARG, "tf32 split: %lld columns padded to %lld in rows of %lld", (long long)cols,
                    (long long)pad, (long long)ldd);
    {
        Launch L("tf32_split", s);
        split_rows_kernel<<<(unsigned)ceil_div(rows * pad, 256), 256, 0, s>>>(rows, cols, src, lds, hi, lo, ldd, pad);
    }
    return check_launch("tf32_split");
}

realq_status_t tc_trail_planes(cudaStream_t s, int64_t m, const float *Et, int64_t ldet, int64_t n, const float *U,
                               int64_t bs, int64_t be, int kb, int B, float *Eh, float *El, float *Ph, float *Pl) {
    if (kb <= 0 || kb % 32 != 0 || kb > B || be > n || bs + kb > n)
        return fail(REALQ_ERR_INVALID_ARG, "trailing planes: bad block (%d of %d at %lld)", kb, B, (long long)bs);
    const int kt = kb / 32;
    const int64_t te = Et ? ceil_div(m, 32) * kt : 0;
    const int64_t tp = ceil_div(n - be, 32) * kt;
    if (te + tp <= 0) return REALQ_OK;
    {
        Launch L("trailing_planes", s);
        trail_planes_kernel<<<(unsigned)(te + tp), dim3(32, 8), 0, s>>>(m, ldet, Et, n, U, bs, be, kt, B, te, Eh, El,
                                                                         Ph, Pl);
    }
    return check_launch("trailing_planes");
}

realq_status_t tc_gsum_adam(cudaStream_t s, int64_t m, int64_t N, int nz, const float *part, const TcEpi &e) {
    if (m <= 0 || N <= 0) return REALQ_OK;
    {
        Launch L("bgd_g_gsum_adam", s);
        gsum_adam_kernel<<<(unsigned)ceil_div(m * N, 256), 256, 0, s>>>(m, N, nz, part, e);
    }
    return check_launch("bgd_g_gsum_adam");
}

realq_status_t tc_make_maps(TcMaps *out, const float *a_hi, const float *a_lo, int64_t a_rows, int64_t a_k,
                            int64_t lda, const float *b_hi, const float *b_lo, int64_t b_rows, int64_t b_k,
                            int64_t ldb) {
    static_assert(sizeof(MapPair) <= sizeof(TcMaps), "map storage");
    MapPair *mp = reinterpret_cast<MapPair *>(out->storage);
    CUresult r = CUDA_SUCCESS;
    // narrow: 32-wide K slices with 128-byte swizzle, 128-row boxes;
    // wide: 16-wide slices with 64-byte swizzle, B boxes of 256 rows
    for (int w = 0; w < 2 && r == CUDA_SUCCESS; ++w) {
        Maps *m = w ? &mp->wide : &mp->narrow;
        const uint32_t ks = w ? Tile<256>::KS : Tile<128>::KS, bn = w ? 256 : 128;
        const int swz = w ? 2 : 1;
        r = encode_tmap_2d_f32(&m->a_hi, a_hi, (uint64_t)a_k, (uint64_t)a_rows, (uint64_t)lda * 4, ks, TB, swz);
        if (r == CUDA_SUCCESS)
            r = encode_tmap_2d_f32(&m->a_lo, a_lo, (uint64_t)a_k, (uint64_t)a_rows, (uint64_t)lda * 4, ks, TB, swz);
        if (r == CUDA_SUCCESS)
            r = encode_tmap_2d_f32(&m->b_hi, b_hi, (uint64_t)b_k, (uint64_t)b_rows, (uint64_t)ldb * 4, ks, bn, swz);
        if (r == CUDA_SUCCESS)
            r = encode_tmap_2d_f32(&m->b_lo, b_lo, (uint64_t)b_k, (uint64_t)b_rows, (uint64_t)ldb * 4, ks, bn, swz);
    }
    if (r != CUDA_SUCCESS) return fail(REALQ_ERR_CUDA, "cuTensorMapEncodeTiled (tf32 planes) failed (%d)", (int)r);
    out->f16 = 0;
    return REALQ_OK;
}

realq_status_t tc_make_maps_f16(TcMaps *out, const __half *a_hi, const __half *a_lo, int64_t a_rows, int64_t a_k,
                                int64_t lda, const __half *b_hi, const __half *b_lo, int64_t b_rows, int64_t b_k,
                                int64_t ldb) {
    MapPair *mp = reinterpret_cast<MapPair *>(out->storage);
    if ((lda & 7) || (ldb & 7) || ((reinterpret_cast<uintptr_t>(a_hi) | reinterpret_cast<uintptr_t>(a_lo) |
                                    reinterpret_cast<uintptr_t>(b_hi) | reinterpret_cast<uintptr_t>(b_lo)) & 15))
        return fail(REALQ_ERR_INVALID_ARG, "f16 planes: row strides of 8 elements and 16-byte bases required");
    CUresult r = CUDA_SUCCESS;
    // the same byte boxes as the tf32 planes': twice the elements per row
    for (int w = 0; w < 2 && r == CUDA_SUCCESS; ++w) {
        Maps *m = w ? &mp->wide : &mp->narrow;
        const uint32_t ks = w ? Tile<256, true>::KS : Tile<128, true>::KS, bn = w ? 256 : 128;
        const int swz = w ? 2 : 1;
        r = encode_tmap_2d_f16(&m->a_hi, a_hi, (uint64_t)a_k, (uint64_t)a_rows, (uint64_t)lda * 2, ks, TB, swz);
        if (r == CUDA_SUCCESS)
            r = encode_tmap_2d_f16(&m->a_lo, a_lo, (uint64_t)a_k, (uint64_t)a_rows, (uint64_t)lda * 2, ks, TB, swz);
        if (r == CUDA_SUCCESS)
            r = encode_tmap_2d_f16(&m->b_hi, b_hi, (uint64_t)b_k, (uint64_t)b_rows, (uint64_t)ldb * 2, ks, bn, swz);
        if (r == CUDA_SUCCESS)
            r = encode_tmap_2d_f16(&m->b_lo, b_lo, (uint64_t)b_k, (uint64_t)b_rows, (uint64_t)ldb * 2, ks, bn, swz);
    }
    if (r != CUDA_SUCCESS) return fail(REALQ_ERR_CUDA, "cuTensorMapEncodeTiled (f16 planes) failed (%d)", (int)r);
    out->f16 = 1;
    return REALQ_OK;
}

namespace {
// One CTA per row: the row's largest magnitude over [c0, c1), the power of
// two s that puts it in [2^14, 2^15) (from its exponent field; clamped so
// that s and 1/s are normal floats), then the fp16 planes of s v.  The
// largest scaled value stays below 2^15 after rounding, within fp16's range.
__global__ void __launch_bounds__(256) split_f16_rows_kernel(int64_t c0, int64_t c1, const float *x, const float *y,
                                                             float alpha, int64_t lds, __half *hi, __half *lo,
                                                             int64_t ldd, float *inv) {
    __shared__ float red[8];
    const int64_t r = blockIdx.x;
    const float *xr = x + r * lds;
    const float *yr = y ? y + r * lds : nullptr;
    float mx = 0.f;
    for (int64_t c = c0 + threadIdx.x; c < c1; c += 256) {
        const float v = yr ? alpha * xr[c] + (1.f - alpha) * yr[c] : xr[c];
        mx = fmaxf(mx, fabsf(v));
    }
    for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = mx;
    __syncthreads();
    mx = red[0];
    for (int w = 1; w < 8; ++w) mx = fmaxf(mx, red[w]);
    // mx < 2^(e - 126) for biased exponent e: s = 2^(141 - e)
    const int e = (int)((__float_as_uint(mx) >> 23) & 0xFFu);
    int k = mx == 0.f ? 0 : 141 - e;
    k = k < -126 ? -126 : (k > 126 ? 126 : k);
    const float sc = __uint_as_float((uint32_t)(k + 127) << 23);
    if (threadIdx.x == 0) inv[r] = __uint_as_float((uint32_t)(127 - k) << 23);
    __half *hr = hi + r * ldd, *lr = lo + r * ldd;
    for (int64_t c = c0 + threadIdx.x; c < c1; c += 256) {
        const float v = (yr ? alpha * xr[c] + (1.f - alpha) * yr[c] : xr[c]) * sc;
        const __half h = __float2half_rn(v);
        hr[c] = h;
        lr[c] = __float2half_rn(v - __half2float(h));
    }
}

int g_bgd_products = 1;   // 1: f16x3 for the plain Block-GD products where the shapes allow, 0: tf32x3
}  // namespace

void bgd_set_products(int mode) { g_bgd_products = mode; }
int bgd_products() { return g_bgd_products; }

realq_status_t tc_split_f16_rows(cudaStream_t s, int64_t rows, int64_t c0, int64_t c1, const float *x, const float *y,
                                 float alpha, int64_t lds, __half *hi, __half *lo, int64_t ldd, float *inv) {
    if (rows <= 0 || c1 <= c0) return REALQ_OK;
    if (rows > 0x7FFFFFFFll) return fail(REALQ_ERR_INVALID_ARG, "f16 split: too many rows");
    {
        Launch L("f16_split", s);
        split_f16_rows_kernel<<<(unsigned)rows, 256, 0, s>>>(c0, c1, x, y, alpha, lds, hi, lo, ldd, inv);
    }
    return check_launch("f16_split");
}

namespace {
template <int MODE, int TN, bool F16>
void launch_mode(cudaStream_t s, const Maps &m, dim3 grid, int64_t M, int64_t N, int64_t K, int k_off, int b_row0,
                 const TcEpi &e, int *err, int a_row0, int kchunk, int exact) {
    gemm_x3_kernel<MODE, TN, F16><<<grid, THREADS, Tile<TN, F16>::SMEM, s>>>(m, M, N, K, k_off, b_row0, a_row0, e,
                                                                             err, kchunk, exact);
}

template <int TN, bool F16>
realq_status_t launch_x3(cudaStream_t s, const Maps &m, int64_t M, int64_t N, int64_t K, int k_off, int b_row0,
                         const TcEpi &e, int *err, int a_row0, int kchunk, int exact) {
    constexpr int SM = Tile<TN, F16>::SMEM;
    const unsigned nz = kchunk > 0 ? (unsigned)ceil_div(K, kchunk) : 1u;
    const dim3 grid((unsigned)ceil_div(N, TN), (unsigned)ceil_div(M, TB), nz);
    if constexpr (F16) {
        // the f16x3 products: the plain Block-GD gradient factor, the G
        // product with its optimizer step, and its K-split slices
        REALQ_TRY(set_smem_limit(reinterpret_cast<const void *>(gemm_x3_kernel<TC_STORE, TN, true>), SM));
        REALQ_TRY(set_smem_limit(reinterpret_cast<const void *>(gemm_x3_kernel<TC_BGD_P, TN, true>), SM));
        REALQ_TRY(set_smem_limit(reinterpret_cast<const void *>(gemm_x3_kernel<TC_ADAM, TN, true>), SM));
        switch (e.mode) {
            case TC_STORE: launch_mode<TC_STORE, TN, true>(s, m, grid, M, N, K, k_off, b_row0, e, err, a_row0, kchunk, exact); break;
            case TC_BGD_P: launch_mode<TC_BGD_P, TN, true>(s, m, grid, M, N, K, k_off, b_row0, e, err, a_row0, kchunk, exact); break;
            case TC_ADAM: launch_mode<TC_ADAM, TN, true>(s, m, grid, M, N, K, k_off, b_row0, e, err, a_row0, kchunk, exact); break;
            default: return fail(REALQ_ERR_INVALID_ARG, "f16x3 product: epilogue mode %d not built", e.mode);
        }
        return REALQ_OK;
    } else {
        REALQ_TRY(set_smem_limit(reinterpret_cast<const void *>(gemm_x3_kernel<TC_STORE, TN, false>), SM));
        REALQ_TRY(set_smem_limit(reinterpret_cast<const void *>(gemm_x3_kernel<TC_BGD_P, TN, false>), SM));
        REALQ_TRY(set_smem_limit(reinterpret_cast<const void *>(gemm_x3_kernel<TC_ADAM, TN, false>), SM));
        REALQ_TRY(set_smem_limit(reinterpret_cast<const void *>(gemm_x3_kernel<TC_ACCUM, TN, false>), SM));
        REALQ_TRY(set_smem_limit(reinterpret_cast<const void *>(gemm_x3_kernel<TC_BGD_PG, TN, false>), SM));
        REALQ_TRY(set_smem_limit(reinterpret_cast<const void *>(gemm_x3_kernel<TC_SYRK, TN, false>), SM));
        switch (e.mode) {
            case TC_STORE: launch_mode<TC_STORE, TN, false>(s, m, grid, M, N, K, k_off, b_row0, e, err, a_row0, kchunk, exact); break;
            case TC_BGD_P: launch_mode<TC_BGD_P, TN, false>(s, m, grid, M, N, K, k_off, b_row0, e, err, a_row0, kchunk, exact); break;
            case TC_ADAM: launch_mode<TC_ADAM, TN, false>(s, m, grid, M, N, K, k_off, b_row0, e, err, a_row0, kchunk, exact); break;
            case TC_ACCUM: launch_mode<TC_ACCUM, TN, false>(s, m, grid, M, N, K, k_off, b_row0, e, err, a_row0, kchunk, exact); break;
            case TC_SYRK: launch_mode<TC_SYRK, TN, false>(s, m, grid, M, N, K, k_off, b_row0, e, err, a_row0, kchunk, exact); break;
            default: launch_mode<TC_BGD_PG, TN, false>(s, m, grid, M, N, K, k_off, b_row0, e, err, a_row0, kchunk, exact); break;
        }
        return REALQ_OK;
    }
}

int g_tile_mode = 0;   // 0: by the grid (wide_tiles_pay), 1: always 128 x 128, 2: always 128 x 256
int g_overlap = 1;     // persistent f16x3 kernels: 1 for the G product, 2 for G and the gradient factor

int sm_count() {
    static int sms = 0;
    if (sms == 0) {
        int dev = 0, c = 0;
        if (cudaGetDevice(&dev) == cudaSuccess &&
            cudaDeviceGetAttribute(&c, cudaDevAttrMultiProcessorCount, dev) == cudaSuccess && c > 0)
            sms = c;
    }
    return sms;
}

template <int MODE>
realq_status_t launch_persistent(cudaStream_t s, const Maps &m, int64_t M, int64_t N, int64_t K, int k_off,
                                 int b_row0, const TcEpi &e, int *err, int a_row0, int kchunk) {
    constexpr int SM = PSTAGES * Tile<256, true>::STAGE_BYTES + PEPI_WARPS * 32 * PSTAGE_PITCH * 4 + 1024 + 256;
    static_assert(SM <= 232448, "shared memory of the persistent kernel");
    REALQ_TRY(set_smem_limit(reinterpret_cast<const void *>(gemm_f16x3_persistent_kernel<MODE>), SM));
    const int64_t tiles_m = ceil_div(M, TB), tiles_n = ceil_div(N, 256);
    const int64_t nz = kchunk > 0 ? ceil_div(K, kchunk) : 1;
    const int64_t ntiles = tiles_m * tiles_n * nz;
    const int sms = sm_count();
    if (sms <= 0) return fail(REALQ_ERR_CUDA, "persistent product: no SM count");
    if (tiles_m > 0x7FFFFFFF || tiles_n > 0x7FFFFFFF || nz > 0x7FFFFFFF)
        return fail(REALQ_ERR_UNSUPPORTED, "persistent product: too many tiles");
    const unsigned grid = (unsigned)(ntiles < sms ? ntiles : sms);
    gemm_f16x3_persistent_kernel<MODE><<<grid, PTHREADS, SM, s>>>(m, M, N, K, k_off, b_row0, a_row0, e, err, kchunk,
                                                                  (int)tiles_m, (int)tiles_n, (int)nz);
    return REALQ_OK;
}

// The 128 x 256 tile does twice a narrow tile's work in about 1.55 narrow
// tile times (its measured rate over the narrow one's, at the shared-memory
// bound above); it pays when that beats the narrow grid's waves on the SMs.
bool wide_tiles_pay(int64_t M, int64_t N, unsigned nz) {
    static int sms = 0;
    if (sms == 0) {
        int dev = 0, c = 0;
        if (cudaGetDevice(&dev) == cudaSuccess &&
            cudaDeviceGetAttribute(&c, cudaDevAttrMultiProcessorCount, dev) == cudaSuccess && c > 0)
            sms = c;
        else
            return false;
    }
    const int64_t rows = ceil_div(M, TB) * (int64_t)nz;
    const int64_t waves_n = ceil_div(rows * ceil_div(N, 128), sms);
    const int64_t waves_w = ceil_div(rows * ceil_div(N, 256), sms);
    return 155 * waves_w < 100 * waves_n;
}
}  // namespace

void tc_set_tile_mode(int mode) { g_tile_mode = mode; }
void tc_set_overlap(int mode) { g_overlap = mode; }

realq_status_t tc_gemm_x3(cudaStream_t s, const TcMaps &maps, int64_t M, int64_t N, int64_t K, int k_off,
                              int b_row0, const TcEpi &e, int *err, const char *name, int a_row0, int kchunk,
                              int exact) {
    if (M <= 0 || N <= 0) return REALQ_OK;
    const bool f16 = maps.f16 != 0;
    // the x coordinate of every TMA box: 16-byte aligned
    if ((k_off & (f16 ? 7 : 3)) != 0)
        return fail(REALQ_ERR_INVALID_ARG, "%s: K offset must be a multiple of %d", name, f16 ? 8 : 4);
    const int ks = f16 ? Tile<128, true>::KS : Tile<128>::KS;
    if (kchunk < 0 || (kchunk % ks) != 0 || (kchunk > 0 && e.mode != TC_STORE))
        return fail(REALQ_ERR_INVALID_ARG, "%s: a K split takes a multiple of %d and the store epilogue", name, ks);
    if (f16 && (e.b_tri || (e.mode != TC_STORE && e.mode != TC_BGD_P && e.mode != TC_ADAM) || !e.ainv || !e.binv))
        return fail(REALQ_ERR_INVALID_ARG, "%s: f16x3 takes the store, gradient-factor or Adam epilogue with row "
                    "scales", name);
    if (e.mode < TC_STORE || e.mode > TC_SYRK) return fail(REALQ_ERR_INVALID_ARG, "%s: bad epilogue mode", name);
    if (e.mode == TC_SYRK && (a_row0 != 0 || b_row0 != 0 || M != N))
        return fail(REALQ_ERR_INVALID_ARG, "%s: a symmetric update takes a square product from row 0", name);
    if (e.b_tri && kchunk > 0) return fail(REALQ_ERR_INVALID_ARG, "%s: a triangular B takes no K split", name);
    if (e.affine && (kchunk > 0 || e.mode != TC_STORE))
        return fail(REALQ_ERR_INVALID_ARG, "%s: the affine store takes no K split", name);
    const MapPair &mp = *reinterpret_cast<const MapPair *>(maps.storage);
    const unsigned nz = kchunk > 0 ? (unsigned)ceil_div(K, kchunk) : 1u;
    const bool wide = g_tile_mode == 2 || (g_tile_mode == 0 && wide_tiles_pay(M, N, nz));
    {
        Launch L(name, s);
        if (f16 && wide && g_overlap >= 1 && e.mode == TC_ADAM) {
            REALQ_TRY(launch_persistent<TC_ADAM>(s, mp.wide, M, N, K, k_off, b_row0, e, err, a_row0, kchunk));
        } else if (f16 && wide && g_overlap == 2 && e.mode == TC_BGD_P) {
            REALQ_TRY(launch_persistent<TC_BGD_P>(s, mp.wide, M, N, K, k_off, b_row0, e, err, a_row0, kchunk));
        } else if (f16) {
            if (wide) REALQ_TRY((launch_x3<256, true>(s, mp.wide, M, N, K, k_off, b_row0, e, err, a_row0, kchunk, exact)));
            else REALQ_TRY((launch_x3<128, true>(s, mp.narrow, M, N, K, k_off, b_row0, e, err, a_row0, kchunk, exact)));
        } else {
            if (wide) REALQ_TRY((launch_x3<256, false>(s, mp.wide, M, N, K, k_off, b_row0, e, err, a_row0, kchunk, exact)));
            else REALQ_TRY((launch_x3<128, false>(s, mp.narrow, M, N, K, k_off, b_row0, e, err, a_row0, kchunk, exact)));
        }
    }
    return check_launch(name);
}

}  // namespace realq
