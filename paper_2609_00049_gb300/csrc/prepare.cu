// Step a3 (Alg. 1: "Compute ... H and its inverse"): H̄ = H_sum / T, dead
// channels, relative damping, and the upper factor U with Hd^-1 = U^T U.
//
// U is obtained without forming Hd^-1: factor Hd = R R^T with R upper
// triangular (Cholesky taken from the last index backwards), then U = R^-1,
// because Hd^-1 = R^-T R^-1 = U^T U.  Row j of U, scaled by U_jj, is row j of
// the inverse Hessian after the Schur-complement downdates of columns < j,
// which is what the OBS step of Eq. (gptq_update) consumes.
//
// Both factorizations are blocked with 64-wide blocks: a one-CTA kernel
// factors / inverts the diagonal block in shared memory, the off-diagonal work
// runs as fp32 GEMMs.  A pivot that is not positive (or not finite) records its
// column in the workspace status word; prepare reads it once at the end, the
// deferred variant leaves it for realq_prepare_status (a captured step reads
// no host memory).
#include "kernels.cuh"

#include <vector>

namespace realq {
namespace {

constexpr int NB = 64;

__global__ void prep_init_kernel(int64_t n, float Tf, const float *H, float *Hbar, float *A, uint8_t *dead) {
    const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= n * n) return;
    const int64_t i = idx / n, j = idx % n;
    const float h = H[idx];
    const float hb = h / Tf;
    float a = 0.f;
    if (j > i) a = hb;
    else if (j == i) {
        const bool d = (h == 0.f);
        dead[i] = d ? 1 : 0;
        a = d ? 1.f : hb;
    }
    if (Hbar) Hbar[idx] = hb;
    A[idx] = a;
}

// lambda = damp * mean(diag A) (fp64 reduction in a fixed order); A_jj += lambda
__global__ void prep_damp_kernel(int64_t n, float *A, float damp, float *lam_out) {
    __shared__ double red[1024];
    double s = 0.0;
    for (int64_t j = threadIdx.x; j < n; j += blockDim.x) s += (double)A[j * n + j];
    red[threadIdx.x] = s;
    __syncthreads();
    for (int w = blockDim.x / 2; w > 0; w >>= 1) {
        if ((int)threadIdx.x < w) red[threadIdx.x] += red[threadIdx.x + w];
        __syncthreads();
    }
    const float lam = (float)((double)damp * (red[0] / (double)n));
    for (int64_t j = threadIdx.x; j < n; j += blockDim.x) A[j * n + j] += lam;
    if (threadIdx.x == 0) *lam_out = lam;
}

// A 32 x 32 block As (pitch 33, upper triangle): reverse-order Cholesky
// As = R R^T (R upper) fused with the back substitution V = R^-1, written to
// Vs (row-major, zeros below the diagonal), by the 128 threads of the CTA.
// Lane j owns column j of the block and row j of V; warp w keeps entries
// 8w .. 8w + 7 of both in registers.  Pivot k needs only column k of R and
// row k of V: lane k of every warp publishes its eight entries of both
// (unscaled) into a double-buffered 64-float slot bf[(k & 1) * 64 ..] with
// one CTA barrier per pivot (the slot of pivot k is next written at pivot
// k - 2, after the barrier of pivot k - 1, which every warp reaches only after
// its reads of pivot k); every thread then applies
//   a_ij -= r_ik r_jk (i <= j < k),   V[j] -= r_jk V[k] (j < k),
// with r_ik = a_ik / sqrt(a_kk), to its entries.  Row k of V is scaled by its
// own 1 / r_kk once, at the end (no later pivot reads it).  A pivot that is
// not positive (or not finite) is recorded (the first one wins; columns >=
// valid are padding) and replaced by 1 to keep going.  (One warp doing all 32
// entries issues a ~100-instruction pivot at about seven cycles each; split
// four ways with a barrier the pivot is about three times shorter.)
__device__ __forceinline__ void cta_rchol_inv32(const float (*As)[33], float (*Vs)[33], float *bf, int warp,
                                                int lane, int *status, int64_t col0, int valid) {
    const int q0 = warp * 8;
    float c[8], v[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        c[i] = As[q0 + i][lane];
        v[i] = (q0 + i == lane) ? 1.f : 0.f;
    }
    float rown = 1.f;
#pragma unroll 1
    for (int k = 31; k >= 0; --k) {
        float *b = bf + (k & 1) * 64;
        if (lane == k) {
            *reinterpret_cast<float4 *>(b + q0) = make_float4(c[0], c[1], c[2], c[3]);
            *reinterpret_cast<float4 *>(b + q0 + 4) = make_float4(c[4], c[5], c[6], c[7]);
            *reinterpret_cast<float4 *>(b + 32 + q0) = make_float4(v[0], v[1], v[2], v[3]);
            *reinterpret_cast<float4 *>(b + 32 + q0 + 4) = make_float4(v[4], v[5], v[6], v[7]);
        }
        __syncthreads();
        float d = b[k];
        if (!(d > 0.f) || !isfinite(d)) {
            if (warp == 0 && lane == 0 && k < valid) atomicCAS(status, -1, (int)(col0 + k));
            d = 1.f;
        }
        const float rinv = rsqrtf(d);
        if (lane == k) rown = rinv;
        const float rjk = lane < k ? b[lane] * rinv : 0.f;
        const float cf = -rjk * rinv;
        const float4 bc0 = *reinterpret_cast<const float4 *>(b + q0);
        const float4 bc1 = *reinterpret_cast<const float4 *>(b + q0 + 4);
        const float4 bv0 = *reinterpret_cast<const float4 *>(b + 32 + q0);
        const float4 bv1 = *reinterpret_cast<const float4 *>(b + 32 + q0 + 4);
        const float bc[8] = {bc0.x, bc0.y, bc0.z, bc0.w, bc1.x, bc1.y, bc1.z, bc1.w};
        const float bv[8] = {bv0.x, bv0.y, bv0.z, bv0.w, bv1.x, bv1.y, bv1.z, bv1.w};
#pragma unroll
        for (int q = 0; q < 8; ++q) {
            if (q0 + q <= lane) c[q] = fmaf(bc[q], cf, c[q]);
            v[q] = fmaf(bv[q], cf, v[q]);
        }
    }
#pragma unroll
    for (int q = 0; q < 8; ++q) Vs[lane][q0 + q] = v[q] * rown;
}

// Diagonal block [k0, k0 + kb) of the reverse-order blocked Cholesky, 128
// threads.  With the block split 2 x 2 into 32 x 32 pieces,
//   A22 = R22 R22^T,  R12 = A12 R22^-T,  A11 - R12 R12^T = R11 R11^T,
//   V = R^-1 = [[V11, -V11 R12 V22], [0, V22]].
// All four warps factor and invert the two diagonal pieces together
// (cta_rchol_inv32) and form the 32 x 32 products.  Out: U_KK = V into
// A[K, K] (upper, in place of the block) and Vt = V^T (dense 64 x 64,
// row-major) for the panel solve.  Rows / columns >= kb are padded with the
// identity.
__global__ void __launch_bounds__(128) chol_diag_kernel(int64_t n, float *A, int64_t k0, int kb, int *status,
                                                        float *Vt) {
    __shared__ float S11[32][33], S22[32][33], A12[32][33];
    __shared__ float V11[32][33], V22[32][33], V12[32][33];
    __shared__ float R12[32][33], X[32][33];   // X = R12 V22
    __shared__ __align__(16) float bf[128];     // pivot broadcast slots
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    {
        // all loads of a thread are issued before the first use
        float x[NB * NB / 128];
#pragma unroll
        for (int t = 0; t < NB * NB / 128; ++t) {
            const int e = tid + t * 128, i = e >> 6, j = e & 63;
            x[t] = (i < kb && j < kb && j >= i) ? A[(k0 + i) * n + k0 + j] : 0.f;
        }
#pragma unroll
        for (int t = 0; t < NB * NB / 128; ++t) {
            const int e = tid + t * 128, i = e >> 6, j = e & 63;
            const float v = (i == j && i >= kb) ? 1.f : x[t];
            if (i < 32) {
                if (j < 32) S11[i][j] = v;
                else A12[i][j - 32] = v;
            } else if (j >= 32) {
                S22[i - 32][j - 32] = v;
            }
        }
    }
    __syncthreads();
    cta_rchol_inv32(S22, V22, bf, warp, lane, status, k0 + 32, kb - 32);
    __syncthreads();
    // R12[i][j] = sum_l A12[i][l] V22[j][l]   (V22 upper, zeros below)
#pragma unroll 1
    for (int e = tid; e < 32 * 32; e += 128) {
        const int i = e >> 5, j = e & 31;
        float acc = 0.f;
#pragma unroll 8
        for (int l = 0; l < 32; ++l) acc = fmaf(A12[i][l], V22[j][l], acc);
        R12[i][j] = acc;
    }
    __syncthreads();
    // A11 -= R12 R12^T and X = R12 V22
#pragma unroll 1
    for (int e = tid; e < 32 * 32; e += 128) {
        const int i = e >> 5, j = e & 31;
        float acc = 0.f, accx = 0.f;
#pragma unroll 8
        for (int l = 0; l < 32; ++l) {
            acc = fmaf(R12[i][l], R12[j][l], acc);
            accx = fmaf(R12[i][l], V22[l][j], accx);
        }
        S11[i][j] -= acc;
        X[i][j] = accx;
    }
    __syncthreads();
    cta_rchol_inv32(S11, V11, bf, warp, lane, status, k0, kb);
    __syncthreads();
    // V12 = -V11 X   (V11 upper, zeros below)
#pragma unroll 1
    for (int e = tid; e < 32 * 32; e += 128) {
        const int i = e >> 5, j = e & 31;
        float acc = 0.f;
#pragma unroll 8
        for (int l = 0; l < 32; ++l) acc = fmaf(V11[i][l], X[l][j], acc);
        V12[i][j] = -acc;
    }
    __syncthreads();
#pragma unroll 4
    for (int e = tid; e < NB * NB; e += 128) {
        const int r = e >> 6, c = e & 63;
        float x;
        if (r < 32) x = c < 32 ? V11[r][c] : V12[r][c - 32];
        else x = c < 32 ? 0.f : V22[r - 32][c - 32];
        if (r < kb && c < kb && c >= r) A[(k0 + r) * n + k0 + c] = x;
        Vt[c * NB + r] = x;
    }
}

// A[i][j] -= sum_c A[i][k0+c] A[j][k0+c] for i <= j < k0 (64 x 64 upper tiles,
// tile idx0 + blockIdx.x of the column-by-column enumeration: tile column tj
// holds tiles (0..tj, tj)).
__global__ void __launch_bounds__(256) chol_update_kernel(int64_t n, float *A, int64_t k0, int kb, int64_t idx0) {
    __shared__ __align__(16) float Pi[NB][NB + 4];
    __shared__ __align__(16) float Pj[NB][NB + 4];
    const int64_t idx = idx0 + blockIdx.x;
    int r = (int)((sqrt(8.0 * (double)idx + 1.0) - 1.0) * 0.5);
    while ((int64_t)(r + 1) * (r + 2) / 2 <= idx) ++r;
    while ((int64_t)r * (r + 1) / 2 > idx) --r;
    const int tj = r, ti = (int)(idx - (int64_t)r * (r + 1) / 2);  // ti <= tj
    const int64_t i0 = (int64_t)ti * NB, j0 = (int64_t)tj * NB;
    {
        // all loads of a thread are issued before the first use
        constexpr int PER = NB * NB / 256;
        float xi[PER], xj[PER];
#pragma unroll
        for (int t = 0; t < PER; ++t) {
            const int e = threadIdx.x + t * 256, rr = e / NB, c = e % NB;
            xi[t] = (c < kb && i0 + rr < k0) ? A[(i0 + rr) * n + k0 + c] : 0.f;
            xj[t] = (c < kb && j0 + rr < k0) ? A[(j0 + rr) * n + k0 + c] : 0.f;
        }
#pragma unroll
        for (int t = 0; t < PER; ++t) {
            const int e = threadIdx.x + t * 256, rr = e / NB, c = e % NB;
            Pi[c][rr] = xi[t];
            Pj[c][rr] = xj[t];
        }
    }
    __syncthreads();
    const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
    float acc[4][4] = {};
    for (int c = 0; c < kb; ++c) {
        const float4 a = *reinterpret_cast<const float4 *>(&Pi[c][ty * 4]);
        const float4 b = *reinterpret_cast<const float4 *>(&Pj[c][tx * 4]);
        const float av[4] = {a.x, a.y, a.z, a.w}, bv[4] = {b.x, b.y, b.z, b.w};
#pragma unroll
        for (int p = 0; p < 4; ++p)
#pragma unroll
            for (int q = 0; q < 4; ++q) acc[p][q] = fmaf(av[p], bv[q], acc[p][q]);
    }
#pragma unroll
    for (int p = 0; p < 4; ++p) {
        const int64_t gi = i0 + ty * 4 + p;
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const int64_t gj = j0 + tx * 4 + q;
            if (gi < k0 && gj < k0 && gj >= gi) A[gi * n + gj] -= acc[p][q];
        }
    }
}

__global__ void scale_kernel(int64_t count, float div, const float *in, float *out) {
    const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (i < count) out[i] = in[i] / div;
}

constexpr size_t align256(size_t x) { return (x + 255) / 256 * 256; }
constexpr int KSPLIT_MAX = 16;   // K slices of the triangular-inverse panel product
constexpr size_t prepare_bytes_split(int64_t n, int slices) {
    return align256(sizeof(int)) + align256(sizeof(float)) + align256((size_t)NB * NB * sizeof(float)) +
           align256((size_t)slices * n * NB * sizeof(float));
}
constexpr size_t prepare_bytes(int64_t n) { return prepare_bytes_split(n, 1); }
// tf32 hi / lo planes of two panels (n x NB each), for the rank-NB updates on
// the tensor cores (two sets: a step's panel is split while the previous
// step's update may still read the other set)
constexpr size_t tc_panel_bytes(int64_t n) { return 4 * align256((size_t)n * NB * sizeof(float)); }
// the triangular inverse's product on the tensor cores: planes of U^T (n x n,
// filled block column by block column as U's row blocks become final) and of
// the row block R[K, K+1:] (NB x n, at its global columns)
constexpr size_t tc_trtri_bytes(int64_t n) {
    return 2 * align256((size_t)n * n * sizeof(float)) + 2 * align256((size_t)NB * n * sizeof(float));
}
// the rank-NB update above the diagonal takes the tensor cores from this many
// rows on (below it the fp32 tiles, whose work is small)
constexpr int64_t kTcUpdateRows = 512;

// Scratch of the allocation-free entry point, sized for n <= REALQ_PREPARE_NOALLOC_MAX_N.
// Every GPU that loads the library holds it until the process exits.
constexpr size_t kNoAllocBytes = prepare_bytes(REALQ_PREPARE_NOALLOC_MAX_N);
static __device__ __align__(256) unsigned char g_prepare_scratch[kNoAllocBytes];

// Device address of g_prepare_scratch on the current device, looked up on
// every call (it allocates nothing): a cached address would outlive a reset
// device or a recreated primary context, after which the module is loaded
// again at another address.
realq_status_t noalloc_scratch(void **out) {
    void *p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_prepare_scratch);
    if (e != cudaSuccess || p == nullptr)
        return fail(REALQ_ERR_CUDA, "cudaGetSymbolAddress(prepare scratch): %s", cudaGetErrorString(e));
    *out = p;
    return REALQ_OK;
}

}  // namespace

size_t prepare_ws_bytes(int64_t n) {
    return prepare_bytes_split(n, KSPLIT_MAX) + tc_panel_bytes(n) + tc_trtri_bytes(n);
}

realq_status_t prepare_impl(cudaStream_t s, int64_t n, double norm, float damp, const float *H, float *U, float *Hbar,
                            uint8_t *dead, int64_t *fail_col, void *ws, size_t ws_bytes, bool overlap, bool sync);

realq_status_t prepare_noalloc(cudaStream_t s, int64_t n, int64_t T, float damp, const float *H, float *U, float *Hbar,
                               uint8_t *dead, int64_t *fail_col) {
    void *scratch = nullptr;
    REALQ_TRY(noalloc_scratch(&scratch));
    // single stream: this entry point creates no stream or event
    return prepare_impl(s, n, (double)T, damp, H, U, Hbar, dead, fail_col, scratch, kNoAllocBytes, false, true);
}

// Auxiliary streams of the calling thread (and their events) for the U row
// work and the look-ahead, one set per (device, caller's stream, its
// priority), created on first use and kept for the life of the thread.  Keyed
// by the caller's stream so that calls on different streams (e.g. enqueued
// one after another into one CUDA graph) share no stream and so no false
// dependency.
struct AuxStream {
    int device = -1, priority = 0;
    cudaStream_t caller = nullptr;
    cudaStream_t stream = nullptr;       // U row work
    cudaStream_t wide = nullptr;         // the look-ahead's wide trailing updates
    cudaEvent_t ev[3] = {nullptr, nullptr, nullptr};
    std::vector<cudaEvent_t> steps, pdone, wdone;
};
static thread_local std::vector<AuxStream> g_aux;

realq_status_t aux_for(cudaStream_t s, int64_t nsteps, AuxStream **out) {
    int dev = 0, prio = 0;
    REALQ_CUDA_TRY(cudaGetDevice(&dev));
    REALQ_CUDA_TRY(cudaStreamGetPriority(s, &prio));
    AuxStream *found = nullptr;
    for (AuxStream &x : g_aux)
        if (x.device == dev && x.priority == prio && x.caller == s) found = &x;
    if (!found) {
        AuxStream a;
        REALQ_CUDA_TRY(cudaStreamCreateWithPriority(&a.stream, cudaStreamNonBlocking, prio));
        REALQ_CUDA_TRY(cudaStreamCreateWithPriority(&a.wide, cudaStreamNonBlocking, prio));
        for (int i = 0; i < 3; ++i) REALQ_CUDA_TRY(cudaEventCreateWithFlags(&a.ev[i], cudaEventDisableTiming));
        a.device = dev;
        a.priority = prio;
        a.caller = s;
        g_aux.push_back(a);
        found = &g_aux.back();
    }
    AuxStream &a = *found;
    for (std::vector<cudaEvent_t> *v : {&a.steps, &a.pdone, &a.wdone}) {
        while ((int64_t)v->size() < nsteps) {
            cudaEvent_t e;
            REALQ_CUDA_TRY(cudaEventCreateWithFlags(&e, cudaEventDisableTiming));
            v->push_back(e);
        }
    }
    *out = &a;
    return REALQ_OK;
}

realq_status_t prepare(cudaStream_t s, int64_t n, double norm, float damp, const float *H, float *U, float *Hbar,
                       uint8_t *dead, int64_t *fail_col, void *ws, size_t ws_bytes) {
    return prepare_impl(s, n, norm, damp, H, U, Hbar, dead, fail_col, ws, ws_bytes, !profiling(), true);
}

realq_status_t prepare_deferred(cudaStream_t s, int64_t n, double norm, float damp, const float *H, float *U,
                                float *Hbar, uint8_t *dead, void *ws, size_t ws_bytes) {
    return prepare_impl(s, n, norm, damp, H, U, Hbar, dead, nullptr, ws, ws_bytes, !profiling(), false);
}

realq_status_t prepare_impl(cudaStream_t s, int64_t n, double norm, float damp, const float *H, float *U, float *Hbar,
                            uint8_t *dead, int64_t *fail_col, void *ws, size_t ws_bytes, bool overlap, bool sync) {
    Carve cv(ws);
    int *status = cv.take<int>(1);
    float *lam = cv.take<float>(1);
    float *Vd = cv.take<float>((size_t)NB * NB);
    float *panel = cv.take<float>(0);
    // the wide rank-NB updates on the tensor cores when the workspace has
    // room for the panel planes besides one panel slice (otherwise the fp32
    // tiles) and n suits the product
    const bool tc_update = n % 4 == 0 && n > kTcUpdateRows && tc_gemm_eligible(n, n) &&
                           ws_bytes >= prepare_bytes_split(n, 1) + tc_panel_bytes(n);
    const bool tc_trtri = tc_update && ws_bytes >= prepare_bytes_split(n, 1) + tc_panel_bytes(n) + tc_trtri_bytes(n);
    const size_t reserve = (tc_update ? tc_panel_bytes(n) : 0) + (tc_trtri ? tc_trtri_bytes(n) : 0);
    // as many K slices of the panel product as the workspace holds
    int slices = 1;
    while (slices < KSPLIT_MAX && prepare_bytes_split(n, slices + 1) + reserve <= ws_bytes) ++slices;
    const int64_t plane = n * NB;
    float *Pp[4] = {nullptr, nullptr, nullptr, nullptr};   // set 0 hi, lo; set 1 hi, lo
    float *UTh = nullptr, *UTl = nullptr, *Rh = nullptr, *Rl = nullptr;
    TcMaps pmaps[2], tmaps;
    if (tc_update) {
        Carve pc(reinterpret_cast<unsigned char *>(ws) + prepare_bytes_split(n, slices));
        for (int i = 0; i < 4; ++i) Pp[i] = pc.take<float>((size_t)n * NB);
        for (int st = 0; st < 2; ++st)
            REALQ_TRY(tc_make_maps(&pmaps[st], Pp[2 * st], Pp[2 * st + 1], n, NB, NB, Pp[2 * st], Pp[2 * st + 1], n,
                                   NB, NB));
        if (tc_trtri) {
            UTh = pc.take<float>((size_t)n * n);
            UTl = pc.take<float>((size_t)n * n);
            Rh = pc.take<float>((size_t)NB * n);
            Rl = pc.take<float>((size_t)NB * n);
            // A: the row block R[K, K+1:] (NB rows, columns at their global
            // index); B: rows of U^T, so that both take K from column k1 on
            REALQ_TRY(tc_make_maps(&tmaps, Rh, Rl, NB, n, n, UTh, UTl, n, n, n));
        }
    }
    // status[0]: the failing column (-1: none); status[1]: timeout bits of
    // the tensor-core updates (the same 256-byte slot of the workspace)
    int *status_tc = status + 1;
    REALQ_CUDA_TRY(cudaMemsetAsync(status, 0xFF, sizeof(int), s));
    REALQ_CUDA_TRY(cudaMemsetAsync(status_tc, 0, sizeof(int), s));
    const int64_t tot = n * n;
    {
        Launch L("prepare_init", s);
        prep_init_kernel<<<(unsigned)((tot + 255) / 256), 256, 0, s>>>(n, (float)norm, H, Hbar, U, dead);
    }
    REALQ_TRY(check_launch("prepare_init"));
    {
        Launch L("prepare_damp", s);
        prep_damp_kernel<<<1, 1024, 0, s>>>(n, U, damp, lam);
    }
    REALQ_TRY(check_launch("prepare_damp"));
    // Reverse-order blocked Cholesky Hd = R R^T, with U = R^-1 formed block row
    // by block row as soon as a row block of R is final: after step K no later
    // step reads row block K of R, and
    //   U[K, K] = R_KK^-1,  U[K, K+1:] = -U[K, K] (R[K, K+1:] U[K+1:, K+1:]).
    const int nbk = ceil_div(n, NB);
    // Row block K of U touches rows >= k0 only, the later Cholesky steps rows
    // < k0 only: with overlap, the U row work runs on an auxiliary stream that
    // starts after the diagonal step of K (which wrote U_KK into A[K, K]).
    if (tc_trtri) {
        // U^T's planes are filled on and below the diagonal, block column by
        // block column; what lies above it is read as zeros
        REALQ_CUDA_TRY(cudaMemsetAsync(UTh, 0, (size_t)n * n * sizeof(float), s));
        REALQ_CUDA_TRY(cudaMemsetAsync(UTl, 0, (size_t)n * n * sizeof(float), s));
    }
    AuxStream *aux = nullptr;
    if (overlap && nbk > 1) REALQ_TRY(aux_for(s, nbk, &aux));
    cudaStream_t rs = aux ? aux->stream : s;
    if (aux) {
        REALQ_CUDA_TRY(cudaEventRecord(aux->ev[0], s));
        REALQ_CUDA_TRY(cudaStreamWaitEvent(rs, aux->ev[0], 0));
    }
    std::vector<char> wide_pending(nbk + 1, 0);
    bool wide_used = false;
    for (int K = nbk - 1; K >= 0; --K) {
        const int64_t k0 = (int64_t)K * NB;
        const int kb = (int)std::min<int64_t>(NB, n - k0);
        const int64_t k1 = k0 + kb;
        {
            Launch L("chol_diag", s);
            chol_diag_kernel<<<1, 128, 0, s>>>(n, U, k0, kb, status, Vd);
        }
        REALQ_TRY(check_launch("chol_diag"));
        if (aux && (k1 < n || tc_trtri)) {
            REALQ_CUDA_TRY(cudaEventRecord(aux->steps[K], s));
            REALQ_CUDA_TRY(cudaStreamWaitEvent(rs, aux->steps[K], 0));
        }
        if (k0 > 0) {
            // rows above the block: R[0:k0, K] = A[0:k0, K] R_KK^-T (in place; one
            // column tile, so every CTA reads only the rows it writes)
            GemmArgs pg{};
            pg.M = k0; pg.N = kb; pg.K = kb;
            pg.A = U + k0; pg.lda = n;
            pg.B = Vd; pg.ldb = NB;
            pg.C = U + k0; pg.ldc = n;
            pg.alpha = 1.f;
            REALQ_TRY(gemm_f32(s, A_ROW, EPI_STORE, pg, "chol_panel"));
            // Rank-kb update of the block above.  Look-ahead: the next step
            // needs only tile column nt0 - 1 (its diagonal block and its
            // panel), which is updated at once; the other columns ("wide")
            // run on a second stream, overlapped with the next diagonal
            // factorisation and panel, and the next narrow update waits for
            // them because it touches their last column.
            const int64_t nt0 = k0 / NB;
            const int64_t nwide = (nt0 - 1) * nt0 / 2;
            if (aux && nwide > 0) {
                REALQ_CUDA_TRY(cudaEventRecord(aux->pdone[K], s));
                REALQ_CUDA_TRY(cudaStreamWaitEvent(aux->wide, aux->pdone[K], 0));
            }
            if (aux && K + 1 < nbk && wide_pending[K + 1]) REALQ_CUDA_TRY(cudaStreamWaitEvent(s, aux->wdone[K + 1], 0));
            {
                Launch L("chol_update", s);
                chol_update_kernel<<<(unsigned)nt0, 256, 0, s>>>(n, U, k0, kb, nwide);
            }
            REALQ_TRY(check_launch("chol_update"));
            if (nwide > 0) {
                cudaStream_t ws_ = aux ? aux->wide : s;
                const int64_t kw = k0 - NB;   // rows and columns of the wide part
                if (tc_update && kw >= kTcUpdateRows) {
                    // U[0:kw, 0:kw] (upper) -= P P^T with P = R[0:kw, K], as
                    // a tf32x3 symmetric product on the tensor cores
                    const int st = K & 1;
                    REALQ_TRY(tc_split_rows(ws_, kw, kb, U + k0, n, Pp[2 * st], Pp[2 * st + 1], NB, NB));
                    TcEpi e{};
                    e.mode = TC_SYRK;
                    e.M = U;
                    e.ldw = n;
                    REALQ_TRY(tc_gemm_x3(ws_, pmaps[st], kw, kw, NB, 0, 0, e, status_tc, "chol_update_tc"));
                } else {
                    Launch L("chol_update", ws_);
                    chol_update_kernel<<<(unsigned)nwide, 256, 0, ws_>>>(n, U, k0, kb, 0);
                }
                REALQ_TRY(check_launch("chol_update"));
                if (aux) {
                    REALQ_CUDA_TRY(cudaEventRecord(aux->wdone[K], aux->wide));
                    wide_pending[K] = 1;
                    wide_used = true;
                }
            }
        }
        if (k1 < n && tc_trtri) {
            const int64_t r = n - k1;
            // X = R[K, K+1:] U[K+1:, K+1:] on the tensor cores: the planes of
            // the row block, then X = R_K (U^T)^T with U^T's rows k1.. (a
            // column tile's K range ends at its last column: U is upper)
            REALQ_TRY(tc_split_rows(rs, kb, r, U + k0 * n + k1, n, Rh + k1, Rl + k1, n, r));
            TcEpi e{};
            e.mode = TC_STORE;
            e.C = panel;
            e.ldc = n;
            e.b_tri = 1;
            REALQ_TRY(tc_gemm_x3(rs, tmaps, kb, r, r, (int)k1, (int)k1, e, status_tc, "trtri_trmm_tc"));
            // U[K, K+1:] = -U_KK X, U_KK read from A[K, K] (upper, zeros below)
            GemmArgs h{};
            h.M = kb; h.N = r; h.K = kb;
            h.A = U + k0 * n + k0; h.lda = n;
            h.B = panel; h.ldb = n; h.nsum_b = 1; h.bplane = plane;
            h.C = U + k0 * n + k1; h.ldc = n;
            h.alpha = -1.f;
            REALQ_TRY(gemm_f32(rs, A_ROW, EPI_STORE, h, "trtri_panel"));
        } else if (k1 < n) {
            const int64_t r = n - k1;
            // X = R[K, K+1:] U[K+1:, K+1:] (U upper: a column tile's K range ends
            // at its last column), K split into fixed-order slices
            const int ks = (int)std::max<int64_t>(1, std::min<int64_t>(slices, r / 256));
            GemmArgs g{};
            g.M = kb; g.N = r; g.K = r;
            g.A = U + k0 * n + k1; g.lda = n;
            g.B = U + k1 * n + k1; g.ldb = n;
            g.C = panel; g.ldc = n;
            g.ksplit = ks; g.cplane = plane; g.b_upper = 1;
            g.alpha = 1.f;
            REALQ_TRY(gemm_f32(rs, A_ROW, EPI_STORE, g, "trtri_trmm"));
            // U[K, K+1:] = -U_KK X, U_KK read from A[K, K] (upper, zeros below)
            GemmArgs h{};
            h.M = kb; h.N = r; h.K = kb;
            h.A = U + k0 * n + k0; h.lda = n;
            h.B = panel; h.ldb = n; h.nsum_b = ks; h.bplane = plane;
            h.C = U + k0 * n + k1; h.ldc = n;
            h.alpha = -1.f;
            REALQ_TRY(gemm_f32(rs, A_ROW, EPI_STORE, h, "trtri_panel"));
        }
        // row block K of U is final: its transpose joins U^T's planes for the
        // later steps' products
        if (tc_trtri)
            REALQ_TRY(tc_trans_planes(rs, kb, n - k0, U + k0 * n + k0, n, UTh + k0 * n + k0, UTl + k0 * n + k0, n));
    }
    if (aux) {
        REALQ_CUDA_TRY(cudaEventRecord(aux->ev[1], rs));
        REALQ_CUDA_TRY(cudaStreamWaitEvent(s, aux->ev[1], 0));
        // join the wide stream only if it forked from s (under stream capture
        // a wait on an event recorded outside the capture is an error)
        if (wide_used) {
            REALQ_CUDA_TRY(cudaEventRecord(aux->ev[2], aux->wide));
            REALQ_CUDA_TRY(cudaStreamWaitEvent(s, aux->ev[2], 0));
        }
    }
    if (!sync) return REALQ_OK;  // the failing column stays in the workspace's first word
    int host_status[2] = {-1, 0};
    REALQ_CUDA_TRY(cudaMemcpyAsync(host_status, status, 2 * sizeof(int), cudaMemcpyDeviceToHost, s));
    REALQ_CUDA_TRY(cudaStreamSynchronize(s));
    *fail_col = host_status[0];
    if (host_status[1] & ST_TIMEOUT) return fail(REALQ_ERR_TIMEOUT, "a bounded device-side wait gave up (prepare)");
    if (host_status[0] >= 0)
        return fail(REALQ_ERR_NOT_SPD, "damped Hessian not positive definite at column %d", host_status[0]);
    return REALQ_OK;
}

realq_status_t scale_copy(cudaStream_t s, int64_t count, float div, const float *in, float *out) {
    if (count == 0) return REALQ_OK;
    {
        Launch L("scale_moment", s);
        scale_kernel<<<(unsigned)((count + 255) / 256), 256, 0, s>>>(count, div, in, out);
    }
    return check_launch("scale_moment");
}

}  // namespace realq
