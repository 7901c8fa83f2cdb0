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
// column in the workspace status word; the host reads it once at the end.
#include "kernels.cuh"

#include <mutex>
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

// The 64 x 64 diagonal-block kernels below use 256 threads as a 16 x 16 grid;
// thread (ty, tx) keeps the 4 x 4 block rows 4ty.., columns 4tx.. in
// registers, and only the pivot and the pivot column / row travel through
// double-buffered shared memory.

// V = R^-1 for the kb x kb upper triangle in Rs, by row operations on the
// identity (back substitution applied to all columns at once); v is this
// thread's 4 x 4 block of V.  One barrier per pivot.
__device__ __forceinline__ void upper_inverse_regs(const float (*Rs)[NB + 1], int kb, float (&v)[4][4],
                                                   float (*rowk)[NB]) {
    const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
#pragma unroll
    for (int a = 0; a < 4; ++a)
#pragma unroll
        for (int b = 0; b < 4; ++b) v[a][b] = (ty * 4 + a == tx * 4 + b && ty * 4 + a < kb) ? 1.f : 0.f;
    for (int k = kb - 1; k >= 0; --k) {
        const int kt = k >> 2, kq = k & 3, p = k & 1;
        if (ty == kt) {
            const float rinv = 1.f / Rs[k][k];
#pragma unroll
            for (int a = 0; a < 4; ++a)
                if (a == kq) {
#pragma unroll
                    for (int b = 0; b < 4; ++b) {
                        v[a][b] = v[a][b] * rinv;
                        rowk[p][tx * 4 + b] = v[a][b];
                    }
                }
        }
        __syncthreads();
        float rv[4];
#pragma unroll
        for (int b = 0; b < 4; ++b) rv[b] = rowk[p][tx * 4 + b];
#pragma unroll
        for (int a = 0; a < 4; ++a) {
            const int i = ty * 4 + a;
            if (i < k) {
                const float rik = Rs[i][k];
#pragma unroll
                for (int b = 0; b < 4; ++b) v[a][b] -= rik * rv[b];
            }
        }
    }
}

// Diagonal block [k0, k0 + kb): A_KK = R_KK R_KK^T with R_KK upper (in place),
// and Vt = (R_KK^-1)^T (dense 64 x 64, row-major) for the panel solve.
// Two barriers per Cholesky pivot, one per inverse pivot.
__global__ void __launch_bounds__(256) chol_diag_kernel(int64_t n, float *A, int64_t k0, int kb, int *status,
                                                        float *Vt) {
    __shared__ float Rs[NB][NB + 1];
    __shared__ float colk[2][NB];
    __shared__ float rk_s[2];
    const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
    float sv[4][4];
#pragma unroll
    for (int a = 0; a < 4; ++a)
#pragma unroll
        for (int b = 0; b < 4; ++b) {
            const int r = ty * 4 + a, c = tx * 4 + b;
            sv[a][b] = (r < kb && c < kb && c >= r) ? A[(k0 + r) * n + k0 + c] : 0.f;
        }
    for (int k = kb - 1; k >= 0; --k) {
        const int kt = k >> 2, kq = k & 3, p = k & 1;
        if (ty == kt && tx == kt) {
#pragma unroll
            for (int a = 0; a < 4; ++a)
                if (a == kq) {
                    float d = sv[a][a];
                    const bool bad = !(d > 0.f) || !isfinite(d);
                    if (bad) {
                        atomicCAS(status, -1, (int)(k0 + k));
                        d = 1.f;
                    }
                    const float rk = sqrtf(d);
                    sv[a][a] = rk;
                    rk_s[p] = rk;
                }
        }
        __syncthreads();
        if (tx == kt) {
            const float rinv = 1.f / rk_s[p];
#pragma unroll
            for (int b = 0; b < 4; ++b)
                if (b == kq) {
#pragma unroll
                    for (int a = 0; a < 4; ++a) {
                        const int i = ty * 4 + a;
                        if (i < k) {
                            sv[a][b] = sv[a][b] * rinv;
                            colk[p][i] = sv[a][b];
                        }
                    }
                }
        }
        __syncthreads();
        if (ty * 4 < k && tx * 4 < k) {
            float ci[4], cj[4];
#pragma unroll
            for (int a = 0; a < 4; ++a) ci[a] = colk[p][ty * 4 + a];
#pragma unroll
            for (int b = 0; b < 4; ++b) cj[b] = colk[p][tx * 4 + b];
#pragma unroll
            for (int a = 0; a < 4; ++a)
#pragma unroll
                for (int b = 0; b < 4; ++b) {
                    const int i = ty * 4 + a, j = tx * 4 + b;
                    if (i <= j && j < k) sv[a][b] -= ci[a] * cj[b];
                }
        }
    }
#pragma unroll
    for (int a = 0; a < 4; ++a)
#pragma unroll
        for (int b = 0; b < 4; ++b) Rs[ty * 4 + a][tx * 4 + b] = sv[a][b];
    __syncthreads();
    __shared__ float rowk[2][NB];
    float v[4][4];
    upper_inverse_regs(Rs, kb, v, rowk);
    // U_KK = R_KK^-1 goes to A[K, K]; Vt = U_KK^T feeds the panel solve
#pragma unroll
    for (int a = 0; a < 4; ++a)
#pragma unroll
        for (int b = 0; b < 4; ++b) {
            const int r = ty * 4 + a, c = tx * 4 + b;
            if (r < kb && c < kb && c >= r) A[(k0 + r) * n + k0 + c] = v[a][b];
            Vt[c * NB + r] = v[a][b];
        }
}

// A[i][j] -= sum_c A[i][k0+c] A[j][k0+c] for i <= j < k0 (64 x 64 upper tiles).
__global__ void __launch_bounds__(256) chol_update_kernel(int64_t n, float *A, int64_t k0, int kb) {
    __shared__ __align__(16) float Pi[NB][NB + 4];
    __shared__ __align__(16) float Pj[NB][NB + 4];
    const int64_t idx = blockIdx.x;
    int r = (int)((sqrt(8.0 * (double)idx + 1.0) - 1.0) * 0.5);
    while ((int64_t)(r + 1) * (r + 2) / 2 <= idx) ++r;
    while ((int64_t)r * (r + 1) / 2 > idx) --r;
    const int tj = r, ti = (int)(idx - (int64_t)r * (r + 1) / 2);  // ti <= tj
    const int64_t i0 = (int64_t)ti * NB, j0 = (int64_t)tj * NB;
    for (int e = threadIdx.x; e < NB * NB; e += blockDim.x) {
        const int rr = e / NB, c = e % NB;
        Pi[c][rr] = (c < kb && i0 + rr < k0) ? A[(i0 + rr) * n + k0 + c] : 0.f;
        Pj[c][rr] = (c < kb && j0 + rr < k0) ? A[(j0 + rr) * n + k0 + c] : 0.f;
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
constexpr int KSPLIT_MAX = 8;    // K slices of the triangular-inverse panel product
constexpr size_t prepare_bytes_split(int64_t n, int slices) {
    return align256(sizeof(int)) + align256(sizeof(float)) + align256((size_t)NB * NB * sizeof(float)) +
           align256((size_t)slices * n * NB * sizeof(float));
}
constexpr size_t prepare_bytes(int64_t n) { return prepare_bytes_split(n, 1); }

// Scratch of the allocation-free entry point, sized for n <= REALQ_PREPARE_NOALLOC_MAX_N.
// Every GPU that loads the library holds it until the process exits.
constexpr size_t kNoAllocBytes = prepare_bytes(REALQ_PREPARE_NOALLOC_MAX_N);
static __device__ __align__(256) unsigned char g_prepare_scratch[kNoAllocBytes];

std::mutex g_noalloc_mu;
void *g_noalloc_ptr[256] = {};

// Device address of g_prepare_scratch on the current device (looked up once per device).
realq_status_t noalloc_scratch(void **out) {
    int dev = 0;
    REALQ_CUDA_TRY(cudaGetDevice(&dev));
    if (dev < 0 || dev >= 256) return fail(REALQ_ERR_UNSUPPORTED, "device ordinal %d out of range", dev);
    std::lock_guard<std::mutex> lk(g_noalloc_mu);
    if (g_noalloc_ptr[dev] == nullptr) {
        void *p = nullptr;
        const cudaError_t e = cudaGetSymbolAddress(&p, g_prepare_scratch);
        if (e != cudaSuccess || p == nullptr)
            return fail(REALQ_ERR_CUDA, "cudaGetSymbolAddress(prepare scratch): %s", cudaGetErrorString(e));
        g_noalloc_ptr[dev] = p;
    }
    *out = g_noalloc_ptr[dev];
    return REALQ_OK;
}

}  // namespace

size_t prepare_ws_bytes(int64_t n) { return prepare_bytes_split(n, KSPLIT_MAX); }

realq_status_t prepare_impl(cudaStream_t s, int64_t n, int64_t T, float damp, const float *H, float *U, float *Hbar,
                            uint8_t *dead, int64_t *fail_col, void *ws, size_t ws_bytes, bool overlap);

realq_status_t prepare_noalloc(cudaStream_t s, int64_t n, int64_t T, float damp, const float *H, float *U, float *Hbar,
                               uint8_t *dead, int64_t *fail_col) {
    void *scratch = nullptr;
    REALQ_TRY(noalloc_scratch(&scratch));
    // single stream: this entry point creates no stream or event
    return prepare_impl(s, n, T, damp, H, U, Hbar, dead, fail_col, scratch, kNoAllocBytes, false);
}

// Auxiliary stream of the calling thread (and its events) for the U row
// work, one per (device, priority of the caller's stream), created on first
// use and kept for the life of the thread.
struct AuxStream {
    int device = -1, priority = 0;
    cudaStream_t stream = nullptr;
    cudaEvent_t ev[2] = {nullptr, nullptr};
    std::vector<cudaEvent_t> steps;
};
static thread_local std::vector<AuxStream> g_aux;

realq_status_t aux_for(cudaStream_t s, int64_t nsteps, AuxStream **out) {
    int dev = 0, prio = 0;
    REALQ_CUDA_TRY(cudaGetDevice(&dev));
    REALQ_CUDA_TRY(cudaStreamGetPriority(s, &prio));
    AuxStream *found = nullptr;
    for (AuxStream &x : g_aux)
        if (x.device == dev && x.priority == prio) found = &x;
    if (!found) {
        AuxStream a;
        REALQ_CUDA_TRY(cudaStreamCreateWithPriority(&a.stream, cudaStreamNonBlocking, prio));
        REALQ_CUDA_TRY(cudaEventCreateWithFlags(&a.ev[0], cudaEventDisableTiming));
        REALQ_CUDA_TRY(cudaEventCreateWithFlags(&a.ev[1], cudaEventDisableTiming));
        a.device = dev;
        a.priority = prio;
        g_aux.push_back(a);
        found = &g_aux.back();
    }
    AuxStream &a = *found;
    while ((int64_t)a.steps.size() < nsteps) {
        cudaEvent_t e;
        REALQ_CUDA_TRY(cudaEventCreateWithFlags(&e, cudaEventDisableTiming));
        a.steps.push_back(e);
    }
    *out = &a;
    return REALQ_OK;
}

realq_status_t prepare(cudaStream_t s, int64_t n, int64_t T, float damp, const float *H, float *U, float *Hbar,
                       uint8_t *dead, int64_t *fail_col, void *ws, size_t ws_bytes) {
    return prepare_impl(s, n, T, damp, H, U, Hbar, dead, fail_col, ws, ws_bytes, true);
}

realq_status_t prepare_impl(cudaStream_t s, int64_t n, int64_t T, float damp, const float *H, float *U, float *Hbar,
                            uint8_t *dead, int64_t *fail_col, void *ws, size_t ws_bytes, bool overlap) {
    Carve cv(ws);
    int *status = cv.take<int>(1);
    float *lam = cv.take<float>(1);
    float *Vd = cv.take<float>((size_t)NB * NB);
    float *panel = cv.take<float>(0);
    // as many K slices of the panel product as the workspace holds
    int slices = 1;
    while (slices < KSPLIT_MAX && prepare_bytes_split(n, slices + 1) <= ws_bytes) ++slices;
    const int64_t plane = n * NB;
    REALQ_CUDA_TRY(cudaMemsetAsync(status, 0xFF, sizeof(int), s));
    const int64_t tot = n * n;
    {
        Launch L("prepare_init", s);
        prep_init_kernel<<<(unsigned)((tot + 255) / 256), 256, 0, s>>>(n, (float)T, H, Hbar, U, dead);
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
    AuxStream *aux = nullptr;
    if (overlap && nbk > 1) REALQ_TRY(aux_for(s, nbk, &aux));
    cudaStream_t rs = aux ? aux->stream : s;
    if (aux) {
        REALQ_CUDA_TRY(cudaEventRecord(aux->ev[0], s));
        REALQ_CUDA_TRY(cudaStreamWaitEvent(rs, aux->ev[0], 0));
    }
    for (int K = nbk - 1; K >= 0; --K) {
        const int64_t k0 = (int64_t)K * NB;
        const int kb = (int)std::min<int64_t>(NB, n - k0);
        const int64_t k1 = k0 + kb;
        {
            Launch L("chol_diag", s);
            chol_diag_kernel<<<1, 256, 0, s>>>(n, U, k0, kb, status, Vd);
        }
        REALQ_TRY(check_launch("chol_diag"));
        if (aux && k1 < n) {
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
            const int64_t nt0 = k0 / NB;
            {
                Launch L("chol_update", s);
                chol_update_kernel<<<(unsigned)(nt0 * (nt0 + 1) / 2), 256, 0, s>>>(n, U, k0, kb);
            }
            REALQ_TRY(check_launch("chol_update"));
        }
        if (k1 < n) {
            const int64_t r = n - k1;
            // X = R[K, K+1:] U[K+1:, K+1:] (U upper: a column tile's K range ends
            // at its last column), K split into fixed-order slices
            const int ks = (int)std::max<int64_t>(1, std::min<int64_t>(slices, r / 512));
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
    }
    if (aux) {
        REALQ_CUDA_TRY(cudaEventRecord(aux->ev[1], rs));
        REALQ_CUDA_TRY(cudaStreamWaitEvent(s, aux->ev[1], 0));
    }
    int host_status = -1;
    REALQ_CUDA_TRY(cudaMemcpyAsync(&host_status, status, sizeof(int), cudaMemcpyDeviceToHost, s));
    REALQ_CUDA_TRY(cudaStreamSynchronize(s));
    *fail_col = host_status;
    if (host_status >= 0) return fail(REALQ_ERR_NOT_SPD, "damped Hessian not positive definite at column %d", host_status);
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
