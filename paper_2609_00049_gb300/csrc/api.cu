// C ABI of the library (include/realq.h): argument validation, workspace
// checks, sequencing of the kernels of one call, error reporting, launch
// accounting and optional per-kernel event timing.
#include "kernels.cuh"

#include <algorithm>
#include <atomic>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <map>
#include <mutex>
#include <set>
#include <tuple>
#include <string>
#include <vector>

namespace realq {

// ------------------------------------------------------------ error text ---
static thread_local char g_err[512] = "";

void set_error(const char *fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_err, sizeof(g_err), fmt, ap);
    va_end(ap);
}

realq_status_t fail(realq_status_t s, const char *fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_err, sizeof(g_err), fmt, ap);
    va_end(ap);
    return s;
}

realq_status_t check_launch(const char *what) {
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return fail(REALQ_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
    return REALQ_OK;
}

realq_status_t set_smem_limit(const void *kernel, int bytes) {
    int dev = 0;
    REALQ_CUDA_TRY(cudaGetDevice(&dev));
    static std::mutex mu;
    static std::set<std::tuple<const void *, int, int>> done;
    std::lock_guard<std::mutex> lk(mu);
    const auto key = std::make_tuple(kernel, dev, bytes);
    if (done.count(key)) return REALQ_OK;
    REALQ_CUDA_TRY(cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes));
    done.insert(key);
    return REALQ_OK;
}

// ------------------------------------------------------ launch accounting ---
static std::atomic<int64_t> g_launches{0};
static std::atomic<int> g_prof_on{0};
bool profiling() { return g_prof_on.load(std::memory_order_relaxed) != 0; }
struct ProfRec {
    const char *name;
    cudaEvent_t a, b;
};
static std::mutex g_prof_mu;
static std::vector<ProfRec> g_pending;
static std::vector<cudaEvent_t> g_pool;

static cudaEvent_t pool_get() {
    if (!g_pool.empty()) {
        cudaEvent_t e = g_pool.back();
        g_pool.pop_back();
        return e;
    }
    cudaEvent_t e = nullptr;
    if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
    return e;
}

Launch::Launch(const char *n, cudaStream_t s) : name(n), stream(s), slot(-1) {
    g_launches.fetch_add(1, std::memory_order_relaxed);
    if (!g_prof_on.load(std::memory_order_relaxed)) return;
    std::lock_guard<std::mutex> lk(g_prof_mu);
    ProfRec r{n, pool_get(), pool_get()};
    if (!r.a || !r.b) return;
    cudaEventRecord(r.a, s);
    g_pending.push_back(r);
    slot = (int)g_pending.size() - 1;
}

Launch::~Launch() {
    if (slot < 0) return;
    std::lock_guard<std::mutex> lk(g_prof_mu);
    if (slot < (int)g_pending.size()) cudaEventRecord(g_pending[slot].b, stream);
}

}  // namespace realq

using namespace realq;

namespace {

cudaStream_t S(realq_stream_t s) { return static_cast<cudaStream_t>(s); }

realq_status_t check_ws(void *ws, size_t have, size_t need, const char *who) {
    if (need == 0) return REALQ_OK;
    if (ws == nullptr) return fail(REALQ_ERR_WORKSPACE, "%s: workspace of %zu bytes required", who, need);
    if (reinterpret_cast<uintptr_t>(ws) % kAlign != 0)
        return fail(REALQ_ERR_WORKSPACE, "%s: workspace must be %zu-byte aligned", who, kAlign);
    if (have < need) return fail(REALQ_ERR_WORKSPACE, "%s: workspace %zu < %zu bytes", who, have, need);
    return REALQ_OK;
}

bool valid_dtype(realq_dtype_t d) { return d == REALQ_F32 || d == REALQ_BF16; }

realq_status_t check_qcfg(const realq_quant_cfg_t *q, int64_t n) {
    if (!q) return fail(REALQ_ERR_INVALID_ARG, "qcfg is NULL");
    if (q->bits < 2 || q->bits > 4) return fail(REALQ_ERR_INVALID_ARG, "bits must be in [2, 4] (got %d)", q->bits);
    if (q->block_size != 32 && q->block_size != 64 && q->block_size != 128)
        return fail(REALQ_ERR_INVALID_ARG, "block_size must be 32, 64 or 128 (got %d)", q->block_size);
    if (q->group_size < 0) return fail(REALQ_ERR_INVALID_ARG, "group_size must be >= 0");
    if (q->symmetric != 0 && q->symmetric != 1) return fail(REALQ_ERR_INVALID_ARG, "symmetric must be 0 or 1");
    if (!(q->damp_frac >= 0.f) || !std::isfinite(q->damp_frac)) return fail(REALQ_ERR_INVALID_ARG, "damp_frac must be >= 0");
    const int B = q->block_size;
    const int g = q->group_size == 0 ? (int)std::min<int64_t>(n, 1 << 30) : q->group_size;
    if (q->group_size != 0) {
        if (g <= B) {
            if (B % g != 0 || (g != B && g != B / 2 && g != B / 4) || g < 32)
                return fail(REALQ_ERR_UNSUPPORTED, "group_size %d inside block %d (supported: B, B/2, B/4, >= 32)", g, B);
        } else if (g % B != 0) {
            return fail(REALQ_ERR_INVALID_ARG, "group_size %d must be a multiple of block_size %d", g, B);
        }
    }
    return REALQ_OK;
}

realq_status_t check_bcfg(const realq_bgd_cfg_t *b) {
    if (!b) return REALQ_OK;
    if (b->steps_per_block < 0) return fail(REALQ_ERR_INVALID_ARG, "steps_per_block must be >= 0");
    if (b->optimizer != REALQ_OPT_ADAM && b->optimizer != REALQ_OPT_SGD)
        return fail(REALQ_ERR_INVALID_ARG, "optimizer must be REALQ_OPT_ADAM or REALQ_OPT_SGD");
    if (!std::isfinite(b->lr) || b->lr < 0.f) return fail(REALQ_ERR_INVALID_ARG, "lr must be finite and >= 0");
    if (b->optimizer == REALQ_OPT_ADAM) {
        if (!(b->beta1 >= 0.f && b->beta1 < 1.f) || !(b->beta2 >= 0.f && b->beta2 < 1.f))
            return fail(REALQ_ERR_INVALID_ARG, "betas must be in [0, 1)");
        if (!(b->eps > 0.f)) return fail(REALQ_ERR_INVALID_ARG, "eps must be > 0");
    }
    if (b->b_global_start < 1 || b->B_total < 1) return fail(REALQ_ERR_INVALID_ARG, "b_global_start and B_total must be >= 1");
    return REALQ_OK;
}

int effective_group(const realq_quant_cfg_t *q, int64_t n) {
    return q->group_size == 0 ? (int)n : q->group_size;
}

}  // namespace

extern "C" {

const char *realq_status_string(realq_status_t s) {
    switch (s) {
        case REALQ_OK: return "ok";
        case REALQ_ERR_INVALID_ARG: return "invalid argument";
        case REALQ_ERR_WORKSPACE: return "workspace missing, too small or misaligned";
        case REALQ_ERR_NOT_SPD: return "damped Hessian not positive definite";
        case REALQ_ERR_NONFINITE: return "non-finite value in the weights";
        case REALQ_ERR_TIMEOUT: return "bounded device wait timed out";
        case REALQ_ERR_CUDA: return "CUDA error";
        case REALQ_ERR_UNSUPPORTED: return "unsupported configuration";
    }
    return "unknown status";
}

const char *realq_last_error(void) { return g_err; }

int64_t realq_launch_count(void) { return g_launches.load(); }

// ------------------------------------------------------------ CUDA graphs ---
struct realq_graph_s {
    cudaGraphExec_t exec = nullptr;
    int64_t kernels = 0;  // this library's kernels in the graph
};
static thread_local int64_t g_capture_start = -1;

realq_status_t realq_graph_begin(realq_stream_t stream) {
    if (!stream) return fail(REALQ_ERR_INVALID_ARG, "graph_begin: the legacy default stream cannot be captured");
    REALQ_CUDA_TRY(cudaStreamBeginCapture(S(stream), cudaStreamCaptureModeThreadLocal));
    g_capture_start = g_launches.load();
    return REALQ_OK;
}

realq_status_t realq_graph_end(realq_stream_t stream, int node_priorities, realq_graph_t *out) {
    if (!out) return fail(REALQ_ERR_INVALID_ARG, "graph_end: NULL output");
    *out = nullptr;
    cudaGraph_t g = nullptr;
    const cudaError_t e = cudaStreamEndCapture(S(stream), &g);
    const int64_t kernels = g_capture_start >= 0 ? g_launches.load() - g_capture_start : 0;
    g_capture_start = -1;
    if (e != cudaSuccess) {
        if (g) cudaGraphDestroy(g);
        return fail(REALQ_ERR_CUDA, "cudaStreamEndCapture: %s", cudaGetErrorString(e));
    }
    cudaGraphExec_t x = nullptr;
    const cudaError_t ei =
        cudaGraphInstantiateWithFlags(&x, g, node_priorities ? cudaGraphInstantiateFlagUseNodePriority : 0);
    cudaGraphDestroy(g);
    if (ei != cudaSuccess) return fail(REALQ_ERR_CUDA, "cudaGraphInstantiate: %s", cudaGetErrorString(ei));
    realq_graph_s *h = new realq_graph_s;
    h->exec = x;
    h->kernels = kernels;
    *out = h;
    return REALQ_OK;
}

realq_status_t realq_graph_launch(realq_graph_t graph, realq_stream_t stream) {
    if (!graph || !graph->exec) return fail(REALQ_ERR_INVALID_ARG, "graph_launch: no graph");
    REALQ_CUDA_TRY(cudaGraphLaunch(graph->exec, S(stream)));
    g_launches.fetch_add(graph->kernels, std::memory_order_relaxed);
    return REALQ_OK;
}

int64_t realq_graph_kernels(realq_graph_t graph) { return graph ? graph->kernels : 0; }

void realq_graph_destroy(realq_graph_t graph) {
    if (!graph) return;
    if (graph->exec) cudaGraphExecDestroy(graph->exec);
    delete graph;
}

void realq_profile_enable(int on) { g_prof_on.store(on ? 1 : 0); }

int realq_profile_collect(realq_kernel_stat_t *out, int max_entries) {
    std::vector<ProfRec> recs;
    {
        std::lock_guard<std::mutex> lk(g_prof_mu);
        recs.swap(g_pending);
    }
    std::map<std::string, std::pair<int64_t, double>> acc;
    for (auto &r : recs) {
        float ms = 0.f;
        if (cudaEventSynchronize(r.b) == cudaSuccess && cudaEventElapsedTime(&ms, r.a, r.b) == cudaSuccess) {
            auto &e = acc[r.name];
            e.first += 1;
            e.second += ms;
        }
    }
    {
        std::lock_guard<std::mutex> lk(g_prof_mu);
        for (auto &r : recs) {
            g_pool.push_back(r.a);
            g_pool.push_back(r.b);
        }
    }
    int k = 0;
    for (auto &kv : acc) {
        if (k >= max_entries || out == nullptr) break;
        std::memset(out[k].name, 0, sizeof(out[k].name));
        std::strncpy(out[k].name, kv.first.c_str(), sizeof(out[k].name) - 1);
        out[k].launches = kv.second.first;
        out[k].total_ms = kv.second.second;
        ++k;
    }
    return k;
}

// -------------------------------------------------------------- Hessian ---
size_t realq_hessian_workspace_size(int64_t n, int64_t T_chunk, realq_dtype_t x_dtype, int has_X_fp) {
    (void)x_dtype;
    if (n <= 0 || T_chunk <= 0) return 0;
    return hessian_ws_bytes(n, T_chunk, has_X_fp);
}

realq_status_t realq_hessian_accumulate(realq_stream_t stream, int64_t n, int64_t T_chunk, const void *X_hat,
                                        const void *X_fp, realq_dtype_t x_dtype, float *H_sum, float *D_sum, void *ws,
                                        size_t ws_bytes) {
    if (n <= 0 || T_chunk < 0) return fail(REALQ_ERR_INVALID_ARG, "hessian_accumulate: n > 0, T_chunk >= 0 required");
    if (!valid_dtype(x_dtype)) return fail(REALQ_ERR_INVALID_ARG, "hessian_accumulate: bad x_dtype");
    if (!H_sum || (T_chunk > 0 && !X_hat)) return fail(REALQ_ERR_INVALID_ARG, "hessian_accumulate: NULL X_hat or H_sum");
    if (X_fp && !D_sum) return fail(REALQ_ERR_INVALID_ARG, "hessian_accumulate: D_sum required with X_fp");
    if (ws && reinterpret_cast<uintptr_t>(ws) % kAlign)
        return fail(REALQ_ERR_WORKSPACE, "hessian_accumulate: workspace must be %zu-byte aligned", kAlign);
    if (T_chunk == 0) return REALQ_OK;
    return hessian_accumulate(S(stream), n, T_chunk, X_hat, X_fp, x_dtype, H_sum, D_sum, ws, ws ? ws_bytes : 0);
}

// -------------------------------------------------------------- prepare ---
size_t realq_prepare_workspace_size(int64_t n) { return n > 0 ? prepare_ws_bytes(n) : 0; }

realq_status_t realq_hessian_prepare(realq_stream_t stream, int64_t n, int64_t T_total, float damp_frac,
                                     const float *H_sum, float *U_out, float *Hbar_out, uint8_t *dead_out,
                                     int64_t *fail_col, void *ws, size_t ws_bytes) {
    if (n <= 0 || T_total <= 0) return fail(REALQ_ERR_INVALID_ARG, "hessian_prepare: n > 0, T_total > 0 required");
    if (!H_sum || !U_out || !dead_out || !fail_col) return fail(REALQ_ERR_INVALID_ARG, "hessian_prepare: NULL argument");
    if ((const void *)U_out == (const void *)H_sum) return fail(REALQ_ERR_INVALID_ARG, "hessian_prepare: U_out may not alias H_sum");
    if (!(damp_frac >= 0.f) || !std::isfinite(damp_frac)) return fail(REALQ_ERR_INVALID_ARG, "hessian_prepare: damp_frac >= 0");
    REALQ_TRY(check_ws(ws, ws_bytes, prepare_ws_bytes(n), "hessian_prepare"));
    *fail_col = -1;
    return prepare(S(stream), n, T_total, damp_frac, H_sum, U_out, Hbar_out, dead_out, fail_col, ws, ws_bytes);
}

realq_status_t realq_hessian_prepare_deferred(realq_stream_t stream, int64_t n, int64_t T_total, float damp_frac,
                                              const float *H_sum, float *U_out, float *Hbar_out, uint8_t *dead_out,
                                              void *ws, size_t ws_bytes) {
    if (n <= 0 || T_total <= 0) return fail(REALQ_ERR_INVALID_ARG, "hessian_prepare_deferred: n > 0, T_total > 0 required");
    if (!H_sum || !U_out || !dead_out) return fail(REALQ_ERR_INVALID_ARG, "hessian_prepare_deferred: NULL argument");
    if ((const void *)U_out == (const void *)H_sum)
        return fail(REALQ_ERR_INVALID_ARG, "hessian_prepare_deferred: U_out may not alias H_sum");
    if (!(damp_frac >= 0.f) || !std::isfinite(damp_frac))
        return fail(REALQ_ERR_INVALID_ARG, "hessian_prepare_deferred: damp_frac >= 0");
    REALQ_TRY(check_ws(ws, ws_bytes, prepare_ws_bytes(n), "hessian_prepare_deferred"));
    return prepare_deferred(S(stream), n, (double)T_total, damp_frac, H_sum, U_out, Hbar_out, dead_out, ws, ws_bytes);
}

realq_status_t realq_prepare_status(realq_stream_t stream, void *ws, size_t ws_bytes, int64_t *fail_col) {
    if (!ws || ws_bytes < 2 * sizeof(int) || !fail_col)
        return fail(REALQ_ERR_INVALID_ARG, "prepare_status: bad argument");
    int st[2] = {-1, 0};
    REALQ_CUDA_TRY(cudaMemcpyAsync(st, ws, 2 * sizeof(int), cudaMemcpyDeviceToHost, S(stream)));
    REALQ_CUDA_TRY(cudaStreamSynchronize(S(stream)));
    *fail_col = st[0];
    if (st[1] & ST_TIMEOUT) return fail(REALQ_ERR_TIMEOUT, "a bounded device-side wait gave up (prepare)");
    if (st[0] >= 0) return fail(REALQ_ERR_NOT_SPD, "damped Hessian not positive definite at column %d", st[0]);
    return REALQ_OK;
}

realq_status_t realq_hessian_prepare_noalloc(realq_stream_t stream, int64_t n, int64_t T_total, float damp_frac,
                                             const float *H_sum, float *U_out, float *Hbar_out, uint8_t *dead_out,
                                             int64_t *fail_col) {
    if (n <= 0 || T_total <= 0) return fail(REALQ_ERR_INVALID_ARG, "hessian_prepare_noalloc: n > 0, T_total > 0 required");
    if (n > REALQ_PREPARE_NOALLOC_MAX_N)
        return fail(REALQ_ERR_INVALID_ARG,
                    "hessian_prepare_noalloc: n = %lld exceeds the allocation-free maximum %d; use "
                    "realq_hessian_prepare with a workspace",
                    (long long)n, REALQ_PREPARE_NOALLOC_MAX_N);
    if (!H_sum || !U_out || !dead_out || !fail_col)
        return fail(REALQ_ERR_INVALID_ARG, "hessian_prepare_noalloc: NULL argument");
    if ((const void *)U_out == (const void *)H_sum)
        return fail(REALQ_ERR_INVALID_ARG, "hessian_prepare_noalloc: U_out may not alias H_sum");
    if (!(damp_frac >= 0.f) || !std::isfinite(damp_frac))
        return fail(REALQ_ERR_INVALID_ARG, "hessian_prepare_noalloc: damp_frac >= 0");
    *fail_col = -1;
    return prepare_noalloc(S(stream), n, T_total, damp_frac, H_sum, U_out, Hbar_out, dead_out, fail_col);
}

realq_status_t realq_quantize_activations(realq_stream_t stream, int64_t T, int64_t n, const void *X,
                                          realq_dtype_t x_dtype, int bits, float a_clip, void *X_q, uint8_t *codes,
                                          float *scale) {
    if (T < 0 || n <= 0 || !X || !X_q) return fail(REALQ_ERR_INVALID_ARG, "quantize_activations: bad argument");
    if (x_dtype != REALQ_BF16 && x_dtype != REALQ_F32)
        return fail(REALQ_ERR_INVALID_ARG, "quantize_activations: x_dtype must be REALQ_BF16 or REALQ_F32");
    if (bits < 2 || bits > 8) return fail(REALQ_ERR_INVALID_ARG, "quantize_activations: bits must be in [2, 8]");
    if (!(a_clip > 0.f && a_clip <= 1.f)) return fail(REALQ_ERR_INVALID_ARG, "quantize_activations: 0 < a_clip <= 1");
    if (T > (int64_t)INT32_MAX * 8) return fail(REALQ_ERR_UNSUPPORTED, "quantize_activations: too many tokens");
    return act_quant(S(stream), T, n, X, x_dtype, bits, a_clip, X_q, codes, scale);
}

realq_status_t realq_saliency_clip(realq_stream_t stream, int64_t T, int n_groups, const float *sal, double pct,
                                   float *sal_out, float *clip_out) {
    if (T <= 0 || n_groups <= 0 || !sal || !clip_out) return fail(REALQ_ERR_INVALID_ARG, "saliency_clip: bad argument");
    if (!(pct > 0.0 && pct <= 1.0)) return fail(REALQ_ERR_INVALID_ARG, "saliency_clip: 0 < pct <= 1");
    return saliency_clip(S(stream), T, n_groups, sal, pct, sal_out, clip_out);
}

size_t realq_hessian_weighted_workspace_size(int64_t n, int64_t T_chunk) {
    return (n > 0 && T_chunk >= 0) ? weighted_ws_bytes(n, T_chunk) : 0;
}

realq_status_t realq_hessian_accumulate_weighted(realq_stream_t stream, int64_t n, int64_t T_chunk,
                                                 const void *X_hat, int n_groups, const float *sal, float *H_g,
                                                 double *wsum, void *ws, size_t ws_bytes) {
    if (n <= 0 || T_chunk < 0 || n_groups <= 0) return fail(REALQ_ERR_INVALID_ARG, "hessian_accumulate_weighted: bad size");
    if (T_chunk > 0 && (!X_hat || !sal)) return fail(REALQ_ERR_INVALID_ARG, "hessian_accumulate_weighted: NULL input");
    if (!H_g || !wsum || !ws) return fail(REALQ_ERR_INVALID_ARG, "hessian_accumulate_weighted: NULL output or workspace");
    if (reinterpret_cast<uintptr_t>(ws) % kAlign)
        return fail(REALQ_ERR_WORKSPACE, "hessian_accumulate_weighted: workspace must be %zu-byte aligned", kAlign);
    if (ws_bytes < weighted_ws_bytes(n, T_chunk))
        return fail(REALQ_ERR_WORKSPACE, "hessian_accumulate_weighted: workspace too small");
    if (T_chunk == 0) return REALQ_OK;
    return hessian_weighted(S(stream), n, T_chunk, X_hat, n_groups, sal, H_g, wsum, ws, ws_bytes);
}

realq_status_t realq_hessian_prepare_scaled(realq_stream_t stream, int64_t n, double norm, float damp_frac,
                                            const float *H_sum, float *U_out, float *Hbar_out, uint8_t *dead_out,
                                            int64_t *fail_col, void *ws, size_t ws_bytes) {
    if (!(norm > 0.0) || !std::isfinite(norm)) return fail(REALQ_ERR_INVALID_ARG, "hessian_prepare_scaled: norm > 0");
    if (n <= 0) return fail(REALQ_ERR_INVALID_ARG, "hessian_prepare_scaled: n > 0 required");
    if (!H_sum || !U_out || !dead_out || !fail_col) return fail(REALQ_ERR_INVALID_ARG, "hessian_prepare_scaled: NULL argument");
    if ((const void *)U_out == (const void *)H_sum) return fail(REALQ_ERR_INVALID_ARG, "hessian_prepare_scaled: U_out may not alias H_sum");
    if (!(damp_frac >= 0.f) || !std::isfinite(damp_frac)) return fail(REALQ_ERR_INVALID_ARG, "hessian_prepare_scaled: damp_frac >= 0");
    REALQ_TRY(check_ws(ws, ws_bytes, prepare_ws_bytes(n), "hessian_prepare_scaled"));
    *fail_col = -1;
    return prepare(S(stream), n, norm, damp_frac, H_sum, U_out, Hbar_out, dead_out, fail_col, ws, ws_bytes);
}

realq_status_t realq_scale_moment(realq_stream_t stream, int64_t n, int64_t T_total, const float *D_sum, float *Dbar) {
    if (n <= 0 || T_total <= 0 || !D_sum || !Dbar) return fail(REALQ_ERR_INVALID_ARG, "scale_moment: bad argument");
    return scale_copy(S(stream), n * n, (float)T_total, D_sum, Dbar);
}

// ---------------------------------------------------------------- sweep ---
size_t realq_quantize_workspace_size(int64_t m, int64_t n, const realq_quant_cfg_t *qcfg, const realq_bgd_cfg_t *bcfg,
                                     int has_F_next, int has_Dbar) {
    if (m <= 0 || n <= 0 || !qcfg) return 0;
    const int bgd = bcfg && bcfg->steps_per_block > 0;
    return sweep_ws_bytes(m, n, qcfg->block_size, bgd, has_F_next, has_Dbar);
}

// The calibration tokens of token-form mini-batch Block-GD (nullptr: the
// moment form).
struct TokArgs {
    const void *X;       // T x n bf16
    int64_t T, tmb;      // tokens, tokens per mini-batch
    double clip;         // per-token output clipping percentile, (0, 1]
};

// Per-block surrogate values (nullptr: not traced).
struct TraceArgs {
    float *block_loss;   // device, nb x 2
    void *ws;
    size_t ws_bytes;
};

// Called after each column block of the sweep (the OBS step and the lazy
// batch update enqueued), on the sweep's stream: an optimizer step whose
// gradient the sweep does not form itself.
struct BlockHook {
    realq_status_t (*fn)(cudaStream_t s, SweepPlan &p, int64_t b, void *ctx);
    void *ctx;
};

static realq_status_t quantize_impl(realq_stream_t stream, int64_t m, int64_t n, const void *W0, realq_dtype_t w_dtype,
                                    int grouped, int rgroups, const float *Ug, const float *Hbar_g,
                                    const uint8_t *dead_g, int nmb, const float *Hbar_mb,
                                    const float *U, const float *Hbar, const float *Dbar, const uint8_t *dead,
                                    const realq_quant_cfg_t *qcfg, const realq_bgd_cfg_t *bcfg, const float *F,
                                    const float *F_next, float *W_work, float *adam_m, float *adam_v, float *bgd_disp,
                                    int64_t *adam_t, uint8_t *codes, float *scale, uint8_t *zero, void *W_deq,
                                    realq_dtype_t deq_dtype, int64_t block_begin, int64_t block_end, void *ws,
                                    size_t ws_bytes, const char *who, const TokArgs *tok = nullptr,
                                    const TraceArgs *trace = nullptr, const BlockHook *hook = nullptr) {
    if (m <= 0 || n <= 0) return fail(REALQ_ERR_INVALID_ARG, "%s: m, n must be > 0", who);
    if (m > (int64_t)1 << 30 || n > (int64_t)1 << 30) return fail(REALQ_ERR_INVALID_ARG, "%s: m, n too large", who);
    if (!valid_dtype(w_dtype) || !valid_dtype(deq_dtype)) return fail(REALQ_ERR_INVALID_ARG, "%s: bad dtype", who);
    if (!W0 || !U || !W_work || !codes || !scale || !zero)
        return fail(REALQ_ERR_INVALID_ARG, "%s: NULL W0, U, W_work, codes, scale or zero", who);
    REALQ_TRY(check_qcfg(qcfg, n));
    REALQ_TRY(check_bcfg(bcfg));
    const int bgd = bcfg && bcfg->steps_per_block > 0;
    if (bgd) {
        if (!Hbar || !F || !adam_t || !bgd_disp)
            return fail(REALQ_ERR_INVALID_ARG, "%s: Block-GD needs Hbar, F, bgd_disp and adam_t", who);
        if (bcfg->optimizer == REALQ_OPT_ADAM && (!adam_m || !adam_v))
            return fail(REALQ_ERR_INVALID_ARG, "%s: Adam needs adam_m and adam_v", who);
        if ((grouped || nmb > 0 || tok) && !(qcfg->block_size > 0 && tc_gemm_eligible(m, n)))
            return fail(REALQ_ERR_UNSUPPORTED,
                        "%s: Block-GD with row groups needs m and n multiples of 4 and at least 32", who);
    }
    const int64_t nb = (n + qcfg->block_size - 1) / qcfg->block_size;
    if (block_begin < 0 || block_end > nb || block_begin > block_end)
        return fail(REALQ_ERR_INVALID_ARG, "%s: block range [%lld, %lld) outside [0, %lld)", who,
                    (long long)block_begin, (long long)block_end, (long long)nb);
    const int has_fn = bgd && F_next != nullptr;
    const int has_db = bgd && Dbar != nullptr;
    if (nmb > 0 && bgd && (Dbar || grouped))
        return fail(REALQ_ERR_UNSUPPORTED, "%s: mini-batch moments with perturbed inputs or row groups", who);
    const int64_t tmb = (bgd && tok) ? tok->tmb : 0;
    REALQ_TRY(check_ws(ws, ws_bytes,
                       sweep_ws_bytes(m, n, qcfg->block_size, bgd, has_fn, has_db, grouped ? rgroups : 0,
                                      bgd ? nmb : 0, tmb), who));

    SweepPlan p{};
    p.m = m; p.n = n; p.W0 = W0; p.w_dtype = w_dtype;
    p.U = U; p.Hbar = Hbar; p.Dbar = has_db ? Dbar : nullptr; p.dead = dead;
    p.rgroups = grouped ? rgroups : 1;
    p.grouped = grouped;
    p.rg_rows = (m + p.rgroups - 1) / p.rgroups;
    p.Ug = grouped ? Ug : U;
    p.Hbar_g = grouped ? Hbar_g : nullptr;
    p.dead_g = grouped ? dead_g : nullptr;
    p.nmb = bgd ? nmb : 0;
    p.Hbar_mb = bgd ? Hbar_mb : nullptr;
    p.bits = qcfg->bits; p.block = qcfg->block_size; p.sym = qcfg->symmetric;
    p.group = effective_group(qcfg, n);
    p.ngroups = (int)((n + p.group - 1) / p.group);
    p.bgd_steps = bgd ? bcfg->steps_per_block : 0;
    if (bgd) {
        p.optimizer = bcfg->optimizer; p.lr = bcfg->lr; p.beta1 = bcfg->beta1; p.beta2 = bcfg->beta2; p.eps = bcfg->eps;
        p.b_global_start = bcfg->b_global_start; p.B_total = bcfg->B_total;
    }
    p.F = F; p.F_next = has_fn ? F_next : nullptr;
    p.W = W_work; p.adam_m = adam_m; p.adam_v = adam_v; p.disp = bgd ? bgd_disp : nullptr; p.adam_t = adam_t;
    p.damp = qcfg->damp_frac;
    p.codes = codes; p.scale = scale; p.zero = zero; p.W_deq = W_deq; p.deq_dtype = deq_dtype;
    if (tmb > 0) {
        p.Xtok = tok->X; p.Ttok = tok->T; p.tmb = tmb;
        p.ntok = (int)((tok->T + tmb - 1) / tmb);
        // nearest-rank threshold: the ceil(pct m)-th smallest |Δ| (pct and
        // the product in double: the exact rank for a percentile such as 0.95)
        const int64_t k = (int64_t)std::ceil(tok->clip * (double)m) - 1;
        p.rank_q = std::min<int64_t>(std::max<int64_t>(k, 0), m - 1);
    }
    if (trace) {
        if (!trace->block_loss) return fail(REALQ_ERR_INVALID_ARG, "%s: NULL block_loss", who);
        if (has_db) return fail(REALQ_ERR_UNSUPPORTED, "%s: the trace takes unperturbed inputs (Dbar = NULL)", who);
        REALQ_TRY(check_ws(trace->ws, trace->ws_bytes, surrogate_ws_bytes(m, n) + 256, who));
        if (bgd) {
            p.block_loss = trace->block_loss;
            p.trace_ws = trace->ws;
        }
    }
    sweep_carve(p, ws, bgd, has_fn, has_db);
    cudaStream_t s = S(stream);
    REALQ_CUDA_TRY(cudaMemsetAsync(p.status, 0, sizeof(int), s));
    if (block_begin == 0) REALQ_TRY(sweep_init(s, p));
    REALQ_TRY(sweep_prologue_r0(s, p, block_begin == 0));
    // (while profiling, everything stays on the caller's stream, so that each
    // launch's event interval is its own time; the arithmetic is the same)
    if (p.tc && p.bgd_steps > 0 && block_end - block_begin > 1 && !profiling()) REALQ_TRY(sweep_side_stream(s, p));
    for (int64_t b = block_begin; b < block_end; ++b) {
        REALQ_TRY(sweep_block(s, p, b));
        if (hook) REALQ_TRY(hook->fn(s, p, b, hook->ctx));
    }
    REALQ_TRY(sweep_join_wide(s, p));
    return REALQ_OK;
}

realq_status_t realq_quantize_layer(realq_stream_t stream, int64_t m, int64_t n, const void *W0, realq_dtype_t w_dtype,
                                    const float *U, const float *Hbar, const float *Dbar, const uint8_t *dead,
                                    const realq_quant_cfg_t *qcfg, const realq_bgd_cfg_t *bcfg, const float *F,
                                    const float *F_next, float *W_work, float *adam_m, float *adam_v, float *bgd_disp,
                                    int64_t *adam_t,
                                    uint8_t *codes, float *scale, uint8_t *zero, void *W_deq, realq_dtype_t deq_dtype,
                                    int64_t block_begin, int64_t block_end, void *ws, size_t ws_bytes) {
    return quantize_impl(stream, m, n, W0, w_dtype, 0, 1, nullptr, nullptr, nullptr, 0, nullptr, U, Hbar, Dbar, dead, qcfg,
                         bcfg, F,
                         F_next, W_work, adam_m, adam_v, bgd_disp, adam_t, codes, scale, zero, W_deq, deq_dtype,
                         block_begin, block_end, ws, ws_bytes, "quantize_layer");
}

size_t realq_quantize_grouped_workspace_size(int64_t m, int64_t n, int n_row_groups, const realq_quant_cfg_t *qcfg,
                                             const realq_bgd_cfg_t *bcfg, int has_F_next, int has_Dbar) {
    if (m <= 0 || n <= 0 || !qcfg || n_row_groups <= 0) return 0;
    const int bgd = bcfg && bcfg->steps_per_block > 0;
    return sweep_ws_bytes(m, n, qcfg->block_size, bgd, has_F_next, has_Dbar, n_row_groups);
}

realq_status_t realq_quantize_layer_grouped(realq_stream_t stream, int64_t m, int64_t n, const void *W0,
                                            realq_dtype_t w_dtype, int n_row_groups, const float *U_g,
                                            const float *Hbar_g, const uint8_t *dead_g, const float *Hbar,
                                            const float *Dbar, const realq_quant_cfg_t *qcfg,
                                            const realq_bgd_cfg_t *bcfg, const float *F, const float *F_next,
                                            float *W_work, float *adam_m, float *adam_v, float *bgd_disp,
                                            int64_t *adam_t, uint8_t *codes, float *scale, uint8_t *zero,
                                            void *W_deq, realq_dtype_t deq_dtype, int64_t block_begin,
                                            int64_t block_end, void *ws, size_t ws_bytes) {
    if (n_row_groups <= 0 || (int64_t)n_row_groups > m)
        return fail(REALQ_ERR_INVALID_ARG, "quantize_layer_grouped: 1 <= n_row_groups <= m required");
    if (!U_g || !dead_g) return fail(REALQ_ERR_INVALID_ARG, "quantize_layer_grouped: NULL U_g or dead_g");
    const int bgd = bcfg && bcfg->steps_per_block > 0;
    if (bgd && !Hbar_g) return fail(REALQ_ERR_INVALID_ARG, "quantize_layer_grouped: Block-GD needs Hbar_g");
    return quantize_impl(stream, m, n, W0, w_dtype, 1, n_row_groups, U_g, Hbar_g, dead_g, 0, nullptr, U_g, Hbar, Dbar,
                         dead_g, qcfg,
                         bcfg, F, F_next, W_work, adam_m, adam_v, bgd_disp, adam_t, codes, scale, zero, W_deq,
                         deq_dtype, block_begin, block_end, ws, ws_bytes, "quantize_layer_grouped");
}

size_t realq_quantize_minibatch_workspace_size(int64_t m, int64_t n, int n_minibatch, const realq_quant_cfg_t *qcfg,
                                               const realq_bgd_cfg_t *bcfg, int has_F_next) {
    if (m <= 0 || n <= 0 || !qcfg || n_minibatch <= 0) return 0;
    const int bgd = bcfg && bcfg->steps_per_block > 0;
    return sweep_ws_bytes(m, n, qcfg->block_size, bgd, has_F_next, 0, 0, bgd ? n_minibatch : 0);
}

realq_status_t realq_quantize_layer_minibatch(realq_stream_t stream, int64_t m, int64_t n, const void *W0,
                                              realq_dtype_t w_dtype, const float *U, const float *Hbar,
                                              const uint8_t *dead, int n_minibatch, const float *Hbar_mb,
                                              const realq_quant_cfg_t *qcfg, const realq_bgd_cfg_t *bcfg,
                                              const float *F, const float *F_next, float *W_work, float *adam_m,
                                              float *adam_v, float *bgd_disp, int64_t *adam_t, uint8_t *codes,
                                              float *scale, uint8_t *zero, void *W_deq, realq_dtype_t deq_dtype,
                                              int64_t block_begin, int64_t block_end, void *ws, size_t ws_bytes) {
    if (n_minibatch <= 0 || !Hbar_mb)
        return fail(REALQ_ERR_INVALID_ARG, "quantize_layer_minibatch: n_minibatch >= 1 and Hbar_mb required");
    return quantize_impl(stream, m, n, W0, w_dtype, 0, 1, nullptr, nullptr, nullptr, n_minibatch, Hbar_mb, U, Hbar,
                         nullptr, dead, qcfg, bcfg, F, F_next, W_work, adam_m, adam_v, bgd_disp, adam_t, codes, scale,
                         zero, W_deq, deq_dtype, block_begin, block_end, ws, ws_bytes, "quantize_layer_minibatch");
}

// Block-GD on the block ops' loss (the exact window of Eq. slide_window or
// the final block's KL of Eq. kl_loss): the after-block step of
// realq_quantize_layer_window.
struct WindowStep {
    realq_stream_t stream;
    const realq_block_dims_t *dims;
    const realq_block_weights_t *this_block, *this_block_hat, *next_block;
    int64_t S, L, n_minibatch;
    const float *x, *x_hat;
    int module;
    const float *F_this, *F_next, *gf, *Wh;
    int64_t vocab;
    realq_bgd_cfg_t cfg;
    float *adam_m, *adam_v;
    int64_t *adam_t;
    float *grad, *block_loss;
    void *mws;
    size_t mws_bytes;
};

// the loss and gradient on calibration mini-batch k of the rotation
// (sequences (k mod n_minibatch) S .. + S of x and x_hat)
static realq_status_t window_loss(const WindowStep &w, const float *W, float alpha, int64_t k, float *loss) {
    const int64_t off = (k % w.n_minibatch) * w.S * w.L * w.dims->d;
    const float *x = w.x + off, *xh = w.x_hat ? w.x_hat + off : nullptr;
    if (w.next_block)
        return realq_block_module_window(w.stream, w.dims, w.this_block, w.this_block_hat, w.next_block, w.S, w.L, x,
                                         xh, w.module, W, alpha, w.F_this, w.F_next, w.grad, loss, w.mws,
                                         w.mws_bytes);
    return realq_block_module_kl(w.stream, w.dims, w.this_block, w.this_block_hat, w.S, w.L, x, xh, w.module, W,
                                 w.gf, w.Wh, w.vocab, w.grad, loss, w.mws, w.mws_bytes);
}

static realq_status_t window_step(cudaStream_t s, SweepPlan &p, int64_t b, void *ctx) {
    const WindowStep &w = *static_cast<const WindowStep *>(ctx);
    const int64_t be = std::min<int64_t>((b + 1) * p.block, p.n);
    if (be >= p.n) return REALQ_OK;   // no free columns after the last block
    const int64_t b_global = w.cfg.b_global_start + b;
    float alpha = 1.f;
    if (w.cfg.B_total > 1) alpha = (float)(1.0 - (double)(b_global - 1) / (double)(w.cfg.B_total - 1));
    float *bl = w.block_loss ? w.block_loss + 2 * b : nullptr;
    const int64_t steps = w.cfg.steps_per_block, k0 = (b_global - 1) * steps;
    const BlockStatusScope into_sweep(p.status);
    for (int64_t k = 0; k < steps; ++k) {
        // the loss and its gradient at the current weights (the dequantized
        // columns < be and the free ones) on the step's mini-batch
        REALQ_TRY(window_loss(w, p.W, alpha, k0 + k, k == 0 ? bl : nullptr));
        const int64_t t = ++(*w.adam_t);
        REALQ_TRY(adam_cols(s, p.m, p.n, be, w.grad, p.W, w.adam_m, w.adam_v, w.cfg.lr, w.cfg.beta1, w.cfg.beta2,
                            w.cfg.eps, t, w.cfg.optimizer == REALQ_OPT_SGD));
    }
    if (bl) REALQ_TRY(window_loss(w, p.W, alpha, k0 + steps - 1, bl + 1));
    return REALQ_OK;
}

size_t realq_quantize_window_workspace_size(const realq_block_dims_t *dims, int64_t S, int64_t L, int module,
                                            int64_t vocab, const realq_quant_cfg_t *qcfg) {
    if (!dims || !qcfg || module < 0 || module > 6 || vocab < 0) return 0;
    const int64_t qw = dims->n_heads * dims->head_dim, kw = dims->n_kv * dims->head_dim;
    const int64_t shape[7][2] = {{qw, dims->d}, {kw, dims->d}, {kw, dims->d}, {dims->d, qw},
                                 {dims->ffn, dims->d}, {dims->ffn, dims->d}, {dims->d, dims->ffn}};
    const int64_t m = shape[module][0], n = shape[module][1];
    if (m <= 0 || n <= 0 || qcfg->block_size <= 0) return 0;
    const size_t mod = realq_block_module_workspace_size(dims, S, L, vocab);
    if (mod == 0) return 0;
    return sweep_ws_bytes(m, n, qcfg->block_size, 0, 0, 0) + align_up((size_t)m * n * sizeof(float)) + mod;
}

realq_status_t realq_quantize_layer_window(realq_stream_t stream, const realq_block_dims_t *dims,
                                           const realq_block_weights_t *this_block,
                                           const realq_block_weights_t *this_block_hat,
                                           const realq_block_weights_t *next_block, int64_t S, int64_t L,
                                           int64_t n_minibatch, const float *x, const float *x_hat, int module,
                                           const float *F_this, const float *F_next,
                                           const float *head_gf, const float *head_Wh, int64_t vocab, const float *U,
                                           const uint8_t *dead, const realq_quant_cfg_t *qcfg,
                                           const realq_bgd_cfg_t *bcfg, float *W_work, float *adam_m, float *adam_v,
                                           int64_t *adam_t, uint8_t *codes, float *scale, uint8_t *zero, void *W_deq,
                                           realq_dtype_t deq_dtype, float *block_loss, int64_t block_begin,
                                           int64_t block_end, void *ws, size_t ws_bytes) {
    const char *who = "quantize_layer_window";
    int64_t m = 0, n = 0;
    size_t mws = 0;
    REALQ_TRY(block_loss_check(dims, this_block, this_block_hat, next_block, S, L, x, module, F_this, F_next, head_gf,
                               head_Wh, next_block ? 0 : vocab, who, &m, &n, &mws));
    if (m * n > ((int64_t)1 << 38)) return fail(REALQ_ERR_UNSUPPORTED, "%s: m n must be below 2^38", who);
    if (n_minibatch < 1 || n_minibatch > ((int64_t)1 << 38) / (S * L * dims->d))
        return fail(REALQ_ERR_INVALID_ARG, "%s: n_minibatch >= 1 and n_minibatch S L d < 2^38 required", who);
    REALQ_TRY(check_qcfg(qcfg, n));
    REALQ_TRY(check_bcfg(bcfg));
    if (!bcfg || bcfg->steps_per_block < 1)
        return fail(REALQ_ERR_INVALID_ARG, "%s: a Block-GD configuration with steps_per_block >= 1 required", who);
    if (!adam_t) return fail(REALQ_ERR_INVALID_ARG, "%s: NULL adam_t", who);
    if (bcfg->optimizer == REALQ_OPT_ADAM && (!adam_m || !adam_v))
        return fail(REALQ_ERR_INVALID_ARG, "%s: Adam needs adam_m and adam_v", who);
    if (!U || !W_work || !codes || !scale || !zero)
        return fail(REALQ_ERR_INVALID_ARG, "%s: NULL U, W_work, codes, scale or zero", who);
    if (!valid_dtype(deq_dtype)) return fail(REALQ_ERR_INVALID_ARG, "%s: bad dtype", who);
    const int64_t nb = (n + qcfg->block_size - 1) / qcfg->block_size;
    if (block_begin < 0 || block_end > nb || block_begin > block_end)
        return fail(REALQ_ERR_INVALID_ARG, "%s: block range [%lld, %lld) outside [0, %lld)", who,
                    (long long)block_begin, (long long)block_end, (long long)nb);
    const size_t sw = sweep_ws_bytes(m, n, qcfg->block_size, 0, 0, 0);
    const size_t gb = align_up((size_t)m * n * sizeof(float));
    REALQ_TRY(check_ws(ws, ws_bytes, sw + gb + mws, who));
    const float *W0 = nullptr;
    switch (module) {
        case 0: W0 = this_block->Wq; break;
        case 1: W0 = this_block->Wk; break;
        case 2: W0 = this_block->Wv; break;
        case 3: W0 = this_block->Wo; break;
        case 4: W0 = this_block->Wg; break;
        case 5: W0 = this_block->Wu; break;
        default: W0 = this_block->Wd; break;
    }
    char *base = static_cast<char *>(ws);
    WindowStep w{stream, dims, this_block, this_block_hat, next_block, S, L, n_minibatch, x, x_hat, module, F_this,
                 F_next, head_gf, head_Wh, vocab, *bcfg, adam_m, adam_v, adam_t, reinterpret_cast<float *>(base + sw),
                 block_loss, base + sw + gb, mws};
    if (block_begin == 0) {
        // (S is the sequence count here; the stream is cast directly)
        cudaStream_t cs = static_cast<cudaStream_t>(stream);
        *adam_t = 0;
        if (bcfg->optimizer == REALQ_OPT_ADAM) {
            REALQ_CUDA_TRY(cudaMemsetAsync(adam_m, 0, (size_t)m * n * sizeof(float), cs));
            REALQ_CUDA_TRY(cudaMemsetAsync(adam_v, 0, (size_t)m * n * sizeof(float), cs));
        }
    }
    const BlockHook hook{window_step, &w};
    // the column sweep itself is the plain one (no layer-level Block-GD); the
    // hook takes each block's optimizer steps
    return quantize_impl(stream, m, n, W0, REALQ_F32, 0, 1, nullptr, nullptr, nullptr, 0, nullptr, U, nullptr, nullptr,
                         dead, qcfg, nullptr, nullptr, nullptr, W_work, nullptr, nullptr, nullptr, nullptr, codes,
                         scale, zero, W_deq, deq_dtype, block_begin, block_end, ws, sw, who, nullptr, nullptr, &hook);
}

size_t realq_quantize_tokens_workspace_size(int64_t m, int64_t n, int64_t T_mb, const realq_quant_cfg_t *qcfg,
                                            const realq_bgd_cfg_t *bcfg, int has_F_next) {
    if (m <= 0 || n <= 0 || !qcfg || T_mb <= 0) return 0;
    const int bgd = bcfg && bcfg->steps_per_block > 0;
    return sweep_ws_bytes(m, n, qcfg->block_size, bgd, has_F_next, 0, 0, 0, bgd ? T_mb : 0);
}

realq_status_t realq_quantize_layer_tokens(realq_stream_t stream, int64_t m, int64_t n, const void *W0,
                                           realq_dtype_t w_dtype, const float *U, const float *Hbar,
                                           const uint8_t *dead, const void *X_hat, int64_t T, int64_t T_mb,
                                           double a_loss_clip, const realq_quant_cfg_t *qcfg,
                                           const realq_bgd_cfg_t *bcfg, const float *F, const float *F_next,
                                           float *W_work, float *adam_m, float *adam_v, float *bgd_disp,
                                           int64_t *adam_t, uint8_t *codes, float *scale, uint8_t *zero, void *W_deq,
                                           realq_dtype_t deq_dtype, int64_t block_begin, int64_t block_end, void *ws,
                                           size_t ws_bytes) {
    if (!X_hat || T <= 0 || T_mb <= 0)
        return fail(REALQ_ERR_INVALID_ARG, "quantize_layer_tokens: X_hat, T > 0 and T_mb > 0 required");
    if (T_mb % 4 != 0) return fail(REALQ_ERR_INVALID_ARG, "quantize_layer_tokens: T_mb must be a multiple of 4");
    // (the mini-batch's layout kernels tile the token axis by 32 on grid y)
    if (T_mb > (int64_t)65535 * 32 || T > ((int64_t)1 << 40))
        return fail(REALQ_ERR_INVALID_ARG, "quantize_layer_tokens: T_mb <= 2097120 and T <= 2^40 required");
    if (reinterpret_cast<uintptr_t>(X_hat) % 16 != 0 || n % 8 != 0)
        return fail(REALQ_ERR_INVALID_ARG, "quantize_layer_tokens: X_hat must be 16-byte aligned with n %% 8 == 0");
    if (!(a_loss_clip > 0.0 && a_loss_clip <= 1.0))
        return fail(REALQ_ERR_INVALID_ARG, "quantize_layer_tokens: 0 < a_loss_clip <= 1");
    const TokArgs tok{X_hat, T, T_mb, a_loss_clip};
    return quantize_impl(stream, m, n, W0, w_dtype, 0, 1, nullptr, nullptr, nullptr, 0, nullptr, U, Hbar, nullptr, dead,
                         qcfg, bcfg, F, F_next, W_work, adam_m, adam_v, bgd_disp, adam_t, codes, scale, zero, W_deq,
                         deq_dtype, block_begin, block_end, ws, ws_bytes, "quantize_layer_tokens", &tok);
}

size_t realq_quantize_trace_workspace_size(int64_t m, int64_t n) {
    return (m > 0 && n > 0) ? surrogate_ws_bytes(m, n) + 256 : 0;
}

realq_status_t realq_quantize_layer_traced(realq_stream_t stream, int64_t m, int64_t n, const void *W0,
                                           realq_dtype_t w_dtype, const float *U, const float *Hbar,
                                           const uint8_t *dead, const realq_quant_cfg_t *qcfg,
                                           const realq_bgd_cfg_t *bcfg, const float *F, const float *F_next,
                                           float *W_work, float *adam_m, float *adam_v, float *bgd_disp,
                                           int64_t *adam_t, uint8_t *codes, float *scale, uint8_t *zero, void *W_deq,
                                           realq_dtype_t deq_dtype, int64_t block_begin, int64_t block_end, void *ws,
                                           size_t ws_bytes, float *block_loss, void *trace_ws,
                                           size_t trace_ws_bytes) {
    const TraceArgs tr{block_loss, trace_ws, trace_ws_bytes};
    return quantize_impl(stream, m, n, W0, w_dtype, 0, 1, nullptr, nullptr, nullptr, 0, nullptr, U, Hbar, nullptr, dead,
                         qcfg, bcfg, F, F_next, W_work, adam_m, adam_v, bgd_disp, adam_t, codes, scale, zero, W_deq,
                         deq_dtype, block_begin, block_end, ws, ws_bytes, "quantize_layer_traced", nullptr, &tr);
}

// ---------------------------------------------------------------- BGD -----
size_t realq_bgd_workspace_size(int64_t m, int64_t n, int has_F_next, int has_Dbar) {
    if (m <= 0 || n <= 0) return 0;
    return sweep_ws_bytes(m, n, 0, 1, has_F_next, has_Dbar);
}

realq_status_t realq_bgd_refine(realq_stream_t stream, int64_t m, int64_t n, int64_t col_start, float *W, const void *W0,
                                realq_dtype_t w_dtype, const float *Hbar, const float *Dbar, const float *F,
                                const float *F_next, float alpha, float *adam_m, float *adam_v, int64_t *adam_t,
                                const realq_bgd_cfg_t *bcfg, void *ws, size_t ws_bytes) {
    if (m <= 0 || n <= 0 || col_start < 0 || col_start > n) return fail(REALQ_ERR_INVALID_ARG, "bgd_refine: bad sizes");
    if (!W || !W0 || !Hbar || !F || !bcfg || !adam_t) return fail(REALQ_ERR_INVALID_ARG, "bgd_refine: NULL argument");
    if (!valid_dtype(w_dtype)) return fail(REALQ_ERR_INVALID_ARG, "bgd_refine: bad dtype");
    REALQ_TRY(check_bcfg(bcfg));
    if (bcfg->optimizer == REALQ_OPT_ADAM && (!adam_m || !adam_v)) return fail(REALQ_ERR_INVALID_ARG, "bgd_refine: Adam state");
    if (!(alpha >= 0.f && alpha <= 1.f)) return fail(REALQ_ERR_INVALID_ARG, "bgd_refine: alpha must be in [0, 1]");
    const int has_fn = F_next != nullptr, has_db = Dbar != nullptr;
    REALQ_TRY(check_ws(ws, ws_bytes, sweep_ws_bytes(m, n, 0, 1, has_fn, has_db), "bgd_refine"));
    SweepPlan p{};
    p.m = m; p.n = n; p.W0 = W0; p.w_dtype = w_dtype; p.Hbar = Hbar; p.Dbar = Dbar;
    p.bgd_steps = bcfg->steps_per_block; p.optimizer = bcfg->optimizer; p.lr = bcfg->lr;
    p.beta1 = bcfg->beta1; p.beta2 = bcfg->beta2; p.eps = bcfg->eps;
    p.F = F; p.F_next = F_next; p.W = W; p.adam_m = adam_m; p.adam_v = adam_v; p.adam_t = adam_t;
    p.block = 0;
    sweep_carve(p, ws, 1, has_fn, has_db);
    return bgd_step(S(stream), p, col_start, alpha);
}

realq_status_t realq_set_tensor_tile(int mode) {
    if (mode < 0 || mode > 2) return fail(REALQ_ERR_INVALID_ARG, "set_tensor_tile: mode 0, 1 or 2");
    tc_set_tile_mode(mode);
    return REALQ_OK;
}

realq_status_t realq_set_tensor_overlap(int mode) {
    if (mode < 0 || mode > 2) return fail(REALQ_ERR_INVALID_ARG, "set_tensor_overlap: mode 0, 1 or 2");
    tc_set_overlap(mode);
    return REALQ_OK;
}

realq_status_t realq_set_bgd_products(int mode) {
    if (mode < 0 || mode > 1) return fail(REALQ_ERR_INVALID_ARG, "set_bgd_products: mode 0 or 1");
    bgd_set_products(mode);
    return REALQ_OK;
}

realq_status_t realq_set_quant_kernel(int mode) {
    if (mode < 0 || mode > 1) return fail(REALQ_ERR_INVALID_ARG, "set_quant_kernel: mode 0 or 1");
    quant_set_kernel(mode);
    return REALQ_OK;
}

// ------------------------------------------------------------ schedules ---
realq_status_t realq_reverse_cosine_lr(int64_t i, int64_t L, double lr_final, double *lr_out) {
    if (!lr_out || L < 1 || i < 1 || i > L || !std::isfinite(lr_final))
        return fail(REALQ_ERR_INVALID_ARG, "reverse_cosine_lr: need 1 <= i <= L and a finite rate");
    if (L == 1) {
        *lr_out = lr_final;
        return REALQ_OK;
    }
    const double base = 0.01 * lr_final;
    const double half_pi = 1.5707963267948966;
    *lr_out = base + (lr_final - base) * std::sin(half_pi * (double)(i - 1) / (double)(L - 1));
    return REALQ_OK;
}

// ------------------------------------------------------------ surrogate ---
size_t realq_surrogate_workspace_size(int64_t m, int64_t n) { return (m > 0 && n > 0) ? surrogate_ws_bytes(m, n) : 0; }

realq_status_t realq_surrogate_loss(realq_stream_t stream, int64_t m, int64_t n, const float *W_hat, const void *W0,
                                    realq_dtype_t w_dtype, const float *Hbar, const float *F, float *loss_out, void *ws,
                                    size_t ws_bytes) {
    if (m <= 0 || n <= 0 || !W_hat || !W0 || !Hbar || !F || !loss_out)
        return fail(REALQ_ERR_INVALID_ARG, "surrogate_loss: bad argument");
    if (!valid_dtype(w_dtype)) return fail(REALQ_ERR_INVALID_ARG, "surrogate_loss: bad dtype");
    REALQ_TRY(check_ws(ws, ws_bytes, surrogate_ws_bytes(m, n), "surrogate_loss"));
    return surrogate(S(stream), m, n, W_hat, W0, w_dtype, Hbar, F, loss_out, ws);
}

realq_status_t realq_workspace_status(realq_stream_t stream, void *ws, size_t ws_bytes) {
    if (!ws || ws_bytes < sizeof(int)) return fail(REALQ_ERR_INVALID_ARG, "workspace_status: bad workspace");
    int st = 0;
    REALQ_CUDA_TRY(cudaMemcpyAsync(&st, ws, sizeof(int), cudaMemcpyDeviceToHost, S(stream)));
    REALQ_CUDA_TRY(cudaStreamSynchronize(S(stream)));
    REALQ_CUDA_TRY(cudaMemsetAsync(ws, 0, sizeof(int), S(stream)));
    if (st & ST_TIMEOUT) return fail(REALQ_ERR_TIMEOUT, "a bounded device-side wait gave up");
    if (st & ST_NONFINITE) return fail(REALQ_ERR_NONFINITE, "non-finite weight met during the sweep");
    return REALQ_OK;
}

}  // extern "C"
