// Shared definitions of the REAL-Q CUDA library (sm_103a).
#pragma once

#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cstdint>
#include <cstddef>

#include "realq.h"

namespace realq {

// ---------------------------------------------------------------- errors ---
// (printf-style: the compiler checks each format against its arguments)
void set_error(const char *fmt, ...) __attribute__((format(printf, 1, 2)));
realq_status_t fail(realq_status_t s, const char *fmt, ...) __attribute__((format(printf, 2, 3)));

// Launch bookkeeping: every kernel launch of the library goes through
// Launch, which counts it and, when profiling is on, brackets it with CUDA
// events recorded on the launch stream.
struct Launch {
    const char *name;
    cudaStream_t stream;
    int slot;
    Launch(const char *name, cudaStream_t s);
    ~Launch();
};

// cudaGetLastError after a launch, as a library status
realq_status_t check_launch(const char *what);
// The dynamic shared-memory limit of a kernel, set once per (kernel, device,
// size); safe to call from several host threads.
realq_status_t set_smem_limit(const void *kernel, int bytes);

// Device status word layout (int32) kept at the start of workspaces.
enum : int {
    ST_OK = 0,
    ST_NONFINITE = 1,
    ST_NOT_SPD = 2,
    ST_TIMEOUT = 4,
};

constexpr size_t kAlign = 256;
inline size_t align_up(size_t x) { return (x + kAlign - 1) / kAlign * kAlign; }

// Simple bump allocator over a caller workspace.
struct Carve {
    char *base;
    size_t off = 0;
    explicit Carve(void *p) : base(static_cast<char *>(p)) {}
    template <class T> T *take(size_t count) {
        T *p = reinterpret_cast<T *>(base ? base + off : nullptr);
        off += align_up(count * sizeof(T));
        return p;
    }
};

__device__ __forceinline__ float load_as_float(const float *p, int64_t i) { return p[i]; }
__device__ __forceinline__ float load_as_float(const __nv_bfloat16 *p, int64_t i) { return __bfloat162float(p[i]); }

inline int ceil_div(int64_t a, int64_t b) { return static_cast<int>((a + b - 1) / b); }

}  // namespace realq

#define REALQ_CUDA_TRY(call)                                                                 \
    do {                                                                                     \
        cudaError_t _e = (call);                                                             \
        if (_e != cudaSuccess)                                                               \
            return ::realq::fail(REALQ_ERR_CUDA, "%s: %s", #call, cudaGetErrorString(_e));   \
    } while (0)

#define REALQ_TRY(expr)                       \
    do {                                      \
        realq_status_t _s = (expr);           \
        if (_s != REALQ_OK) return _s;        \
    } while (0)
