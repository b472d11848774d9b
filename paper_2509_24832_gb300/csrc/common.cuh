// common.cuh -- host-side helpers shared by the entry points.
#pragma once

#include <cuda_runtime.h>

#include <cstdint>
#include <cstdlib>
#include <utility>

#include "semshare.h"

namespace semshare {

inline cudaStream_t as_stream(void* s) { return static_cast<cudaStream_t>(s); }

inline bool aligned(const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

// Streaming multiprocessors of the current device (queried per call: cheap, no cached state).
inline semshare_status current_sm_count(int* sms, int* device) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return SEMSHARE_ECUDA;
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return SEMSHARE_ECUDA;
    *sms = n;
    if (device) *device = dev;
    return SEMSHARE_OK;
}

// Programmatic dependent launch.  grid_dependency_wait: returns once every grid this one depends
// on has completed and its memory is visible (immediately when launched without the programmatic
// attribute).  grid_dependents_launch: lets the next grid in the stream be scheduled once every
// CTA of this grid has executed it (or exited); that grid still waits for this one to complete
// before touching memory.
__device__ __forceinline__ void grid_dependency_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void grid_dependents_launch() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

// Every kernel of the library calls grid_dependency_wait before it touches global memory: most as
// their first statement, the tensor-core search after its shared- and tensor-memory set-up.  The
// short kernels release their dependents right away (pdl_prologue); the persistent ones that fill
// every SM (the hash kernels, the tensor-core search) release them only at their end, since
// dependents released early queue behind them for their whole run (measured slower).
__device__ __forceinline__ void pdl_prologue() {
    grid_dependency_wait();
    grid_dependents_launch();
}

// Launches kernel<<<grid, block, smem, s>>>(args...) as a programmatic dependent of the work
// before it in the stream: its CTAs may be scheduled while the previous kernel drains, and they
// wait (griddepcontrol.wait, before any global memory access) until it has completed.
template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                              Args&&... args) {
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

inline semshare_status launch_status() {
    return cudaGetLastError() == cudaSuccess ? SEMSHARE_OK : SEMSHARE_ECUDA;
}

// ---- the checked build (-DSEMSHARE_CHECKED) ----
// SEMSHARE_CHECK(cond, err, kernel): in the checked build, a false cond ORs SEMSHARE_FLAG_CHECK into
// *err and, if no check has failed before, stores the kernel id (bits 8..15) and the source line
// (bits 16..31); the kernel carries on.  In the plain build it compiles to nothing (cond is not
// evaluated).
#ifdef SEMSHARE_CHECKED
constexpr bool kChecked = true;
__device__ __forceinline__ void check_fail(uint32_t* err, uint32_t kernel, uint32_t line) {
    if (err == nullptr) return;
    const uint32_t old = atomicOr(err, SEMSHARE_FLAG_CHECK);
    if ((old >> 8) == 0u) {
        const uint32_t base = old | SEMSHARE_FLAG_CHECK;
        atomicCAS(err, base, base | (kernel << 8) | (line << 16));
    }
}
#define SEMSHARE_CHECK(cond, err, kernel)                                   \
    do {                                                                    \
        if (!(cond)) ::semshare::check_fail((err), (kernel), __LINE__);     \
    } while (0)
#else
constexpr bool kChecked = false;
#define SEMSHARE_CHECK(cond, err, kernel) \
    do {                                  \
    } while (0)
#endif

// Limit of every bounded pipeline wait inside a kernel (the host never sees a longer stall).
constexpr uint64_t kWaitLimitNs = 2000000000ull;

// The pipeline-wait limit of one call: kWaitLimitNs, or the nanoseconds in the environment
// variable SEMSHARE_WAIT_LIMIT_NS (a diagnostic knob, read at every call; tests use a tiny
// value to drive the timeout path).  The waits that let copies in flight land before a CTA
// exits always keep kWaitLimitNs.
inline uint64_t wait_limit_ns() {
    const char* e = getenv("SEMSHARE_WAIT_LIMIT_NS");
    if (e == nullptr || *e == 0) return kWaitLimitNs;
    char* end = nullptr;
    const unsigned long long v = strtoull(e, &end, 10);
    return (end != e && v > 0) ? static_cast<uint64_t>(v) : kWaitLimitNs;
}

}  // namespace semshare
