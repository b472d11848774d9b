// common.cuh -- host-side helpers shared by the entry points.
#pragma once

#include <cuda_runtime.h>

#include <cstdint>
#include <cstdlib>

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

inline semshare_status launch_status() {
    return cudaGetLastError() == cudaSuccess ? SEMSHARE_OK : SEMSHARE_ECUDA;
}

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
