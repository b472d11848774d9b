// common.cuh -- host-side helpers shared by the entry points.
#pragma once

#include <cuda_runtime.h>

#include <cstdint>

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

}  // namespace semshare
