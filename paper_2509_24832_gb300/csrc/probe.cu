// probe.cu -- semshare_probe_hamming_rate: the sustained rate of the Hamming search's word
// operation (xor two code words, population count, add to the distance) on this device.
//
// Each thread runs SEMSHARE_PROBE_CHAINS independent chains in registers; a chain's code word
// changes every iteration by an add, so no count can be hoisted out of the loop.  Per word op:
// one xor, one popc, two adds -- the population count is the narrowest of the pipes involved.
// Enough warps are resident that the chains' latency is hidden and the issue of popc binds.
//
// Built into its own library, libsemshare_probe.so (measurement support for bench.py), not into
// libsemshare.so.
#include "common.cuh"
#include "ptx.cuh"
#include "semshare_probe.h"

namespace semshare {
namespace {

constexpr int kThreads = 256;
constexpr int kChains = SEMSHARE_PROBE_CHAINS;

__global__ void __launch_bounds__(kThreads) hamming_rate_kernel(int64_t iters, uint32_t* __restrict__ sink) {
    const uint32_t t = blockIdx.x * kThreads + threadIdx.x;
    uint32_t x[kChains], y[kChains], acc[kChains];
#pragma unroll
    for (int c = 0; c < kChains; ++c) {
        x[c] = (t * 0x9E3779B9u) ^ (0x85EBCA6Bu * static_cast<uint32_t>(c + 1));
        y[c] = x[c] * 0xC2B2AE35u + static_cast<uint32_t>(c);
        acc[c] = 0u;
    }
    for (int64_t i = 0; i < iters; ++i) {
#pragma unroll
        for (int c = 0; c < kChains; ++c) {
            acc[c] += static_cast<uint32_t>(__popc(x[c] ^ y[c]));
            y[c] += 0x9E3779B9u;
        }
    }
    uint32_t r = 0u;
#pragma unroll
    for (int c = 0; c < kChains; ++c) r ^= acc[c] + static_cast<uint32_t>(c);
    sink[t] = r;
}

bool probe_grid(int* blocks) {
    int sms = 0, per_sm = 0;
    if (current_sm_count(&sms, nullptr) != SEMSHARE_OK) return false;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, hamming_rate_kernel, kThreads, 0) != cudaSuccess ||
        per_sm < 1)
        return false;
    *blocks = sms * per_sm;
    return true;
}

}  // namespace
}  // namespace semshare

extern "C" int64_t semshare_probe_hamming_threads(void) {
    int blocks = 0;
    if (!semshare::probe_grid(&blocks)) return -1;
    return static_cast<int64_t>(blocks) * semshare::kThreads;
}

extern "C" semshare_status semshare_probe_hamming_rate(int64_t iters, uint32_t* sink, int64_t sink_words,
                                                       void* stream) {
    using namespace semshare;
    if (iters < 1 || iters > (int64_t(1) << 24) || !sink || !aligned(sink, 4)) return SEMSHARE_EINVAL;
    int blocks = 0;
    if (!probe_grid(&blocks)) return SEMSHARE_ECUDA;
    if (sink_words < static_cast<int64_t>(blocks) * kThreads) return SEMSHARE_EINVAL;
    hamming_rate_kernel<<<blocks, kThreads, 0, as_stream(stream)>>>(iters, sink);
    return launch_status();
}
