// probe.cu -- semshare_probe_hamming_rate: the sustained rate of the Hamming search's word
// operation (xor two code words, population count, add to the distance) on this device.
//
// Each thread runs SEMSHARE_PROBE_CHAINS independent chains in registers; a chain's code word
// changes every iteration by an add, so no count can be hoisted out of the loop.  Per word op:
// one xor, one popc, two adds -- the population count is the narrowest of the pipes involved.
// Enough warps are resident that the chains' latency is hidden and the issue of popc binds.
//
// semshare_probe_operand_stream: the LSH projection's operand stream on its own.  One CTA per
// SM takes the same equal contiguous share of the (128-row tile, 64-wide K block) iterations as
// semshare_hash and moves each iteration's blocks into a ring of shared-memory slots with the
// same TMA boxes (128 x 64 bf16 embedding block, nbits x 64 hyperplane block, 128-byte swizzle)
// and, optionally, the same L2 prefetch; one thread releases each slot as soon as it lands.  No
// rotation, no MMA: the launch time is what the operand traffic alone costs.
#include "common.cuh"
#include "ptx.cuh"
#include "semshare_probe.h"
#include "tma_host.cuh"

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

struct StreamArgs {
    int64_t total;  // n_tiles * n_kblocks
    int32_t n_kblocks;
    int32_t slots;
    int32_t prefetch;
    int32_t with_hyp;
    uint32_t slot_bytes;
    uint32_t* err_flag;
    uint64_t limit_ns;
};

__device__ __forceinline__ bool stream_wait(uint32_t bar, uint32_t parity, uint64_t limit_ns) {
    if (mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = global_timer_ns();
    while (!mbar_try_wait(bar, parity))
        if (global_timer_ns() - t0 > limit_ns) return false;
    return true;
}

__global__ void __launch_bounds__(64, 1)
    operand_stream_kernel(const __grid_constant__ CUtensorMap tmap_emb, const __grid_constant__ CUtensorMap tmap_hyp,
                          const StreamArgs a) {
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_addr(smem_raw);
    const uint32_t sbase = (raw + 1023u) & ~1023u;
    const uint32_t S = static_cast<uint32_t>(a.slots);
    const uint32_t full = sbase + S * a.slot_bytes, empty = full + 8u * S;
    const int64_t G = gridDim.x;
    const int64_t i0 = (static_cast<int64_t>(blockIdx.x) * a.total) / G;
    const int64_t i1 = ((static_cast<int64_t>(blockIdx.x) + 1) * a.total) / G;
    const int nkb = a.n_kblocks;
    if (threadIdx.x == 0) {
        for (uint32_t s = 0; s < S; ++s) {
            mbar_init(full + 8u * s, 1);
            mbar_init(empty + 8u * s, 1);
        }
        fence_barrier_init();
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        // producer: the hash kernel's loads, slot by slot
        int64_t pf = i0;
        for (int i = 0; i < a.prefetch && pf < i1; ++i, ++pf)
            tma_prefetch_l2_2d(&tmap_emb, static_cast<int32_t>(pf % nkb) * 64, static_cast<int32_t>(pf / nkb) * 128);
        uint32_t q = 0;
        for (int64_t it = i0; it < i1; ++it, ++q) {
            const uint32_t s = q % S, ph = (q / S) & 1u;
            if (!stream_wait(empty + 8u * s, ph ^ 1u, a.limit_ns)) {
                if (a.err_flag) atomicOr(a.err_flag, SEMSHARE_FLAG_TIMEOUT);
                break;
            }
            const uint32_t dst = sbase + s * a.slot_bytes;
            mbar_arrive_expect_tx(full + 8u * s, a.slot_bytes);
            const int32_t x = static_cast<int32_t>(it % nkb) * 64;
            tma_load_2d(dst, &tmap_emb, full + 8u * s, x, static_cast<int32_t>(it / nkb) * 128);
            if (a.with_hyp) tma_load_2d(dst + 16384u, &tmap_hyp, full + 8u * s, x, 0);
            if (a.prefetch && pf < i1) {
                tma_prefetch_l2_2d(&tmap_emb, static_cast<int32_t>(pf % nkb) * 64, static_cast<int32_t>(pf / nkb) * 128);
                ++pf;
            }
        }
    } else if (threadIdx.x == 32) {
        // consumer: frees each slot once its copy has landed.  It waits for every issued copy
        // (in order), so none is in flight when the CTA exits; after a producer timeout the first
        // copy never issued ends the loop through the same bounded wait.
        uint32_t q = 0;
        for (int64_t it = i0; it < i1; ++it, ++q) {
            const uint32_t s = q % S, ph = (q / S) & 1u;
            if (!stream_wait(full + 8u * s, ph, a.limit_ns)) {
                if (a.err_flag) atomicOr(a.err_flag, SEMSHARE_FLAG_TIMEOUT);
                break;
            }
            mbar_arrive(empty + 8u * s);
        }
    }
    __syncthreads();
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

extern "C" semshare_status semshare_probe_operand_stream(const uint16_t* emb, int64_t n, int32_t d,
                                                         const uint16_t* hyperplanes, int32_t nbits, int32_t slots,
                                                         int32_t prefetch, uint32_t* err_flag, void* stream) {
    using namespace semshare;
    if (!emb || n < 128 || n % 128 != 0 || n >= (int64_t(1) << 31) || d < 64 || d % 64 != 0 || !aligned(emb, 16))
        return SEMSHARE_EINVAL;
    if (slots < 1 || slots > 12 || prefetch < 0 || prefetch > 64 || (err_flag && !aligned(err_flag, 4)))
        return SEMSHARE_EINVAL;
    if (hyperplanes && (nbits < 32 || nbits > 256 || nbits % 32 != 0)) return SEMSHARE_EUNSUPPORTED;
    if (hyperplanes && !aligned(hyperplanes, 16)) return SEMSHARE_EINVAL;
    int sms = 0, dev = 0, smem_optin = 0;
    if (current_sm_count(&sms, &dev) != SEMSHARE_OK ||
        cudaDeviceGetAttribute(&smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess)
        return SEMSHARE_ECUDA;
    StreamArgs a{};
    a.n_kblocks = d / 64;
    a.total = (n / 128) * a.n_kblocks;
    a.slots = slots;
    a.prefetch = prefetch;
    a.with_hyp = hyperplanes != nullptr;
    a.slot_bytes = 16384u + (hyperplanes ? static_cast<uint32_t>(nbits) * 128u : 0u);
    a.err_flag = err_flag;
    a.limit_ns = wait_limit_ns();
    const size_t smem = 1024 + static_cast<size_t>(slots) * a.slot_bytes + 16 * static_cast<size_t>(slots);
    if (smem > static_cast<size_t>(smem_optin)) return SEMSHARE_EUNSUPPORTED;
    CUtensorMap tm_e, tm_h;
    if (!encode_tma_2d(&tm_e, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, emb, static_cast<uint64_t>(d), static_cast<uint64_t>(n),
                       static_cast<uint64_t>(d) * 2, 64, 128))
        return SEMSHARE_ECUDA;
    tm_h = tm_e;  // unused without hyperplanes
    if (hyperplanes && !encode_tma_2d(&tm_h, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, hyperplanes, static_cast<uint64_t>(d),
                                      static_cast<uint64_t>(nbits), static_cast<uint64_t>(d) * 2, 64,
                                      static_cast<uint32_t>(nbits)))
        return SEMSHARE_ECUDA;
    if (cudaFuncSetAttribute(operand_stream_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(smem)) != cudaSuccess)
        return SEMSHARE_ECUDA;
    operand_stream_kernel<<<sms, 64, smem, as_stream(stream)>>>(tm_e, tm_h, a);
    return launch_status();
}
