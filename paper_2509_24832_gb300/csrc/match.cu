// match.cu -- semshare_match: all-pairs Hamming nearest neighbour of every target code
// among the reference codes, ties to the lowest reference index.
//
// What it computes (SemShareKV, arXiv 2509.24832, Sec. 3.3): for each token of the target
// prompt, the most similar token of the reference prompt, here the reference row whose LSH
// code differs from the target's in the fewest bits.
//
// Kernel design.  The (target block, reference row) pairs, target blocks outermost, are split
// into one equal contiguous range per CTA (a stream-K style partition: every CTA does the same
// number of pair evaluations whatever n_tgt and n_ref are).  A CTA holds 512 target codes in
// registers (2 per thread), stages up to 256 reference codes at a time in shared memory, and
// each thread scans them with xor + popc against its targets (shared-memory broadcast reads),
// keeping a running minimum of (distance << 16 | local index).  When the range leaves a target
// block, each target's best (distance << 32 | global index) goes to a 64-bit atomicMin in the
// workspace.  atomicMin of that key is exactly "smallest distance, then lowest index", so the
// result does not depend on the partition.  A final pass splits the keys into idx and dist.
#include <cuda.h>

#include <mutex>

#include "common.cuh"

namespace semshare {
namespace {

constexpr int kThreads = 256;
constexpr int kTPT = 2;                     // target codes per thread
constexpr int kTB = kThreads * kTPT;        // targets per target block
constexpr int kRC = 256;                    // reference codes per staging round (local index < 2^16)
constexpr unsigned long long kNoKey = ~0ull;

__global__ void keys_init_kernel(unsigned long long* __restrict__ keys, int64_t n) {
    pdl_prologue();
    for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < n;
         i += static_cast<int64_t>(gridDim.x) * blockDim.x)
        keys[i] = kNoKey;
}

__global__ void keys_split_kernel(const unsigned long long* __restrict__ keys, int64_t n, int32_t* __restrict__ idx,
                                  int32_t* __restrict__ dist) {
    pdl_prologue();
    for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < n;
         i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const unsigned long long k = keys[i];
        idx[i] = static_cast<int32_t>(static_cast<uint32_t>(k));
        if (dist) dist[i] = static_cast<int32_t>(static_cast<uint32_t>(k >> 32));
    }
}

template <int W>
__device__ __forceinline__ void load_code(const uint32_t* p, uint32_t (&c)[W]) {
    if constexpr (W % 4 == 0) {
#pragma unroll
        for (int q = 0; q < W; q += 4) {
            const uint4 v = *reinterpret_cast<const uint4*>(p + q);
            c[q] = v.x; c[q + 1] = v.y; c[q + 2] = v.z; c[q + 3] = v.w;
        }
    } else {
#pragma unroll
        for (int q = 0; q < W; ++q) c[q] = p[q];
    }
}

template <int W>
__global__ void __launch_bounds__(kThreads)
    hamming_nn_kernel(const uint32_t* __restrict__ tgt, int64_t n_tgt, const uint32_t* __restrict__ ref, int64_t n_ref,
                      unsigned long long* __restrict__ keys, int64_t n_tblocks) {
    pdl_prologue();
    __shared__ __align__(16) uint32_t sref[kRC * W];

    // this CTA's share of the n_tblocks * n_ref (target block, reference row) pairs
    const int64_t total = n_tblocks * n_ref;
    const int64_t G = gridDim.x, q = total / G, rem = total % G, b = blockIdx.x;
    const int64_t p_begin = q * b + (b < rem ? b : rem);
    const int64_t p_end = p_begin + q + (b < rem ? 1 : 0);

    int64_t cur_tb = -1;
    uint32_t tc[kTPT][W];
    unsigned long long best[kTPT];

    for (int64_t p = p_begin; p < p_end;) {
        const int64_t tb = p / n_ref;
        const int64_t j0 = p - tb * n_ref;
        int64_t span = n_ref - j0;
        if (p_end - p < span) span = p_end - p;
        const int nr = static_cast<int>(span < kRC ? span : kRC);

        if (tb != cur_tb) {
            if (cur_tb >= 0) {
#pragma unroll
                for (int t = 0; t < kTPT; ++t) {
                    const int64_t g = cur_tb * kTB + t * kThreads + threadIdx.x;
                    if (g < n_tgt && best[t] != kNoKey) atomicMin(keys + g, best[t]);
                }
            }
            cur_tb = tb;
#pragma unroll
            for (int t = 0; t < kTPT; ++t) {
                const int64_t g = tb * kTB + t * kThreads + threadIdx.x;
                if (g < n_tgt) {
                    load_code<W>(tgt + g * W, tc[t]);
                } else {
#pragma unroll
                    for (int w = 0; w < W; ++w) tc[t][w] = 0u;
                }
                best[t] = kNoKey;
            }
        }

        __syncthreads();  // the previous round's readers are done with sref
        if constexpr (W % 4 == 0) {
            const uint4* src = reinterpret_cast<const uint4*>(ref + j0 * W);
            uint4* dst = reinterpret_cast<uint4*>(sref);
            for (int e = threadIdx.x; e < nr * (W / 4); e += kThreads) dst[e] = __ldg(src + e);
        } else {
            for (int e = threadIdx.x; e < nr * W; e += kThreads) sref[e] = __ldg(ref + j0 * W + e);
        }
        __syncthreads();

        uint32_t local[kTPT];
#pragma unroll
        for (int t = 0; t < kTPT; ++t) local[t] = 0xFFFFFFFFu;
#pragma unroll 4
        for (int j = 0; j < nr; ++j) {
            uint32_t r[W];
            load_code<W>(sref + j * W, r);
#pragma unroll
            for (int t = 0; t < kTPT; ++t) {
                uint32_t dsum = 0;
#pragma unroll
                for (int w = 0; w < W; ++w) dsum += __popc(tc[t][w] ^ r[w]);
                local[t] = min(local[t], (dsum << 16) | static_cast<uint32_t>(j));
            }
        }
#pragma unroll
        for (int t = 0; t < kTPT; ++t) {
            if (local[t] != 0xFFFFFFFFu) {
                const unsigned long long cand = (static_cast<unsigned long long>(local[t] >> 16) << 32) |
                                                static_cast<unsigned long long>(j0 + (local[t] & 0xFFFFu));
                best[t] = cand < best[t] ? cand : best[t];
            }
        }
        p += nr;
    }
    if (cur_tb >= 0) {
#pragma unroll
        for (int t = 0; t < kTPT; ++t) {
            const int64_t g = cur_tb * kTB + t * kThreads + threadIdx.x;
            if (g < n_tgt && best[t] != kNoKey) atomicMin(keys + g, best[t]);
        }
    }
}

template <int W>
semshare_status launch_search(const uint32_t* tgt, int64_t n_tgt, const uint32_t* ref, int64_t n_ref,
                              unsigned long long* keys, int sms, cudaStream_t s) {
    int per_sm = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, hamming_nn_kernel<W>, kThreads, 0) != cudaSuccess)
        return SEMSHARE_ECUDA;
    if (per_sm < 1) per_sm = 1;
    const int64_t n_tblocks = (n_tgt + kTB - 1) / kTB;
    const int64_t total = n_tblocks * n_ref;
    int64_t grid = static_cast<int64_t>(sms) * per_sm;
    if (grid > total) grid = total;
    if (launch_pdl(hamming_nn_kernel<W>, dim3(static_cast<unsigned>(grid)), dim3(kThreads), 0, s, tgt, n_tgt, ref, n_ref,
                   keys, n_tblocks) != cudaSuccess)
        return SEMSHARE_ECUDA;
    return launch_status();
}

}  // namespace
}  // namespace semshare

extern "C" size_t semshare_match_workspace_size(int64_t n_tgt) {
    return n_tgt > 0 ? static_cast<size_t>(n_tgt) * sizeof(unsigned long long) : 0;
}

extern "C" semshare_status semshare_match(const uint32_t* tgt_codes, int64_t n_tgt, const uint32_t* ref_codes,
                                          int64_t n_ref, int32_t nbits, int32_t* idx, int32_t* dist,
                                          void* workspace, size_t workspace_bytes, void* stream) {
    using namespace semshare;
    if (n_tgt < 0 || n_ref < 1) return SEMSHARE_EINVAL;
    if (nbits < 32 || nbits > 256 || nbits % 32 != 0) return SEMSHARE_EUNSUPPORTED;
    if (n_tgt >= (int64_t(1) << 31) || n_ref >= (int64_t(1) << 31)) return SEMSHARE_EUNSUPPORTED;
    if (n_tgt == 0) return SEMSHARE_OK;
    if (!tgt_codes || !ref_codes || !idx || !workspace) return SEMSHARE_EINVAL;
    if (!aligned(tgt_codes, 16) || !aligned(ref_codes, 16) || !aligned(idx, 4) || !aligned(workspace, 8) ||
        (dist && !aligned(dist, 4)))
        return SEMSHARE_EINVAL;
    if (workspace_bytes < semshare_match_workspace_size(n_tgt)) return SEMSHARE_EINVAL;

    int sms = 0;
    if (current_sm_count(&sms, nullptr) != SEMSHARE_OK) return SEMSHARE_ECUDA;
    cudaStream_t s = as_stream(stream);
    auto* keys = static_cast<unsigned long long*>(workspace);
    const int small_grid = static_cast<int>((n_tgt + 255) / 256 < sms * 4 ? (n_tgt + 255) / 256 : sms * 4);

    if (launch_pdl(keys_init_kernel, dim3(small_grid), dim3(256), 0, s, keys, n_tgt) != cudaSuccess) return SEMSHARE_ECUDA;
    if (launch_status() != SEMSHARE_OK) return SEMSHARE_ECUDA;
    semshare_status st = SEMSHARE_EUNSUPPORTED;
    switch (nbits / 32) {
        case 1: st = launch_search<1>(tgt_codes, n_tgt, ref_codes, n_ref, keys, sms, s); break;
        case 2: st = launch_search<2>(tgt_codes, n_tgt, ref_codes, n_ref, keys, sms, s); break;
        case 3: st = launch_search<3>(tgt_codes, n_tgt, ref_codes, n_ref, keys, sms, s); break;
        case 4: st = launch_search<4>(tgt_codes, n_tgt, ref_codes, n_ref, keys, sms, s); break;
        case 5: st = launch_search<5>(tgt_codes, n_tgt, ref_codes, n_ref, keys, sms, s); break;
        case 6: st = launch_search<6>(tgt_codes, n_tgt, ref_codes, n_ref, keys, sms, s); break;
        case 7: st = launch_search<7>(tgt_codes, n_tgt, ref_codes, n_ref, keys, sms, s); break;
        case 8: st = launch_search<8>(tgt_codes, n_tgt, ref_codes, n_ref, keys, sms, s); break;
    }
    if (st != SEMSHARE_OK) return st;
    if (launch_pdl(keys_split_kernel, dim3(small_grid), dim3(256), 0, s, keys, n_tgt, idx, dist) != cudaSuccess)
        return SEMSHARE_ECUDA;
    return launch_status();
}

// ---- semshare_match_static: the same search with library-owned scratch ------------------------
//
// For callers that cannot allocate device memory themselves (for example code embedded in a
// host framework that owns the whole device memory pool and forbids allocations, or a serving
// loop that must not allocate on its hot path).  The per-target keys live in one file-scope
// device array instead of a caller workspace; every device that loads this library holds it
// (SEMSHARE_MATCH_STATIC_MAX_TARGETS x 8 bytes = 2 MiB) until the process exits.

static __device__ __align__(256) unsigned long long g_static_match_keys[SEMSHARE_MATCH_STATIC_MAX_TARGETS];

namespace semshare {
namespace {

constexpr int kStaticMaxDevices = 64;
std::mutex g_static_keys_mutex;
struct StaticKeysEntry {
    unsigned long long ctx_id;  // the context the address belongs to (0: none looked up yet)
    unsigned long long* addr;
};
StaticKeysEntry g_static_keys[kStaticMaxDevices] = {};

// Unique id of the calling thread's current CUDA context (0 if there is none or the driver
// cannot say).  Ids are never reused within a process, unlike context handles.
unsigned long long current_context_id() {
    using GetCurrentFn = CUresult (*)(CUcontext*);
    using GetIdFn = CUresult (*)(CUcontext, unsigned long long*);
    static GetCurrentFn get_current = nullptr;  // resolved once per process
    static GetIdFn get_id = nullptr;
    if (get_current == nullptr || get_id == nullptr) {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q = cudaDriverEntryPointSymbolNotFound;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) != cudaSuccess ||
            q != cudaDriverEntryPointSuccess)
            return 0;
        get_current = reinterpret_cast<GetCurrentFn>(p);
        if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &p, 12000, cudaEnableDefault, &q) != cudaSuccess ||
            q != cudaDriverEntryPointSuccess)
            return 0;
        get_id = reinterpret_cast<GetIdFn>(p);
    }
    CUcontext ctx = nullptr;
    unsigned long long id = 0;
    if (get_current(&ctx) != CUDA_SUCCESS || ctx == nullptr || get_id(ctx, &id) != CUDA_SUCCESS) return 0;
    return id;
}

// Device address of g_static_match_keys in the current device's current context.  In host code
// the array's name is only a host-side stand-in, so the address is looked up (with the device
// current) the first time a device is used, and again whenever the device's current context is
// not the one the cached address belongs to (after cudaDeviceReset, or when the caller switches
// to a context of its own), since the array lives at a per-context address.
semshare_status static_keys_on_current_device(unsigned long long** keys) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return SEMSHARE_ECUDA;
    if (dev < 0 || dev >= kStaticMaxDevices) return SEMSHARE_EUNSUPPORTED;
    std::lock_guard<std::mutex> lock(g_static_keys_mutex);
    StaticKeysEntry& e = g_static_keys[dev];
    unsigned long long ctx_id = current_context_id();
    if (ctx_id == 0 || e.ctx_id != ctx_id || e.addr == nullptr) {
        // the lookup also makes the device's primary context current when no context is yet
        void* p = nullptr;
        if (cudaGetSymbolAddress(&p, g_static_match_keys) != cudaSuccess || p == nullptr) return SEMSHARE_ECUDA;
        if (ctx_id == 0) ctx_id = current_context_id();
        if (ctx_id == 0) return SEMSHARE_ECUDA;
        e.addr = static_cast<unsigned long long*>(p);
        e.ctx_id = ctx_id;
    }
    *keys = e.addr;
    return SEMSHARE_OK;
}

}  // namespace
}  // namespace semshare

extern "C" semshare_status semshare_match_static(const uint32_t* tgt_codes, int64_t n_tgt, const uint32_t* ref_codes,
                                                 int64_t n_ref, int32_t nbits, int32_t* idx, int32_t* dist,
                                                 void* stream) {
    using namespace semshare;
    if (n_tgt < 0 || n_ref < 1) return SEMSHARE_EINVAL;
    if (nbits < 32 || nbits > 256 || nbits % 32 != 0) return SEMSHARE_EUNSUPPORTED;
    if (n_ref >= (int64_t(1) << 31)) return SEMSHARE_EUNSUPPORTED;
    if (n_tgt > SEMSHARE_MATCH_STATIC_MAX_TARGETS) return SEMSHARE_ETOOLARGE;
    if (n_tgt == 0) return SEMSHARE_OK;
    if (!tgt_codes || !ref_codes || !idx) return SEMSHARE_EINVAL;
    if (!aligned(tgt_codes, 16) || !aligned(ref_codes, 16) || !aligned(idx, 4) || (dist && !aligned(dist, 4)))
        return SEMSHARE_EINVAL;

    unsigned long long* keys = nullptr;
    semshare_status st = static_keys_on_current_device(&keys);
    if (st != SEMSHARE_OK) return st;
    int sms = 0;
    if (current_sm_count(&sms, nullptr) != SEMSHARE_OK) return SEMSHARE_ECUDA;
    cudaStream_t s = as_stream(stream);
    const int small_grid = static_cast<int>((n_tgt + 255) / 256 < sms * 4 ? (n_tgt + 255) / 256 : sms * 4);

    // the array keeps the previous call's keys: reset the ones this call uses
    if (launch_pdl(keys_init_kernel, dim3(small_grid), dim3(256), 0, s, keys, n_tgt) != cudaSuccess) return SEMSHARE_ECUDA;
    if (launch_status() != SEMSHARE_OK) return SEMSHARE_ECUDA;
    st = SEMSHARE_EUNSUPPORTED;
    switch (nbits / 32) {
        case 1: st = launch_search<1>(tgt_codes, n_tgt, ref_codes, n_ref, keys, sms, s); break;
        case 2: st = launch_search<2>(tgt_codes, n_tgt, ref_codes, n_ref, keys, sms, s); break;
        case 3: st = launch_search<3>(tgt_codes, n_tgt, ref_codes, n_ref, keys, sms, s); break;
        case 4: st = launch_search<4>(tgt_codes, n_tgt, ref_codes, n_ref, keys, sms, s); break;
        case 5: st = launch_search<5>(tgt_codes, n_tgt, ref_codes, n_ref, keys, sms, s); break;
        case 6: st = launch_search<6>(tgt_codes, n_tgt, ref_codes, n_ref, keys, sms, s); break;
        case 7: st = launch_search<7>(tgt_codes, n_tgt, ref_codes, n_ref, keys, sms, s); break;
        case 8: st = launch_search<8>(tgt_codes, n_tgt, ref_codes, n_ref, keys, sms, s); break;
    }
    if (st != SEMSHARE_OK) return st;
    if (launch_pdl(keys_split_kernel, dim3(small_grid), dim3(256), 0, s, keys, n_tgt, idx, dist) != cudaSuccess)
        return SEMSHARE_ECUDA;
    return launch_status();
}
