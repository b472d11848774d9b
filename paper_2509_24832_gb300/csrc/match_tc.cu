// match_tc.cu -- semshare_match_tc: the Hamming nearest-neighbour search of semshare_match
// computed on the tcgen05 tensor cores.
//
// What it computes (SemShareKV, arXiv 2509.24832, Sec. 3.3): for each target token, the
// reference token whose LSH code differs from the target's in the fewest bits, ties to the
// lowest reference index -- exactly semshare_match's result.
//
// Method.  With s = 2*bit - 1 in {-1, +1}, popcount(a XOR b) = (nbits - <s_a, s_b>) / 2, so the
// all-pairs distances are one dense contraction over the code bits.  Codes are expanded to
// e4m3 +-1 rows (zero-padded to a multiple of 128 bytes), multiplied as a GEMM with fp32
// accumulation (every partial sum is a small integer, so the products are exact), and each
// accumulator row is reduced on the fly to its best reference with the exact fp32 key
// 256*dot - j (largest dot first, then lowest j within the 256-wide tile).  The best
// (distance << 32 | index) of a target over the tiles a CTA visits goes to a 64-bit atomicMin,
// which is "smallest distance, then lowest index" whatever the split.
//
// Roles (256 threads): warp 0 TMA producer (the 128-target A tile, reloaded only when the
// target block changes, and the 256-reference B tile, double-buffered); warp 1 TMEM allocator
// and MMA issuer (tcgen05.mma kind::f8f6f4, M=128, N=256, K=32); warps 4-7 epilogue
// (tcgen05.ld, lane = target, running arg-max).  The (target block, reference block) tiles are
// split into one equal contiguous range per CTA, target blocks outermost.  Every pipeline wait
// is bounded (SEMSHARE_FLAG_TIMEOUT), nothing traps.
#include <cuda.h>

#include "common.cuh"
#include "ptx.cuh"
#include "tma_host.cuh"

namespace semshare {
namespace {

constexpr int kTM = 128;        // targets per tile (TMEM lanes)
constexpr int kTN = 256;        // references per tile (MMA N)
constexpr int kChunk = 128;     // bytes per 128-byte swizzle chunk along the code
constexpr int kThreads = 256;
constexpr int kEpiWarp0 = 4;
constexpr unsigned long long kNoKey = ~0ull;
constexpr size_t kFixedSmem = 1024 + 256;

struct TcArgs {
    int64_t n_tgt;
    int64_t n_ref;
    int64_t n_rb;
    int64_t total;  // target blocks x reference blocks
    int32_t nbits;
    int32_t kchunks;
    uint32_t a_bytes;  // one A buffer: 128 rows x kchunks*128 bytes
    uint32_t b_bytes;  // one B buffer: 256 rows x kchunks*128 bytes
    unsigned long long* keys;
    uint32_t* err_flag;
    uint64_t wait_limit_ns;
};

// e4m3 +1 is 0x38, -1 is 0xB8: byte = 0xB8 ^ (bit << 7).  Rows are padded with zero bytes to
// kpad; the keys of the search are reset on the way.
__global__ void expand_codes_kernel(const uint32_t* __restrict__ tgt, int64_t n_tgt, const uint32_t* __restrict__ ref,
                                    int64_t n_ref, int32_t nbits, int32_t kpad, uint8_t* __restrict__ tpm,
                                    uint8_t* __restrict__ rpm, unsigned long long* __restrict__ keys) {
    const int W = nbits >> 5;
    const int per_row = kpad >> 4;  // 16-byte pieces per row
    const int64_t total = (n_tgt + n_ref) * per_row;
    const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
    for (int64_t e = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; e < total; e += stride) {
        const int64_t row = e / per_row;
        const int piece = static_cast<int>(e - row * per_row);
        const int b0 = piece * 16;
        uint4 out = make_uint4(0u, 0u, 0u, 0u);
        if (b0 < nbits) {
            const uint32_t* src = row < n_tgt ? tgt + row * W : ref + (row - n_tgt) * W;
            const uint32_t bits = __ldg(src + (b0 >> 5)) >> (b0 & 31);
            uint32_t w[4];
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                uint32_t v = 0;
#pragma unroll
                for (int i = 0; i < 4; ++i) v |= (0xB8u ^ (((bits >> (4 * q + i)) & 1u) << 7)) << (8 * i);
                w[q] = v;
            }
            out = make_uint4(w[0], w[1], w[2], w[3]);
        }
        uint8_t* dst = row < n_tgt ? tpm + row * kpad : rpm + (row - n_tgt) * kpad;
        *reinterpret_cast<uint4*>(dst + b0) = out;
    }
    for (int64_t t = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; t < n_tgt; t += stride) keys[t] = kNoKey;
}

__global__ void tc_keys_split_kernel(const unsigned long long* __restrict__ keys, int64_t n, int32_t* __restrict__ idx,
                                     int32_t* __restrict__ dist) {
    for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < n;
         i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const unsigned long long k = keys[i];
        idx[i] = static_cast<int32_t>(static_cast<uint32_t>(k));
        if (dist) dist[i] = static_cast<int32_t>(static_cast<uint32_t>(k >> 32));
    }
}

__device__ __forceinline__ bool drain_wait(uint32_t bar, uint32_t parity, uint64_t limit_ns) {
    if (mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = global_timer_ns();
    while (!mbar_try_wait(bar, parity))
        if (global_timer_ns() - t0 > limit_ns) return false;
    return true;
}

__global__ void __launch_bounds__(kThreads, 1)
    hamming_tc_kernel(const __grid_constant__ CUtensorMap tm_t, const __grid_constant__ CUtensorMap tm_r,
                      const TcArgs a) {
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_addr(smem_raw);
    const uint32_t sbase = (raw + 1023u) & ~1023u;
    uint8_t* const gbase = smem_raw + (sbase - raw);
    const uint32_t a_buf0 = sbase;                    // 2 A buffers
    const uint32_t b_buf0 = sbase + 2u * a.a_bytes;   // 2 B buffers
    const uint32_t bars = b_buf0 + 2u * a.b_bytes;
    const uint32_t bar_afull = bars, bar_aempty = bars + 16, bar_bfull = bars + 32, bar_bempty = bars + 48;
    const uint32_t bar_accfull = bars + 64, bar_accempty = bars + 80, bar_done = bars + 96;
    const uint32_t tmem_slot = bars + 104;
    volatile uint32_t* const tmem_slot_ptr = reinterpret_cast<volatile uint32_t*>(gbase + (tmem_slot - sbase));
    volatile int* const abort_flag = reinterpret_cast<volatile int*>(gbase + (tmem_slot + 4u - sbase));

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t G = gridDim.x, b = blockIdx.x;
    const int64_t u0 = (b * a.total) / G, u1 = ((b + 1) * a.total) / G;

    if (threadIdx.x == 0) {
        for (int i = 0; i < 2; ++i) {
            mbar_init(bar_afull + 8 * i, 1);
            mbar_init(bar_aempty + 8 * i, 1);
            mbar_init(bar_bfull + 8 * i, 1);
            mbar_init(bar_bempty + 8 * i, 1);
            mbar_init(bar_accfull + 8 * i, 1);
            mbar_init(bar_accempty + 8 * i, 4);
        }
        mbar_init(bar_done, 1);
        *abort_flag = 0;
        fence_barrier_init();
    }
    if (warp == 0 && lane == 0) {
        tma_prefetch_desc(&tm_t);
        tma_prefetch_desc(&tm_r);
    }
    if (warp == 1) {
        tmem_alloc(tmem_slot, 512);
        tmem_relinquish();
    }
    tc_fence_before_sync();
    __syncthreads();
    tc_fence_after_sync();
    const uint32_t tmem_base = *tmem_slot_ptr;
    const uint64_t lim = a.wait_limit_ns;
    uint32_t* const err = a.err_flag;

    if (warp == 0) {
        // ---------------- TMA producer ----------------
        if (lane == 0) {
            uint32_t na = 0, nb = 0;
            int64_t cur_tb = -1;
            bool ok = true;
            for (int64_t u = u0; u < u1 && ok; ++u) {
                const int64_t tb = u / a.n_rb, rb = u - tb * a.n_rb;
                if (tb != cur_tb) {
                    const uint32_t s = na & 1u, ph = (na >> 1) & 1u;
                    if (!mbar_wait_bounded(bar_aempty + 8 * s, ph ^ 1u, abort_flag, err, SEMSHARE_FLAG_TIMEOUT, lim)) {
                        ok = false;
                        break;
                    }
                    mbar_arrive_expect_tx(bar_afull + 8 * s, a.a_bytes);
                    for (int c = 0; c < a.kchunks; ++c)
                        tma_load_2d(a_buf0 + s * a.a_bytes + c * (kTM * kChunk), &tm_t, bar_afull + 8 * s, c * kChunk,
                                    static_cast<int32_t>(tb * kTM));
                    ++na;
                    cur_tb = tb;
                }
                const uint32_t s = nb & 1u, ph = (nb >> 1) & 1u;
                if (!mbar_wait_bounded(bar_bempty + 8 * s, ph ^ 1u, abort_flag, err, SEMSHARE_FLAG_TIMEOUT, lim)) {
                    ok = false;
                    break;
                }
                mbar_arrive_expect_tx(bar_bfull + 8 * s, a.b_bytes);
                for (int c = 0; c < a.kchunks; ++c)
                    tma_load_2d(b_buf0 + s * a.b_bytes + c * (kTN * kChunk), &tm_r, bar_bfull + 8 * s, c * kChunk,
                                static_cast<int32_t>(rb * kTN));
                ++nb;
            }
            if (!ok) {
                // loads already issued may still be landing: wait for them before exit
                if (na > 0) drain_wait(bar_afull + 8 * ((na - 1) & 1u), ((na - 1) >> 1) & 1u, kWaitLimitNs);
                if (na > 1) drain_wait(bar_afull + 8 * ((na - 2) & 1u), ((na - 2) >> 1) & 1u, kWaitLimitNs);
                if (nb > 0) drain_wait(bar_bfull + 8 * ((nb - 1) & 1u), ((nb - 1) >> 1) & 1u, kWaitLimitNs);
                if (nb > 1) drain_wait(bar_bfull + 8 * ((nb - 2) & 1u), ((nb - 2) >> 1) & 1u, kWaitLimitNs);
            }
        }
        __syncwarp();
    } else if (warp == 1) {
        // ---------------- MMA issuer ----------------
        if (lane == 0) {
            const uint32_t idesc = umma_idesc_e4m3_f32(kTM, kTN);
            uint32_t na = 0, nb = 0, acc = 0, a_slot = 0;
            int64_t cur_tb = -1;
            for (int64_t u = u0; u < u1; ++u) {
                const int64_t tb = u / a.n_rb;
                if (tb != cur_tb) {
                    if (cur_tb >= 0) umma_commit(bar_aempty + 8 * a_slot);  // free once its MMAs are done
                    a_slot = na & 1u;
                    if (!mbar_wait_bounded(bar_afull + 8 * a_slot, (na >> 1) & 1u, abort_flag, err,
                                           SEMSHARE_FLAG_TIMEOUT, lim))
                        break;
                    ++na;
                    cur_tb = tb;
                }
                const uint32_t buf = acc & 1u;
                if (!mbar_wait_bounded(bar_accempty + 8 * buf, ((acc >> 1) & 1u) ^ 1u, abort_flag, err,
                                       SEMSHARE_FLAG_TIMEOUT, lim))
                    break;
                const uint32_t s = nb & 1u;
                if (!mbar_wait_bounded(bar_bfull + 8 * s, (nb >> 1) & 1u, abort_flag, err, SEMSHARE_FLAG_TIMEOUT, lim))
                    break;
                tc_fence_after_sync();
                const uint32_t d_tmem = tmem_base + buf * kTN;
                const uint32_t abase = a_buf0 + a_slot * a.a_bytes, bbase = b_buf0 + s * a.b_bytes;
                for (int c = 0; c < a.kchunks; ++c)
#pragma unroll
                    for (int k = 0; k < kChunk / 32; ++k)
                        umma_f8_ss(d_tmem, sw128_kmajor_desc(abase + c * (kTM * kChunk) + k * 32),
                                   sw128_kmajor_desc(bbase + c * (kTN * kChunk) + k * 32), idesc,
                                   (c | k) != 0 ? 1u : 0u);
                umma_commit(bar_bempty + 8 * s);
                umma_commit(bar_accfull + 8 * buf);
                ++nb;
                ++acc;
            }
            umma_commit(bar_done);
            drain_wait(bar_done, 0, kWaitLimitNs);
        }
        __syncwarp();
    } else if (warp >= kEpiWarp0) {
        // ---------------- epilogue: best reference of every target row ----------------
        const int ew = warp - kEpiWarp0;
        const int r = ew * 32 + lane;
        uint32_t acc = 0;
        int64_t cur_tb = -1;
        unsigned long long best = kNoKey;
        for (int64_t u = u0; u < u1; ++u, ++acc) {
            const int64_t tb = u / a.n_rb, rb = u - tb * a.n_rb;
            if (tb != cur_tb) {
                if (cur_tb >= 0) {
                    const int64_t g = cur_tb * kTM + r;
                    if (g < a.n_tgt && best != kNoKey) atomicMin(a.keys + g, best);
                }
                cur_tb = tb;
                best = kNoKey;
            }
            const uint32_t buf = acc & 1u;
            const bool got = mbar_wait_bounded(bar_accfull + 8 * buf, (acc >> 1) & 1u, abort_flag, err,
                                               SEMSHARE_FLAG_TIMEOUT, lim);
            if (!__all_sync(0xFFFFFFFFu, got)) {
                cur_tb = -1;
                break;
            }
            tc_fence_after_sync();
            const int64_t rem = a.n_ref - rb * kTN;
            const int valid = rem < kTN ? static_cast<int>(rem) : kTN;
            const uint32_t taddr = tmem_base + (static_cast<uint32_t>(ew * 32) << 16) + buf * kTN;
            float bk = -3.0e38f;  // best key 256*dot - j of this tile
#pragma unroll
            for (int q = 0; q < kTN / 32; ++q) {
                uint32_t v[32];
                tmem_load_32cols(taddr + q * 32, v);
                tmem_load_wait();
                if (q * 32 + 32 <= valid) {
#pragma unroll
                    for (int j = 0; j < 32; ++j)
                        bk = fmaxf(bk, fmaf(__uint_as_float(v[j]), 256.0f, -static_cast<float>(q * 32 + j)));
                } else if (q * 32 < valid) {
#pragma unroll
                    for (int j = 0; j < 32; ++j)
                        if (q * 32 + j < valid)
                            bk = fmaxf(bk, fmaf(__uint_as_float(v[j]), 256.0f, -static_cast<float>(q * 32 + j)));
                }
            }
            tc_fence_before_sync();
            __syncwarp();
            if (lane == 0) mbar_arrive(bar_accempty + 8 * buf);
            const int ik = __float2int_rn(bk);
            const int dot = -((-ik) >> 8);   // ceil(ik / 256)
            const int j = 256 * dot - ik;     // 0..255
            const unsigned long long dist = static_cast<unsigned long long>((a.nbits - dot) >> 1);
            const unsigned long long cand = (dist << 32) | static_cast<unsigned long long>(rb * kTN + j);
            best = cand < best ? cand : best;
        }
        if (cur_tb >= 0) {
            const int64_t g = cur_tb * kTM + r;
            if (g < a.n_tgt && best != kNoKey) atomicMin(a.keys + g, best);
        }
    }

    tc_fence_before_sync();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after_sync();
        tmem_dealloc(tmem_base, 512);
    }
}

struct TcPlan {
    int32_t kpad;
    size_t keys_bytes, t_bytes, r_bytes;
};

void plan_tc(int64_t n_tgt, int64_t n_ref, int32_t nbits, TcPlan* p) {
    p->kpad = ((nbits + kChunk - 1) / kChunk) * kChunk;
    p->keys_bytes = ((static_cast<size_t>(n_tgt) * 8 + 255) / 256) * 256;
    p->t_bytes = ((static_cast<size_t>(n_tgt) * p->kpad + 255) / 256) * 256;
    p->r_bytes = ((static_cast<size_t>(n_ref) * p->kpad + 255) / 256) * 256;
}

}  // namespace
}  // namespace semshare

extern "C" size_t semshare_match_tc_workspace_size(int64_t n_tgt, int64_t n_ref, int32_t nbits) {
    using namespace semshare;
    if (n_tgt <= 0 || n_ref <= 0 || nbits < 32 || nbits > 256 || nbits % 32 != 0) return 0;
    TcPlan p;
    plan_tc(n_tgt, n_ref, nbits, &p);
    return p.keys_bytes + p.t_bytes + p.r_bytes;
}

extern "C" semshare_status semshare_match_tc(const uint32_t* tgt_codes, int64_t n_tgt, const uint32_t* ref_codes,
                                             int64_t n_ref, int32_t nbits, int32_t* idx, int32_t* dist,
                                             void* workspace, size_t workspace_bytes, uint32_t* err_flag,
                                             void* stream) {
    using namespace semshare;
    if (n_tgt < 0 || n_ref < 1) return SEMSHARE_EINVAL;
    if (nbits < 32 || nbits > 256 || nbits % 32 != 0) return SEMSHARE_EUNSUPPORTED;
    if (n_tgt >= (int64_t(1) << 31) || n_ref >= (int64_t(1) << 31)) return SEMSHARE_EUNSUPPORTED;
    if (n_tgt == 0) return SEMSHARE_OK;
    if (!tgt_codes || !ref_codes || !idx || !workspace) return SEMSHARE_EINVAL;
    if (!aligned(tgt_codes, 4) || !aligned(ref_codes, 4) || !aligned(idx, 4) || !aligned(workspace, 256) ||
        (dist && !aligned(dist, 4)) || (err_flag && !aligned(err_flag, 4)))
        return SEMSHARE_EINVAL;
    TcPlan plan;
    plan_tc(n_tgt, n_ref, nbits, &plan);
    if (workspace_bytes < plan.keys_bytes + plan.t_bytes + plan.r_bytes) return SEMSHARE_EINVAL;

    int sms = 0, dev = 0, smem_optin = 0;
    if (current_sm_count(&sms, &dev) != SEMSHARE_OK) return SEMSHARE_ECUDA;
    if (cudaDeviceGetAttribute(&smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess)
        return SEMSHARE_ECUDA;
    cudaStream_t s = as_stream(stream);
    auto* keys = static_cast<unsigned long long*>(workspace);
    uint8_t* tpm = static_cast<uint8_t*>(workspace) + plan.keys_bytes;
    uint8_t* rpm = tpm + plan.t_bytes;

    const int64_t pieces = (n_tgt + n_ref) * (plan.kpad / 16);
    const int64_t eg = (pieces + 255) / 256;
    expand_codes_kernel<<<static_cast<unsigned>(eg < sms * 8 ? eg : sms * 8), 256, 0, s>>>(
        tgt_codes, n_tgt, ref_codes, n_ref, nbits, plan.kpad, tpm, rpm, keys);
    if (launch_status() != SEMSHARE_OK) return SEMSHARE_ECUDA;

    TcArgs a{};
    a.n_tgt = n_tgt;
    a.n_ref = n_ref;
    a.n_rb = (n_ref + kTN - 1) / kTN;
    a.total = ((n_tgt + kTM - 1) / kTM) * a.n_rb;
    a.nbits = nbits;
    a.kchunks = plan.kpad / kChunk;
    a.a_bytes = static_cast<uint32_t>(kTM * plan.kpad);
    a.b_bytes = static_cast<uint32_t>(kTN * plan.kpad);
    a.keys = keys;
    a.err_flag = err_flag;
    a.wait_limit_ns = wait_limit_ns();
    const size_t smem = kFixedSmem + 2 * static_cast<size_t>(a.a_bytes) + 2 * static_cast<size_t>(a.b_bytes);
    if (smem > static_cast<size_t>(smem_optin)) return SEMSHARE_EUNSUPPORTED;

    CUtensorMap tm_t, tm_r;
    if (!encode_tma_2d(&tm_t, CU_TENSOR_MAP_DATA_TYPE_UINT8, tpm, static_cast<uint64_t>(plan.kpad),
                       static_cast<uint64_t>(n_tgt), static_cast<uint64_t>(plan.kpad), kChunk, kTM) ||
        !encode_tma_2d(&tm_r, CU_TENSOR_MAP_DATA_TYPE_UINT8, rpm, static_cast<uint64_t>(plan.kpad),
                       static_cast<uint64_t>(n_ref), static_cast<uint64_t>(plan.kpad), kChunk, kTN))
        return SEMSHARE_ECUDA;
    if (cudaFuncSetAttribute(hamming_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(smem)) != cudaSuccess)
        return SEMSHARE_ECUDA;
    const int64_t grid = a.total < sms ? a.total : sms;
    hamming_tc_kernel<<<static_cast<unsigned>(grid), kThreads, smem, s>>>(tm_t, tm_r, a);
    if (launch_status() != SEMSHARE_OK) return SEMSHARE_ECUDA;
    const int small = static_cast<int>((n_tgt + 255) / 256 < sms * 4 ? (n_tgt + 255) / 256 : sms * 4);
    tc_keys_split_kernel<<<small, 256, 0, s>>>(keys, n_tgt, idx, dist);
    return launch_status();
}
