// hash.cu -- semshare_hash: rotary position encoding fused into a random-hyperplane LSH
// projection on the tcgen05 tensor cores, with a sign-bit packing epilogue.
//
// What it computes (SemShareKV, arXiv 2509.24832): Sec. 3.3.1 applies RoPE (Eq. 1, App. A.1)
// to the E cache of both prompts, then Sec. 3.3 / App. A.2 hash the rotated rows with LSH.
// For row i at position m: y = RoPE(x_i, m) (pair (2k, 2k+1) turned by m * theta_k),
// p = R * bf16(y) with fp32 accumulation, code bit j = [p_j > 0].
//
// Kernel design (one persistent CTA per SM, 128-row tiles, 512 threads):
//   warp 0        TMA producer: the tile's 128 x 64 embedding block (bf16 in place, or fp32
//                 into a staging buffer) and the nbits x 64 hyperplane block, 128-byte swizzle
//   warp 1        TMEM allocator and MMA issuer: 4 x tcgen05.mma (M=128, N=nbits, K=16) per
//                 stage into one of two fp32 TMEM accumulators
//   warps 4-11    RoPE: rotate each staged pair in shared memory, round to bf16 in the
//                 operand tile, then hand the stage to the MMA warp
//   warps 12-15   epilogue: tcgen05.ld of the accumulator (lane = row), sign bits packed into
//                 32-bit words per 32 columns, coalesced stores of codes (and projections)
// Every pipeline wait is bounded; on timeout the CTA raises SEMSHARE_FLAG_TIMEOUT, lets its
// copies and MMAs in flight finish, frees TMEM and returns.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_bf16.h>

#include "common.cuh"
#include "ptx.cuh"

namespace semshare {
namespace {

constexpr int kBM = 128;                       // rows per tile (MMA M, one TMEM lane per row)
constexpr int kBK = 64;                        // K elements per stage: one 128-byte row of bf16
constexpr int kUmmaK = 16;                     // K of one tcgen05.mma kind::f16
constexpr int kThreads = 512;
constexpr int kRopeWarp0 = 4;
constexpr int kRopeWarps = 8;
constexpr int kEpiWarp0 = 12;                  // 12 % 4 == 0: epilogue warp w reads TMEM lanes 32*(w%4)
constexpr int kEpiWarps = 4;
constexpr uint32_t kABytes = kBM * kBK * 2;    // bf16 operand tile, 16 KB
constexpr uint32_t kF32Bytes = kBM * kBK * 4;  // fp32 staging: two 128-byte-wide boxes, 32 KB

struct HashArgs {
    int64_t n;
    int32_t nbits;
    int32_t n_kblocks;
    int32_t n_tiles;
    int32_t is_f32;
    int32_t stages;
    uint32_t stage_bytes;
    uint32_t b_bytes;
    uint32_t tx_bytes;
    uint32_t tmem_cols;
    const int32_t* positions;
    const uint64_t* rope_table;
    uint32_t* codes;
    float* proj;
    uint32_t* err_flag;
    uint64_t wait_limit_ns;
};

// cos and sin of the rotation angle m * theta_k (Eq. 1).  turns_q64 = theta_k/(2*pi) as a
// 0.64 fixed-point fraction, so bits 32..63 of m * turns_q64 (mod 2^64) are the angle's
// fraction of a full turn: the reduction modulo 2*pi is exact integer arithmetic for every
// int32 position.  The fraction, centred on [-1/2, 1/2) and rounded to 23 bits, becomes a
// float through the mantissa (a wrap from +1/2 to -1/2 is the same angle).
__device__ __forceinline__ void rotation(uint32_t m, uint64_t turns_q64, float& c, float& s) {
    const uint32_t lo = static_cast<uint32_t>(turns_q64);
    const uint32_t hi = static_cast<uint32_t>(turns_q64 >> 32);
    const uint32_t frac = __umulhi(m, lo) + m * hi;
    const float t = __uint_as_float(0x3F800000u | ((frac + 0x80000100u) >> 9)) - 1.5f;
    __sincosf(t * 6.28318530717958647692f, &s, &c);
}

// (x0, x1) turned counter-clockwise by the angle with cosine c and sine s, rounded to a bf16
// pair (x0 in the low half, the lower address).
__device__ __forceinline__ uint32_t rotate_to_bf16(float x0, float x1, float c, float s) {
    const float y0 = fmaf(x0, c, -x1 * s);
    const float y1 = fmaf(x0, s, x1 * c);
    __nv_bfloat162 r = __floats2bfloat162_rn(y0, y1);
    return *reinterpret_cast<uint32_t*>(&r);
}

__device__ __forceinline__ bool drain_wait(uint32_t bar, uint32_t parity, uint64_t limit_ns) {
    if (mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = global_timer_ns();
    while (!mbar_try_wait(bar, parity))
        if (global_timer_ns() - t0 > limit_ns) return false;
    return true;
}

__global__ void __launch_bounds__(kThreads, 1)
    lsh_hash_kernel(const __grid_constant__ CUtensorMap tmap_emb, const __grid_constant__ CUtensorMap tmap_hyp,
                    const HashArgs a) {
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_addr(smem_raw);
    const uint32_t sbase = (raw + 1023u) & ~1023u;  // stage tiles on the swizzle-atom boundary
    uint8_t* const gbase = smem_raw + (sbase - raw);
    const uint32_t S = static_cast<uint32_t>(a.stages);
    const uint32_t bars = sbase + S * a.stage_bytes;
    const uint32_t bar_full = bars;                  // [S] TMA landed (count 1 + tx bytes)
    const uint32_t bar_ready = bars + 8u * S;        // [S] operand tile rotated (count kRopeWarps)
    const uint32_t bar_empty = bars + 16u * S;       // [S] MMAs done with the stage (commit)
    const uint32_t bar_accfull = bars + 24u * S;     // [2] accumulator complete (commit)
    const uint32_t bar_accempty = bar_accfull + 16u; // [2] accumulator drained (count kEpiWarps)
    const uint32_t bar_mma_done = bar_accempty + 16u;
    const uint32_t tmem_slot = bar_mma_done + 8u;
    volatile uint32_t* const tmem_slot_ptr = reinterpret_cast<volatile uint32_t*>(gbase + (tmem_slot - sbase));
    volatile int* const abort_flag = reinterpret_cast<volatile int*>(gbase + (tmem_slot + 4u - sbase));

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (uint32_t s = 0; s < S; ++s) {
            mbar_init(bar_full + 8u * s, 1);
            mbar_init(bar_ready + 8u * s, kRopeWarps);
            mbar_init(bar_empty + 8u * s, 1);
        }
        for (uint32_t b = 0; b < 2; ++b) {
            mbar_init(bar_accfull + 8u * b, 1);
            mbar_init(bar_accempty + 8u * b, kEpiWarps);
        }
        mbar_init(bar_mma_done, 1);
        *abort_flag = 0;
        fence_barrier_init();
    }
    if (warp == 0 && lane == 0) {
        tma_prefetch_desc(&tmap_emb);
        tma_prefetch_desc(&tmap_hyp);
    }
    if (warp == 1) {
        tmem_alloc(tmem_slot, a.tmem_cols);
        tmem_relinquish();
    }
    tc_fence_before_sync();
    __syncthreads();
    tc_fence_after_sync();
    const uint32_t tmem_base = *tmem_slot_ptr;

    if (warp == 0) {
        // ---------------- TMA producer ----------------
        if (lane == 0) {
            uint32_t it = 0;
            bool ok = true;
            for (int tile = blockIdx.x; ok && tile < a.n_tiles; tile += gridDim.x) {
                const int32_t row0 = tile * kBM;
                for (int kb = 0; kb < a.n_kblocks; ++kb, ++it) {
                    const uint32_t s = it % S, ph = (it / S) & 1u;
                    if (!mbar_wait_bounded(bar_empty + 8u * s, ph ^ 1u, abort_flag, a.err_flag, SEMSHARE_FLAG_TIMEOUT,
                                           a.wait_limit_ns)) {
                        ok = false;
                        break;
                    }
                    const uint32_t st = sbase + s * a.stage_bytes;
                    const uint32_t full = bar_full + 8u * s;
                    mbar_arrive_expect_tx(full, a.tx_bytes);
                    if (a.is_f32) {
                        const uint32_t stg = st + kABytes + a.b_bytes;
                        tma_load_2d(stg, &tmap_emb, full, kb * kBK, row0);
                        tma_load_2d(stg + kF32Bytes / 2, &tmap_emb, full, kb * kBK + 32, row0);
                    } else {
                        tma_load_2d(st, &tmap_emb, full, kb * kBK, row0);
                    }
                    tma_load_2d(st + kABytes, &tmap_hyp, full, kb * kBK, 0);
                }
            }
            if (!ok) {
                // the last issue of every stage may still be landing: wait for it before exit
                for (uint32_t i = (it > S ? it - S : 0); i < it; ++i)
                    drain_wait(bar_full + 8u * (i % S), (i / S) & 1u, kWaitLimitNs);
            }
        }
        __syncwarp();
    } else if (warp == 1) {
        // ---------------- MMA issuer ----------------
        if (lane == 0) {
            const uint32_t idesc = umma_idesc_bf16_f32(kBM, a.nbits);
            uint32_t it = 0, acc = 0;
            bool ok = true;
            for (int tile = blockIdx.x; ok && tile < a.n_tiles; tile += gridDim.x, ++acc) {
                const uint32_t buf = acc & 1u, aph = (acc >> 1) & 1u;
                if (!mbar_wait_bounded(bar_accempty + 8u * buf, aph ^ 1u, abort_flag, a.err_flag,
                                       SEMSHARE_FLAG_TIMEOUT, a.wait_limit_ns)) {
                    ok = false;
                    break;
                }
                tc_fence_after_sync();
                const uint32_t d_tmem = tmem_base + buf * (a.tmem_cols >> 1);
                for (int kb = 0; kb < a.n_kblocks; ++kb, ++it) {
                    const uint32_t s = it % S, ph = (it / S) & 1u;
                    if (!mbar_wait_bounded(bar_ready + 8u * s, ph, abort_flag, a.err_flag, SEMSHARE_FLAG_TIMEOUT,
                                           a.wait_limit_ns)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after_sync();
                    const uint32_t st = sbase + s * a.stage_bytes;
#pragma unroll
                    for (int k = 0; k < kBK / kUmmaK; ++k) {
                        const uint64_t adesc = sw128_kmajor_desc(st + k * kUmmaK * 2);
                        const uint64_t bdesc = sw128_kmajor_desc(st + kABytes + k * kUmmaK * 2);
                        umma_bf16_ss(d_tmem, adesc, bdesc, idesc, (kb | k) != 0 ? 1u : 0u);
                    }
                    umma_commit(bar_empty + 8u * s);
                }
                if (ok) umma_commit(bar_accfull + 8u * buf);
            }
            // every MMA issued above has finished once this arrives: TMEM may then be freed
            umma_commit(bar_mma_done);
            drain_wait(bar_mma_done, 0, kWaitLimitNs);
        }
        __syncwarp();
    } else if (warp >= kRopeWarp0 && warp < kRopeWarp0 + kRopeWarps) {
        // ---------------- RoPE (Eq. 1) on the staged tile ----------------
        const int rt = threadIdx.x - kRopeWarp0 * 32;  // 0..255
        const int c = rt & 7;                          // 16-byte chunk of the 128-byte row: pairs 4c..4c+3
        const int rg = rt >> 3;                        // rows rg + 32*i, i < 4 (all with row & 7 == rg & 7)
        const uint32_t swz = static_cast<uint32_t>(rg & 7);
        uint32_t it = 0;
        bool ok = true;
        for (int tile = blockIdx.x; ok && tile < a.n_tiles; tile += gridDim.x) {
            const int64_t row0 = static_cast<int64_t>(tile) * kBM;
            uint32_t m[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const int64_t row = row0 + rg + 32 * i;
                m[i] = row < a.n ? (a.positions ? static_cast<uint32_t>(__ldg(a.positions + row))
                                                : static_cast<uint32_t>(row))
                                 : 0u;
            }
            for (int kb = 0; kb < a.n_kblocks; ++kb, ++it) {
                const uint32_t s = it % S, ph = (it / S) & 1u;
                const bool got = mbar_wait_bounded(bar_full + 8u * s, ph, abort_flag, a.err_flag,
                                                   SEMSHARE_FLAG_TIMEOUT, a.wait_limit_ns);
                if (!__all_sync(0xFFFFFFFFu, got)) {
                    ok = false;
                    break;
                }
                const ulonglong2* tp = reinterpret_cast<const ulonglong2*>(a.rope_table + kb * (kBK / 2) + c * 4);
                const ulonglong2 t01 = __ldg(tp), t23 = __ldg(tp + 1);
                const uint64_t T[4] = {t01.x, t01.y, t23.x, t23.y};
                uint8_t* const st = gbase + s * a.stage_bytes;
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const int r = rg + 32 * i;
                    uint4* const dst = reinterpret_cast<uint4*>(st + r * 128 + ((static_cast<uint32_t>(c) ^ swz) << 4));
                    float x[8];
                    if (a.is_f32) {
                        const uint8_t* stg = st + kABytes + a.b_bytes + (c >> 2) * (kF32Bytes / 2) + r * 128;
                        const uint32_t c0 = static_cast<uint32_t>((c & 3) * 2);
                        const float4 f0 = *reinterpret_cast<const float4*>(stg + ((c0 ^ swz) << 4));
                        const float4 f1 = *reinterpret_cast<const float4*>(stg + (((c0 + 1u) ^ swz) << 4));
                        x[0] = f0.x; x[1] = f0.y; x[2] = f0.z; x[3] = f0.w;
                        x[4] = f1.x; x[5] = f1.y; x[6] = f1.z; x[7] = f1.w;
                    } else {
                        const uint4 v = *dst;
                        const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
                        for (int q = 0; q < 4; ++q) {
                            x[2 * q] = __uint_as_float(w[q] << 16);
                            x[2 * q + 1] = __uint_as_float(w[q] & 0xFFFF0000u);
                        }
                    }
                    uint32_t y[4];
#pragma unroll
                    for (int q = 0; q < 4; ++q) {
                        float cs, sn;
                        rotation(m[i], T[q], cs, sn);
                        y[q] = rotate_to_bf16(x[2 * q], x[2 * q + 1], cs, sn);
                    }
                    *dst = make_uint4(y[0], y[1], y[2], y[3]);
                }
                fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0) mbar_arrive(bar_ready + 8u * s);
            }
        }
    } else if (warp >= kEpiWarp0) {
        // ---------------- epilogue: signs -> packed codes ----------------
        const int ew = warp - kEpiWarp0;
        const int W = a.nbits >> 5;
        uint32_t acc = 0;
        for (int tile = blockIdx.x; tile < a.n_tiles; tile += gridDim.x, ++acc) {
            const uint32_t buf = acc & 1u, aph = (acc >> 1) & 1u;
            const bool got = mbar_wait_bounded(bar_accfull + 8u * buf, aph, abort_flag, a.err_flag,
                                               SEMSHARE_FLAG_TIMEOUT, a.wait_limit_ns);
            if (!__all_sync(0xFFFFFFFFu, got)) break;
            tc_fence_after_sync();
            const int64_t row = static_cast<int64_t>(tile) * kBM + ew * 32 + lane;
            const uint32_t taddr =
                tmem_base + (static_cast<uint32_t>(ew * 32) << 16) + buf * (a.tmem_cols >> 1);
            uint32_t words[8];
#pragma unroll
            for (int q = 0; q < 8; ++q) {
                words[q] = 0u;
                if (q < W) {
                    uint32_t v[32];
                    tmem_load_32cols(taddr + q * 32, v);
                    tmem_load_wait();
                    uint32_t bits = 0u;
#pragma unroll
                    for (int j = 0; j < 32; ++j) bits |= (static_cast<int32_t>(v[j]) > 0 ? 1u : 0u) << j;
                    words[q] = bits;
                    if (a.proj != nullptr && row < a.n) {
                        float4* pp = reinterpret_cast<float4*>(a.proj + row * a.nbits + q * 32);
#pragma unroll
                        for (int j = 0; j < 8; ++j)
                            pp[j] = make_float4(__uint_as_float(v[4 * j]), __uint_as_float(v[4 * j + 1]),
                                                __uint_as_float(v[4 * j + 2]), __uint_as_float(v[4 * j + 3]));
                    }
                }
            }
            tc_fence_before_sync();
            __syncwarp();
            if (lane == 0) mbar_arrive(bar_accempty + 8u * buf);
            if (row < a.n) {
                uint32_t* cp = a.codes + row * W;
                if ((W & 3) == 0) {
#pragma unroll
                    for (int q = 0; q < 8; q += 4)
                        if (q < W) *reinterpret_cast<uint4*>(cp + q) = make_uint4(words[q], words[q + 1], words[q + 2], words[q + 3]);
                } else {
#pragma unroll
                    for (int q = 0; q < 8; ++q)
                        if (q < W) cp[q] = words[q];
                }
            }
        }
    }

    tc_fence_before_sync();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after_sync();
        tmem_dealloc(tmem_base, a.tmem_cols);
    }
}

PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;  // resolved once per process
    if (fn == nullptr) {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q = cudaDriverEntryPointSymbolNotFound;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    }
    return fn;
}

bool encode_2d(CUtensorMap* map, CUtensorMapDataType type, const void* base, uint64_t inner, uint64_t outer,
               uint64_t row_bytes, uint32_t box_inner, uint32_t box_outer) {
    PFN_cuTensorMapEncodeTiled_v12000 enc = tensor_map_encoder();
    if (enc == nullptr) return false;
    const cuuint64_t dims[2] = {inner, outer};
    const cuuint64_t strides[1] = {row_bytes};
    const cuuint32_t box[2] = {box_inner, box_outer};
    const cuuint32_t estr[2] = {1, 1};
    return enc(map, type, 2, const_cast<void*>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
               CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace
}  // namespace semshare

extern "C" semshare_status semshare_hash(const void* emb, semshare_dtype dtype, int64_t n, int32_t d,
                                         int64_t row_stride, const int32_t* positions, const uint64_t* rope_table,
                                         const uint16_t* hyperplanes, int32_t nbits, uint32_t* codes,
                                         float* proj_out, uint32_t* err_flag, void* stream) {
    using namespace semshare;
    if (dtype != SEMSHARE_BF16 && dtype != SEMSHARE_F32) return SEMSHARE_EINVAL;
    if (n < 0 || d <= 0 || (d & 1) || row_stride < d) return SEMSHARE_EINVAL;
    if (d % kBK != 0 || d > 65536) return SEMSHARE_EUNSUPPORTED;
    if (nbits < 32 || nbits > 256 || nbits % 32 != 0) return SEMSHARE_EUNSUPPORTED;
    if (n >= (int64_t(1) << 31)) return SEMSHARE_EUNSUPPORTED;
    const int64_t esize = dtype == SEMSHARE_BF16 ? 2 : 4;
    if ((row_stride * esize) % 16 != 0) return SEMSHARE_EINVAL;
    if (n == 0) return SEMSHARE_OK;
    if (!emb || !rope_table || !hyperplanes || !codes) return SEMSHARE_EINVAL;
    if (!aligned(emb, 16) || !aligned(rope_table, 16) || !aligned(hyperplanes, 16) || !aligned(codes, 16))
        return SEMSHARE_EINVAL;
    if ((proj_out && !aligned(proj_out, 16)) || (positions && !aligned(positions, 4)) ||
        (err_flag && !aligned(err_flag, 4)))
        return SEMSHARE_EINVAL;

    int sms = 0, dev = 0;
    if (current_sm_count(&sms, &dev) != SEMSHARE_OK) return SEMSHARE_ECUDA;
    int smem_optin = 0;
    if (cudaDeviceGetAttribute(&smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess)
        return SEMSHARE_ECUDA;

    HashArgs a{};
    a.n = n;
    a.nbits = nbits;
    a.n_kblocks = d / kBK;
    a.n_tiles = static_cast<int32_t>((n + kBM - 1) / kBM);
    a.is_f32 = dtype == SEMSHARE_F32;
    a.b_bytes = static_cast<uint32_t>(nbits) * kBK * 2;
    a.stage_bytes = kABytes + a.b_bytes + (a.is_f32 ? kF32Bytes : 0u);
    a.tx_bytes = (a.is_f32 ? kF32Bytes : kABytes) + a.b_bytes;
    uint32_t cols = 32;
    while (cols < 2u * static_cast<uint32_t>(nbits)) cols <<= 1;
    a.tmem_cols = cols;
    const size_t fixed = 1024 + 256;  // alignment slack + barriers + TMEM slot + abort flag
    int stages = static_cast<int>((static_cast<size_t>(smem_optin) - fixed) / a.stage_bytes);
    if (stages > 6) stages = 6;
    if (stages < 2) return SEMSHARE_EUNSUPPORTED;
    a.stages = stages;
    a.positions = positions;
    a.rope_table = rope_table;
    a.codes = codes;
    a.proj = proj_out;
    a.err_flag = err_flag;
    a.wait_limit_ns = kWaitLimitNs;
    const size_t smem = fixed + static_cast<size_t>(stages) * a.stage_bytes;

    CUtensorMap tm_emb, tm_hyp;
    if (!encode_2d(&tm_emb, a.is_f32 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, emb,
                   static_cast<uint64_t>(d), static_cast<uint64_t>(n), static_cast<uint64_t>(row_stride * esize),
                   a.is_f32 ? 32u : 64u, kBM))
        return SEMSHARE_ECUDA;
    if (!encode_2d(&tm_hyp, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, hyperplanes, static_cast<uint64_t>(d),
                   static_cast<uint64_t>(nbits), static_cast<uint64_t>(d) * 2, 64u, static_cast<uint32_t>(nbits)))
        return SEMSHARE_ECUDA;

    if (cudaFuncSetAttribute(lsh_hash_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem)) !=
        cudaSuccess)
        return SEMSHARE_ECUDA;
    const int grid = a.n_tiles < sms ? a.n_tiles : sms;
    lsh_hash_kernel<<<grid, kThreads, smem, as_stream(stream)>>>(tm_emb, tm_hyp, a);
    return launch_status();
}
