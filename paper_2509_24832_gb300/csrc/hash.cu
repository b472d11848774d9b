// hash.cu -- semshare_hash: rotary position encoding fused into a random-hyperplane LSH
// projection on the tcgen05 tensor cores, with a sign-bit packing epilogue.
//
// What it computes (SemShareKV, arXiv 2509.24832): Sec. 3.3.1 applies RoPE (Eq. 1, App. A.1)
// to the E cache of both prompts, then Sec. 3.3 / App. A.2 hash the rotated rows with LSH.
// For row i at position m: y = RoPE(x_i, m) (pair (2k, 2k+1) turned by m * theta_k),
// p = R * bf16(y) with fp32 accumulation, code bit j = [p_j > 0].
//
// Work split (stream-K).  The n_tiles x n_kblocks (128-row tile, 64-wide K block) iterations
// are cut into one equal contiguous range per CTA, one persistent CTA per SM, so every SM does
// the same amount of rotation and MMA work even when there are fewer tiles than SMs.  A tile
// covered by one CTA is finished in place.  A tile shared by several CTAs is finished by the
// last of them to arrive: each writes its fp32 partial accumulator to its workspace slot,
// fences, and bumps the tile's counter; the CTA that sees the count complete adds the partials
// in K order (so the sum, and the codes, do not depend on arrival order), packs the signs and
// puts the counter back to zero.  Nobody waits for another CTA.  The hand-off of a CTA's last
// segment and every fix-up run after its main loop, shared by all 512 threads (the final
// partial is staged through the then idle pipeline buffers).
//
// Roles inside a CTA (512 threads):
//   warp 0        TMA producer: the 128 x 64 embedding block (bf16 in place, fp32 into a
//                 staging buffer) and the nbits x 64 hyperplane block, 128-byte swizzle; the
//                 embedding blocks are also prefetched into L2 two pipeline depths ahead
//   warp 1        TMEM allocator and MMA issuer: 4 x tcgen05.mma (M=128, N=nbits, K=16) per
//                 stage into one of two fp32 TMEM accumulators
//   warps 4-11    RoPE: rotate each staged pair in shared memory, round to bf16 in the operand
//                 tile, hand the stage to the MMA warp.  Two groups of four warps take alternate
//                 stages (interleaved pairing), so two stages are rotated at once; a group's next
//                 rotation table entries are fetched while the other group works.  A thread owns
//                 2 chunks (8 pairs) of 4 rows 32 apart: when their positions are 32 apart too,
//                 only the first row's angles go through sincos and the others step by the
//                 32-position rotation.  (Rotate-half pairing: all eight warps on every stage.)
//   warps 12-15   epilogue: tcgen05.ld of the accumulator (lane = row), sign bits packed into
//                 32-bit words, or the partial-sum hand-off of a shared tile
// Every pipeline wait is bounded; on timeout the CTA raises SEMSHARE_FLAG_TIMEOUT, lets its
// copies and MMAs in flight finish, frees TMEM and returns.
//
// Rotate-half pairing (semshare_hash_ex, SEMSHARE_ROPE_HALF): pair k is (k, k + d/2).  A stage
// then also loads the partner block (columns kb*64 +- d/2, the same 128-byte swizzled box) into
// its staging slot, and the RoPE warps write each of the stage's own 64 columns from its own
// value and its partner's: y = x*c - x_partner*s in the first half, x*c + x_partner*s in the
// second, at angle index (column mod d/2).  The hyperplane tiles and the MMA are unchanged.
#include <cuda.h>

#include <cstdlib>
#include <cstring>
#include <cudaTypedefs.h>
#include <cuda_bf16.h>

#include "common.cuh"
#include "hash_2sm.cuh"
#include "hash_common.cuh"
#include "ptx.cuh"
#include "tma_host.cuh"

namespace semshare {
namespace {

using namespace hashk;

constexpr int kBM = 128;                       // rows per tile (MMA M, one TMEM lane per row)
constexpr int kBK = 64;                        // K elements per stage: one 128-byte row of bf16
constexpr int kUmmaK = 16;                     // K of one tcgen05.mma kind::f16
constexpr int kRopeWarp0 = 4;
constexpr int kRopeWarps = 8;
// (row, 16-byte chunk) items of a stage per RoPE thread: rows rbase + 32*i, i < kRopeRows
constexpr int kRopeRows = kBM * (kBK * 2 / 16) / (kRopeWarps * 32);
static_assert(kRopeRows >= 1 && kRopeRows <= 4 && kRopeRows * kRopeWarps * 32 == kBM * (kBK * 2 / 16), "RoPE split");
// Interleaved pairing: the RoPE warps form kRopeGroups groups that rotate alternate stages; a
// thread of a group covers kRopeRows rows and kGroupChunks of the 8 chunks of each.
// Two groups measured fastest on GB300 (5k hash 47.3 us; one group 49.6, four 55.4).
constexpr int kRopeGroups = 2;
constexpr int kGroupThreads = kRopeWarps * 32 / kRopeGroups;
constexpr int kGroupChunks = kRopeGroups;
constexpr int kChunkStride = 8 / kGroupChunks;
constexpr int kRowsPerPhase = 8 / kChunkStride;  // rows in one 8-thread shared-memory phase
static_assert(kGroupThreads == kChunkStride * 32 && kRopeRows == 4, "grouped RoPE split: 32 row groups x chunks");
constexpr int kEpiWarp0 = kRopeWarp0 + kRopeWarps;  // a multiple of 4: epilogue warp w reads TMEM lanes 32*(w%4)
constexpr int kEpiWarps = 4;
constexpr int kThreads = (kEpiWarp0 + kEpiWarps) * 32;
static_assert(kEpiWarp0 % 4 == 0, "epilogue warps must start on a warpgroup");
constexpr uint32_t kABytes = kBM * kBK * 2;    // bf16 operand tile, 16 KB
constexpr uint32_t kF32Bytes = kBM * kBK * 4;  // fp32 staging: two 128-byte-wide boxes, 32 KB
constexpr int kEpiBarrier = 1;                 // named barrier of the epilogue warps
// alignment slack + barriers + TMEM slot + flags (+ the checked build's counters)
constexpr size_t kFixedSmem = 1024 + 512 + (kChecked ? 256 : 0);

struct HashArgs {
    int64_t n;
    int64_t total_iters;  // n_tiles * n_kblocks
    int32_t nbits;
    int32_t n_kblocks;
    int32_t n_tiles;
    int32_t is_f32;
    int32_t stages;
    int64_t pair_rows;  // semshare_hash_pair: n rounded up to a tile; logical tiles below it hash the rows
                        // as they are into codes, those above it (the same rows again) rotated into codes2
    uint32_t* codes2;
    uint32_t stage_bytes;
    uint32_t b_bytes;
    uint32_t tx_bytes;
    uint32_t tmem_cols;
    const int32_t* positions;
    const uint64_t* rope_table;
    uint32_t* codes;
    float* proj;
    uint8_t* signs;  // nullable: [n][signs_pitch] e4m3 +-1 bytes of the code bits, zero-padded
    int32_t signs_pitch;
    uint32_t* err_flag;
    uint32_t* tile_count;  // workspace: [n_tiles] arrivals of shared tiles, zero between calls
    float4* partials;      // workspace: [2 * gridDim.x][nbits/32][8][128] partial accumulators
    uint64_t wait_limit_ns;
};


// First source row of logical tile `tile`, whether its rows are rotated, and where its codes go.
template <int kRot>
__device__ __forceinline__ int64_t tile_src_row(const HashArgs& a, int64_t tile) {
    const int64_t r = tile * kBM;
    return (kRot == kRotPair && r >= a.pair_rows) ? r - a.pair_rows : r;
}
template <int kRot>
__device__ __forceinline__ bool tile_rotates(const HashArgs& a, int64_t tile) {
    return kRot == kRotAll || (kRot == kRotPair && tile * kBM >= a.pair_rows);
}
template <int kRot>
__device__ __forceinline__ uint32_t* tile_codes(const HashArgs& a, int64_t tile) {
    return (kRot == kRotPair && tile * kBM >= a.pair_rows) ? a.codes2 : a.codes;
}

// The K block holding the rotate-half partners of block kb's columns (d/2 = nkb/2 blocks away).
__device__ __forceinline__ int partner_kb(int kb, int nkb) { return kb < nkb / 2 ? kb + nkb / 2 : kb - nkb / 2; }

// Rotate-half outputs of one column from its own value and its partner's (the two lines of the
// pair rotation, with the operands in the order the column takes in the pair).
__device__ __forceinline__ float rotate_half_col(float own, float partner, float c, float s, bool first_half) {
    return first_half ? fmaf(own, c, -partner * s) : fmaf(partner, s, own * c);
}

__device__ __forceinline__ bool drain_wait(uint32_t bar, uint32_t parity, uint64_t limit_ns) {
    if (mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = global_timer_ns();
    while (!mbar_try_wait(bar, parity))
        if (global_timer_ns() - t0 > limit_ns) return false;
    return true;
}

__device__ __forceinline__ void epilogue_sync() {
    asm volatile("bar.sync %0, %1;" ::"n"(kEpiBarrier), "n"(kEpiWarps * 32) : "memory");
}

// AND of v over the epilogue warps (also a barrier among them): they continue or stop together,
// so none can be left waiting at the hand-off barrier.
__device__ __forceinline__ bool epilogue_all(bool v) {
    uint32_t r;
    asm volatile(
        "{\n\t.reg .pred p, q;\n\t"
        "setp.ne.u32 p, %1, 0;\n\t"
        "bar.red.and.pred q, %2, %3, p;\n\t"
        "selp.u32 %0, 1, 0, q;\n\t}\n"
        : "=r"(r)
        : "r"(static_cast<uint32_t>(v)), "n"(kEpiBarrier), "n"(kEpiWarps * 32)
        : "memory");
    return r != 0;
}

// Table entries of 8 consecutive angle indices j0 .. j0+7 (rotate-half pairing).
struct Pairs8 {
    uint64_t turns[8];
    uint64_t cis32[8];
};

__device__ __forceinline__ void load_pairs8(const uint64_t* table, int half, int j0, Pairs8& t) {
    const ulonglong2* tp = reinterpret_cast<const ulonglong2*>(table + j0);
    const ulonglong2* cp = reinterpret_cast<const ulonglong2*>(table + half + j0);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const ulonglong2 a = __ldg(tp + i), b = __ldg(cp + i);
        t.turns[2 * i] = a.x;
        t.turns[2 * i + 1] = a.y;
        t.cis32[2 * i] = b.x;
        t.cis32[2 * i + 1] = b.y;
    }
}

// Table entries of the 4 pairs (kb*32 + 4c .. +3): turn fractions, and the rotation between
// positions 32 apart (cos in the low word, sin in the high word).
struct Pairs4 {
    uint64_t turns[4];
    uint64_t cis32[4];
};

__device__ __forceinline__ void load_pairs4(const uint64_t* table, int half, int kb, int c, Pairs4& t) {
    const ulonglong2* tp = reinterpret_cast<const ulonglong2*>(table + kb * (kBK / 2) + c * 4);
    const ulonglong2* cp = reinterpret_cast<const ulonglong2*>(table + half + kb * (kBK / 2) + c * 4);
    const ulonglong2 t01 = __ldg(tp), t23 = __ldg(tp + 1), c01 = __ldg(cp), c23 = __ldg(cp + 1);
    t.turns[0] = t01.x; t.turns[1] = t01.y; t.turns[2] = t23.x; t.turns[3] = t23.y;
    t.cis32[0] = c01.x; t.cis32[1] = c01.y; t.cis32[2] = c23.x; t.cis32[3] = c23.y;
}

template <bool kHalf, int kRot>
__global__ void __launch_bounds__(kThreads, 1)
    lsh_hash_kernel(const __grid_constant__ CUtensorMap tmap_emb, const __grid_constant__ CUtensorMap tmap_hyp,
                    const HashArgs a) {
    // the next kernel is released at the end (below), as in hash_2sm.cu
    grid_dependency_wait();
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_addr(smem_raw);
    const uint32_t sbase = (raw + 1023u) & ~1023u;  // stage tiles on the swizzle-atom boundary
    uint8_t* const gbase = smem_raw + (sbase - raw);
    const uint32_t S = static_cast<uint32_t>(a.stages);
    const uint32_t bars = sbase + S * a.stage_bytes;
    const uint32_t bar_full = bars;                  // [S] TMA landed (count 1 + tx bytes)
    const uint32_t bar_ready = bars + 8u * S;        // [S] operand tile rotated (count: the warps of a stage)
    const uint32_t bar_empty = bars + 16u * S;       // [S] MMAs done with the stage (commit)
    const uint32_t bar_accfull = bars + 24u * S;     // [2] accumulator complete (commit)
    const uint32_t bar_accempty = bar_accfull + 16u; // [2] accumulator drained (count kEpiWarps)
    const uint32_t bar_mma_done = bar_accempty + 16u;
    const uint32_t tmem_slot = bar_mma_done + 8u;
    volatile uint32_t* const tmem_slot_ptr = reinterpret_cast<volatile uint32_t*>(gbase + (tmem_slot - sbase));
    volatile int* const abort_flag = reinterpret_cast<volatile int*>(gbase + (tmem_slot + 4u - sbase));
    // hand-off bookkeeping shared with the end phase: [0] final partial staged (0/1), [1] its tile,
    // [2] its slot, [3] b_lo, [4] b_hi, [5] fix-ups pending, [6 + 3f ..] tile, b_lo, b_hi of fix-up f
    volatile int64_t* const ctl = reinterpret_cast<volatile int64_t*>(gbase + (tmem_slot + 16u - sbase));
    // checked build: fills [0, 8) and rotations [8, 16) per ring slot, producer stages [16], MMA
    // stages [17], epilogue segments [18]
    volatile uint32_t* const chk = reinterpret_cast<volatile uint32_t*>(gbase + (bars + 512u - sbase));
    constexpr uint32_t kRopeArrivals = kHalf ? kRopeWarps : kRopeWarps / kRopeGroups;  // per stage

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const int64_t G = gridDim.x;
    const int64_t i0 = range_begin(blockIdx.x, a.total_iters, G);
    const int64_t i1 = range_begin(static_cast<int64_t>(blockIdx.x) + 1, a.total_iters, G);
    const int nkb = a.n_kblocks;

    if (threadIdx.x == 0) {
        for (uint32_t s = 0; s < S; ++s) {
            mbar_init(bar_full + 8u * s, 1);
            mbar_init(bar_ready + 8u * s, kHalf ? kRopeWarps : kRopeWarps / kRopeGroups);
            mbar_init(bar_empty + 8u * s, 1);
        }
        for (uint32_t b = 0; b < 2; ++b) {
            mbar_init(bar_accfull + 8u * b, 1);
            mbar_init(bar_accempty + 8u * b, kEpiWarps);
        }
        mbar_init(bar_mma_done, 1);
        *abort_flag = 0;
        ctl[0] = 0;
        ctl[5] = 0;
        if (kChecked)
            for (int i = 0; i < 32; ++i) chk[i] = 0u;
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
    if (threadIdx.x == 0) SEMSHARE_CHECK(tmem_base == 0u, a.err_flag, SEMSHARE_KERNEL_HASH);  // lane 0, column 0

    if (warp == 0) {
        // ---------------- TMA producer ----------------
        if (lane == 0) {
            uint32_t q = 0;
            bool ok = true;
            int tile = static_cast<int>(i0 / nkb), kb = static_cast<int>(i0 % nkb);
            // L2 prefetch of the embedding blocks, 2*S iterations ahead of the loads
            int pf_tile = tile, pf_kb = kb;
            int64_t pf_it = i0;
            auto prefetch_next = [&]() {
                if (pf_it >= i1) return;
                tma_prefetch_l2_2d(&tmap_emb, pf_kb * kBK, static_cast<int32_t>(tile_src_row<kRot>(a, pf_tile)));
                if (a.is_f32) tma_prefetch_l2_2d(&tmap_emb, pf_kb * kBK + 32, static_cast<int32_t>(tile_src_row<kRot>(a, pf_tile)));
                if (kHalf) tma_prefetch_l2_2d(&tmap_emb, partner_kb(pf_kb, nkb) * kBK, pf_tile * kBM);
                ++pf_it;
                if (++pf_kb == nkb) {
                    pf_kb = 0;
                    ++pf_tile;
                }
            };
            for (uint32_t i = 0; i < 2 * S; ++i) prefetch_next();
            for (int64_t it = i0; it < i1; ++it, ++q) {
                const uint32_t s = q % S, ph = (q / S) & 1u;
                if (!mbar_wait_bounded(bar_empty + 8u * s, ph ^ 1u, abort_flag, a.err_flag, SEMSHARE_FLAG_TIMEOUT,
                                       a.wait_limit_ns)) {
                    ok = false;
                    break;
                }
                if (kChecked) {
                    // every earlier fill of the slot was rotated by all its warps
                    SEMSHARE_CHECK(chk[8 + s] == kRopeArrivals * (q / S), a.err_flag, SEMSHARE_KERNEL_HASH);
                    chk[s] = chk[s] + 1u;
                }
                const uint32_t st = sbase + s * a.stage_bytes;
                const uint32_t full = bar_full + 8u * s;
                mbar_arrive_expect_tx(full, a.tx_bytes);
                if (a.is_f32) {
                    const uint32_t stg = st + kABytes + a.b_bytes;
                    tma_load_2d(stg, &tmap_emb, full, kb * kBK, static_cast<int32_t>(tile_src_row<kRot>(a, tile)));
                    tma_load_2d(stg + kF32Bytes / 2, &tmap_emb, full, kb * kBK + 32, static_cast<int32_t>(tile_src_row<kRot>(a, tile)));
                } else {
                    tma_load_2d(st, &tmap_emb, full, kb * kBK, static_cast<int32_t>(tile_src_row<kRot>(a, tile)));
                    if (kHalf) tma_load_2d(st + kABytes + a.b_bytes, &tmap_emb, full, partner_kb(kb, nkb) * kBK,
                                           tile * kBM);
                }
                tma_load_2d(st + kABytes, &tmap_hyp, full, kb * kBK, 0);
                prefetch_next();
                if (++kb == nkb) {
                    kb = 0;
                    ++tile;
                }
            }
            if (kChecked && ok) chk[16] = q;
            if (!ok) {
                // the last issue of every stage may still be landing: wait for it before exit
                for (uint32_t i = (q > S ? q - S : 0); i < q; ++i)
                    drain_wait(bar_full + 8u * (i % S), (i / S) & 1u, kWaitLimitNs);
            }
        }
        __syncwarp();
    } else if (warp == 1) {
        // ---------------- MMA issuer ----------------
        if (lane == 0) {
            const uint32_t idesc = umma_idesc_bf16_f32(kBM, a.nbits);
            uint32_t q = 0, acc = 0, d_tmem = 0;
            bool seg_first = true;
            int kb = static_cast<int>(i0 % nkb);
            for (int64_t it = i0; it < i1; ++it, ++q) {
                if (seg_first) {
                    const uint32_t buf = acc & 1u, aph = (acc >> 1) & 1u;
                    if (!mbar_wait_bounded(bar_accempty + 8u * buf, aph ^ 1u, abort_flag, a.err_flag,
                                           SEMSHARE_FLAG_TIMEOUT, a.wait_limit_ns))
                        break;
                    tc_fence_after_sync();
                    d_tmem = tmem_base + buf * (a.tmem_cols >> 1);
                }
                const uint32_t s = q % S, ph = (q / S) & 1u;
                if (!mbar_wait_bounded(bar_ready + 8u * s, ph, abort_flag, a.err_flag, SEMSHARE_FLAG_TIMEOUT,
                                       a.wait_limit_ns))
                    break;
                // the operand tile is this stage's: all its warps have rotated this fill of the slot
                SEMSHARE_CHECK(chk[8 + s] == kRopeArrivals * (q / S + 1u) && chk[s] == q / S + 1u, a.err_flag, SEMSHARE_KERNEL_HASH);
                tc_fence_after_sync();
                const uint32_t st = sbase + s * a.stage_bytes;
#pragma unroll
                for (int k = 0; k < kBK / kUmmaK; ++k) {
                    const uint64_t adesc = sw128_kmajor_desc(st + k * kUmmaK * 2);
                    const uint64_t bdesc = sw128_kmajor_desc(st + kABytes + k * kUmmaK * 2);
                    umma_bf16_ss(d_tmem, adesc, bdesc, idesc, (seg_first && k == 0) ? 0u : 1u);
                }
                umma_commit(bar_empty + 8u * s);
                const bool seg_last = (kb == nkb - 1) || (it == i1 - 1);
                if (seg_last) {
                    umma_commit(bar_accfull + 8u * (acc & 1u));
                    ++acc;
                }
                seg_first = seg_last;
                if (++kb == nkb) kb = 0;
            }
            if (kChecked) chk[17] = q;
            // every MMA issued above has finished once this arrives: TMEM may then be freed
            umma_commit(bar_mma_done);
            drain_wait(bar_mma_done, 0, kWaitLimitNs);
        }
        __syncwarp();
    } else if (kHalf && warp >= kRopeWarp0 && warp < kRopeWarp0 + kRopeWarps) {
        // ---------------- RoPE, rotate-half pairing ----------------
        // A thread owns the 8 columns of one 16-byte chunk (c) of 4 rows 32 apart; their partners
        // sit at the same place in the staged partner block.
        const int rt = threadIdx.x - kRopeWarp0 * 32;
        const int c = rt & 7;
        const int rg = (rt >> 3) & 31;
        const int rbase = rg + 32 * kRopeRows * (rt >> 8);  // rows rbase + 32*i, i < kRopeRows
        const uint32_t chunk_off = (static_cast<uint32_t>(c) ^ static_cast<uint32_t>(rg & 7)) << 4;
        const int hk = nkb / 2;
        const int half = nkb * (kBK / 2);
        uint32_t q = 0;
        int tile = static_cast<int>(i0 / nkb), kb = static_cast<int>(i0 % nkb), cur_tile = -1;
        uint32_t m[kRopeRows];
        bool steps32 = false;
        Pairs8 tn;
        load_pairs8(a.rope_table, half, (kb % hk) * kBK + 8 * c, tn);
        for (int64_t it = i0; it < i1; ++it, ++q) {
            if (tile != cur_tile) {
                cur_tile = tile;
                const int64_t r0 = static_cast<int64_t>(tile) * kBM + rbase;
                steps32 = true;
#pragma unroll
                for (int i = 0; i < kRopeRows; ++i) {
                    const int64_t row = r0 + 32 * i;
                    m[i] = row < a.n ? (a.positions ? static_cast<uint32_t>(__ldg(a.positions + row))
                                                    : static_cast<uint32_t>(row))
                                     : (i == 0 ? 0u : m[0] + 32u * i);
                    steps32 = steps32 && m[i] == m[0] + 32u * i;
                }
            }
            const Pairs8 tc = tn;
            const bool first_half = kb < hk;
            const int kb_next = kb + 1 == nkb ? 0 : kb + 1;
            if (it + 1 < i1) load_pairs8(a.rope_table, half, (kb_next % hk) * kBK + 8 * c, tn);

            const uint32_t s = q % S, ph = (q / S) & 1u;
            const bool got = mbar_wait_bounded(bar_full + 8u * s, ph, abort_flag, a.err_flag, SEMSHARE_FLAG_TIMEOUT,
                                               a.wait_limit_ns);
            if (!__all_sync(0xFFFFFFFFu, got)) break;
            if (kChecked && lane == 0) SEMSHARE_CHECK(chk[s] == q / S + 1u, a.err_flag, SEMSHARE_KERNEL_HASH);  // this stage's fill
            uint8_t* const st = gbase + s * a.stage_bytes;
            const uint8_t* const pt = st + kABytes + a.b_bytes;  // partner block
            float cs[8], sn[8];
            if (steps32) {
#pragma unroll
                for (int e = 0; e < 8; ++e) rotation(m[0], tc.turns[e], cs[e], sn[e]);
            }
#pragma unroll
            for (int i = 0; i < kRopeRows; ++i) {
                const uint32_t off = (rbase + 32 * i) * 128 + chunk_off;
                const uint4 vo = *reinterpret_cast<const uint4*>(st + off);
                const uint4 vp = *reinterpret_cast<const uint4*>(pt + off);
                const uint32_t wo[4] = {vo.x, vo.y, vo.z, vo.w}, wp[4] = {vp.x, vp.y, vp.z, vp.w};
                if (!steps32) {
#pragma unroll
                    for (int e = 0; e < 8; ++e) rotation(m[i], tc.turns[e], cs[e], sn[e]);
                }
                uint32_t y[4];
#pragma unroll
                for (int w = 0; w < 4; ++w) {
                    const float o0 = __uint_as_float(wo[w] << 16), o1 = __uint_as_float(wo[w] & 0xFFFF0000u);
                    const float p0 = __uint_as_float(wp[w] << 16), p1 = __uint_as_float(wp[w] & 0xFFFF0000u);
                    const float y0 = rotate_half_col(o0, p0, cs[2 * w], sn[2 * w], first_half);
                    const float y1 = rotate_half_col(o1, p1, cs[2 * w + 1], sn[2 * w + 1], first_half);
                    __nv_bfloat162 r = __floats2bfloat162_rn(y0, y1);
                    y[w] = *reinterpret_cast<uint32_t*>(&r);
                }
                *reinterpret_cast<uint4*>(st + off) = make_uint4(y[0], y[1], y[2], y[3]);
                if (steps32 && i < kRopeRows - 1) {
#pragma unroll
                    for (int e = 0; e < 8; ++e) {
                        const float c32 = __uint_as_float(static_cast<uint32_t>(tc.cis32[e]));
                        const float s32 = __uint_as_float(static_cast<uint32_t>(tc.cis32[e] >> 32));
                        const float nc = fmaf(cs[e], c32, -sn[e] * s32);
                        sn[e] = fmaf(cs[e], s32, sn[e] * c32);
                        cs[e] = nc;
                    }
                }
            }
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) {
                    if (kChecked) atomicAdd(const_cast<uint32_t*>(chk + 8 + s), 1u);
                    mbar_arrive(bar_ready + 8u * s);
                }
            kb = kb_next;
            if (kb == 0) ++tile;
        }
    } else if (!kHalf && warp >= kRopeWarp0 && warp < kRopeWarp0 + kRopeWarps) {
        // ---------------- RoPE (Eq. 1) on the staged tile ----------------
        // kRopeGroups groups take turns: group g rotates the stages q = g, g + G, ..., so G stages
        // are in flight at once and one group's chain of waits and latencies overlaps the others'.
        // A thread of a group owns kRopeRows rows 32 apart and kGroupChunks 16-byte chunks of them.
        const int rt = threadIdx.x - kRopeWarp0 * 32;
        const int g = rt / kGroupThreads;
        const int gt = rt - g * kGroupThreads;
        const int c0 = gt % kChunkStride;             // chunks c0 + kChunkStride*j: pairs 4c .. 4c+3
        // rows rbase + 32*i, i < kRopeRows.  The 8 threads of one 16-byte shared-memory access phase
        // take chunks c0 .. c0 + kChunkStride - 1 of kRowsPerPhase rows whose swizzle phases
        // (row & 7) differ by multiples of kChunkStride, so together they touch all 32 banks
        const int u = gt / kChunkStride;
        const int lowr = u % kRowsPerPhase, hir = u / kRowsPerPhase;
        const int rbase = (hir / kChunkStride) * 8 + (hir % kChunkStride) + lowr * kChunkStride;
        const uint32_t swz = static_cast<uint32_t>(rbase & 7);
        const int half = nkb * (kBK / 2);  // d/2: start of the 32-position rotations in the table
        uint32_t m[kRopeRows];
        bool steps32 = false, rot = true;
        int cur_tile = -1;
        Pairs4 tn[kGroupChunks];
        if (i0 + g < i1 && kRot != kRotNone) {
            const int kb = static_cast<int>((i0 + g) % nkb);
#pragma unroll
            for (int j = 0; j < kGroupChunks; ++j) load_pairs4(a.rope_table, half, kb, c0 + kChunkStride * j, tn[j]);
        }
        for (int64_t it = i0 + g; it < i1; it += kRopeGroups) {
            const uint32_t q = static_cast<uint32_t>(it - i0);
            const int tile = static_cast<int>(it / nkb);
            if (tile != cur_tile) {
                cur_tile = tile;
                rot = tile_rotates<kRot>(a, tile);
                const int64_t r0 = tile_src_row<kRot>(a, tile) + rbase;
                m[0] = r0 < a.n ? (a.positions ? static_cast<uint32_t>(__ldg(a.positions + r0)) : static_cast<uint32_t>(r0))
                                : 0u;
                steps32 = true;
#pragma unroll
                for (int i = 1; i < kRopeRows; ++i) {
                    // rows past n are zero-filled by TMA: any angle will do, keep the 32-step pattern
                    const int64_t row = r0 + 32 * i;
                    m[i] = row < a.n ? (a.positions ? static_cast<uint32_t>(__ldg(a.positions + row))
                                                    : static_cast<uint32_t>(row))
                                     : m[0] + 32u * i;
                    steps32 = steps32 && m[i] == m[0] + 32u * i;
                }
            }
            const uint32_t s = q % S, ph = (q / S) & 1u;
            const bool got = mbar_wait_bounded(bar_full + 8u * s, ph, abort_flag, a.err_flag, SEMSHARE_FLAG_TIMEOUT,
                                               a.wait_limit_ns);
            if (!__all_sync(0xFFFFFFFFu, got)) break;
            if (kChecked && lane == 0) SEMSHARE_CHECK(chk[s] == q / S + 1u, a.err_flag, SEMSHARE_KERNEL_HASH);  // this stage's fill
            uint8_t* const st = gbase + s * a.stage_bytes;
            if (kRot != kRotAll && !rot) {
                // rows hashed as they are: bf16 rows already are the MMA operand; fp32 rows are only
                // rounded to bf16 (the rotation at position 0, which is the identity)
                if (a.is_f32) {
#pragma unroll
                    for (int j = 0; j < kGroupChunks; ++j) {
                        const int c = c0 + kChunkStride * j;
                        const uint32_t chunk_off = (static_cast<uint32_t>(c) ^ swz) << 4;
                        const uint32_t cc = static_cast<uint32_t>((c & 3) * 2);
#pragma unroll
                        for (int i = 0; i < kRopeRows; ++i) {
                            const uint8_t* stg =
                                st + kABytes + a.b_bytes + (c >> 2) * (kF32Bytes / 2) + (rbase + 32 * i) * 128;
                            const float4 f0 = *reinterpret_cast<const float4*>(stg + ((cc ^ swz) << 4));
                            const float4 f1 = *reinterpret_cast<const float4*>(stg + (((cc + 1u) ^ swz) << 4));
                            const float xs[8] = {f0.x, f0.y, f0.z, f0.w, f1.x, f1.y, f1.z, f1.w};
                            uint32_t y[4];
#pragma unroll
                            for (int p = 0; p < 4; ++p) {
                                __nv_bfloat162 r = __floats2bfloat162_rn(xs[2 * p], xs[2 * p + 1]);
                                y[p] = *reinterpret_cast<uint32_t*>(&r);
                            }
                            *reinterpret_cast<uint4*>(st + (rbase + 32 * i) * 128 + chunk_off) =
                                make_uint4(y[0], y[1], y[2], y[3]);
                        }
                    }
                    fence_proxy_async_smem();
                }
                __syncwarp();
                if (lane == 0) {
                    if (kChecked) atomicAdd(const_cast<uint32_t*>(chk + 8 + s), 1u);
                    mbar_arrive(bar_ready + 8u * s);
                }
                // a pair call's range may go on into rotated tiles: this group's next stage needs its
                // table entries whichever kind of tile this one was
                if (kRot == kRotPair && it + kRopeGroups < i1) {
                    const int kb = static_cast<int>((it + kRopeGroups) % nkb);
#pragma unroll
                    for (int j = 0; j < kGroupChunks; ++j)
                        load_pairs4(a.rope_table, half, kb, c0 + kChunkStride * j, tn[j]);
                }
                continue;
            }
#pragma unroll
            for (int j = 0; j < kGroupChunks; ++j) {
                const int c = c0 + kChunkStride * j;
                const uint32_t chunk_off = (static_cast<uint32_t>(c) ^ swz) << 4;
                float x[kRopeRows][8];
                if (a.is_f32) {
                    const uint32_t cc = static_cast<uint32_t>((c & 3) * 2);
#pragma unroll
                    for (int i = 0; i < kRopeRows; ++i) {
                        const uint8_t* stg =
                            st + kABytes + a.b_bytes + (c >> 2) * (kF32Bytes / 2) + (rbase + 32 * i) * 128;
                        const float4 f0 = *reinterpret_cast<const float4*>(stg + ((cc ^ swz) << 4));
                        const float4 f1 = *reinterpret_cast<const float4*>(stg + (((cc + 1u) ^ swz) << 4));
                        x[i][0] = f0.x; x[i][1] = f0.y; x[i][2] = f0.z; x[i][3] = f0.w;
                        x[i][4] = f1.x; x[i][5] = f1.y; x[i][6] = f1.z; x[i][7] = f1.w;
                    }
                } else {
#pragma unroll
                    for (int i = 0; i < kRopeRows; ++i) {
                        const uint4 v = *reinterpret_cast<const uint4*>(st + (rbase + 32 * i) * 128 + chunk_off);
                        const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
                        for (int p = 0; p < 4; ++p) {
                            x[i][2 * p] = __uint_as_float(w[p] << 16);
                            x[i][2 * p + 1] = __uint_as_float(w[p] & 0xFFFF0000u);
                        }
                    }
                }
                const Pairs4& tc = tn[j];
                uint32_t y[kRopeRows][4];
                if (steps32) {
                    // row i+1 sits 32 positions after row i: turn the angle on by the 32-step rotation
                    float cs[4], sn[4];
#pragma unroll
                    for (int p = 0; p < 4; ++p) rotation(m[0], tc.turns[p], cs[p], sn[p]);
#pragma unroll
                    for (int i = 0; i < kRopeRows; ++i)
#pragma unroll
                        for (int p = 0; p < 4; ++p) {
                            y[i][p] = rotate_to_bf16(x[i][2 * p], x[i][2 * p + 1], cs[p], sn[p]);
                            if (i < kRopeRows - 1) {
                                const float c32 = __uint_as_float(static_cast<uint32_t>(tc.cis32[p]));
                                const float s32 = __uint_as_float(static_cast<uint32_t>(tc.cis32[p] >> 32));
                                const float nc = fmaf(cs[p], c32, -sn[p] * s32);
                                sn[p] = fmaf(cs[p], s32, sn[p] * c32);
                                cs[p] = nc;
                            }
                        }
                } else {
#pragma unroll
                    for (int i = 0; i < kRopeRows; ++i)
#pragma unroll
                        for (int p = 0; p < 4; ++p) {
                            float cs, sn;
                            rotation(m[i], tc.turns[p], cs, sn);
                            y[i][p] = rotate_to_bf16(x[i][2 * p], x[i][2 * p + 1], cs, sn);
                        }
                }
#pragma unroll
                for (int i = 0; i < kRopeRows; ++i)
                    *reinterpret_cast<uint4*>(st + (rbase + 32 * i) * 128 + chunk_off) =
                        make_uint4(y[i][0], y[i][1], y[i][2], y[i][3]);
            }
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) {
                    if (kChecked) atomicAdd(const_cast<uint32_t*>(chk + 8 + s), 1u);
                    mbar_arrive(bar_ready + 8u * s);
                }
            // this group's next stage: its table entries load while the other groups work
            if (it + kRopeGroups < i1 && kRot != kRotNone) {
                const int kb = static_cast<int>((it + kRopeGroups) % nkb);
#pragma unroll
                for (int j = 0; j < kGroupChunks; ++j)
                    load_pairs4(a.rope_table, half, kb, c0 + kChunkStride * j, tn[j]);
            }
        }
    } else if (warp >= kEpiWarp0) {
        // ---------------- epilogue: signs -> packed codes, or partial hand-off ----------------
        const int ew = warp - kEpiWarp0;
        const int r = ew * 32 + lane;  // row within the tile == TMEM lane
        const int W = a.nbits >> 5;
        uint32_t acc = 0;
        for (int64_t it = i0; it < i1; ++acc) {
            const int tile = static_cast<int>(it / nkb);
            const int kb_begin = static_cast<int>(it - static_cast<int64_t>(tile) * nkb);
            const int64_t seg_len = (i1 - it) < (nkb - kb_begin) ? (i1 - it) : (nkb - kb_begin);
            const bool whole = kb_begin == 0 && seg_len == nkb;
            const bool last_seg = it + seg_len == i1;
            const int64_t tile_it0 = static_cast<int64_t>(tile) * nkb;
            int64_t b_lo = 0, b_hi = 0;
            if (!whole) {  // contributors of this tile, worked out while its MMAs run
                b_lo = range_owner(tile_it0, a.total_iters, G);
                b_hi = range_owner(tile_it0 + nkb - 1, a.total_iters, G);
            }
            const uint32_t buf = acc & 1u, aph = (acc >> 1) & 1u;
            const bool got = mbar_wait_bounded(bar_accfull + 8u * buf, aph, abort_flag, a.err_flag,
                                               SEMSHARE_FLAG_TIMEOUT, a.wait_limit_ns);
            if (!epilogue_all(got)) break;
            if (kChecked && threadIdx.x == kEpiWarp0 * 32) chk[18] = chk[18] + 1u;
            tc_fence_after_sync();
            const int64_t row = tile_src_row<kRot>(a, tile) + r;
            uint32_t* const out_codes = tile_codes<kRot>(a, tile);
            const uint32_t taddr = tmem_base + (static_cast<uint32_t>(ew * 32) << 16) + buf * (a.tmem_cols >> 1);
            if (whole) {
                uint32_t words[8];
#pragma unroll
                for (int qq = 0; qq < 8; ++qq) {
                    words[qq] = 0u;
                    if (qq < W) {
                        uint32_t v[32];
                        tmem_load_32cols_sync(taddr + qq * 32, v);
                        words[qq] = sign_word(v);
                        if (a.proj != nullptr && row < a.n) store_proj(a.proj, row, a.nbits, qq, v);
                    }
                }
                tc_fence_before_sync();
                __syncwarp();
                if (lane == 0) mbar_arrive(bar_accempty + 8u * buf);
                if (row < a.n) {
                    store_codes(out_codes, row, W, words);
                    if (a.signs != nullptr) store_sign_row(a.signs, row, a.signs_pitch, W, words);
                }
            } else {
                // shared tile: this CTA's partial sum goes to its workspace slot.  The last segment's
                // is staged in the idle pipeline buffers and published by the whole CTA at the end.
                const int64_t slot = 2 * static_cast<int64_t>(blockIdx.x) + (i0 >= tile_it0 ? 0 : 1);
                float4* dst = last_seg ? reinterpret_cast<float4*>(gbase) : a.partials + slot * W * 8 * kBM;
#pragma unroll
                for (int qq = 0; qq < 8; ++qq) {
                    if (qq < W) {
                        uint32_t v[32];
                        tmem_load_32cols_sync(taddr + qq * 32, v);
#pragma unroll
                        for (int j = 0; j < 8; ++j)
                            dst[(qq * 8 + j) * kBM + r] =
                                make_float4(__uint_as_float(v[4 * j]), __uint_as_float(v[4 * j + 1]),
                                            __uint_as_float(v[4 * j + 2]), __uint_as_float(v[4 * j + 3]));
                    }
                }
                tc_fence_before_sync();
                __syncwarp();
                if (lane == 0) mbar_arrive(bar_accempty + 8u * buf);
                if (last_seg) {
                    if (threadIdx.x == kEpiWarp0 * 32) {
                        ctl[1] = tile;
                        ctl[2] = slot;
                        ctl[3] = b_lo;
                        ctl[4] = b_hi;
                        ctl[0] = 1;
                    }
                } else {
                    __threadfence();
                    epilogue_sync();
                    if (threadIdx.x == kEpiWarp0 * 32) {
                        if (atomicAdd(a.tile_count + tile, 1u) == static_cast<uint32_t>(b_hi - b_lo)) {
                            const int64_t f = ctl[5];
                            ctl[6 + 3 * f] = tile;
                            ctl[7 + 3 * f] = b_lo;
                            ctl[8 + 3 * f] = b_hi;
                            ctl[5] = f + 1;
                        }
                    }
                }
            }
            it += seg_len;
        }
    }

    tc_fence_before_sync();
    __syncthreads();
    if (kChecked && threadIdx.x == 0 && *abort_flag == 0) {
        // every role handled the whole range: i1 - i0 stages, one accumulator per K-block segment
        const uint32_t stages = static_cast<uint32_t>(i1 - i0);
        const uint32_t segs = i1 > i0 ? static_cast<uint32_t>((i1 - 1) / nkb - i0 / nkb + 1) : 0u;
        uint32_t rotated = 0;
        for (uint32_t q = 0; q < S; ++q) rotated += chk[8 + q];
        SEMSHARE_CHECK(chk[16] == stages && chk[17] == stages, a.err_flag, SEMSHARE_KERNEL_HASH);
        SEMSHARE_CHECK(rotated == kRopeArrivals * stages, a.err_flag, SEMSHARE_KERNEL_HASH);
        SEMSHARE_CHECK(chk[18] == segs, a.err_flag, SEMSHARE_KERNEL_HASH);
    }

    // ---------------- end phase: publish the final partial, finish the tiles this CTA closes ----
    if (*abort_flag == 0) {
        const int W = a.nbits >> 5;
        const int items = W * 8 * kBM;  // float4 per partial slot
        if (ctl[0]) {
            const float4* stage = reinterpret_cast<const float4*>(gbase);
            float4* dst = a.partials + ctl[2] * items;
            for (int e = threadIdx.x; e < items; e += kThreads) dst[e] = stage[e];
            __threadfence();
            __syncthreads();
            if (threadIdx.x == 0) {
                const int64_t tile = ctl[1];
                if (atomicAdd(a.tile_count + tile, 1u) == static_cast<uint32_t>(ctl[4] - ctl[3])) {
                    const int64_t f = ctl[5];
                    ctl[6 + 3 * f] = tile;
                    ctl[7 + 3 * f] = ctl[3];
                    ctl[8 + 3 * f] = ctl[4];
                    ctl[5] = f + 1;
                }
            }
            __syncthreads();
        }
        const int n_fix = static_cast<int>(ctl[5]);
        for (int f = 0; f < n_fix; ++f) {
            // every partial of the tile is in place: add them in K order (contributor order)
            __threadfence();
            const int tile = static_cast<int>(ctl[6 + 3 * f]);
            const int64_t b_lo = ctl[7 + 3 * f], b_hi = ctl[8 + 3 * f];
            const int64_t tile_it0 = static_cast<int64_t>(tile) * nkb;
            for (int e = threadIdx.x; e < W * kBM; e += kThreads) {
                const int qq = e / kBM, rr = e % kBM;
                float sum[32];
#pragma unroll
                for (int j = 0; j < 32; ++j) sum[j] = 0.0f;
                int64_t bb = b_lo;
                for (; bb + 1 <= b_hi; bb += 2) {  // two contributors' loads in flight at once
                    const int64_t s0 = 2 * bb + (range_begin(bb, a.total_iters, G) >= tile_it0 ? 0 : 1);
                    const int64_t s1 = 2 * (bb + 1) + (range_begin(bb + 1, a.total_iters, G) >= tile_it0 ? 0 : 1);
                    const float4* p0 = a.partials + s0 * items + qq * 8 * kBM + rr;
                    const float4* p1 = a.partials + s1 * items + qq * 8 * kBM + rr;
                    float4 f0[8], f1[8];
#pragma unroll
                    for (int j = 0; j < 8; ++j) {
                        f0[j] = __ldcg(p0 + j * kBM);
                        f1[j] = __ldcg(p1 + j * kBM);
                    }
#pragma unroll
                    for (int j = 0; j < 8; ++j) {
                        sum[4 * j] += f0[j].x;
                        sum[4 * j + 1] += f0[j].y;
                        sum[4 * j + 2] += f0[j].z;
                        sum[4 * j + 3] += f0[j].w;
                    }
#pragma unroll
                    for (int j = 0; j < 8; ++j) {
                        sum[4 * j] += f1[j].x;
                        sum[4 * j + 1] += f1[j].y;
                        sum[4 * j + 2] += f1[j].z;
                        sum[4 * j + 3] += f1[j].w;
                    }
                }
                if (bb <= b_hi) {
                    const int64_t s0 = 2 * bb + (range_begin(bb, a.total_iters, G) >= tile_it0 ? 0 : 1);
                    const float4* p0 = a.partials + s0 * items + qq * 8 * kBM + rr;
#pragma unroll
                    for (int j = 0; j < 8; ++j) {
                        const float4 f0 = __ldcg(p0 + j * kBM);
                        sum[4 * j] += f0.x;
                        sum[4 * j + 1] += f0.y;
                        sum[4 * j + 2] += f0.z;
                        sum[4 * j + 3] += f0.w;
                    }
                }
                uint32_t v[32];
#pragma unroll
                for (int j = 0; j < 32; ++j) v[j] = __float_as_uint(sum[j]);
                const int64_t row = tile_src_row<kRot>(a, tile) + rr;
                if (row < a.n) {
                    const uint32_t bits = sign_word(v);
                    tile_codes<kRot>(a, tile)[row * W + qq] = bits;
                    if (a.proj != nullptr) store_proj(a.proj, row, a.nbits, qq, v);
                    if (a.signs != nullptr) store_sign_bytes(a.signs + row * a.signs_pitch + 32 * qq, bits);
                }
            }
            if (a.signs != nullptr) {
                // the pad of the sign rows past the code bits
                const int pads = a.signs_pitch / 32 - W;
                for (int e = threadIdx.x; e < pads * kBM; e += kThreads) {
                    const int64_t row = tile_src_row<kRot>(a, tile) + e % kBM;
                    if (row < a.n) store_sign_pad(a.signs + row * a.signs_pitch + 32 * (W + e / kBM));
                }
            }
            if (threadIdx.x == 0) a.tile_count[tile] = 0u;  // leave the workspace zeroed
        }
    }

    __syncthreads();
    grid_dependents_launch();  // every CTA, at its end
    if (warp == 1) {
        tc_fence_after_sync();
        tmem_dealloc(tmem_base, a.tmem_cols);
    }
}

// Grid and workspace of one call: one CTA per SM (fewer if there are fewer iterations).
// Workspace layout: the partial-accumulator slots (two per CTA) first, in a region sized for
// the largest call on this device (one CTA per SM, 256-bit codes), then the per-tile counters.
// The counters therefore start at the same offset for every call on a device and never overlap
// the slots of any other call: the counters are the only part that must be zero on entry, the
// slots are written before they are read, and calls of different sizes can share a workspace.
struct HashPlan {
    int64_t n_tiles;
    int64_t total_iters;
    int grid;
    size_t partial_bytes;  // the slot region (fixed per device)
    size_t count_bytes;
};

constexpr int kMaxBits = 256;

semshare_status plan_hash(int64_t n, int32_t d, HashPlan* p) {
    int sms = 0;
    if (current_sm_count(&sms, nullptr) != SEMSHARE_OK) return SEMSHARE_ECUDA;
    p->n_tiles = (n + kBM - 1) / kBM;
    p->total_iters = p->n_tiles * (d / kBK);
    // SEMSHARE_HASH_CTAS (read per call, a test knob) lowers the number of CTAs, so that tests can
    // make a CTA's range cross from the plain into the rotated tiles of a pair call
    int ctas = sms;
    const char* e = getenv("SEMSHARE_HASH_CTAS");
    if (e != nullptr && *e != 0) {
        const long v = strtol(e, nullptr, 10);
        if (v >= 1 && v < sms) ctas = static_cast<int>(v);
    }
    p->grid = static_cast<int>(p->total_iters < ctas ? p->total_iters : ctas);
    p->partial_bytes = static_cast<size_t>(2) * sms * kBM * static_cast<size_t>(kMaxBits) * 4;
    // counters of 128-row tiles (this kernel) or of the two halves of 256-row pair tiles
    // (hash_2sm.cu): n_tiles + 4 words covers both, for single and pair calls
    p->count_bytes = (((static_cast<size_t>(p->n_tiles) + 4) * 4 + 255) / 256) * 256;
    return SEMSHARE_OK;
}

}  // namespace
}  // namespace semshare

extern "C" size_t semshare_hash_workspace_size(int64_t n, int32_t d, int32_t nbits) {
    using namespace semshare;
    if (n <= 0 || d < kBK || d % kBK != 0 || nbits < 32 || nbits > 256 || nbits % 32 != 0) return 0;
    HashPlan p;
    if (plan_hash(n, d, &p) != SEMSHARE_OK) return 0;
    return p.partial_bytes + p.count_bytes;
}

namespace semshare {
namespace {

// bf16 rows with the interleaved pairing (or none) run on SM pairs unless the call is small: below
// 8 stages (256-row pair tile x 64-wide K block) per SM pair the pair kernel's pipeline fill and end
// phase outweigh its faster stages (on GB300, 2048 rows x 4096: 27.3 us on pairs against 25.2 us on
// single SMs; 4096 rows: equal; 10240 rows: 41.6 against 47.7 us).  SEMSHARE_HASH_KERNEL=pair|one
// (read per call, a test knob) forces one of the two.
bool use_pair_kernel(int64_t rows, int32_t d) {
    const char* e = getenv("SEMSHARE_HASH_KERNEL");
    if (e != nullptr && strcmp(e, "pair") == 0) return true;
    if (e != nullptr && strcmp(e, "one") == 0) return false;
    int sms = 0;
    if (current_sm_count(&sms, nullptr) != SEMSHARE_OK) return true;
    const int64_t stages = ((rows + 255) / 256) * (d / kBK);
    return stages >= 4 * static_cast<int64_t>(sms);
}

// semshare_hash_ex, and with codes2 non-null semshare_hash_pair (the rows as they are into codes,
// rotated into codes2, in one launch over twice the tiles).
semshare_status hash_impl(const void* emb, semshare_dtype dtype, int64_t n, int32_t d, int64_t row_stride,
                          const int32_t* positions, const uint64_t* rope_table, const uint16_t* hyperplanes,
                          int32_t nbits, uint32_t rope_layout, uint32_t* codes, uint32_t* codes2, float* proj_out,
                          uint8_t* signs, void* workspace, size_t workspace_bytes, uint32_t* err_flag, void* stream) {
    const bool pair = codes2 != nullptr;
    if (dtype != SEMSHARE_BF16 && dtype != SEMSHARE_F32) return SEMSHARE_EINVAL;
    if (rope_layout != SEMSHARE_ROPE_INTERLEAVED && rope_layout != SEMSHARE_ROPE_HALF &&
        rope_layout != SEMSHARE_ROPE_NONE)
        return SEMSHARE_EINVAL;
    const bool half = rope_layout == SEMSHARE_ROPE_HALF;
    const bool none = rope_layout == SEMSHARE_ROPE_NONE;
    if (half && (dtype != SEMSHARE_BF16 || d % (2 * kBK) != 0)) return SEMSHARE_EUNSUPPORTED;
    if (n < 0 || d <= 0 || (d & 1) || row_stride < d) return SEMSHARE_EINVAL;
    if (d % kBK != 0 || d > 65536) return SEMSHARE_EUNSUPPORTED;
    if (nbits < 32 || nbits > 256 || nbits % 32 != 0) return SEMSHARE_EUNSUPPORTED;
    if (n >= (int64_t(1) << 31)) return SEMSHARE_EUNSUPPORTED;
    const int64_t esize = dtype == SEMSHARE_BF16 ? 2 : 4;
    if ((row_stride * esize) % 16 != 0) return SEMSHARE_EINVAL;
    if (n == 0) return SEMSHARE_OK;
    if (!emb || (!rope_table && !none) || !hyperplanes || !codes || !workspace) return SEMSHARE_EINVAL;
    if (!aligned(emb, 16) || (!none && !aligned(rope_table, 16)) || !aligned(hyperplanes, 16) || !aligned(codes, 16) ||
        !aligned(workspace, 256))
        return SEMSHARE_EINVAL;
    if ((proj_out && !aligned(proj_out, 16)) || (positions && !aligned(positions, 4)) ||
        (err_flag && !aligned(err_flag, 4)))
        return SEMSHARE_EINVAL;
    if (pair && (rope_layout != SEMSHARE_ROPE_INTERLEAVED || proj_out || signs || !aligned(codes2, 16)))
        return SEMSHARE_EINVAL;
    if (signs && !aligned(signs, 16)) return SEMSHARE_EINVAL;
    const int32_t signs_pitch = semshare_signs_pitch(nbits);
    const int64_t n_pad = ((n + kBM - 1) / kBM) * kBM;

    HashPlan plan;
    if (plan_hash(pair ? 2 * n_pad : n, d, &plan) != SEMSHARE_OK) return SEMSHARE_ECUDA;
    if (workspace_bytes < plan.partial_bytes + plan.count_bytes) return SEMSHARE_EINVAL;
    if (dtype == SEMSHARE_BF16 && !half && use_pair_kernel(pair ? 2 * n : n, d)) {
        // bf16 rows, interleaved pairing or none: the CTA-pair kernel (hash_2sm.cu)
        Hash2smCall c{};
        c.emb = emb;
        c.n = n;
        c.d = d;
        c.row_stride = row_stride;
        c.positions = none ? nullptr : positions;
        c.rope_table = rope_table;
        c.hyperplanes = hyperplanes;
        c.nbits = nbits;
        c.none = none;
        c.pair = pair;
        c.pair_rows = ((n + 255) / 256) * 256;
        c.codes = codes;
        c.codes2 = codes2;
        c.proj = proj_out;
        c.signs = signs;
        c.signs_pitch = signs_pitch;
        c.err_flag = err_flag;
        c.partials = workspace;
        c.partial_bytes = plan.partial_bytes;
        c.tile_count = reinterpret_cast<uint32_t*>(static_cast<uint8_t*>(workspace) + plan.partial_bytes);
        c.count_bytes = plan.count_bytes;
        c.stream = stream;
        return launch_hash_2sm(c);
    }
    int dev = 0, smem_optin = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess)
        return SEMSHARE_ECUDA;

    HashArgs a{};
    a.n = n;
    a.total_iters = plan.total_iters;
    a.nbits = nbits;
    a.n_kblocks = d / kBK;
    a.n_tiles = static_cast<int32_t>(plan.n_tiles);
    a.is_f32 = dtype == SEMSHARE_F32;
    a.b_bytes = static_cast<uint32_t>(nbits) * kBK * 2;
    // the staging slot after the hyperplane block: fp32 rows, or the rotate-half partner block
    a.stage_bytes = kABytes + a.b_bytes + (a.is_f32 ? kF32Bytes : (half ? kABytes : 0u));
    a.tx_bytes = (a.is_f32 ? kF32Bytes : kABytes) + a.b_bytes + (half ? kABytes : 0u);
    uint32_t cols = 32;
    while (cols < 2u * static_cast<uint32_t>(nbits)) cols <<= 1;
    a.tmem_cols = cols;
    const size_t fixed = kFixedSmem;
    int stages = static_cast<int>((static_cast<size_t>(smem_optin) - fixed) / a.stage_bytes);
    if (stages > 6) stages = 6;
    // Interleaved pairing: RoPE group g rotates the stages q = g (mod kRopeGroups), which sit in
    // slot q mod S.  With S a multiple of kRopeGroups every slot belongs to one group, so a group
    // never waits on a slot whose previous stage it has not seen land; otherwise it could wait
    // two phases ahead, where the full barrier's parity test cannot tell the phases apart.
    if (!half) stages -= stages % kRopeGroups;
    if (stages < 2) return SEMSHARE_EUNSUPPORTED;
    // the last segment's partial accumulator (128 x nbits fp32) is staged in the stage buffers
    if (static_cast<size_t>(stages) * a.stage_bytes < static_cast<size_t>(kBM) * nbits * 4) return SEMSHARE_EUNSUPPORTED;
    a.stages = stages;
    a.positions = none ? nullptr : positions;
    a.rope_table = rope_table;
    a.pair_rows = pair ? n_pad : 0;
    a.codes2 = codes2;
    a.codes = codes;
    a.proj = proj_out;
    a.signs = signs;
    a.signs_pitch = signs_pitch;
    a.err_flag = err_flag;
    a.partials = static_cast<float4*>(workspace);
    a.tile_count = reinterpret_cast<uint32_t*>(static_cast<uint8_t*>(workspace) + plan.partial_bytes);
    a.wait_limit_ns = wait_limit_ns();
    const size_t smem = fixed + static_cast<size_t>(stages) * a.stage_bytes;

    CUtensorMap tm_emb, tm_hyp;
    if (!encode_tma_2d(&tm_emb, a.is_f32 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, emb,
                   static_cast<uint64_t>(d), static_cast<uint64_t>(n), static_cast<uint64_t>(row_stride * esize),
                   a.is_f32 ? 32u : 64u, kBM))
        return SEMSHARE_ECUDA;
    if (!encode_tma_2d(&tm_hyp, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, hyperplanes, static_cast<uint64_t>(d),
                   static_cast<uint64_t>(nbits), static_cast<uint64_t>(d) * 2, 64u, static_cast<uint32_t>(nbits)))
        return SEMSHARE_ECUDA;

    auto kernel = half   ? lsh_hash_kernel<true, kRotAll>
                  : pair ? lsh_hash_kernel<false, kRotPair>
                  : none ? lsh_hash_kernel<false, kRotNone>
                         : lsh_hash_kernel<false, kRotAll>;
    if (cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem)) != cudaSuccess)
        return SEMSHARE_ECUDA;
    if (launch_pdl(kernel, dim3(plan.grid), dim3(kThreads), smem, as_stream(stream), tm_emb, tm_hyp, a) != cudaSuccess)
        return SEMSHARE_ECUDA;
    return launch_status();
}

}  // namespace
}  // namespace semshare

extern "C" semshare_status semshare_hash_ex(const void* emb, semshare_dtype dtype, int64_t n, int32_t d,
                                            int64_t row_stride, const int32_t* positions, const uint64_t* rope_table,
                                            const uint16_t* hyperplanes, int32_t nbits, uint32_t rope_layout,
                                            uint32_t* codes, float* proj_out, void* workspace,
                                            size_t workspace_bytes, uint32_t* err_flag, void* stream) {
    return semshare::hash_impl(emb, dtype, n, d, row_stride, positions, rope_table, hyperplanes, nbits, rope_layout,
                               codes, nullptr, proj_out, nullptr, workspace, workspace_bytes, err_flag, stream);
}

extern "C" int32_t semshare_signs_pitch(int32_t nbits) {
    if (nbits < 32 || nbits > 256 || nbits % 32 != 0) return 0;
    return ((nbits + 127) / 128) * 128;
}

extern "C" semshare_status semshare_hash_signs(const void* emb, semshare_dtype dtype, int64_t n, int32_t d,
                                               int64_t row_stride, const int32_t* positions,
                                               const uint64_t* rope_table, const uint16_t* hyperplanes, int32_t nbits,
                                               uint32_t rope_layout, uint32_t* codes, uint8_t* signs,
                                               float* proj_out, void* workspace, size_t workspace_bytes,
                                               uint32_t* err_flag, void* stream) {
    if (n > 0 && !signs) return SEMSHARE_EINVAL;
    return semshare::hash_impl(emb, dtype, n, d, row_stride, positions, rope_table, hyperplanes, nbits, rope_layout,
                               codes, nullptr, proj_out, signs, workspace, workspace_bytes, err_flag, stream);
}

extern "C" size_t semshare_hash_pair_workspace_size(int64_t n, int32_t d, int32_t nbits) {
    if (n <= 0) return 0;
    const int64_t n_pad = ((n + semshare::kBM - 1) / semshare::kBM) * semshare::kBM;
    return semshare_hash_workspace_size(2 * n_pad, d, nbits);
}

extern "C" semshare_status semshare_hash_pair(const void* emb, semshare_dtype dtype, int64_t n, int32_t d,
                                              int64_t row_stride, const int32_t* positions, const uint64_t* rope_table,
                                              const uint16_t* hyperplanes, int32_t nbits, uint32_t* codes_plain,
                                              uint32_t* codes_rotary, void* workspace, size_t workspace_bytes,
                                              uint32_t* err_flag, void* stream) {
    if (n > 0 && !codes_rotary) return SEMSHARE_EINVAL;
    if (n >= (int64_t(1) << 30)) return SEMSHARE_EUNSUPPORTED;  // twice the rows stay below 2^31
    return semshare::hash_impl(emb, dtype, n, d, row_stride, positions, rope_table, hyperplanes, nbits,
                               SEMSHARE_ROPE_INTERLEAVED, codes_plain, n > 0 ? codes_rotary : nullptr, nullptr,
                               nullptr, workspace, workspace_bytes, err_flag, stream);
}

extern "C" semshare_status semshare_hash(const void* emb, semshare_dtype dtype, int64_t n, int32_t d,
                                         int64_t row_stride, const int32_t* positions, const uint64_t* rope_table,
                                         const uint16_t* hyperplanes, int32_t nbits, uint32_t* codes,
                                         float* proj_out, void* workspace, size_t workspace_bytes,
                                         uint32_t* err_flag, void* stream) {
    return semshare_hash_ex(emb, dtype, n, d, row_stride, positions, rope_table, hyperplanes, nbits,
                            SEMSHARE_ROPE_INTERLEAVED, codes, proj_out, workspace, workspace_bytes, err_flag, stream);
}
