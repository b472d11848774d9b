// hash_2sm.cu -- semshare_hash for bf16 rows on pairs of SMs: rotary position encoding written
// into tensor memory, the random-hyperplane projection as tcgen05.mma.cta_group::2, sign packing.
//
// What it computes is what hash.cu's kernel computes (SemShareKV, arXiv 2509.24832: Sec. 3.3.1
// and Eq. 1 rotate every row of the E cache, Sec. 3.3 and App. A.2 hash it with LSH): for row i
// at position m, y = bf16(RoPE(x_i, m)) with pair (2k, 2k+1) turned by m * theta_k, then
// p = R * y in fp32 and code bit j = [p_j > 0].
//
// Why a second kernel.  In the one-SM kernel a 64-wide K stage of a 128-row tile moves ~128 KB
// through shared memory (the TMA writes of the embedding and hyperplane blocks, the rotation's
// reads and writes, the MMA's operand reads) against 512 cycles of tensor work.  Here:
//   * two CTAs on two SMs (a cluster) share one M = 256 MMA: each holds its own 128 rows and
//     half of the hyperplane block (nbits/2 rows), so each SM loads and feeds half the
//     hyperplanes per stage;
//   * the RoPE warps read the raw rows from shared memory and write the rotated bf16 rows
//     straight into tensor memory (tcgen05.st), where the MMA reads its A operand: no
//     shared-memory write-back, no proxy fence.
// A stage then moves 64 KB through each SM's shared memory (16 KB embedding block in, its 16 KB
// read by the RoPE warps, 16 KB of hyperplanes in, their 16 KB read by the MMA).
//
// Work split (stream-K over pair tiles).  The n_ptiles x n_kblocks (256-row pair tile, 64-wide
// K block) iterations are cut into one equal contiguous range per cluster; both CTAs of a
// cluster walk the same range, each on its 128-row half.  A tile shared by several clusters is
// closed by the cluster that owns its first K blocks: every later contributor publishes the fp32
// partial of its half and counts it; the closer waits (bounded) for the count, adds the partials
// to its own accumulator in K order and packs the signs.  All clusters are resident at once (the
// grid is the occupancy figure), so that wait depends only on work already running.
//
// Rotation layout.  A RoPE thread owns 4 rows 32 apart and 8 bf16 pairs of each (the .16x256b
// tensor-memory store gives a thread lanes 8 apart and two adjacent columns of every 8-column
// group).  TMEM lane L = 32q + 8j + i of a CTA holds tile row 8q + phi(i) + 32j, phi(i) = 2i
// for i < 4, 2(i-4)+1 otherwise: a thread's rows are 32 positions apart (only the first goes
// through sincos, the others step by the 32-position rotation), and the 16 threads of each half
// warp read 16 different 8-byte bank slots of the 128-byte-swizzled rows (no bank conflict).
// The epilogue reads the accumulator lane by lane with the same map.
//
// Roles of each CTA (512 threads):
//   warp 0       TMA producer of its 128 rows x 64 of the embedding block; the first two
//                blocks are requested before the pair's set-up barrier, and the ring fills
//                behind them at most two blocks ahead of the last one that has landed
//   warp 2       TMA producer of its half of the hyperplane block
//   warp 1       TMEM allocation (both CTAs); MMA issue (even CTA): 4 x tcgen05.mma per stage,
//                commits multicast to both CTAs' barriers
//   warps 4-11   RoPE, two groups of four warps on alternate stages
//   warps 12-15  epilogue: accumulator lanes -> sign bits, or the partial hand-off
// Every wait is bounded; a CTA that gives up raises its own and its peer's abort flag, lets its
// copies and MMAs in flight finish and frees tensor memory after the pair has met at a cluster
// barrier.
#include <cuda.h>
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

constexpr int kPM = 256;                    // rows of a pair tile: M of one cta_group::2 MMA
constexpr int kCM = 128;                    // rows of each CTA's half, one TMEM lane each
constexpr int kBK = 64;                     // K elements per stage: one 128-byte row of bf16
constexpr int kUmmaK = 16;                  // K of one tcgen05.mma kind::f16
static_assert(kBK / kUmmaK == 4, "the MMA loop issues four instructions per stage");
constexpr int kRopeWarp0 = 4;
constexpr int kRopeGroups = 2;              // groups of four warps (one per TMEM lane quadrant)
constexpr int kEpiWarp0 = kRopeWarp0 + 4 * kRopeGroups;
constexpr int kEpiWarps = 4;
constexpr int kThreads = (kEpiWarp0 + kEpiWarps) * 32;
static_assert(kEpiWarp0 % 4 == 0 && kRopeWarp0 % 4 == 0, "warp w reaches TMEM lanes 32*(w%4)..+31");
constexpr uint32_t kABytes = kCM * kBK * 2;  // one CTA's raw embedding block, 16 KB
constexpr uint32_t kAccCols = 256;           // accumulator columns (nbits <= 256), from column 0
constexpr uint32_t kAStageCols = kBK / 2;    // TMEM columns of one stage's A operand (2 bf16 each)
constexpr uint32_t kTmemCols = 512;
constexpr int kBSlots = 4;                   // hyperplane halves and TMEM operand slots in flight
constexpr int kMaxASlots = 10;               // raw embedding blocks in flight
// Embedding blocks requested while the ring first fills: at most this many beyond the last block
// that has landed.  Every SM starts at once on a cold L2 full of dirty lines (the previous work's
// writes); requesting the whole ring at once makes the first block wait for the others, and the
// first stage is on the critical path.
constexpr uint32_t kRampLoads = 2;
constexpr int kRopeBarrier = 2;              // named barrier of the RoPE warps
constexpr uint32_t kMaxTableSmem = 32768;    // rotation tables up to d = 4096 are staged in shared memory
static_assert(kAccCols + kBSlots * kAStageCols <= kTmemCols, "TMEM budget");
static_assert(kBSlots % 2 == 0, "each TMEM operand slot belongs to one RoPE group");
constexpr int kEpiBarrier = 1;
constexpr size_t kFixedSmem = 1024 + 512;    // alignment slack + barriers, TMEM slot, flags, control
constexpr int kMaxBits = 256;

struct Hash2smArgs {
    int64_t n;
    int64_t total_iters;  // n_ptiles * n_kblocks
    int64_t pair_rows;    // kRotPair: pair tiles at rows >= pair_rows rotate rows (row - pair_rows)
    int32_t nbits;
    int32_t n_kblocks;
    int32_t n_ptiles;
    int32_t a_slots;      // raw embedding ring (freed by the RoPE warps once they have read a block)
    int32_t b_slots;      // hyperplane ring and TMEM operand ring (freed by the MMAs)
    uint32_t bh_bytes;    // one CTA's half hyperplane block: nbits/2 rows of 128 bytes
    uint32_t table_bytes; // the rotation table staged in shared memory (d * 8 bytes), or 0: read from L2
    const int32_t* positions;
    const uint64_t* rope_table;
    uint32_t* codes;
    uint32_t* codes2;
    float* proj;
    uint8_t* signs;       // nullable: [n][signs_pitch] e4m3 +-1 bytes of the code bits, zero-padded
    int32_t signs_pitch;
    uint32_t* err_flag;
    uint32_t* tile_count;  // workspace: [2 * n_ptiles] arrivals at each CTA half of a shared pair tile
    float4* partials;      // workspace: [2 per CTA][nbits/32 * 8][128] partial accumulators
    uint64_t wait_limit_ns;
};

template <int kRot>
__device__ __forceinline__ int64_t ptile_src_row(const Hash2smArgs& a, int64_t tile) {
    const int64_t r = tile * kPM;
    return (kRot == kRotPair && r >= a.pair_rows) ? r - a.pair_rows : r;
}
template <int kRot>
__device__ __forceinline__ bool ptile_rotates(const Hash2smArgs& a, int64_t tile) {
    return kRot == kRotAll || (kRot == kRotPair && tile * kPM >= a.pair_rows);
}
template <int kRot>
__device__ __forceinline__ uint32_t* ptile_codes(const Hash2smArgs& a, int64_t tile) {
    return (kRot == kRotPair && tile * kPM >= a.pair_rows) ? a.codes2 : a.codes;
}

// Workspace slot of cluster b's partial of CTA half `rank`.  The workspace plan has two slots per
// CTA; this kernel uses the first only: a cluster publishes a partial only for a segment that
// starts its range inside a tile (the tile's first K block belongs to an earlier cluster, its
// closer), so every partial of a shared tile comes from a different cluster.
__device__ __forceinline__ int64_t partial_slot(int64_t b, uint32_t rank) { return 2 * (2 * b + rank); }

// phi: the rows of one half warp's threads fall on swizzle phases 0,2,4,6 and 1,3,5,7.
__device__ __forceinline__ int row_phase(int i) { return i < 4 ? 2 * i : 2 * i - 7; }

// Row (of the CTA's 128) held in TMEM lane L.
__device__ __forceinline__ int lane_row(int L) {
    return 8 * (L >> 5) + row_phase(L & 7) + 32 * ((L >> 3) & 3);
}

// Bounded wait for barriers that the peer CTA or the pair's MMAs arrive on.  Gives up when this
// CTA's abort flag is up or after limit_ns; in the second case it raises this CTA's flag and the
// peer's (so the peer stops waiting for work that will not come) and records the timeout.
__device__ __forceinline__ bool pair_wait(uint32_t bar, uint32_t parity, volatile int* abort_flag, uint32_t peer_abort,
                                          uint32_t* err, uint64_t limit_ns) {
    if (mbar_try_wait_cluster(bar, parity)) return true;
    const uint64_t t0 = global_timer_ns();
    for (;;) {
        if (*abort_flag) return false;
        if (global_timer_ns() - t0 > limit_ns) {
            *abort_flag = 1;
            st_shared_cluster_u32(peer_abort, 1u);
            if (err) atomicOr(err, SEMSHARE_FLAG_TIMEOUT);
            return false;
        }
        if (mbar_try_wait_cluster_sleep(bar, parity, 20000u)) return true;
    }
}

// Waits (bounded, ignoring the abort flag) for a phase that is certain to complete: copies and
// MMAs already issued.
__device__ __forceinline__ void settle_wait(uint32_t bar, uint32_t parity) {
    if (mbar_try_wait_cluster(bar, parity)) return;
    const uint64_t t0 = global_timer_ns();
    while (!mbar_try_wait_cluster_sleep(bar, parity, 20000u))
        if (global_timer_ns() - t0 > kWaitLimitNs) return;
}

__device__ __forceinline__ void epilogue_sync() {
    asm volatile("bar.sync %0, %1;" ::"n"(kEpiBarrier), "n"(kEpiWarps * 32) : "memory");
}

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

// Arrive on a barrier of the even CTA: locally there, remotely from the odd CTA.  What the
// barrier's waiter consumes was written by tcgen05 instructions that the arriving warp has
// already waited for and fenced (tcgen05.wait + tcgen05.fence::before_thread_sync), so the arrive
// needs no cluster-scope release (which costs a memory barrier per stage).
__device__ __forceinline__ void arrive_lead(uint32_t local_bar, uint32_t lead_addr, bool leader) {
    if (leader)
        mbar_arrive(local_bar);
    else
        mbar_arrive_remote(lead_addr);
}

// Poll (bounded) until *count reaches want; one thread.  The contributors fence their partials
// before they count.
__device__ __forceinline__ bool count_wait(const uint32_t* count, uint32_t want, volatile int* abort_flag,
                                           uint32_t peer_abort, uint32_t* err, uint64_t limit_ns) {
    if (ld_acquire_gpu(count) >= want) return true;
    const uint64_t t0 = global_timer_ns();
    for (;;) {
        if (*abort_flag) return false;
        if (global_timer_ns() - t0 > limit_ns) {
            *abort_flag = 1;
            st_shared_cluster_u32(peer_abort, 1u);
            if (err) atomicOr(err, SEMSHARE_FLAG_TIMEOUT);
            return false;
        }
        __nanosleep(64);
        if (ld_acquire_gpu(count) >= want) return true;
    }
}

__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

template <int kRot>
__global__ void __launch_bounds__(kThreads, 1)
    lsh_hash_2sm_kernel(const __grid_constant__ CUtensorMap tmap_emb, const __grid_constant__ CUtensorMap tmap_hyp,
                        const Hash2smArgs a) {
    // The next kernel is released at the end (below), not here: released at the start, its CTAs
    // queued behind this grid for its whole run and the batched step (135 K rows, then the match
    // and the gather) measured 3.04 ms against 2.91 ms.
    grid_dependency_wait();
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_addr(smem_raw);
    const uint32_t sbase = (raw + 1023u) & ~1023u;  // stage tiles on the swizzle-atom boundary
    uint8_t* const gbase = smem_raw + (sbase - raw);
    const uint32_t SA = static_cast<uint32_t>(a.a_slots);
    const uint32_t SB = static_cast<uint32_t>(a.b_slots);
    const uint32_t a_ring = sbase;                     // [SA] raw 128 x 64 embedding blocks
    const uint32_t b_ring = sbase + SA * kABytes;      // [SB] half hyperplane blocks
    const uint32_t table_s = b_ring + SB * a.bh_bytes;  // the rotation table (when staged)
    const uint32_t bars = table_s + a.table_bytes;
    const uint32_t bar_afull = bars;                   // [SA] embedding block landed (count 1 + tx bytes)
    const uint32_t bar_aempty = bar_afull + 8u * SA;   // [SA] the RoPE group has read it (4 warps)
    const uint32_t bar_bfull = bar_aempty + 8u * SA;   // [SB] hyperplane half landed (count 1 + tx bytes)
    const uint32_t bar_done = bar_bfull + 8u * SB;     // [SB] the pair's MMAs of the stage finished (commit):
                                                       //      frees the hyperplane slot and the TMEM operand slot
    const uint32_t bar_ready = bar_done + 8u * SB;     // [SB] even CTA: both CTAs' rotated rows in TMEM and
                                                       //      their hyperplane halves landed (8 warps)
    const uint32_t bar_accfull = bar_ready + 8u * SB;  // accumulator complete (commit)
    const uint32_t bar_accempty = bar_accfull + 8u;    // even CTA: both CTAs drained the accumulator
    const uint32_t bar_mma_done = bar_accempty + 8u;   // even CTA: every MMA finished
    const uint32_t tmem_slot = bar_mma_done + 8u;
    const uint32_t abort_addr = tmem_slot + 4u;
    volatile uint32_t* const tmem_slot_ptr = reinterpret_cast<volatile uint32_t*>(gbase + (tmem_slot - sbase));
    volatile int* const abort_flag = reinterpret_cast<volatile int*>(gbase + (abort_addr - sbase));
    // the CTA's last segment when it is part of a shared tile, finished by all warps after the
    // main loop: [0] 0 none, 1 publish this half's partial, 2 close the half; [1] pair tile,
    // [2] b_lo, [3] b_hi
    volatile int64_t* const defer = reinterpret_cast<volatile int64_t*>(gbase + (tmem_slot + 8u - sbase));
    // checked build: the bookkeeping counters (fills and releases per ring slot, stages and
    // segments per role), in the fixed region after the barriers
    volatile uint32_t* const chk = reinterpret_cast<volatile uint32_t*>(gbase + (tmem_slot + 64u - sbase));
    constexpr int kChkAFill = 0, kChkARel = 10, kChkBFill = 20, kChkProdA = 24, kChkProdB = 25, kChkMma = 26,
                  kChkRope = 27, kChkMmaSeg = 28, kChkEpiSeg = 29;

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const uint32_t rank = cluster_ctarank();
    const bool leader = rank == 0;
    const int64_t P = cluster_count_x();
    const int64_t pid = cluster_id_x();
    const int64_t i0 = range_begin(pid, a.total_iters, P);
    const int64_t i1 = range_begin(pid + 1, a.total_iters, P);
    const int nkb = a.n_kblocks;
    const uint32_t ready_lead = mapa_shared(bar_ready, 0);
    const uint32_t accempty_lead = mapa_shared(bar_accempty, 0);
    const uint32_t peer_abort = mapa_shared(abort_addr, rank ^ 1u);

    if (threadIdx.x == 0) {
        for (uint32_t i = 0; i < SA; ++i) {
            mbar_init(bar_afull + 8u * i, 1);
            mbar_init(bar_aempty + 8u * i, 4);  // the four RoPE warps of the stage's group
        }
        for (uint32_t i = 0; i < SB; ++i) {
            mbar_init(bar_bfull + 8u * i, 1);
            mbar_init(bar_done + 8u * i, 1);
            mbar_init(bar_ready + 8u * i, 2 * 4);  // four RoPE warps of one group, in each CTA
        }
        mbar_init(bar_accfull, 1);
        mbar_init(bar_accempty, 2 * kEpiWarps);
        mbar_init(bar_mma_done, 1);
        *abort_flag = 0;
        defer[0] = 0;
        if (kChecked)
            for (int i = 0; i < 32; ++i) chk[i] = 0u;
        fence_barrier_init();
    }
    // the first embedding blocks are requested now: this CTA's own ring and barriers, so they
    // need nothing from the peer (the producer loop below continues after them)
    const uint32_t n_early = static_cast<uint32_t>((i1 - i0) < static_cast<int64_t>(kRampLoads) ? (i1 - i0) : kRampLoads);
    auto issue_a = [&](int64_t tile, int kb, uint32_t slot) {
        const uint32_t full = bar_afull + 8u * slot;
        mbar_arrive_expect_tx(full, kABytes);
        tma_load_2d(a_ring + slot * kABytes, &tmap_emb, full, kb * kBK,
                    static_cast<int32_t>(ptile_src_row<kRot>(a, tile)) + static_cast<int32_t>(rank) * kCM);
    };
    if (warp == 0 && lane == 0) {
        tma_prefetch_desc(&tmap_emb);
        tma_prefetch_desc(&tmap_hyp);
        for (uint32_t q = 0; q < n_early; ++q) {
            if (kChecked) chk[kChkAFill + q] = chk[kChkAFill + q] + 1u;
            issue_a((i0 + q) / nkb, static_cast<int>((i0 + q) % nkb), q);
        }
    }
    if (warp == 1) {
        tmem_alloc_pair(tmem_slot, kTmemCols);
        tmem_relinquish_pair();
    }
    tc_fence_before_sync();
    cluster_sync_all();  // both CTAs' barriers exist before any remote arrive or multicast commit
    tc_fence_after_sync();
    const uint32_t tmem_base = *tmem_slot_ptr;
    if (threadIdx.x == 0) SEMSHARE_CHECK(tmem_base == 0u, a.err_flag, SEMSHARE_KERNEL_HASH_2SM);  // lane 0, column 0

    if (warp == 0) {
        // ---------------- TMA producer of the embedding blocks (both CTAs) ----------------
        if (lane == 0) {
            // stage q = n_early on (the first blocks went out before the set-up barrier); its slot
            // and phase parity are kept incrementally (no divisions)
            uint32_t q = n_early;
            uint32_t s = n_early, ph = 0;  // n_early < SA
            int64_t tile = (i0 + n_early) / nkb;
            int kb = static_cast<int>((i0 + n_early) % nkb);
            for (int64_t it = i0 + n_early; it < i1; ++it, ++q) {
                if (q < SA) {
                    // the ring's first fill: ramp behind the blocks that have landed
                    if (q >= kRampLoads &&
                        !pair_wait(bar_afull + 8u * (q - kRampLoads), 0u, abort_flag, peer_abort, a.err_flag, a.wait_limit_ns))
                        break;
                } else if (!pair_wait(bar_aempty + 8u * s, ph ^ 1u, abort_flag, peer_abort, a.err_flag, a.wait_limit_ns)) {
                    break;
                }
                if (kChecked) {
                    // the slot's four RoPE warps released every earlier fill of it
                    SEMSHARE_CHECK(chk[kChkARel + s] == 4u * (q / SA), a.err_flag, SEMSHARE_KERNEL_HASH_2SM);
                    chk[kChkAFill + s] = chk[kChkAFill + s] + 1u;
                }
                issue_a(tile, kb, s);
                if (++kb == nkb) {
                    kb = 0;
                    ++tile;
                }
                if (++s == SA) {
                    s = 0;
                    ph ^= 1u;
                }
            }
            if (kChecked) chk[kChkProdA] = q;
            // the copies issued last may still be landing
            for (uint32_t i = (q > SA ? q - SA : 0); i < q; ++i) settle_wait(bar_afull + 8u * (i % SA), (i / SA) & 1u);
        }
        __syncwarp();
    } else if (warp == 2) {
        // ---------------- TMA producer of the hyperplane halves (both CTAs) ----------------
        if (lane == 0) {
            uint32_t q = 0;
            bool ok = true;
            int kb = static_cast<int>(i0 % nkb);
            const int32_t hyp_row = static_cast<int32_t>(rank) * (a.nbits / 2);
            uint32_t s = 0, ph = 0;
            for (int64_t it = i0; it < i1; ++it, ++q) {
                if (!pair_wait(bar_done + 8u * s, ph ^ 1u, abort_flag, peer_abort, a.err_flag, a.wait_limit_ns)) {
                    ok = false;
                    break;
                }
                if (kChecked) chk[kChkBFill + s] = chk[kChkBFill + s] + 1u;
                const uint32_t full = bar_bfull + 8u * s;
                mbar_arrive_expect_tx(full, a.bh_bytes);
                tma_load_2d(b_ring + s * a.bh_bytes, &tmap_hyp, full, kb * kBK, hyp_row);
                if (++kb == nkb) kb = 0;
                if (++s == SB) {
                    s = 0;
                    ph ^= 1u;
                }
            }
            if (kChecked) chk[kChkProdB] = q;
            for (uint32_t i = (q > SB ? q - SB : 0); i < q; ++i) settle_wait(bar_bfull + 8u * (i % SB), (i / SB) & 1u);
            if (ok) {
                // the pair's MMAs on the last stages may still be running: their commits arrive on
                // this CTA's barriers, so wait for them before the CTA moves on
                for (uint32_t i = (q > SB ? q - SB : 0); i < q; ++i)
                    if (!pair_wait(bar_done + 8u * (i % SB), (i / SB) & 1u, abort_flag, peer_abort, a.err_flag,
                                   a.wait_limit_ns))
                        break;
            }
        }
        __syncwarp();
    } else if (warp == 1) {
        // ---------------- MMA issuer (even CTA) ----------------
        if (leader && lane == 0) {
            // Slot addresses and descriptors advance by constant strides and wrap with the ring.
            const uint32_t idesc = umma_idesc_bf16_f32(kPM, a.nbits);
            const uint64_t bdesc0 = sw128_kmajor_desc(b_ring);
            const uint64_t bstride = a.bh_bytes >> 4;  // descriptor start address is in 16-byte units
            uint64_t bd = bdesc0;
            uint32_t a_tmem = tmem_base + kAccCols, bar_s = 0, s = 0, ph = 0, acc = 0;
            bool seg_first = true;
            int kb = static_cast<int>(i0 % nkb);
            uint32_t n_st = 0, n_seg = 0;  // checked build: stages and segments issued
            for (int64_t it = i0; it < i1; ++it) {
                if (seg_first) {
                    if (!pair_wait(bar_accempty, (acc & 1u) ^ 1u, abort_flag, peer_abort, a.err_flag, a.wait_limit_ns))
                        break;
                    tc_fence_after_sync();
                }
                if (!pair_wait(bar_ready + bar_s, ph, abort_flag, peer_abort, a.err_flag, a.wait_limit_ns)) break;
                tc_fence_after_sync();
                // K = 16 per instruction: 8 TMEM columns of A, 32 bytes (2 descriptor units) of B
                umma_bf16_ts_pair(tmem_base, a_tmem, bd, idesc, seg_first ? 0u : 1u);
                umma_bf16_ts_pair(tmem_base, a_tmem + 8, bd + 2, idesc, 1u);
                umma_bf16_ts_pair(tmem_base, a_tmem + 16, bd + 4, idesc, 1u);
                umma_bf16_ts_pair(tmem_base, a_tmem + 24, bd + 6, idesc, 1u);
                umma_commit_pair_multicast(bar_done + bar_s, 0x3);
                const bool seg_last = (++kb == nkb) || (it == i1 - 1);
                if (kb == nkb) kb = 0;
                if (seg_last) {
                    umma_commit_pair_multicast(bar_accfull, 0x3);
                    ++acc;
                    ++n_seg;
                }
                ++n_st;
                seg_first = seg_last;
                if (++s == SB) {
                    s = 0;
                    ph ^= 1u;
                    bd = bdesc0;
                    a_tmem = tmem_base + kAccCols;
                    bar_s = 0;
                } else {
                    bd += bstride;
                    a_tmem += kAStageCols;
                    bar_s += 8u;
                }
            }
            if (kChecked) {
                chk[kChkMma] = n_st;
                chk[kChkMmaSeg] = n_seg;
            }
            // every MMA issued above has finished once this arrives: TMEM may then be freed
            umma_commit_pair(bar_mma_done);
            settle_wait(bar_mma_done, 0);
        }
        __syncwarp();
    } else if (warp >= kRopeWarp0 && warp < kEpiWarp0) {
        // ---------------- RoPE (Eq. 1) into tensor memory (both CTAs) ----------------
        const int g = (warp - kRopeWarp0) >> 2;   // group: stages q = g, g + 2, ...
        const uint32_t qd = static_cast<uint32_t>(warp & 3);
        const int i = lane >> 2, t4 = lane & 3;
        const int phase = row_phase(i);
        const int rbase = 8 * static_cast<int>(qd) + phase;  // rows rbase + 32*j, j < 4
        const uint32_t row_off = static_cast<uint32_t>(rbase) * 128u;
        const uint32_t lo8 = static_cast<uint32_t>(t4 & 1) << 3;
        const uint32_t chsel = static_cast<uint32_t>(t4 >> 1);
        const uint32_t lane_field = (32u * qd) << 16;
        const int half = nkb * (kBK / 2);  // d/2: start of the 32-position rotations in the table
        uint32_t m[4] = {0u, 0u, 0u, 0u};
        bool steps32 = false, rot = true;
        int64_t cur_tile = -1;
        // The rotation table, a few tens of KB that every stage reads from, does not fit in the L1
        // left beside the pipeline's shared memory: the RoPE warps copy it into shared memory first.
        const bool staged = a.table_bytes != 0;
        const uint64_t* const tbl_sh = reinterpret_cast<const uint64_t*>(gbase + (table_s - sbase));
        if (staged) {
            const uint4* src = reinterpret_cast<const uint4*>(a.rope_table);
            uint4* dst = reinterpret_cast<uint4*>(gbase + (table_s - sbase));
            for (uint32_t e = threadIdx.x - kRopeWarp0 * 32; e < a.table_bytes / 16; e += 4 * kRopeGroups * 32)
                dst[e] = __ldg(src + e);
            asm volatile("bar.sync %0, %1;" ::"n"(kRopeBarrier), "n"(4 * kRopeGroups * 32) : "memory");
        }
        // table words k, k+1 (k even), from shared memory when staged
        auto table_pair = [&](int k) -> ulonglong2 {
            return staged ? *reinterpret_cast<const ulonglong2*>(tbl_sh + k)
                          : __ldg(reinterpret_cast<const ulonglong2*>(a.rope_table + k));
        };
        // this thread's turn entries of a stage, pairs k, k+1 (k = kb*32 + 8c + 2*t4) for c < 4, are
        // fetched a stage ahead; their 32-step rotations are fetched when used
        ulonglong2 tturn[4];
        int kb_table = 0;
        auto load_table = [&](int kb) {
            kb_table = kb;
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                const int k = kb * (kBK / 2) + 8 * c + 2 * t4;
                tturn[c] = table_pair(k);
            }
        };
        // stage q = g, g+2, ...: its tile and K block, and its slots and phase parities, kept
        // incrementally (no divisions on the way)
        int64_t tile = (i0 + g) / nkb;
        int kb = static_cast<int>((i0 + g) % nkb);
        uint32_t sa = static_cast<uint32_t>(g), pa = 0, sb = static_cast<uint32_t>(g), pb = 0;
        if (kRot != kRotNone && i0 + g < i1) load_table(kb);
        for (int64_t it = i0 + g; it < i1; it += kRopeGroups) {
            if (tile != cur_tile) {
                cur_tile = tile;
                rot = ptile_rotates<kRot>(a, tile);
                const int64_t r0 = ptile_src_row<kRot>(a, tile) + static_cast<int64_t>(rank) * kCM + rbase;
                m[0] = r0 < a.n ? (a.positions ? static_cast<uint32_t>(__ldg(a.positions + r0)) : static_cast<uint32_t>(r0))
                                : 0u;
                steps32 = true;
#pragma unroll
                for (int j = 1; j < 4; ++j) {
                    // rows past n are zero-filled by TMA: any angle will do, keep the 32-step pattern
                    const int64_t row = r0 + 32 * j;
                    m[j] = row < a.n ? (a.positions ? static_cast<uint32_t>(__ldg(a.positions + row))
                                                    : static_cast<uint32_t>(row))
                                     : m[0] + 32u * j;
                    steps32 = steps32 && m[j] == m[0] + 32u * j;
                }
                // one path per warp: the branches below hold warp-wide tcgen05.st instructions, which
                // all lanes must execute together (rows past n can make the pattern differ by lane)
                steps32 = __all_sync(0xFFFFFFFFu, steps32);
            }
            const bool got = pair_wait(bar_afull + 8u * sa, pa, abort_flag, peer_abort, a.err_flag, a.wait_limit_ns);
            if (!__all_sync(0xFFFFFFFFu, got)) break;
            // the raw block in the slot is this stage's: the slot's fill count is the stage's turn
            if (kChecked && lane == 0)
                SEMSHARE_CHECK(chk[kChkAFill + sa] == static_cast<uint32_t>((it - i0) / SA) + 1u, a.err_flag, SEMSHARE_KERNEL_HASH_2SM);
            // the thread's 16 words of the stage into registers, then the raw block is free again
            const uint8_t* const st = gbase + sa * kABytes + row_off;
            uint32_t y[4][4][2];  // [row j][column group c][pair e]: raw pairs, rotated in place
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                const uint32_t off = (((2u * c + chsel) ^ static_cast<uint32_t>(phase)) << 4) | lo8;
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    const uint2 w = *reinterpret_cast<const uint2*>(st + j * 32 * 128 + off);
                    y[j][c][0] = w.x;
                    y[j][c][1] = w.y;
                }
            }
            __syncwarp();
            if (kChecked && lane == 0) atomicAdd(const_cast<uint32_t*>(chk + kChkARel + sa), 1u);
            if (lane == 0) mbar_arrive(bar_aempty + 8u * sa);
            // The TMEM operand slot is free once the MMAs of the stage SB before have finished.  The
            // rows are rotated first and the wait comes just before the first store, so that the
            // rotation overlaps those MMAs.
            bool slot_ok = true, slot_waited = false;
            auto wait_slot = [&]() -> bool {
                if (!slot_waited) {
                    slot_waited = true;
                    slot_ok = __all_sync(0xFFFFFFFFu, pair_wait(bar_done + 8u * sb, pb ^ 1u, abort_flag, peer_abort,
                                                                a.err_flag, a.wait_limit_ns));
                    tc_fence_after_sync();
                }
                return slot_ok;
            };
            const uint32_t tcol = tmem_base + kAccCols + sb * kAStageCols + lane_field;
            if ((kRot == kRotAll || rot) && steps32) {
                // the usual case, one branch for the whole stage so that the four column groups'
                // independent chains interleave: row j+1 sits 32 positions after row j, so only
                // row 0's angles go through sincos and the others turn on by the 32-step rotation
#pragma unroll
                for (int ch = 0; ch < 4; ch += 2) {  // two column groups at a time (registers)
                    float cs[2][2], sn[2][2];
                    ulonglong2 tstep[2];
#pragma unroll
                    for (int cc = 0; cc < 2; ++cc)
                        tstep[cc] = table_pair(half + kb_table * (kBK / 2) + 8 * (ch + cc) + 2 * t4);
#pragma unroll
                    for (int cc = 0; cc < 2; ++cc) {
                        rotation(m[0], tturn[ch + cc].x, cs[cc][0], sn[cc][0]);
                        rotation(m[0], tturn[ch + cc].y, cs[cc][1], sn[cc][1]);
                    }
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
#pragma unroll
                        for (int cc = 0; cc < 2; ++cc) {
                            const int c = ch + cc;
#pragma unroll
                            for (int e = 0; e < 2; ++e) {
                                y[j][c][e] =
                                    rotate_to_bf16(bf16_lo(y[j][c][e]), bf16_hi(y[j][c][e]), cs[cc][e], sn[cc][e]);
                                if (j < 3) {
                                    const uint64_t st32 = e ? tstep[cc].y : tstep[cc].x;
                                    const float c32 = __uint_as_float(static_cast<uint32_t>(st32));
                                    const float s32 = __uint_as_float(static_cast<uint32_t>(st32 >> 32));
                                    const float nc = fmaf(cs[cc][e], c32, -sn[cc][e] * s32);
                                    sn[cc][e] = fmaf(cs[cc][e], s32, sn[cc][e] * c32);
                                    cs[cc][e] = nc;
                                }
                            }
                        }
                    }
                    if (!wait_slot()) break;
                    // these two column groups go to tensor memory while the next two are rotated
#pragma unroll
                    for (int h = 0; h < 2; ++h)
#pragma unroll
                        for (int cc = 0; cc < 2; ++cc)
                            tmem_st_16x256b(tcol + ((16u * h) << 16) + 8u * (ch + cc), y[2 * h][ch + cc][0],
                                            y[2 * h][ch + cc][1], y[2 * h + 1][ch + cc][0], y[2 * h + 1][ch + cc][1]);
                }
            } else {
                if (kRot == kRotAll || rot) {
                // positions not 32 apart: every row's own angles
#pragma unroll
                for (int c = 0; c < 4; ++c)
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        float cs0, sn0, cs1, sn1;
                        rotation(m[j], tturn[c].x, cs0, sn0);
                        rotation(m[j], tturn[c].y, cs1, sn1);
                        y[j][c][0] = rotate_to_bf16(bf16_lo(y[j][c][0]), bf16_hi(y[j][c][0]), cs0, sn0);
                        y[j][c][1] = rotate_to_bf16(bf16_lo(y[j][c][1]), bf16_hi(y[j][c][1]), cs1, sn1);
                    }
                }  // rows hashed as they are: the bf16 pairs already are the MMA operand
                if (wait_slot())
#pragma unroll
                for (int h = 0; h < 2; ++h)
#pragma unroll
                    for (int c = 0; c < 4; ++c)
                        tmem_st_16x256b(tcol + ((16u * h) << 16) + 8u * c, y[2 * h][c][0], y[2 * h][c][1],
                                        y[2 * h + 1][c][0], y[2 * h + 1][c][1]);
            }
            tmem_st_wait();
            if (!slot_ok) break;
            // this CTA's hyperplane half of the stage must have landed before the MMA reads it
            const bool b_in = pair_wait(bar_bfull + 8u * sb, pb, abort_flag, peer_abort, a.err_flag, a.wait_limit_ns);
            if (!__all_sync(0xFFFFFFFFu, b_in)) break;
            if (kChecked && lane == 0) {
                SEMSHARE_CHECK(chk[kChkBFill + sb] == static_cast<uint32_t>((it - i0) / SB) + 1u, a.err_flag, SEMSHARE_KERNEL_HASH_2SM);
                if (qd == 0u) atomicAdd(const_cast<uint32_t*>(chk + kChkRope), 1u);
            }
            tc_fence_before_sync();
            __syncwarp();
            if (lane == 0) arrive_lead(bar_ready + 8u * sb, ready_lead + 8u * sb, leader);
            // this group's next stage
            kb += kRopeGroups;
            while (kb >= nkb) {
                kb -= nkb;
                ++tile;
            }
            sa += kRopeGroups;
            if (sa >= SA) {
                sa -= SA;
                pa ^= 1u;
            }
            sb += kRopeGroups;
            if (sb >= SB) {
                sb -= SB;
                pb ^= 1u;
            }
            // its table entries load while it waits for that stage
            if (kRot != kRotNone && it + kRopeGroups < i1) load_table(kb);
        }
    } else if (warp >= kEpiWarp0) {
        // ---------------- epilogue: signs -> packed codes, or partial hand-off (both CTAs) ----
        const int ew = warp & 3;
        const int r = ew * 32 + lane;  // TMEM lane
        const int trow = lane_row(r);  // the row of this CTA's half that the lane holds
        const int W = a.nbits >> 5;
        const int items = W * 8 * kCM;  // float4 per partial slot
        uint32_t acc = 0;
        for (int64_t it = i0; it < i1; ++acc) {
            const int64_t tile = it / nkb;
            const int kb_begin = static_cast<int>(it - tile * nkb);
            const int64_t seg_len = (i1 - it) < (nkb - kb_begin) ? (i1 - it) : (nkb - kb_begin);
            const bool whole = kb_begin == 0 && seg_len == nkb;
            const int64_t tile_it0 = tile * nkb;
            int64_t b_lo = 0, b_hi = 0;
            if (!whole) {  // contributing clusters of this tile, worked out while its MMAs run
                b_lo = range_owner(tile_it0, a.total_iters, P);
                b_hi = range_owner(tile_it0 + nkb - 1, a.total_iters, P);
            }
            const bool got = pair_wait(bar_accfull, acc & 1u, abort_flag, peer_abort, a.err_flag, a.wait_limit_ns);
            if (!epilogue_all(got)) break;
            if (kChecked && threadIdx.x == kEpiWarp0 * 32) chk[kChkEpiSeg] = chk[kChkEpiSeg] + 1u;
            tc_fence_after_sync();
            const int64_t row = ptile_src_row<kRot>(a, tile) + static_cast<int64_t>(rank) * kCM + trow;
            uint32_t* const out_codes = ptile_codes<kRot>(a, tile);
            const uint32_t taddr = tmem_base + (static_cast<uint32_t>(ew * 32) << 16);
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
                if (lane == 0) arrive_lead(bar_accempty, accempty_lead, leader);
                if (row < a.n) {
                    store_codes(out_codes, row, W, words);
                    if (a.signs != nullptr) store_sign_row(a.signs, row, a.signs_pitch, W, words);
                }
            } else if (it + seg_len == i1) {
                // the CTA's last segment, part of a shared tile: closed (this cluster owns the tile's
                // first K blocks) or published (it does not) by all warps after the main loop,
                // straight from the accumulator, which nothing overwrites any more
                if (threadIdx.x == kEpiWarp0 * 32) {
                    defer[1] = tile;
                    defer[2] = b_lo;
                    defer[3] = b_hi;
                    defer[0] = b_lo == pid ? 2 : 1;
                }
            } else {
                // the CTA's first segment, the tail of a tile another cluster started: publish this
                // half's partial and count it
                float4* dst = a.partials + partial_slot(pid, rank) * items;
#pragma unroll
                for (int qq = 0; qq < 8; ++qq) {
                    if (qq < W) {
                        uint32_t v[32];
                        tmem_load_32cols_sync(taddr + qq * 32, v);
#pragma unroll
                        for (int j = 0; j < 8; ++j)
                            dst[(qq * 8 + j) * kCM + r] =
                                make_float4(__uint_as_float(v[4 * j]), __uint_as_float(v[4 * j + 1]),
                                            __uint_as_float(v[4 * j + 2]), __uint_as_float(v[4 * j + 3]));
                    }
                }
                tc_fence_before_sync();
                __syncwarp();
                if (lane == 0) arrive_lead(bar_accempty, accempty_lead, leader);
                __threadfence();
                epilogue_sync();
                if (threadIdx.x == kEpiWarp0 * 32) atomicAdd(a.tile_count + 2 * tile + rank, 1u);
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
        SEMSHARE_CHECK(chk[kChkProdA] == stages, a.err_flag, SEMSHARE_KERNEL_HASH_2SM);
        SEMSHARE_CHECK(chk[kChkProdB] == stages, a.err_flag, SEMSHARE_KERNEL_HASH_2SM);
        SEMSHARE_CHECK(chk[kChkRope] == stages, a.err_flag, SEMSHARE_KERNEL_HASH_2SM);
        SEMSHARE_CHECK(chk[kChkEpiSeg] == segs, a.err_flag, SEMSHARE_KERNEL_HASH_2SM);
        if (leader) {
            SEMSHARE_CHECK(chk[kChkMma] == stages, a.err_flag, SEMSHARE_KERNEL_HASH_2SM);
            SEMSHARE_CHECK(chk[kChkMmaSeg] == segs, a.err_flag, SEMSHARE_KERNEL_HASH_2SM);
        }
    }

    // ---------------- end phase: the deferred shared segment, by all 16 warps ----------------
    // Warp w reads TMEM lanes 32*(w%4).. (its quadrant) and code words 2*(w/4), 2*(w/4)+1.  The
    // decision is taken once (the peer may raise this CTA's abort flag at any moment).
    __shared__ int end_kind;
    if (threadIdx.x == 0) end_kind = *abort_flag == 0 ? static_cast<int>(defer[0]) : 0;
    __syncthreads();
    const int dkind = end_kind;
    if (dkind != 0) {
        tc_fence_after_sync();
        const int W = a.nbits >> 5;
        const int items = W * 8 * kCM;
        const int64_t tile = defer[1], b_lo = defer[2], b_hi = defer[3];
        const int64_t tile_it0 = tile * nkb;
        const int r = (warp & 3) * 32 + lane;
        const uint32_t taddr = tmem_base + (static_cast<uint32_t>((warp & 3) * 32) << 16);
        const int q0 = 2 * (warp >> 2);
        if (dkind == 1) {
            float4* dst = a.partials + partial_slot(pid, rank) * items;
#pragma unroll
            for (int qi = 0; qi < 2; ++qi) {
                const int qq = q0 + qi;
                if (qq < W) {
                    uint32_t v[32];
                    tmem_load_32cols_sync(taddr + qq * 32, v);
#pragma unroll
                    for (int j = 0; j < 8; ++j)
                        dst[(qq * 8 + j) * kCM + r] = make_float4(__uint_as_float(v[4 * j]), __uint_as_float(v[4 * j + 1]),
                                                                  __uint_as_float(v[4 * j + 2]), __uint_as_float(v[4 * j + 3]));
                }
            }
            __threadfence();
            __syncthreads();
            if (threadIdx.x == 0) atomicAdd(a.tile_count + 2 * tile + rank, 1u);
        } else {
            __shared__ int close_ok;
            if (threadIdx.x == 0)
                close_ok = count_wait(a.tile_count + 2 * tile + rank, static_cast<uint32_t>(b_hi - b_lo), abort_flag,
                                      peer_abort, a.err_flag, a.wait_limit_ns);
            __syncthreads();
            if (kChecked && close_ok && threadIdx.x == 0)  // every later contributor counted once
                SEMSHARE_CHECK(ld_acquire_gpu(a.tile_count + 2 * tile + rank) == static_cast<uint32_t>(b_hi - b_lo),
                               a.err_flag, SEMSHARE_KERNEL_HASH_2SM);
            if (close_ok) {
                const int64_t row = ptile_src_row<kRot>(a, tile) + static_cast<int64_t>(rank) * kCM + lane_row(r);
                uint32_t* const out_codes = ptile_codes<kRot>(a, tile);
                // This CTA's K blocks (the tile's first) are in the accumulator; the later
                // contributors' partials are added in K order.  They come through the raw embedding
                // ring, idle now (its copies all landed before the barrier above): copy e = 8 qi + j
                // (float4 j of the thread's word qi) sits at (e * kThreads + threadIdx.x) * 16 bytes.
                // A contributor's sixteen copies are in flight together (cp.async holds no
                // registers), the first contributor's while the accumulator is read.
                const uint32_t stage0 = a_ring + static_cast<uint32_t>(threadIdx.x) * 16u;
                const float4* const staged = reinterpret_cast<const float4*>(gbase + (a_ring - sbase)) + threadIdx.x;
                // word qi's copies of contributor bb into the slots of word `slot_qi`
                auto request = [&](int64_t bb, int qi, int slot_qi) {
                    const float4* p0 = a.partials + partial_slot(bb, rank) * items + r + (q0 + qi) * 8 * kCM;
#pragma unroll
                    for (int j = 0; j < 8; ++j)
                        cp_async_16(stage0 + static_cast<uint32_t>((8 * slot_qi + j) * kThreads) * 16u, p0 + j * kCM);
                };
                const bool two_words = q0 + 1 < W;
                if (b_hi > b_lo && q0 < W) {
                    request(b_lo + 1, 0, 0);
                    if (two_words) request(b_lo + 1, 1, 1);
                }
                // with a second later contributor, its word-1 copies go into word 0's slots as soon
                // as word 0 is summed, and land while word 0 is packed and word 1's first partial added
                bool w1_second_early = false;
#pragma unroll 1
                for (int qi = 0; qi < 2; ++qi) {
                    const int qq = q0 + qi;
                    if (qq >= W) {
                        // the pad of the sign rows past the code bits
                        if (a.signs != nullptr && 32 * qq < a.signs_pitch && row < a.n)
                            store_sign_pad(a.signs + row * a.signs_pitch + 32 * qq);
                        continue;
                    }
                    uint32_t v[32];
                    tmem_load_32cols_sync(taddr + qq * 32, v);
                    float sum[32];
#pragma unroll
                    for (int j = 0; j < 32; ++j) sum[j] = __uint_as_float(v[j]);
                    for (int64_t bb = b_lo + 1; bb <= b_hi; ++bb) {
                        int slot_qi = qi;
                        if (bb == b_lo + 2 && qi == 1 && w1_second_early)
                            slot_qi = 0;  // requested after word 0
                        else if (bb > b_lo + 1)
                            request(bb, qi, qi);  // into the slots its previous values were read from
                        cp_async_wait_all();
#pragma unroll
                        for (int j = 0; j < 8; ++j) {
                            const float4 f = staged[(8 * slot_qi + j) * kThreads];
                            sum[4 * j] += f.x;
                            sum[4 * j + 1] += f.y;
                            sum[4 * j + 2] += f.z;
                            sum[4 * j + 3] += f.w;
                        }
                    }
                    if (qi == 0 && two_words && b_hi >= b_lo + 2) {
                        request(b_lo + 2, 1, 0);
                        w1_second_early = true;
                    }
#pragma unroll
                    for (int j = 0; j < 32; ++j) v[j] = __float_as_uint(sum[j]);
                    if (row < a.n) {
                        const uint32_t bits = sign_word(v);
                        out_codes[row * W + qq] = bits;
                        if (a.proj != nullptr) store_proj(a.proj, row, a.nbits, qq, v);
                        if (a.signs != nullptr) store_sign_bytes(a.signs + row * a.signs_pitch + 32 * qq, bits);
                    }
                }
                if (threadIdx.x == 0) a.tile_count[2 * tile + rank] = 0u;  // leave the workspace zeroed
            }
        }
        tc_fence_before_sync();
    }

    // the pair meets before tensor memory is freed: the even CTA's MMAs read both CTAs' tensor
    // and shared memory, and have all finished once its MMA thread has passed its last wait
    cluster_sync_all();
    if (warp == 1) {
        tc_fence_after_sync();
        tmem_dealloc_pair(tmem_base, kTmemCols);
    }
    grid_dependents_launch();  // every CTA, after it has freed its tensor memory
}

// Clusters of the launch: as many pairs as can be resident at once (one CTA per SM), no more
// than there are iterations.  SEMSHARE_HASH_CLUSTERS (read per call, a test knob) lowers it.
template <typename K>
semshare_status plan_clusters(K kernel, size_t smem, int64_t total_iters, int* clusters) {
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = dim3(2);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = smem;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 2;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, kernel, &cfg) != cudaSuccess || n < 1) return SEMSHARE_ECUDA;
    const char* e = getenv("SEMSHARE_HASH_CLUSTERS");
    if (e != nullptr && *e != 0) {
        const long v = strtol(e, nullptr, 10);
        if (v >= 1 && v < n) n = static_cast<int>(v);
    }
    *clusters = static_cast<int>(total_iters < n ? total_iters : n);
    return SEMSHARE_OK;
}

}  // namespace

semshare_status launch_hash_2sm(const Hash2smCall& c) {
    const int64_t n_rows = c.pair ? 2 * c.pair_rows : c.n;
    const int64_t n_ptiles = (n_rows + kPM - 1) / kPM;
    Hash2smArgs a{};
    a.n = c.n;
    a.n_kblocks = c.d / kBK;
    a.total_iters = n_ptiles * a.n_kblocks;
    a.pair_rows = c.pair ? c.pair_rows : 0;
    a.nbits = c.nbits;
    a.n_ptiles = static_cast<int32_t>(n_ptiles);
    a.bh_bytes = static_cast<uint32_t>(c.nbits) * kBK;  // nbits/2 rows of 128 bytes
    if (c.count_bytes < static_cast<size_t>(2 * n_ptiles) * 4) return SEMSHARE_EINVAL;
    int dev = 0, smem_optin = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess)
        return SEMSHARE_ECUDA;
    a.b_slots = kBSlots;
    a.table_bytes = (!c.none && static_cast<uint32_t>(c.d) * 8u <= kMaxTableSmem) ? static_cast<uint32_t>(c.d) * 8u : 0u;
    const size_t room = static_cast<size_t>(smem_optin) - kFixedSmem - static_cast<size_t>(kBSlots) * a.bh_bytes -
                        a.table_bytes;
    int a_slots = static_cast<int>(room / kABytes);
    if (a_slots > kMaxASlots) a_slots = kMaxASlots;
    a_slots -= a_slots % kRopeGroups;  // each slot belongs to one RoPE group
    // the ring must also hold the close's staging area: 16 copies of 16 bytes per thread
    if (a_slots < 2 || static_cast<size_t>(a_slots) * kABytes < static_cast<size_t>(kThreads) * 16 * 16)
        return SEMSHARE_EUNSUPPORTED;
    a.a_slots = a_slots;
    a.positions = c.positions;
    a.rope_table = c.rope_table;
    a.codes = c.codes;
    a.codes2 = c.codes2;
    a.proj = c.proj;
    a.signs = c.signs;
    a.signs_pitch = c.signs_pitch;
    a.err_flag = c.err_flag;
    a.partials = static_cast<float4*>(c.partials);
    a.tile_count = c.tile_count;
    a.wait_limit_ns = wait_limit_ns();
    const size_t smem = kFixedSmem + static_cast<size_t>(a_slots) * kABytes + static_cast<size_t>(kBSlots) * a.bh_bytes +
                        a.table_bytes;

    CUtensorMap tm_emb, tm_hyp;
    if (!encode_tma_2d(&tm_emb, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, c.emb, static_cast<uint64_t>(c.d),
                       static_cast<uint64_t>(c.n), static_cast<uint64_t>(c.row_stride) * 2, 64u, kCM))
        return SEMSHARE_ECUDA;
    if (!encode_tma_2d(&tm_hyp, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, c.hyperplanes, static_cast<uint64_t>(c.d),
                       static_cast<uint64_t>(c.nbits), static_cast<uint64_t>(c.d) * 2, 64u,
                       static_cast<uint32_t>(c.nbits / 2)))
        return SEMSHARE_ECUDA;

    auto kernel = c.pair ? lsh_hash_2sm_kernel<kRotPair> : c.none ? lsh_hash_2sm_kernel<kRotNone> : lsh_hash_2sm_kernel<kRotAll>;
    if (cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem)) != cudaSuccess)
        return SEMSHARE_ECUDA;
    int clusters = 0;
    semshare_status st = plan_clusters(kernel, smem, a.total_iters, &clusters);
    if (st != SEMSHARE_OK) return st;
    if (2 * static_cast<size_t>(clusters) * 2 * kCM * kMaxBits * 4 > c.partial_bytes) return SEMSHARE_EINVAL;

    cudaLaunchConfig_t cfg{};
    cfg.gridDim = dim3(2 * clusters);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = as_stream(c.stream);
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 2;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    if (cudaLaunchKernelEx(&cfg, kernel, tm_emb, tm_hyp, a) != cudaSuccess) return SEMSHARE_ECUDA;
    return launch_status();
}

}  // namespace semshare
