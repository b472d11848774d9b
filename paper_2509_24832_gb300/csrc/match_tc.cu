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
// 256*dot - j (largest dot first, then the lowest column j of the epilogue warp's 128-column
// half of the tile).  The best
// (distance << 32 | index) of a target over the tiles a CTA visits goes to a 64-bit atomicMin,
// which is "smallest distance, then lowest index" whatever the split.
//
// Roles (384 threads): warp 0 TMA producer (the 128-target A tile, reloaded only when the
// target block changes, and the 256-reference B tile, double-buffered); warp 1 TMEM allocator
// and MMA issuer (tcgen05.mma kind::f8f6f4, M=128, N=256, K=32); warps 4-11 epilogue
// (tcgen05.ld, lane = target, running arg-max), two warps per TMEM lane quadrant, each reducing
// one 128-column half of every tile.  The (target block, reference block) tiles are
// split into one equal contiguous range per CTA, target blocks outermost.  Every pipeline wait
// is bounded (SEMSHARE_FLAG_TIMEOUT), nothing traps.
//
// Segmented mode (semshare_retrieve).  The reference rows are the concatenated codes of several
// candidate prompts; the epilogue keeps one best key per (candidate, target) instead of one per
// target.  Candidate boundaries are the same for every lane of a warp (lanes are targets,
// columns are references), so the boundary tests are warp-uniform: a 32-column chunk without a
// boundary takes the plain arg-max, one with a boundary is cut into runs and the key of the
// finished candidate is flushed with the atomicMin.  A reduction over targets then gives each
// candidate's summed nearest distance, its similarity (App. A.3) and the arg-max candidate.
//
// Selected mode (semshare_match_tc_selected).  The reference rows are one candidate of a pool,
// chosen by a device value (the retrieval's `best`): the expand kernel reads the choice, expands
// that candidate's rows and publishes its length and first pool row; the search, sized for the
// longest candidate, masks the columns past that length; the split adds the first pool row.
//
// Sign-row mode (semshare_match_tc_signs).  The operands are the caller's e4m3 rows written by
// semshare_hash_signs (no expand kernel); the search's last CTA to finish (an arrival counter, no
// CTA waits for another) splits the keys into idx/dist and resets them for the next call.
#include <cuda.h>

#include "common.cuh"
#include "ptx.cuh"
#include "tma_host.cuh"

namespace semshare {
namespace {

constexpr int kTM = 128;        // targets per tile (TMEM lanes)
constexpr int kTN = 256;        // references per tile (MMA N)
constexpr int kChunk = 128;     // bytes per 128-byte swizzle chunk along the code
constexpr int kEpiWarp0 = 4;   // a multiple of 4: epilogue warp w reads TMEM lanes 32*(w%4)
constexpr int kEpiWarps = 8;   // two per lane quadrant, one per 128-column half of every tile
constexpr int kHalfCols = kTN / 2;
constexpr int kThreads = (kEpiWarp0 + kEpiWarps) * 32;
constexpr unsigned long long kNoKey = ~0ull;
constexpr unsigned int kNoArrivals = ~0u;  // the fused search's arrival counter between calls
// Targets up to which the last CTA of the search splits the keys itself (a few per thread);
// larger searches hand them to tc_keys_split_kernel, which spreads them over the GPU.
constexpr int64_t kFusedSplitMaxTargets = 16384;
constexpr size_t kFixedSmem = 1024 + 256 + (kChecked ? 128 : 0);

// Candidate (segment) boundaries of the reference rows, passed by value: off[0] = 0 <
// off[1] < ... < off[n_seg] = n_ref.  kMax = 1 for the plain search.
template <int kMax>
struct SegTable {
    int32_t n_seg;
    int64_t off[kMax + 1];
};

struct TcArgs {
    int64_t n_tgt;
    int64_t n_ref;
    const int64_t* n_ref_dev;  // non-null: the columns actually searched, [0, *n_ref_dev) (<= n_ref)
    int64_t n_rb;
    int64_t total;  // target blocks x reference blocks
    int32_t nbits;
    int32_t kchunks;
    uint32_t a_bytes;  // one A buffer: 128 rows x kchunks*128 bytes
    uint32_t b_bytes;  // one B buffer: 256 rows x kchunks*128 bytes
    unsigned long long* keys;  // [n_seg][n_tgt]
    uint32_t* err_flag;
    uint64_t wait_limit_ns;
    // fused split (kFused): the last CTA to finish writes idx/dist from the keys and resets them
    int32_t* idx;
    int32_t* dist;
    unsigned int* counter;     // arrivals, kNoArrivals between calls
};

// Offsets of the candidates of a pool, passed by value (semshare_match_tc_selected; kMax = 1
// for the other searches, which do not read it).
template <int kMax>
struct CandTable {
    int32_t n_cand;
    int64_t off[kMax + 1];
};
constexpr int kSelMax = SEMSHARE_RETRIEVE_MAX_CANDIDATES;
template <bool kSelect>
using CandTableFor = CandTable<kSelect ? kSelMax : 1>;

// e4m3 +1 is 0x38, -1 is 0xB8: byte = 0xB8 ^ (bit << 7).  Rows are padded with zero bytes to
// kpad; the keys of the search are reset on the way.  kSelect: the reference rows are those of
// candidate *best of the pool `ref` (offsets `cand`), read on the device; rows past its length
// are zero, and sel[0] = its length, sel[1] = its first pool row (0 and -1 for an invalid
// *best, which also raises SEMSHARE_FLAG_INDEX).
template <bool kSelect>
__global__ void expand_codes_kernel(const uint32_t* __restrict__ tgt, int64_t n_tgt, const uint32_t* __restrict__ ref,
                                    int64_t n_ref, int32_t nbits, int32_t kpad, uint8_t* __restrict__ tpm,
                                    uint8_t* __restrict__ rpm, unsigned long long* __restrict__ keys, int64_t n_keys,
                                    unsigned int* __restrict__ counter, const int32_t* __restrict__ best,
                                    const __grid_constant__ CandTableFor<kSelect> cand, int64_t* __restrict__ sel,
                                    uint32_t* err_flag) {
    pdl_prologue();
    const int W = nbits >> 5;
    const int per_row = kpad >> 4;  // 16-byte pieces per row
    int64_t len = n_ref;
    if (kSelect) {
        const int32_t b = __ldg(best);
        const bool ok = b >= 0 && b < cand.n_cand;
        len = ok ? cand.off[b + 1] - cand.off[b] : 0;
        ref += ok ? cand.off[b] * W : 0;
        if (blockIdx.x == 0 && threadIdx.x == 0) {
            sel[0] = len;
            sel[1] = ok ? cand.off[b] : -1;
            if (!ok && err_flag) atomicOr(err_flag, SEMSHARE_FLAG_INDEX);
        }
    }
    const int64_t total = (n_tgt + n_ref) * per_row;
    const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
    for (int64_t e = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; e < total; e += stride) {
        const int64_t row = e / per_row;
        const int piece = static_cast<int>(e - row * per_row);
        const int b0 = piece * 16;
        uint4 out = make_uint4(0u, 0u, 0u, 0u);
        if (b0 < nbits && (!kSelect || row < n_tgt + len)) {
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
    for (int64_t t = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; t < n_keys; t += stride) keys[t] = kNoKey;
    if (counter != nullptr && blockIdx.x == 0 && threadIdx.x == 0) *counter = 0u;
}

// sel non-null: idx are pool rows, local + sel[1]; a target with no key (an invalid candidate)
// gets idx = dist = -1.
// reset: leave every key at kNoKey again (the searches over caller sign rows expect it on entry).
__global__ void tc_keys_split_kernel(unsigned long long* __restrict__ keys, int64_t n, int32_t* __restrict__ idx,
                                     int32_t* __restrict__ dist, const int64_t* __restrict__ sel, bool reset) {
    pdl_prologue();
    const int64_t base = sel ? sel[1] : 0;
    for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < n;
         i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const unsigned long long k = keys[i];
        if (reset) keys[i] = kNoKey;
        const bool none = k == kNoKey;
        idx[i] = none ? -1 : static_cast<int32_t>(static_cast<uint32_t>(k) + base);
        if (dist) dist[i] = none ? -1 : static_cast<int32_t>(static_cast<uint32_t>(k >> 32));
    }
}

__device__ __forceinline__ bool drain_wait(uint32_t bar, uint32_t parity, uint64_t limit_ns) {
    if (mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = global_timer_ns();
    while (!mbar_try_wait(bar, parity))
        if (global_timer_ns() - t0 > limit_ns) return false;
    return true;
}

// kFused (plain search only): the keys are kNoKey on entry; the last CTA to finish writes idx and
// dist from them and resets them (and the arrival counter) for the next call.
template <int kMaxSeg, bool kFused = false>
__global__ void __launch_bounds__(kThreads, 1)
    hamming_tc_kernel(const __grid_constant__ CUtensorMap tm_t, const __grid_constant__ CUtensorMap tm_r,
                      const TcArgs a, const __grid_constant__ SegTable<kMaxSeg> seg) {
    static_assert(!kFused || kMaxSeg == 1, "the fused split is for the plain search");
    // The next kernel is released at the end (below), after the fused split: released at the
    // start, its CTAs queue behind this persistent grid for its whole run (the 5k-token step with
    // the fused search measured 253 us that way against 218 us; the batched step 2.91 against
    // 2.89 ms with the plain search).
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
    // checked build: fills of the two A [0, 2) and two B [2, 4) buffers, releases of the two
    // accumulators by the epilogue warps [4, 6), tiles issued by the producer [6], the MMA [7] and
    // drained by the epilogue [8]
    volatile uint32_t* const chk = reinterpret_cast<volatile uint32_t*>(gbase + (bars + 256u - sbase));

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
            mbar_init(bar_accempty + 8 * i, kEpiWarps);
        }
        mbar_init(bar_done, 1);
        *abort_flag = 0;
        if (kChecked)
            for (int i = 0; i < 16; ++i) chk[i] = 0u;
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
    // The set-up above touches only this CTA's shared and tensor memory, so it overlaps the
    // previous kernel's drain; global memory is read and written only from here on.
    grid_dependency_wait();
    const uint32_t tmem_base = *tmem_slot_ptr;
    const uint64_t lim = a.wait_limit_ns;
    uint32_t* const err = a.err_flag;
    if (threadIdx.x == 0) SEMSHARE_CHECK(tmem_base == 0u, err, SEMSHARE_KERNEL_HAMMING_TC);  // lane 0, column 0

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
                    if (kChecked) chk[s] = chk[s] + 1u;
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
                if (kChecked) chk[2 + s] = chk[2 + s] + 1u;
                mbar_arrive_expect_tx(bar_bfull + 8 * s, a.b_bytes);
                for (int c = 0; c < a.kchunks; ++c)
                    tma_load_2d(b_buf0 + s * a.b_bytes + c * (kTN * kChunk), &tm_r, bar_bfull + 8 * s, c * kChunk,
                                static_cast<int32_t>(rb * kTN));
                ++nb;
            }
            if (kChecked && ok) chk[6] = nb;
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
                    SEMSHARE_CHECK(chk[a_slot] == (na >> 1) + 1u, err, SEMSHARE_KERNEL_HAMMING_TC);  // this target block's fill
                    ++na;
                    cur_tb = tb;
                }
                const uint32_t buf = acc & 1u;
                if (!mbar_wait_bounded(bar_accempty + 8 * buf, ((acc >> 1) & 1u) ^ 1u, abort_flag, err,
                                       SEMSHARE_FLAG_TIMEOUT, lim))
                    break;
                // every epilogue warp released each earlier use of the accumulator
                SEMSHARE_CHECK(chk[4 + buf] == static_cast<uint32_t>(kEpiWarps) * (acc >> 1), err, SEMSHARE_KERNEL_HAMMING_TC);
                const uint32_t s = nb & 1u;
                if (!mbar_wait_bounded(bar_bfull + 8 * s, (nb >> 1) & 1u, abort_flag, err, SEMSHARE_FLAG_TIMEOUT, lim))
                    break;
                SEMSHARE_CHECK(chk[2 + s] == (nb >> 1) + 1u, err, SEMSHARE_KERNEL_HAMMING_TC);  // this tile's reference block
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
            if (kChecked) chk[7] = acc;
            umma_commit(bar_done);
            drain_wait(bar_done, 0, kWaitLimitNs);
        }
        __syncwarp();
    } else if (warp >= kEpiWarp0) {
        // ---------------- epilogue: best reference of every target row ----------------
        // (per candidate in segmented mode; candidate cs covers columns [off[cs], next_b)).  This
        // warp reduces lanes 32*quad.. of columns [half*128, half*128 + 128) of every tile.
        const int ew = warp - kEpiWarp0;
        const int quad = ew & 3;
        const int half = ew >> 2;
        const int r = quad * 32 + lane;
        uint32_t acc = 0;
        int64_t cur_tb = -1, col0 = 0, next_b = 0;
        int32_t cs = 0;
        unsigned long long best = kNoKey;
        const int64_t n_cols = a.n_ref_dev ? *a.n_ref_dev : a.n_ref;  // columns searched
        // fold the best key 256*dot - j (j = column within this warp's half of the tile) into `best`
        auto fold = [&](float bk) {
            if (bk > -1.0e38f) {
                const int ik = __float2int_rn(bk);
                const int dot = -((-ik) >> 8);  // ceil(ik / 256)
                const int j = 256 * dot - ik;    // 0..127
                const unsigned long long dist = static_cast<unsigned long long>((a.nbits - dot) >> 1);
                const unsigned long long cand =
                    (dist << 32) | static_cast<unsigned long long>(col0 + half * kHalfCols + j);
                best = cand < best ? cand : best;
            }
        };
        auto flush = [&]() {
            const int64_t g = cur_tb * kTM + r;
            if (g < a.n_tgt && best != kNoKey && cs < seg.n_seg)
                atomicMin(a.keys + static_cast<int64_t>(cs) * a.n_tgt + g, best);
            best = kNoKey;
        };
        auto advance = [&]() {
            ++cs;
            next_b = cs + 1 <= seg.n_seg ? seg.off[cs + 1] : a.n_ref;
        };
        for (int64_t u = u0; u < u1; ++u, ++acc) {
            const int64_t tb = u / a.n_rb, rb = u - tb * a.n_rb;
            col0 = rb * kTN;
            const int64_t h0 = col0 + half * kHalfCols;  // this warp's first column of the tile
            if (tb != cur_tb) {
                if (cur_tb >= 0) flush();
                cur_tb = tb;
                best = kNoKey;
                // candidate holding column h0: the largest cs with off[cs] <= h0
                int lo = 0, hi = seg.n_seg - 1;
                while (lo < hi) {
                    const int mid = (lo + hi + 1) >> 1;
                    if (seg.off[mid] <= h0) lo = mid; else hi = mid - 1;
                }
                cs = lo;
                next_b = seg.off[lo + 1];
            } else {
                // the other half's columns lie in between: leave every candidate that ended there
                while (next_b <= h0 && cs + 1 < seg.n_seg) {
                    flush();
                    advance();
                }
            }
            const uint32_t buf = acc & 1u;
            const bool got = mbar_wait_bounded(bar_accfull + 8 * buf, (acc >> 1) & 1u, abort_flag, err,
                                               SEMSHARE_FLAG_TIMEOUT, lim);
            if (!__all_sync(0xFFFFFFFFu, got)) {
                cur_tb = -1;
                break;
            }
            tc_fence_after_sync();
            const int64_t rem = n_cols - col0;
            const int valid = rem < kTN ? static_cast<int>(rem) : kTN;
            const int hv = valid - half * kHalfCols;  // valid columns of this half (may be <= 0)
            const uint32_t taddr =
                tmem_base + (static_cast<uint32_t>(quad * 32) << 16) + buf * kTN + half * kHalfCols;
            float bk = -3.0e38f;  // best key 256*dot - j of this tile's half (current candidate)
            if (hv > 0) {
                // 32-column chunks, double-buffered: the load of chunk q+1 is in flight while
                // chunk q is reduced
                uint32_t va[32], vb[32];
                tmem_load_32cols(taddr, va);
                tmem_load_wait_fence(va);
#pragma unroll
                for (int q = 0; q < kHalfCols / 32; ++q) {
                    uint32_t(&v)[32] = (q & 1) ? vb : va;
                    uint32_t(&vn)[32] = (q & 1) ? va : vb;
                    if (q + 1 < kHalfCols / 32) tmem_load_32cols(taddr + (q + 1) * 32, vn);
                    const int tq = half * (kHalfCols / 32) + q;  // chunk index within the tile
                    const int64_t c0 = col0 + tq * 32;
                    if (q * 32 + 32 <= hv && c0 + 32 <= next_b) {
                        // four independent max chains (the keys are distinct: order does not matter)
                        float m0 = -3.0e38f, m1 = -3.0e38f, m2 = -3.0e38f, m3 = -3.0e38f;
#pragma unroll
                        for (int j = 0; j < 32; j += 4) {
                            m0 = fmaxf(m0, fmaf(__uint_as_float(v[j]), 256.0f, -static_cast<float>(q * 32 + j)));
                            m1 = fmaxf(m1, fmaf(__uint_as_float(v[j + 1]), 256.0f, -static_cast<float>(q * 32 + j + 1)));
                            m2 = fmaxf(m2, fmaf(__uint_as_float(v[j + 2]), 256.0f, -static_cast<float>(q * 32 + j + 2)));
                            m3 = fmaxf(m3, fmaf(__uint_as_float(v[j + 3]), 256.0f, -static_cast<float>(q * 32 + j + 3)));
                        }
                        bk = fmaxf(bk, fmaxf(fmaxf(m0, m1), fmaxf(m2, m3)));
                    } else if (q * 32 < hv) {
                        // ragged end and/or candidate boundaries inside the chunk: runs [js, je)
                        const int jend = hv - q * 32 < 32 ? hv - q * 32 : 32;
                        int js = 0;
                        for (;;) {
                            const int64_t lim_b = next_b - c0;  // >= js: the boundary is not passed yet
                            const int je = lim_b < jend ? static_cast<int>(lim_b) : jend;
#pragma unroll
                            for (int j = 0; j < 32; ++j)
                                if (j >= js && j < je)
                                    bk = fmaxf(bk, fmaf(__uint_as_float(v[j]), 256.0f, -static_cast<float>(q * 32 + j)));
                            if (je == jend) break;
                            // column c0 + je opens candidate cs + 1
                            fold(bk);
                            bk = -3.0e38f;
                            flush();
                            advance();
                            js = je;
                        }
                    }
                    if (q + 1 < kHalfCols / 32) tmem_load_wait_fence(vn);
                }
            }
            tc_fence_before_sync();
            __syncwarp();
            if (lane == 0) {
                if (kChecked) atomicAdd(const_cast<uint32_t*>(chk + 4 + buf), 1u);
                mbar_arrive(bar_accempty + 8 * buf);
            }
            fold(bk);
            if (kChecked && ew == 0 && lane == 0) chk[8] = chk[8] + 1u;
        }
        if (cur_tb >= 0) flush();
        if (kFused) __threadfence();  // this thread's keys are in place before the CTA counts itself
    }

    tc_fence_before_sync();
    __syncthreads();
    if (kChecked && threadIdx.x == 0 && *abort_flag == 0) {
        // every role handled every tile of the range
        const uint32_t tiles = static_cast<uint32_t>(u1 - u0);
        SEMSHARE_CHECK(chk[6] == tiles && chk[7] == tiles && chk[8] == tiles, err, SEMSHARE_KERNEL_HAMMING_TC);
        SEMSHARE_CHECK(chk[4] + chk[5] == static_cast<uint32_t>(kEpiWarps) * tiles, err, SEMSHARE_KERNEL_HAMMING_TC);
    }
    if (warp == 1) {
        tc_fence_after_sync();
        tmem_dealloc(tmem_base, 512);
    }
    if (kFused) {
        // The last CTA to arrive has every key: it splits them into idx/dist and resets them.
        // (No CTA waits for another: the others have finished when the last one counts itself.)
        __shared__ bool last;
        if (threadIdx.x == 0)
            last = atomicAdd(a.counter, 1u) == static_cast<unsigned int>(gridDim.x) + kNoArrivals - 1u;
        __syncthreads();
        if (last) {
            __threadfence();
            // kSplitBatch keys per thread are loaded before any is written, so the split waits for
            // L2 once per batch (a load per iteration would wait once per key)
            constexpr int kSplitBatch = 16;
            for (int64_t t0 = threadIdx.x; t0 < a.n_tgt; t0 += kSplitBatch * kThreads) {
                unsigned long long k[kSplitBatch];
#pragma unroll
                for (int i = 0; i < kSplitBatch; ++i) {
                    const int64_t t = t0 + static_cast<int64_t>(i) * kThreads;
                    k[i] = t < a.n_tgt ? __ldcg(a.keys + t) : kNoKey;
                }
#pragma unroll
                for (int i = 0; i < kSplitBatch; ++i) {
                    const int64_t t = t0 + static_cast<int64_t>(i) * kThreads;
                    if (t < a.n_tgt) {
                        a.keys[t] = kNoKey;
                        const bool none = k[i] == kNoKey;
                        a.idx[t] = none ? -1 : static_cast<int32_t>(static_cast<uint32_t>(k[i]));
                        if (a.dist) a.dist[t] = none ? -1 : static_cast<int32_t>(static_cast<uint32_t>(k[i] >> 32));
                    }
                }
            }
            if (threadIdx.x == 0) *a.counter = kNoArrivals;
        }
    }
    grid_dependents_launch();  // every CTA, the last after its split
}

struct TcPlan {
    int32_t kpad;
    size_t keys_bytes, t_bytes, r_bytes, sums_bytes;
    size_t total() const { return keys_bytes + t_bytes + r_bytes + sums_bytes; }
};

size_t round256(size_t x) { return ((x + 255) / 256) * 256; }

// n_seg = 0: the plain search (one key per target, no reduction scratch).
void plan_tc(int64_t n_tgt, int64_t n_ref, int32_t nbits, int32_t n_seg, TcPlan* p) {
    p->kpad = ((nbits + kChunk - 1) / kChunk) * kChunk;
    p->keys_bytes = round256(static_cast<size_t>(n_tgt) * 8 * static_cast<size_t>(n_seg > 0 ? n_seg : 1));
    p->t_bytes = round256(static_cast<size_t>(n_tgt) * p->kpad);
    p->r_bytes = round256(static_cast<size_t>(n_ref) * p->kpad);
    // per-candidate sums, then the arrival counter
    p->sums_bytes = n_seg > 0 ? round256(static_cast<size_t>(n_seg) * 8 + 8) : 0;
}

// Per-candidate reduction (Sec. 3.2, App. A.3, Sec. 4.4): block s sums the nearest distances
// of all targets to candidate s (exact, int64); the last block to finish turns the sums into
// mean distances and similarities, picks the arg-max candidate (lowest index on ties) and
// decides whether reuse applies.  fp64 throughout: the same rounding as a plain host program.
__global__ void __launch_bounds__(256)
    retrieve_finalize_kernel(const unsigned long long* __restrict__ keys, int64_t n_tgt, int32_t n_seg,
                             double max_dist, double threshold, long long* sums, unsigned int* counter,
                             double* __restrict__ mean_dist, double* __restrict__ similarity,
                             int32_t* __restrict__ best, int32_t* __restrict__ applies) {
    pdl_prologue();
    __shared__ long long warp_sum[8];
    __shared__ bool last;
    const int s = blockIdx.x;
    long long acc = 0;
    const unsigned long long* k = keys + static_cast<int64_t>(s) * n_tgt;
    for (int64_t t = threadIdx.x; t < n_tgt; t += blockDim.x) acc += static_cast<long long>(k[t] >> 32);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xFFFFFFFFu, acc, o);
    if ((threadIdx.x & 31) == 0) warp_sum[threadIdx.x >> 5] = acc;
    __syncthreads();
    if (threadIdx.x == 0) {
        long long tot = 0;
        for (int w = 0; w < static_cast<int>(blockDim.x >> 5); ++w) tot += warp_sum[w];
        sums[s] = tot;
        __threadfence();
        last = atomicAdd(counter, 1u) == static_cast<unsigned>(n_seg - 1);
    }
    __syncthreads();
    if (!last) return;
    // the last block: thread c handles candidate c (fp64 is slow on this part: run the
    // divisions side by side), then a tree arg-max over (similarity, lowest index)
    __shared__ double red_sim[256];
    __shared__ int red_idx[256];
    __threadfence();
    const volatile long long* vs = sums;
    const int c = threadIdx.x;
    double sim = -1.0;
    if (c < n_seg) {
        const double m = static_cast<double>(vs[c]) / static_cast<double>(n_tgt);
        sim = 1.0 - m / max_dist;
        sim = sim < 0.0 ? 0.0 : (sim > 1.0 ? 1.0 : sim);
        if (mean_dist) mean_dist[c] = m;
        if (similarity) similarity[c] = sim;
    }
    red_sim[c] = sim;
    red_idx[c] = c;
    __syncthreads();
    for (int o = 128; o > 0; o >>= 1) {
        if (c < o) {
            const double s2 = red_sim[c + o];
            const int i2 = red_idx[c + o];
            if (s2 > red_sim[c] || (s2 == red_sim[c] && i2 < red_idx[c])) {
                red_sim[c] = s2;
                red_idx[c] = i2;
            }
        }
        __syncthreads();
    }
    if (c == 0) {
        *best = red_idx[0];
        if (applies) *applies = red_sim[0] > threshold ? 1 : 0;
        *counter = 0u;
    }
}

// idx/dist of every target against the chosen candidate (global reference rows).
__global__ void retrieve_select_kernel(const unsigned long long* __restrict__ keys, int64_t n_tgt,
                                       const int32_t* __restrict__ best, int32_t* __restrict__ idx,
                                       int32_t* __restrict__ dist) {
    pdl_prologue();
    const unsigned long long* k = keys + static_cast<int64_t>(*best) * n_tgt;
    for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < n_tgt;
         i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const unsigned long long v = k[i];
        if (idx) idx[i] = static_cast<int32_t>(static_cast<uint32_t>(v));
        if (dist) dist[i] = static_cast<int32_t>(static_cast<uint32_t>(v >> 32));
    }
}

// Expand the codes and run the search; leaves keys[n_seg][n_tgt] in the workspace.  kSelect:
// the reference rows are candidate *best of the pool (cand), n_ref its longest candidate, and
// sel (two int64 in device memory) receives the candidate's length and first pool row.
// Sign rows given (tsig/rsig, [n][kpad] bytes from semshare_hash_signs): no expansion; the keys
// (and, with fused_idx, the arrival counter) must then hold kNoKey (kNoArrivals) on entry, and
// with fused_idx the search's last CTA writes idx/dist and resets them.
template <int kMaxSeg, bool kSelect = false>
semshare_status launch_search(const uint32_t* tgt_codes, int64_t n_tgt, const uint32_t* ref_codes, int64_t n_ref,
                              int32_t nbits, const SegTable<kMaxSeg>& seg, const TcPlan& plan, void* workspace,
                              uint32_t* err_flag, cudaStream_t s, int sms, int dev, const int32_t* best = nullptr,
                              const CandTableFor<kSelect>* cand = nullptr, int64_t* sel = nullptr,
                              const uint8_t* tsig = nullptr, const uint8_t* rsig = nullptr, int32_t* fused_idx = nullptr,
                              int32_t* fused_dist = nullptr, unsigned int* fused_counter = nullptr) {
    int smem_optin = 0;
    if (cudaDeviceGetAttribute(&smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess)
        return SEMSHARE_ECUDA;
    auto* keys = static_cast<unsigned long long*>(workspace);
    uint8_t* tpm = static_cast<uint8_t*>(workspace) + plan.keys_bytes;
    uint8_t* rpm = tpm + plan.t_bytes;
    unsigned int* counter = nullptr;
    if (plan.sums_bytes > 0)
        counter = reinterpret_cast<unsigned int*>(rpm + plan.r_bytes + static_cast<size_t>(seg.n_seg) * 8);

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
    a.n_ref_dev = kSelect ? sel : nullptr;
    a.err_flag = err_flag;
    a.wait_limit_ns = wait_limit_ns();
    a.idx = fused_idx;
    a.dist = fused_dist;
    a.counter = fused_counter;
    const bool signs = tsig != nullptr;
    const bool fused = fused_idx != nullptr;
    if (signs) {
        tpm = const_cast<uint8_t*>(tsig);
        rpm = const_cast<uint8_t*>(rsig);
    }
    const size_t smem = kFixedSmem + 2 * static_cast<size_t>(a.a_bytes) + 2 * static_cast<size_t>(a.b_bytes);
    if (smem > static_cast<size_t>(smem_optin)) return SEMSHARE_EUNSUPPORTED;

    CUtensorMap tm_t, tm_r;
    if (!encode_tma_2d(&tm_t, CU_TENSOR_MAP_DATA_TYPE_UINT8, tpm, static_cast<uint64_t>(plan.kpad),
                       static_cast<uint64_t>(n_tgt), static_cast<uint64_t>(plan.kpad), kChunk, kTM) ||
        !encode_tma_2d(&tm_r, CU_TENSOR_MAP_DATA_TYPE_UINT8, rpm, static_cast<uint64_t>(plan.kpad),
                       static_cast<uint64_t>(n_ref), static_cast<uint64_t>(plan.kpad), kChunk, kTN))
        return SEMSHARE_ECUDA;
    auto kernel = fused ? hamming_tc_kernel<kMaxSeg, kMaxSeg == 1> : hamming_tc_kernel<kMaxSeg, false>;
    if (cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem)) != cudaSuccess)
        return SEMSHARE_ECUDA;
    const int64_t grid = a.total < sms ? a.total : sms;
    if (signs) {
        if (launch_pdl(kernel, dim3(static_cast<unsigned>(grid)), dim3(kThreads), smem, s, tm_t, tm_r, a, seg) !=
            cudaSuccess)
            return SEMSHARE_ECUDA;
        return launch_status();
    }

    const int64_t pieces = (n_tgt + n_ref) * (plan.kpad / 16);
    const int64_t eg = (pieces + 255) / 256;
    CandTableFor<kSelect> none{};
    if (launch_pdl(expand_codes_kernel<kSelect>, dim3(static_cast<unsigned>(eg < sms * 8 ? eg : sms * 8)), dim3(256), 0,
                   s, tgt_codes, n_tgt, ref_codes, n_ref, nbits, plan.kpad, tpm, rpm, keys, n_tgt * seg.n_seg, counter,
                   best, cand ? *cand : none, sel, err_flag) != cudaSuccess)
        return SEMSHARE_ECUDA;
    if (launch_pdl(kernel, dim3(static_cast<unsigned>(grid)), dim3(kThreads), smem, s, tm_t, tm_r, a, seg) !=
        cudaSuccess)
        return SEMSHARE_ECUDA;
    return launch_status();
}

}  // namespace
}  // namespace semshare

extern "C" size_t semshare_match_tc_workspace_size(int64_t n_tgt, int64_t n_ref, int32_t nbits) {
    using namespace semshare;
    if (n_tgt <= 0 || n_ref <= 0 || nbits < 32 || nbits > 256 || nbits % 32 != 0) return 0;
    TcPlan p;
    plan_tc(n_tgt, n_ref, nbits, 0, &p);
    return p.total();
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
    plan_tc(n_tgt, n_ref, nbits, 0, &plan);
    if (workspace_bytes < plan.total()) return SEMSHARE_EINVAL;

    int sms = 0, dev = 0;
    if (current_sm_count(&sms, &dev) != SEMSHARE_OK) return SEMSHARE_ECUDA;
    cudaStream_t s = as_stream(stream);
    SegTable<1> seg{};
    seg.n_seg = 1;
    seg.off[0] = 0;
    seg.off[1] = n_ref;
    const semshare_status st = launch_search(tgt_codes, n_tgt, ref_codes, n_ref, nbits, seg, plan, workspace,
                                             err_flag, s, sms, dev);
    if (st != SEMSHARE_OK) return st;
    const int small = static_cast<int>((n_tgt + 255) / 256 < sms * 4 ? (n_tgt + 255) / 256 : sms * 4);
    if (launch_pdl(tc_keys_split_kernel, dim3(small), dim3(256), 0, s, static_cast<unsigned long long*>(workspace),
                   n_tgt, idx, dist, static_cast<const int64_t*>(nullptr), false) != cudaSuccess)
        return SEMSHARE_ECUDA;
    return launch_status();
}

extern "C" size_t semshare_match_tc_signs_workspace_size(int64_t n_tgt) {
    using namespace semshare;
    if (n_tgt <= 0) return 0;
    return round256(static_cast<size_t>(n_tgt) * 8) + 256;  // keys, then the arrival counter
}

extern "C" semshare_status semshare_match_tc_signs(const uint8_t* tgt_signs, int64_t n_tgt, const uint8_t* ref_signs,
                                                   int64_t n_ref, int32_t nbits, int32_t* idx, int32_t* dist,
                                                   void* workspace, size_t workspace_bytes, uint32_t* err_flag,
                                                   void* stream) {
    using namespace semshare;
    if (n_tgt < 0 || n_ref < 1) return SEMSHARE_EINVAL;
    if (nbits < 32 || nbits > 256 || nbits % 32 != 0) return SEMSHARE_EUNSUPPORTED;
    if (n_tgt >= (int64_t(1) << 31) || n_ref >= (int64_t(1) << 31)) return SEMSHARE_EUNSUPPORTED;
    if (n_tgt == 0) return SEMSHARE_OK;
    if (!tgt_signs || !ref_signs || !idx || !workspace) return SEMSHARE_EINVAL;
    if (!aligned(tgt_signs, 16) || !aligned(ref_signs, 16) || !aligned(idx, 4) || !aligned(workspace, 256) ||
        (dist && !aligned(dist, 4)) || (err_flag && !aligned(err_flag, 4)))
        return SEMSHARE_EINVAL;
    if (workspace_bytes < semshare_match_tc_signs_workspace_size(n_tgt)) return SEMSHARE_EINVAL;
    TcPlan plan;
    plan_tc(n_tgt, n_ref, nbits, 0, &plan);

    int sms = 0, dev = 0;
    if (current_sm_count(&sms, &dev) != SEMSHARE_OK) return SEMSHARE_ECUDA;
    cudaStream_t s = as_stream(stream);
    SegTable<1> seg{};
    seg.n_seg = 1;
    seg.off[0] = 0;
    seg.off[1] = n_ref;
    auto* keys = static_cast<unsigned long long*>(workspace);
    auto* counter = reinterpret_cast<unsigned int*>(static_cast<uint8_t*>(workspace) + round256(static_cast<size_t>(n_tgt) * 8));
    const bool fused = n_tgt <= kFusedSplitMaxTargets;
    const semshare_status st = launch_search(static_cast<const uint32_t*>(nullptr), n_tgt,
                                             static_cast<const uint32_t*>(nullptr), n_ref, nbits, seg, plan, workspace,
                                             err_flag, s, sms, dev, nullptr, nullptr, nullptr, tgt_signs, ref_signs,
                                             fused ? idx : nullptr, fused ? dist : nullptr, fused ? counter : nullptr);
    if (st != SEMSHARE_OK || fused) return st;
    const int small = static_cast<int>((n_tgt + 255) / 256 < sms * 4 ? (n_tgt + 255) / 256 : sms * 4);
    if (launch_pdl(tc_keys_split_kernel, dim3(small), dim3(256), 0, s, keys, n_tgt, idx, dist,
                   static_cast<const int64_t*>(nullptr), true) != cudaSuccess)
        return SEMSHARE_ECUDA;
    return launch_status();
}

namespace {
// Longest candidate of a pool, or -1 for bad offsets.
int64_t longest_candidate(const int64_t* off, int32_t n_cand) {
    if (off[0] != 0) return -1;
    int64_t m = 0;
    for (int32_t c = 0; c < n_cand; ++c) {
        if (off[c + 1] <= off[c]) return -1;
        m = off[c + 1] - off[c] > m ? off[c + 1] - off[c] : m;
    }
    return m;
}
}  // namespace

extern "C" size_t semshare_match_tc_selected_workspace_size(int64_t n_tgt, const int64_t* cand_offsets, int32_t n_cand,
                                                           int32_t nbits) {
    using namespace semshare;
    if (n_tgt <= 0 || !cand_offsets || n_cand < 1 || n_cand > SEMSHARE_RETRIEVE_MAX_CANDIDATES || nbits < 32 ||
        nbits > 256 || nbits % 32 != 0)
        return 0;
    const int64_t len = longest_candidate(cand_offsets, n_cand);
    if (len < 1) return 0;
    TcPlan p;
    plan_tc(n_tgt, len, nbits, 0, &p);
    return p.total() + 256;  // + the chosen candidate's length and first row
}

extern "C" semshare_status semshare_match_tc_selected(const uint32_t* tgt_codes, int64_t n_tgt,
                                                      const uint32_t* pool_codes, const int64_t* cand_offsets,
                                                      int32_t n_cand, const int32_t* best, int32_t nbits,
                                                      int32_t* idx, int32_t* dist, void* workspace,
                                                      size_t workspace_bytes, uint32_t* err_flag, void* stream) {
    using namespace semshare;
    if (n_cand < 1 || !cand_offsets || n_tgt < 0) return SEMSHARE_EINVAL;
    if (n_cand > SEMSHARE_RETRIEVE_MAX_CANDIDATES) return SEMSHARE_EUNSUPPORTED;
    if (nbits < 32 || nbits > 256 || nbits % 32 != 0) return SEMSHARE_EUNSUPPORTED;
    const int64_t len = longest_candidate(cand_offsets, n_cand);
    if (len < 1) return SEMSHARE_EINVAL;
    if (n_tgt >= (int64_t(1) << 31) || cand_offsets[n_cand] >= (int64_t(1) << 31)) return SEMSHARE_EUNSUPPORTED;
    if (n_tgt == 0) return SEMSHARE_OK;
    if (!tgt_codes || !pool_codes || !best || !idx || !workspace) return SEMSHARE_EINVAL;
    if (!aligned(tgt_codes, 4) || !aligned(pool_codes, 4) || !aligned(best, 4) || !aligned(idx, 4) ||
        !aligned(workspace, 256) || (dist && !aligned(dist, 4)) || (err_flag && !aligned(err_flag, 4)))
        return SEMSHARE_EINVAL;
    TcPlan plan;
    plan_tc(n_tgt, len, nbits, 0, &plan);
    if (workspace_bytes < plan.total() + 256) return SEMSHARE_EINVAL;

    int sms = 0, dev = 0;
    if (current_sm_count(&sms, &dev) != SEMSHARE_OK) return SEMSHARE_ECUDA;
    cudaStream_t s = as_stream(stream);
    SegTable<1> seg{};
    seg.n_seg = 1;
    seg.off[0] = 0;
    seg.off[1] = len;
    CandTableFor<true> cand{};
    cand.n_cand = n_cand;
    for (int32_t c = 0; c <= n_cand; ++c) cand.off[c] = cand_offsets[c];
    auto* sel = reinterpret_cast<int64_t*>(static_cast<uint8_t*>(workspace) + plan.total());
    const semshare_status st = launch_search<1, true>(tgt_codes, n_tgt, pool_codes, len, nbits, seg, plan, workspace,
                                                      err_flag, s, sms, dev, best, &cand, sel);
    if (st != SEMSHARE_OK) return st;
    const int small = static_cast<int>((n_tgt + 255) / 256 < sms * 4 ? (n_tgt + 255) / 256 : sms * 4);
    if (launch_pdl(tc_keys_split_kernel, dim3(small), dim3(256), 0, s, static_cast<unsigned long long*>(workspace),
                   n_tgt, idx, dist, static_cast<const int64_t*>(sel), false) != cudaSuccess)
        return SEMSHARE_ECUDA;
    return launch_status();
}

extern "C" size_t semshare_retrieve_workspace_size(int64_t n_tgt, int64_t n_pool, int32_t n_cand, int32_t nbits) {
    using namespace semshare;
    if (n_tgt <= 0 || n_pool <= 0 || n_cand < 1 || n_cand > SEMSHARE_RETRIEVE_MAX_CANDIDATES || nbits < 32 ||
        nbits > 256 || nbits % 32 != 0)
        return 0;
    TcPlan p;
    plan_tc(n_tgt, n_pool, nbits, n_cand, &p);
    return p.total();
}

extern "C" semshare_status semshare_retrieve(const uint32_t* tgt_codes, int64_t n_tgt, const uint32_t* pool_codes,
                                             const int64_t* cand_offsets, int32_t n_cand, int32_t nbits,
                                             double max_dist, double threshold, double* mean_dist,
                                             double* similarity, int32_t* best, int32_t* applies, int32_t* idx,
                                             int32_t* dist, void* workspace, size_t workspace_bytes,
                                             uint32_t* err_flag, void* stream) {
    using namespace semshare;
    if (n_cand < 1 || !cand_offsets || n_tgt < 1) return SEMSHARE_EINVAL;
    if (n_cand > SEMSHARE_RETRIEVE_MAX_CANDIDATES) return SEMSHARE_EUNSUPPORTED;
    if (nbits < 32 || nbits > 256 || nbits % 32 != 0) return SEMSHARE_EUNSUPPORTED;
    if (!(max_dist > 0.0) || !(max_dist <= 1.0e300) || threshold != threshold) return SEMSHARE_EINVAL;
    if (cand_offsets[0] != 0) return SEMSHARE_EINVAL;
    for (int32_t c = 0; c < n_cand; ++c)
        if (cand_offsets[c + 1] <= cand_offsets[c]) return SEMSHARE_EINVAL;
    const int64_t n_pool = cand_offsets[n_cand];
    if (n_tgt >= (int64_t(1) << 31) || n_pool >= (int64_t(1) << 31)) return SEMSHARE_EUNSUPPORTED;
    if (!tgt_codes || !pool_codes || !best || !workspace) return SEMSHARE_EINVAL;
    if (!aligned(tgt_codes, 4) || !aligned(pool_codes, 4) || !aligned(best, 4) || !aligned(workspace, 256) ||
        (applies && !aligned(applies, 4)) || (mean_dist && !aligned(mean_dist, 8)) ||
        (similarity && !aligned(similarity, 8)) || (idx && !aligned(idx, 4)) || (dist && !aligned(dist, 4)) ||
        (err_flag && !aligned(err_flag, 4)))
        return SEMSHARE_EINVAL;
    TcPlan plan;
    plan_tc(n_tgt, n_pool, nbits, n_cand, &plan);
    if (workspace_bytes < plan.total()) return SEMSHARE_EINVAL;

    int sms = 0, dev = 0;
    if (current_sm_count(&sms, &dev) != SEMSHARE_OK) return SEMSHARE_ECUDA;
    cudaStream_t s = as_stream(stream);
    SegTable<SEMSHARE_RETRIEVE_MAX_CANDIDATES> seg{};
    seg.n_seg = n_cand;
    for (int32_t c = 0; c <= n_cand; ++c) seg.off[c] = cand_offsets[c];
    semshare_status st = launch_search(tgt_codes, n_tgt, pool_codes, n_pool, nbits, seg, plan, workspace, err_flag,
                                       s, sms, dev);
    if (st != SEMSHARE_OK) return st;
    auto* keys = static_cast<const unsigned long long*>(workspace);
    auto* sums = reinterpret_cast<long long*>(static_cast<uint8_t*>(workspace) + plan.keys_bytes + plan.t_bytes +
                                              plan.r_bytes);
    auto* counter = reinterpret_cast<unsigned int*>(sums + n_cand);
    if (launch_pdl(retrieve_finalize_kernel, dim3(n_cand), dim3(256), 0, s, keys, n_tgt, n_cand, max_dist, threshold, sums,
                   counter, mean_dist, similarity, best, applies) != cudaSuccess)
        return SEMSHARE_ECUDA;
    if (launch_status() != SEMSHARE_OK) return SEMSHARE_ECUDA;
    if (idx || dist) {
        const int small = static_cast<int>((n_tgt + 255) / 256 < sms * 4 ? (n_tgt + 255) / 256 : sms * 4);
        if (launch_pdl(retrieve_select_kernel, dim3(small), dim3(256), 0, s, keys, n_tgt, best, idx, dist) !=
            cudaSuccess)
            return SEMSHARE_ECUDA;
        st = launch_status();
    }
    return st;
}
