// deviation.cu -- semshare_kv_deviation and semshare_select_hd: the Key-Value deviation of the
// reused (rearranged) cache against the recomputed one, and the high-deviation (HD) tokens.
//
// What it computes (SemShareKV, arXiv 2509.24832): App. A.4 defines sigma_K = ||K_reused -
// K_recomputed||_2, sigma_V likewise and sigma_KV = sigma_K + sigma_V; here per layer and token,
// the norm running over all KV heads and head dimensions of that token.  On the first layer
// every token is recomputed and compared with the rearranged cache (Sec. 3.2); the tokens of
// highest deviation -- 40% of them in Insight 1 -- are the HD tokens handed to recomputation.
//
// kv_deviation_kernel: one warp per (layer, token), grid-stride over a grid of resident CTAs.  The warp streams the token's H rows of K
// and V from both caches with 16-byte non-allocating loads (all of a lane's loads issued before
// its arithmetic), squares the differences in fp32 and reduces with a fixed shuffle tree, so the
// result does not depend on timing.  HBM-bound: 4 x H x hd x element bytes per token.
//
// hd_select_kernel: one CTA per layer.  A 4-pass radix select (8 bits per pass, from the top)
// over the order-preserving integer image of the fp32 deviations finds the k-th largest value;
// a block scan then lists, in ascending token order, every token above it and the lowest-index
// tokens equal to it until k are taken.  The deviations of a layer are staged in shared memory
// when they fit, else re-read from global memory (L2) in every pass.
#include <cuda_runtime.h>

#include "common.cuh"

namespace semshare {
namespace {

constexpr int kDevThreads = 256;
constexpr int kSelThreads = 1024;
constexpr int kMaxRowChunks = 16;  // 16-byte chunks per lane held in flight per array

struct DevArgs {
    const uint8_t* k_re;
    const uint8_t* v_re;
    const uint8_t* k_rc;
    const uint8_t* v_rc;
    int64_t re_layer, re_head, re_tok;  // strides in bytes
    int64_t rc_layer, rc_head, rc_tok;
    int32_t n_layers, n_heads, row_chunks;  // row_chunks = 16-byte chunks per head row
    int32_t is_f32;
    int64_t n_tok;
    float* sigma_k;
    float* sigma_v;
    float* sigma_kv;
};

__device__ __forceinline__ uint4 ld_stream(const uint8_t* p) {
    uint4 v;
    asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(p));
    return v;
}

// Sum of squared differences of the 8 bf16 (or 4 fp32) values in two 16-byte chunks.
__device__ __forceinline__ float sq_diff(uint4 a, uint4 b, int is_f32, float acc) {
    const uint32_t x[4] = {a.x, a.y, a.z, a.w}, y[4] = {b.x, b.y, b.z, b.w};
    if (is_f32) {
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const float d = __uint_as_float(x[i]) - __uint_as_float(y[i]);
            acc = fmaf(d, d, acc);
        }
    } else {
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const float d0 = __uint_as_float(x[i] << 16) - __uint_as_float(y[i] << 16);
            const float d1 = __uint_as_float(x[i] & 0xFFFF0000u) - __uint_as_float(y[i] & 0xFFFF0000u);
            acc = fmaf(d0, d0, acc);
            acc = fmaf(d1, d1, acc);
        }
    }
    return acc;
}

__device__ __forceinline__ void deviation_of_token(const DevArgs& a, int64_t w, int lane) {
    const int64_t l = w / a.n_tok, t = w - l * a.n_tok;
    const int total = a.n_heads * a.row_chunks;  // chunks per token per array
    const uint8_t* kre = a.k_re + l * a.re_layer + t * a.re_tok;
    const uint8_t* vre = a.v_re + l * a.re_layer + t * a.re_tok;
    const uint8_t* krc = a.k_rc + l * a.rc_layer + t * a.rc_tok;
    const uint8_t* vrc = a.v_rc + l * a.rc_layer + t * a.rc_tok;
    float sk = 0.0f, sv = 0.0f;
    for (int c0 = lane; c0 < total; c0 += 32 * kMaxRowChunks / 4) {
        uint4 xk[kMaxRowChunks / 4], yk[kMaxRowChunks / 4], xv[kMaxRowChunks / 4], yv[kMaxRowChunks / 4];
#pragma unroll
        for (int i = 0; i < kMaxRowChunks / 4; ++i) {
            const int c = c0 + 32 * i;
            if (c < total) {
                const int h = c / a.row_chunks, q = c - h * a.row_chunks;
                const int64_t ore = h * a.re_head + q * 16, orc = h * a.rc_head + q * 16;
                xk[i] = ld_stream(kre + ore);
                yk[i] = ld_stream(krc + orc);
                xv[i] = ld_stream(vre + ore);
                yv[i] = ld_stream(vrc + orc);
            }
        }
#pragma unroll
        for (int i = 0; i < kMaxRowChunks / 4; ++i)
            if (c0 + 32 * i < total) {
                sk = sq_diff(xk[i], yk[i], a.is_f32, sk);
                sv = sq_diff(xv[i], yv[i], a.is_f32, sv);
            }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        sk += __shfl_xor_sync(0xFFFFFFFFu, sk, o);
        sv += __shfl_xor_sync(0xFFFFFFFFu, sv, o);
    }
    if (lane == 0) {
        const float rk = sqrtf(sk), rv = sqrtf(sv);
        const int64_t o = l * a.n_tok + t;
        if (a.sigma_k) a.sigma_k[o] = rk;
        if (a.sigma_v) a.sigma_v[o] = rv;
        a.sigma_kv[o] = rk + rv;
    }
}

// Grid-stride over (layer, token) items, one warp each; the grid is the resident CTAs.
__global__ void __launch_bounds__(kDevThreads) kv_deviation_kernel(const DevArgs a) {
    pdl_prologue();
    const int lane = threadIdx.x & 31;
    const int64_t n_items = static_cast<int64_t>(a.n_layers) * a.n_tok;
    const int64_t n_warps = static_cast<int64_t>(gridDim.x) * (kDevThreads / 32);
    for (int64_t w = (static_cast<int64_t>(blockIdx.x) * kDevThreads + threadIdx.x) >> 5; w < n_items; w += n_warps)
        deviation_of_token(a, w, lane);
}

// Order-preserving image of an fp32 value as an unsigned integer under the selection's total
// order: every NaN, of either sign and any payload, maps to the one largest key (above +inf, and
// tied with every other NaN, so the lower token wins); -0 maps to the key of +0.
__device__ __forceinline__ uint32_t order_key(float f) {
    uint32_t u = __float_as_uint(f);
    if ((u & 0x7FFFFFFFu) > 0x7F800000u) return 0xFFFFFFFFu;  // NaN (exponent all ones, mantissa != 0)
    if (u == 0x80000000u) u = 0u;
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// Block-wide exclusive scan of one int per thread (kSelThreads threads); returns the
// exclusive prefix and writes the block total.
__device__ __forceinline__ int block_exclusive_scan(int v, int* warp_tot, int* total) {
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    int inc = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int n = __shfl_up_sync(0xFFFFFFFFu, inc, o);
        if (lane >= o) inc += n;
    }
    if (lane == 31) warp_tot[wid] = inc;
    __syncthreads();
    if (wid == 0) {
        int s = lane < kSelThreads / 32 ? warp_tot[lane] : 0;
        int si = s;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int n = __shfl_up_sync(0xFFFFFFFFu, si, o);
            if (lane >= o) si += n;
        }
        if (lane < kSelThreads / 32) warp_tot[lane] = si - s;  // exclusive warp offsets
        if (lane == 31) *total = si;
    }
    __syncthreads();
    const int r = warp_tot[wid] + inc - v;
    __syncthreads();
    return r;
}

template <bool kStaged>
__global__ void __launch_bounds__(kSelThreads)
    hd_select_kernel(const float* __restrict__ sigma, int64_t n_tok, int64_t k, int32_t* __restrict__ hd_idx,
                     uint8_t* __restrict__ hd_mask) {
    pdl_prologue();
    extern __shared__ uint32_t staged[];
    __shared__ unsigned int hist[256];
    __shared__ int warp_tot[kSelThreads / 32];
    __shared__ int scan_total;
    __shared__ uint32_t s_prefix;
    __shared__ long long s_remaining;
    __shared__ unsigned s_count_eq;
    const int64_t l = blockIdx.x;
    const float* row = sigma + l * n_tok;
    if (kStaged) {
        for (int64_t t = threadIdx.x; t < n_tok; t += kSelThreads) staged[t] = order_key(row[t]);
        __syncthreads();
    }
    auto key = [&](int64_t t) -> uint32_t { return kStaged ? staged[t] : order_key(__ldg(row + t)); };

    uint32_t prefix = 0, mask = 0;
    long long remaining = k;  // tokens still to take among those matching the prefix
    if (k > 0) {
        for (int shift = 24; shift >= 0; shift -= 8) {
            for (int i = threadIdx.x; i < 256; i += kSelThreads) hist[i] = 0u;
            __syncthreads();
            // warp-aggregated: deviations of one range share their top digits, so lanes with the
            // same digit add once (one shared atomic per distinct digit per warp)
            for (int64_t base = 0; base < n_tok; base += kSelThreads) {
                const int64_t t = base + threadIdx.x;
                const uint32_t kk = t < n_tok ? key(t) : 0u;
                const bool in = t < n_tok && (kk & mask) == prefix;
                const uint32_t digit = in ? (kk >> shift) & 0xFFu : 0x100u;
                const unsigned peers = __match_any_sync(0xFFFFFFFFu, digit);
                if (in && (threadIdx.x & 31) == __ffs(peers) - 1) atomicAdd(&hist[digit], __popc(peers));
            }
            __syncthreads();
            if (threadIdx.x < 32) {
                // lane i owns digits 255-8i .. 248-8i; a suffix scan over lanes finds the digit d
                // with count(digits > d) < remaining <= count(digits >= d)
                const int lane = threadIdx.x;
                unsigned own = 0;
#pragma unroll
                for (int j = 0; j < 8; ++j) own += hist[255 - 8 * lane - j];
                unsigned incl = own;
#pragma unroll
                for (int o = 1; o < 32; o <<= 1) {
                    const unsigned n = __shfl_up_sync(0xFFFFFFFFu, incl, o);
                    if (lane >= o) incl += n;
                }
                const unsigned excl = incl - own;
                const bool hit = excl < remaining && static_cast<long long>(incl) >= remaining;
                const unsigned who = __ballot_sync(0xFFFFFFFFu, hit);
                if (lane == __ffs(who) - 1) {
                    long long above = excl;
                    int d = 255 - 8 * lane;
                    for (int j = 0; j < 7; ++j, --d) {
                        if (above + hist[d] >= remaining) break;
                        above += hist[d];
                    }
                    s_prefix = prefix | (static_cast<uint32_t>(d) << shift);
                    s_remaining = remaining - above;
                    s_count_eq = hist[d];  // after the last pass: the keys equal to the k-th
                }
            }
            __syncthreads();
            prefix = s_prefix;
            remaining = s_remaining;
            mask |= 0xFFu << shift;
        }
    }
    // prefix is now the k-th largest key; take every key above it and the first `remaining`
    // (lowest-index) keys equal to it.  Each thread takes 4 consecutive tokens per chunk, so the
    // output stays in token order; when every equal key is taken (the usual case) the scan of
    // equal-key ranks is skipped.
    const uint32_t kth = prefix;
    const bool take_all_eq = k == 0 || static_cast<long long>(s_count_eq) == remaining;
    int64_t eq_before = 0, sel_before = 0;
    for (int64_t base = 0; base < n_tok; base += 4 * kSelThreads) {
        const int64_t t0 = base + 4 * static_cast<int64_t>(threadIdx.x);
        int gt[4], eq[4], n_eq = 0;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int64_t t = t0 + j;
            const bool live = t < n_tok && k > 0;
            const uint32_t kk = live ? key(t) : 0u;
            gt[j] = live && kk > kth;
            eq[j] = live && kk == kth;
            n_eq += eq[j];
        }
        int eq_rank = 0, eq_total = 0;
        if (!take_all_eq) {
            eq_rank = block_exclusive_scan(n_eq, warp_tot, &scan_total);
            eq_total = scan_total;
        }
        int sel[4], n_sel = 0;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            sel[j] = gt[j] || (eq[j] && (take_all_eq || eq_before + eq_rank < remaining));
            eq_rank += eq[j];
            n_sel += sel[j];
        }
        int pos = block_exclusive_scan(n_sel, warp_tot, &scan_total);
        const int sel_total = scan_total;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int64_t t = t0 + j;
            if (sel[j]) hd_idx[l * k + sel_before + pos++] = static_cast<int32_t>(t);
            if (hd_mask && t < n_tok) hd_mask[l * n_tok + t] = static_cast<uint8_t>(sel[j]);
        }
        eq_before += eq_total;
        sel_before += sel_total;
    }
}

bool layouts_match(const semshare_kv_layout& a, const semshare_kv_layout& b) {
    return a.n_layers == b.n_layers && a.n_heads == b.n_heads && a.head_dim == b.head_dim &&
           a.elem_bytes == b.elem_bytes;
}

bool layout_aligned(const semshare_kv_layout& y) {
    const int64_t e = y.elem_bytes;
    return (y.stride_layer * e) % 16 == 0 && (y.stride_head * e) % 16 == 0 && (y.stride_token * e) % 16 == 0 &&
           y.stride_layer >= 0 && y.stride_head >= 0 && y.stride_token >= 0;
}

}  // namespace
}  // namespace semshare

extern "C" semshare_status semshare_kv_deviation(const void* k_reused, const void* v_reused,
                                                 semshare_kv_layout reused, const void* k_recomp,
                                                 const void* v_recomp, semshare_kv_layout recomp,
                                                 semshare_dtype dtype, int64_t n_tok, float* sigma_k,
                                                 float* sigma_v, float* sigma_kv, void* stream) {
    using namespace semshare;
    if (dtype != SEMSHARE_BF16 && dtype != SEMSHARE_F32) return SEMSHARE_EINVAL;
    const int32_t esize = dtype == SEMSHARE_BF16 ? 2 : 4;
    if (!layouts_match(reused, recomp) || reused.elem_bytes != esize) return SEMSHARE_EINVAL;
    if (reused.n_layers < 0 || reused.n_heads < 1 || reused.head_dim < 1 || n_tok < 0) return SEMSHARE_EINVAL;
    const int64_t row_bytes = static_cast<int64_t>(reused.head_dim) * esize;
    if (row_bytes % 16 != 0 || !layout_aligned(reused) || !layout_aligned(recomp)) return SEMSHARE_EINVAL;
    if (static_cast<int64_t>(reused.n_heads) * (row_bytes / 16) >= (int64_t(1) << 30)) return SEMSHARE_EUNSUPPORTED;
    if (n_tok == 0 || reused.n_layers == 0) return SEMSHARE_OK;
    if (!k_reused || !v_reused || !k_recomp || !v_recomp || !sigma_kv) return SEMSHARE_EINVAL;
    for (const void* p : {k_reused, v_reused, k_recomp, v_recomp})
        if (!aligned(p, 16)) return SEMSHARE_EINVAL;
    if (!aligned(sigma_kv, 4) || (sigma_k && !aligned(sigma_k, 4)) || (sigma_v && !aligned(sigma_v, 4)))
        return SEMSHARE_EINVAL;
    DevArgs a{};
    a.k_re = static_cast<const uint8_t*>(k_reused);
    a.v_re = static_cast<const uint8_t*>(v_reused);
    a.k_rc = static_cast<const uint8_t*>(k_recomp);
    a.v_rc = static_cast<const uint8_t*>(v_recomp);
    a.re_layer = reused.stride_layer * esize;
    a.re_head = reused.stride_head * esize;
    a.re_tok = reused.stride_token * esize;
    a.rc_layer = recomp.stride_layer * esize;
    a.rc_head = recomp.stride_head * esize;
    a.rc_tok = recomp.stride_token * esize;
    a.n_layers = reused.n_layers;
    a.n_heads = reused.n_heads;
    a.row_chunks = static_cast<int32_t>(row_bytes / 16);
    a.is_f32 = dtype == SEMSHARE_F32;
    a.n_tok = n_tok;
    a.sigma_k = sigma_k;
    a.sigma_v = sigma_v;
    a.sigma_kv = sigma_kv;
    int sms = 0, per_sm = 0;
    if (current_sm_count(&sms, nullptr) != SEMSHARE_OK ||
        cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kv_deviation_kernel, kDevThreads, 0) != cudaSuccess)
        return SEMSHARE_ECUDA;
    const int64_t warps = static_cast<int64_t>(reused.n_layers) * n_tok;
    const int64_t need = (warps * 32 + kDevThreads - 1) / kDevThreads;
    const int64_t resident = static_cast<int64_t>(sms) * (per_sm > 0 ? per_sm : 1);
    const int64_t grid = need < resident ? need : resident;
    if (launch_pdl(kv_deviation_kernel, dim3(static_cast<unsigned>(grid)), dim3(kDevThreads), 0, as_stream(stream), a) !=
        cudaSuccess)
        return SEMSHARE_ECUDA;
    return launch_status();
}

extern "C" semshare_status semshare_select_hd(const float* sigma, int32_t n_layers, int64_t n_tok, int64_t k,
                                              int32_t* hd_idx, uint8_t* hd_mask, void* stream) {
    using namespace semshare;
    if (n_layers < 0 || n_tok < 0 || k < 0 || k > n_tok) return SEMSHARE_EINVAL;
    if (n_tok >= (int64_t(1) << 31) || n_layers > 65535) return SEMSHARE_EUNSUPPORTED;
    if (n_layers == 0 || n_tok == 0) return SEMSHARE_OK;
    if (!sigma || (k > 0 && !hd_idx)) return SEMSHARE_EINVAL;
    if (!aligned(sigma, 4) || (hd_idx && !aligned(hd_idx, 4))) return SEMSHARE_EINVAL;
    int dev = 0, smem_optin = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess)
        return SEMSHARE_ECUDA;
    const size_t stage = static_cast<size_t>(n_tok) * 4;
    const size_t static_smem = 256 * 4 + (kSelThreads / 32) * 4 + 64;
    cudaStream_t s = as_stream(stream);
    if (stage + static_smem <= static_cast<size_t>(smem_optin)) {
        if (stage > 48 * 1024 && cudaFuncSetAttribute(hd_select_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                      static_cast<int>(stage)) != cudaSuccess)
            return SEMSHARE_ECUDA;
        if (launch_pdl(hd_select_kernel<true>, dim3(n_layers), dim3(kSelThreads), stage, s, sigma, n_tok, k, hd_idx,
                       hd_mask) != cudaSuccess)
            return SEMSHARE_ECUDA;
    } else {
        if (launch_pdl(hd_select_kernel<false>, dim3(n_layers), dim3(kSelThreads), 0, s, sigma, n_tok, k, hd_idx,
                       hd_mask) != cudaSuccess)
            return SEMSHARE_ECUDA;
    }
    return launch_status();
}
