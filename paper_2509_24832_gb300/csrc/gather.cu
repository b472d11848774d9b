// gather.cu -- semshare_gather_kv: rearrange the reference K/V cache into the target's token
// order with 16-byte vector copies.
//
// What it computes (SemShareKV, arXiv 2509.24832): Sec. 3.3 reorders the reference prompt's
// KV cache token by token so that it has the target's length and every pair comes from the
// reference cache; Sec. 3.3.2 stores K/V after RoPE, so rows move bit for bit.  For prompt b,
// layer l, KV head h, token t:  out[b][l][h][t] = ref[l][h][idx[b][t]]  (K and V alike).
//
// Kernel design.  Pure streaming copy, bound by HBM bandwidth.  A CTA owns 64 target tokens
// of one (b, l, h) plane and moves their 64 K rows and 64 V rows: it resolves the 64 indices
// once (segment and local row, bounds-checked) into shared memory, then every thread issues
// all of its 16-byte loads (read-only path) before any of its stores, so each thread keeps
// 2*64*row_bytes/(16*256) requests in flight.  Consecutive threads touch consecutive 16-byte
// chunks of a row and consecutive rows of the destination.  The loads are cached in L1: the
// CTAs resident on one SM often read the same reference rows (a row several targets select;
// with several target prompts, the same token block of each prompt, which similar prompts map
// to nearby reference rows).  With several target prompts the stores are marked evict-first,
// so the reference planes that every prompt re-reads stay in L2 while the output streams out.
//
// Retention (semshare_gather_kv_retained; Sec. 3.3.4, App. A: Retain[i] = T * prod alpha_retain,
// evicted tokens dropped): each layer keeps only the target tokens of its list, and its cache
// holds just their rows, packed in list order -- out[l][h][r] = ref[l][h][idx[ret_l[r]]].  The
// same kernels run with the token index remapped through the layer's list; CTAs past a layer's
// count exit at once, so evicted tokens cost neither reads nor writes.
#include "common.cuh"

namespace semshare {
namespace {

constexpr int kThreads = 256;
constexpr int kTokens = 64;  // target tokens per CTA
constexpr int kMaxSeg = 64;

// Per-layer retained-token lists (ret[off[l] .. off[l+1]) for layer l), passed by value.
template <int kMax>
struct RetTable {
    const int32_t* ret;
    int64_t off[kMax + 1];
};
using NoRet = RetTable<1>;
using Ret = RetTable<SEMSHARE_RETAIN_MAX_LAYERS>;

struct GatherArgs {
    const uint8_t* src_k[kMaxSeg];
    const uint8_t* src_v[kMaxSeg];
    int64_t seg_off[kMaxSeg + 1];
    int32_t n_seg;
    int32_t n_layers;
    int32_t n_heads;
    int32_t n_batch;
    int32_t stream_out;  // 1: evict-first stores (several target prompts share the reference)
    int64_t n_tgt;
    int64_t s_layer, s_head, s_token;           // source strides, bytes
    int64_t d_batch, d_layer, d_head, d_token;  // destination strides, bytes
    const int32_t* idx;
    uint8_t* dst_k;
    uint8_t* dst_v;
    uint32_t* err_flag;
};

__device__ __forceinline__ uint4 load_row(const void* p) {
    uint4 v;
    asm volatile("ld.global.nc.v4.u32 {%0, %1, %2, %3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "l"(p));
    return v;
}

// stream = 1: evict-first (st.global.cs), the output is not re-read soon.  Uniform over the grid.
__device__ __forceinline__ void store_vec(void* p, const uint4& v, int32_t stream) {
    if (stream)
        asm volatile("st.global.cs.v4.u32 [%0], {%1, %2, %3, %4};" ::"l"(p), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w)
                     : "memory");
    else
        asm volatile("st.global.v4.u32 [%0], {%1, %2, %3, %4};" ::"l"(p), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w)
                     : "memory");
}

// Resolves the CTA's kTokens rows into their source row addresses in shared memory (K and V;
// nullptr = skip: tail or bad index).  Returns false when the CTA has nothing to move (past its
// layer's retained count).
template <bool kRetain, typename RT>
__device__ __forceinline__ bool resolve_rows(const GatherArgs& a, const RT& rt, int l, int h, int64_t b, int64_t t0,
                                             const uint8_t** s_src_k, const uint8_t** s_src_v) {
    int64_t count = a.n_tgt, base = 0;
    if (kRetain) {
        base = rt.off[l];
        count = rt.off[l + 1] - base;
        if (t0 >= count) return false;  // uniform over the CTA
    }
    if (threadIdx.x < kTokens) {
        const int64_t t = t0 + threadIdx.x;
        const uint8_t* pk = nullptr;
        const uint8_t* pv = nullptr;
        if (t < count) {
            int64_t tok = t;
            bool ok = true;
            if (kRetain) {
                tok = __ldg(rt.ret + base + t);
                ok = tok >= 0 && tok < a.n_tgt;
            }
            const int64_t r = ok ? __ldg(a.idx + b * a.n_tgt + tok) : -1;
            if (ok && r >= 0 && r < a.seg_off[a.n_seg]) {
                int seg = 0;
                while (r >= a.seg_off[seg + 1]) ++seg;
                const int64_t off = l * a.s_layer + h * a.s_head + (r - a.seg_off[seg]) * a.s_token;
                pk = a.src_k[seg] + off;
                pv = a.src_v[seg] + off;
            } else if (a.err_flag) {
                atomicOr(a.err_flag, SEMSHARE_FLAG_INDEX);
            }
        }
        s_src_k[threadIdx.x] = pk;
        s_src_v[threadIdx.x] = pv;
    }
    __syncthreads();
    return true;
}

// Rows of up to 16 chunks: at most 48 registers, so that 5 CTAs (1280 threads, 160 KB of loads in
// flight) are resident per SM; measured on GB300 against 4 CTAs (58 registers): equal at one
// prompt, 5% faster with 64 prompts sharing the reference; 6 CTAs spill.
template <int C>
constexpr int gather_min_ctas() { return C <= 16 ? 5 : 2; }

// C = 16-byte chunks per row (row_bytes / 16).
template <int C, bool kRetain, typename RT>
__global__ void __launch_bounds__(kThreads, gather_min_ctas<C>())
    kv_gather_kernel(const __grid_constant__ GatherArgs a, const __grid_constant__ RT rt) {
    pdl_prologue();
    constexpr int kRowsPerPass = kThreads / C;
    constexpr int kPasses = 2 * kTokens / kRowsPerPass;  // K rows then V rows
    static_assert(kThreads % C == 0 && (2 * kTokens) % kRowsPerPass == 0, "row split");

    __shared__ const uint8_t* s_src_k[kTokens];  // source rows, nullptr = skip (tail or bad index)
    __shared__ const uint8_t* s_src_v[kTokens];

    // planes in (l, h, b) order, b fastest: the target prompts that read one reference plane
    // (l, h) run back to back, so the plane's rows are still in L2 for all of them.  Layers go
    // last to first, so the first layer's rearranged rows -- which the KV deviation of App. A.4
    // reads next -- are the most recently written, still in L2.
    const int64_t plane = blockIdx.y + static_cast<int64_t>(gridDim.y) * blockIdx.z;
    const int64_t b = plane % a.n_batch;
    const int64_t lh = plane / a.n_batch;
    const int h = static_cast<int>(lh % a.n_heads);
    const int l = a.n_layers - 1 - static_cast<int>(lh / a.n_heads);
    const int64_t t0 = static_cast<int64_t>(blockIdx.x) * kTokens;
    if (!resolve_rows<kRetain>(a, rt, l, h, b, t0, s_src_k, s_src_v)) return;

    const int c = threadIdx.x % C;
    const int rr = threadIdx.x / C;
    uint4 v[kPasses];
#pragma unroll
    for (int p = 0; p < kPasses; ++p) {  // passes below kPasses/2 move K rows, the rest V rows
        const int tt = (rr + p * kRowsPerPass) % kTokens;
        const uint8_t* src = p < kPasses / 2 ? s_src_k[tt] : s_src_v[tt];
        if (src) v[p] = load_row(src + c * 16);
    }
    uint8_t* const dst_k = a.dst_k + b * a.d_batch + l * a.d_layer + h * a.d_head + t0 * a.d_token + c * 16;
    uint8_t* const dst_v = a.dst_v + (dst_k - a.dst_k);
#pragma unroll
    for (int p = 0; p < kPasses; ++p) {
        const int tt = (rr + p * kRowsPerPass) % kTokens;
        if (s_src_k[tt]) store_vec((p < kPasses / 2 ? dst_k : dst_v) + tt * a.d_token, v[p], a.stream_out);
    }
}

// Rows whose size is not a power-of-two number of 16-byte chunks: one chunk per thread per
// step over the CTA's rows.
template <bool kRetain, typename RT>
__global__ void __launch_bounds__(kThreads)
    kv_gather_generic_kernel(const __grid_constant__ GatherArgs a, const __grid_constant__ RT rt, int chunks) {
    pdl_prologue();
    __shared__ const uint8_t* s_src_k[kTokens];
    __shared__ const uint8_t* s_src_v[kTokens];
    const int64_t plane = blockIdx.y + static_cast<int64_t>(gridDim.y) * blockIdx.z;  // (l, h, b), b fastest
    const int64_t b = plane % a.n_batch;
    const int64_t lh = plane / a.n_batch;
    const int h = static_cast<int>(lh % a.n_heads);
    const int l = a.n_layers - 1 - static_cast<int>(lh / a.n_heads);  // last layer first
    const int64_t t0 = static_cast<int64_t>(blockIdx.x) * kTokens;
    if (!resolve_rows<kRetain>(a, rt, l, h, b, t0, s_src_k, s_src_v)) return;
    const int64_t dst_plane = b * a.d_batch + l * a.d_layer + h * a.d_head;
    const int total = 2 * kTokens * chunks;
    for (int e = threadIdx.x; e < total; e += kThreads) {
        const int row = e / chunks, c = e - row * chunks;
        const int tt = row % kTokens;
        const uint8_t* src = row < kTokens ? s_src_k[tt] : s_src_v[tt];
        if (!src) continue;
        uint8_t* dst = ((row < kTokens) ? a.dst_k : a.dst_v) + dst_plane + (t0 + tt) * a.d_token + c * 16;
        store_vec(dst, load_row(src + c * 16), a.stream_out);
    }
}

bool stride_ok(int64_t s, int64_t elem) { return s >= 0 && ((s * elem) % 16) == 0; }

// Validates the arguments shared by both entry points and fills `a` (n_batch, n_tgt, idx set
// by the caller).
semshare_status build_args(const void* const* ref_k, const void* const* ref_v, const int64_t* seg_offsets,
                           int32_t n_seg, const semshare_kv_layout& src, void* out_k, void* out_v,
                           const semshare_kv_layout& dst, uint32_t* err_flag, GatherArgs* a) {
    if (n_seg < 1 || n_seg > kMaxSeg || !ref_k || !ref_v || !seg_offsets) return SEMSHARE_EINVAL;
    if (src.n_layers < 1 || src.n_heads < 1 || src.head_dim < 1) return SEMSHARE_EINVAL;
    if (src.elem_bytes != 1 && src.elem_bytes != 2 && src.elem_bytes != 4 && src.elem_bytes != 8)
        return SEMSHARE_EINVAL;
    if (dst.n_layers != src.n_layers || dst.n_heads != src.n_heads || dst.head_dim != src.head_dim ||
        dst.elem_bytes != src.elem_bytes)
        return SEMSHARE_EINVAL;
    const int64_t eb = src.elem_bytes;
    const int64_t row_bytes = static_cast<int64_t>(src.head_dim) * eb;
    if (row_bytes % 16 != 0) return SEMSHARE_EINVAL;
    if (!stride_ok(src.stride_layer, eb) || !stride_ok(src.stride_head, eb) || !stride_ok(src.stride_token, eb) ||
        !stride_ok(dst.stride_batch, eb) || !stride_ok(dst.stride_layer, eb) || !stride_ok(dst.stride_head, eb) ||
        !stride_ok(dst.stride_token, eb))
        return SEMSHARE_EINVAL;
    if (seg_offsets[0] != 0) return SEMSHARE_EINVAL;
    for (int s = 0; s < n_seg; ++s) {
        if (seg_offsets[s + 1] < seg_offsets[s]) return SEMSHARE_EINVAL;
        if (seg_offsets[s + 1] > seg_offsets[s] && (!ref_k[s] || !ref_v[s] || !aligned(ref_k[s], 16) || !aligned(ref_v[s], 16)))
            return SEMSHARE_EINVAL;
    }
    if (seg_offsets[n_seg] >= (int64_t(1) << 31)) return SEMSHARE_EUNSUPPORTED;
    for (int s = 0; s < n_seg; ++s) {
        a->src_k[s] = static_cast<const uint8_t*>(ref_k[s]);
        a->src_v[s] = static_cast<const uint8_t*>(ref_v[s]);
    }
    for (int s = 0; s <= n_seg; ++s) a->seg_off[s] = seg_offsets[s];
    a->n_seg = n_seg;
    a->n_layers = src.n_layers;
    a->n_heads = src.n_heads;
    a->s_layer = src.stride_layer * eb;
    a->s_head = src.stride_head * eb;
    a->s_token = src.stride_token * eb;
    a->d_batch = dst.stride_batch * eb;
    a->d_layer = dst.stride_layer * eb;
    a->d_head = dst.stride_head * eb;
    a->d_token = dst.stride_token * eb;
    a->dst_k = static_cast<uint8_t*>(out_k);
    a->dst_v = static_cast<uint8_t*>(out_v);
    a->err_flag = err_flag;
    return SEMSHARE_OK;
}

template <bool kRetain, typename RT>
semshare_status launch_gather(const GatherArgs& a, const RT& rt, int64_t planes, int64_t tokens, int64_t row_bytes,
                              cudaStream_t s) {
    const int64_t tblocks = (tokens + kTokens - 1) / kTokens;
    if (tblocks > 0x7FFFFFFF) return SEMSHARE_EUNSUPPORTED;
    // planes tile the (y, z) grid exactly: y = the largest divisor of planes within 65535
    int64_t gy = planes < 65535 ? planes : 65535;
    while (planes % gy != 0) --gy;
    if (planes / gy > 65535) return SEMSHARE_EUNSUPPORTED;
    const dim3 grid(static_cast<unsigned>(tblocks), static_cast<unsigned>(gy), static_cast<unsigned>(planes / gy));
    const int chunks = static_cast<int>(row_bytes / 16);
    cudaError_t e;
    switch (chunks) {
        case 4: e = launch_pdl(kv_gather_kernel<4, kRetain, RT>, grid, dim3(kThreads), 0, s, a, rt); break;
        case 8: e = launch_pdl(kv_gather_kernel<8, kRetain, RT>, grid, dim3(kThreads), 0, s, a, rt); break;
        case 16: e = launch_pdl(kv_gather_kernel<16, kRetain, RT>, grid, dim3(kThreads), 0, s, a, rt); break;
        case 32: e = launch_pdl(kv_gather_kernel<32, kRetain, RT>, grid, dim3(kThreads), 0, s, a, rt); break;
        default: e = launch_pdl(kv_gather_generic_kernel<kRetain, RT>, grid, dim3(kThreads), 0, s, a, rt, chunks); break;
    }
    if (e != cudaSuccess) return SEMSHARE_ECUDA;
    return launch_status();
}

}  // namespace
}  // namespace semshare

extern "C" semshare_status semshare_gather_kv(const void* const* ref_k, const void* const* ref_v,
                                              const int64_t* seg_offsets, int32_t n_seg, semshare_kv_layout src,
                                              const int32_t* idx, int64_t n_tgt, int32_t n_batch, void* out_k,
                                              void* out_v, semshare_kv_layout dst, uint32_t* err_flag,
                                              void* stream) {
    using namespace semshare;
    if (n_tgt < 0 || n_batch < 0) return SEMSHARE_EINVAL;
    GatherArgs a{};
    const semshare_status st = build_args(ref_k, ref_v, seg_offsets, n_seg, src, out_k, out_v, dst, err_flag, &a);
    if (st != SEMSHARE_OK) return st;
    if (n_tgt == 0 || n_batch == 0) return SEMSHARE_OK;
    if (!idx || !out_k || !out_v || !aligned(idx, 4) || !aligned(out_k, 16) || !aligned(out_v, 16) ||
        (err_flag && !aligned(err_flag, 4)))
        return SEMSHARE_EINVAL;
    a.n_batch = n_batch;
    a.stream_out = n_batch > 1 ? 1 : 0;
    a.n_tgt = n_tgt;
    a.idx = idx;
    NoRet none{};
    const int64_t planes = static_cast<int64_t>(n_batch) * src.n_layers * src.n_heads;
    return launch_gather<false>(a, none, planes, n_tgt, static_cast<int64_t>(src.head_dim) * src.elem_bytes,
                                as_stream(stream));
}

extern "C" semshare_status semshare_gather_kv_retained(const void* const* ref_k, const void* const* ref_v,
                                                       const int64_t* seg_offsets, int32_t n_seg,
                                                       semshare_kv_layout src, const int32_t* idx, int64_t n_tgt,
                                                       const int32_t* retained, const int64_t* ret_offsets,
                                                       void* out_k, void* out_v, semshare_kv_layout dst,
                                                       uint32_t* err_flag, void* stream) {
    using namespace semshare;
    if (n_tgt < 0 || !ret_offsets) return SEMSHARE_EINVAL;
    if (src.n_layers > SEMSHARE_RETAIN_MAX_LAYERS) return SEMSHARE_EUNSUPPORTED;
    GatherArgs a{};
    const semshare_status st = build_args(ref_k, ref_v, seg_offsets, n_seg, src, out_k, out_v, dst, err_flag, &a);
    if (st != SEMSHARE_OK) return st;
    Ret rt{};
    if (ret_offsets[0] != 0) return SEMSHARE_EINVAL;
    int64_t longest = 0;
    for (int l = 0; l < src.n_layers; ++l) {
        const int64_t c = ret_offsets[l + 1] - ret_offsets[l];
        if (c < 0) return SEMSHARE_EINVAL;
        longest = c > longest ? c : longest;
    }
    for (int l = 0; l <= src.n_layers; ++l) rt.off[l] = ret_offsets[l];
    if (longest == 0) return SEMSHARE_OK;
    if (!retained || !idx || !out_k || !out_v || !aligned(retained, 4) || !aligned(idx, 4) || !aligned(out_k, 16) ||
        !aligned(out_v, 16) || (err_flag && !aligned(err_flag, 4)))
        return SEMSHARE_EINVAL;
    rt.ret = retained;
    a.n_batch = 1;
    a.n_tgt = n_tgt;
    a.idx = idx;
    const int64_t planes = static_cast<int64_t>(src.n_layers) * src.n_heads;
    return launch_gather<true>(a, rt, planes, longest, static_cast<int64_t>(src.head_dim) * src.elem_bytes,
                               as_stream(stream));
}
