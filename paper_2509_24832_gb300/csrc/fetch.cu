// fetch.cu -- semshare_fetch_rows: bring the reference K/V rows a match selects into device
// memory, each selected row once.
//
// Sec. 3.2 loads the retrieved reference prompt onto the GPU with its KV cache before the
// cache is rearranged (Sec. 3.3).  Only the rows the match selects are ever read by the
// rearrangement, and targets often select the same row, so this copies exactly the selected
// rows -- each once -- from caches that may live in page-locked host memory into device caches
// of the same layout; semshare_gather_kv then runs on the device copy.  The copy is bitwise.
//
// mark_rows_kernel: one byte per reference row, set where some target selects it (an index
// outside the reference sets SEMSHARE_FLAG_INDEX).  fetch_rows_kernel: for each 64 reference rows
// of one (layer, head) plane, the marked rows' K and V move as 16-byte vectors, all loads of a
// thread issued before its stores; unmarked rows are neither read nor written.
#include "common.cuh"

namespace semshare {
namespace {

constexpr int kThreads = 256;
constexpr int kRows = 64;  // reference rows per CTA
constexpr int kMaxSeg = 64;
constexpr int kCtasPerSm = 4;  // resident copy CTAs per SM: 4 x 16 KB of requests in flight per SM

struct FetchArgs {
    const uint8_t* src_k[kMaxSeg];
    const uint8_t* src_v[kMaxSeg];
    uint8_t* dst_k[kMaxSeg];
    uint8_t* dst_v[kMaxSeg];
    int64_t seg_off[kMaxSeg + 1];
    int32_t n_seg, n_layers, n_heads, chunks;  // chunks: 16-byte pieces per row
    int64_t s_layer, s_head, s_token;          // strides of every segment, bytes
    const uint8_t* map;                        // [n_rows] 1 = selected
    const uint8_t* block_map;                  // [rblocks] 1 = some row of the block is selected
};

__global__ void clear_map_kernel(uint8_t* __restrict__ map, int64_t n) {
    pdl_prologue();
    for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < n;
         i += static_cast<int64_t>(gridDim.x) * blockDim.x)
        map[i] = 0;
}

// map[r] = 1 for every selected row r, and block_map[r / kRows] = 1 for its block of rows.
__global__ void mark_rows_kernel(const int32_t* __restrict__ idx, int64_t n, int64_t n_rows, uint8_t* __restrict__ map,
                                 uint8_t* __restrict__ block_map, uint32_t* err_flag) {
    pdl_prologue();
    for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < n;
         i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int32_t r = __ldg(idx + i);
        if (r >= 0 && r < n_rows) {
            map[r] = 1;
            block_map[r / kRows] = 1;
        } else if (err_flag) {
            atomicOr(err_flag, SEMSHARE_FLAG_INDEX);
        }
    }
}

__device__ __forceinline__ uint4 ld_nc(const void* p) {
    uint4 v;
    asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(p));
    return v;
}

// Work item w = (plane, row block): plane = w / rblocks is one (layer, head), row block w % rblocks
// holds reference rows [64*rb, 64*rb + 64).  A persistent grid of a few CTAs per SM strides over
// the items: enough requests stay in flight to fill the host link (or HBM), and the SMs keep
// room for kernels of other streams (a gather of rows already fetched) to run alongside.
__global__ void __launch_bounds__(kThreads) fetch_rows_kernel(const __grid_constant__ FetchArgs a, int64_t n_rows,
                                                              int64_t rblocks, int64_t n_items) {
    pdl_prologue();
    __shared__ int64_t s_off[kRows];  // byte offset of the row inside its segment
    __shared__ int32_t s_seg[kRows];  // segment, -1 = not selected
    const int total = 2 * kRows * a.chunks;  // 2 * kRows rows (K then V) x chunks pieces
    for (int64_t w = blockIdx.x; w < n_items; w += gridDim.x) {
        const int64_t plane = w / rblocks;  // (l, h)
        const int64_t rb = w - plane * rblocks;
        if (!a.block_map[rb]) continue;  // no selected row here (the same for the whole CTA)
        const int h = static_cast<int>(plane % a.n_heads);
        const int l = static_cast<int>(plane / a.n_heads);
        const int64_t r0 = rb * kRows;
        if (threadIdx.x < kRows) {
            const int64_t r = r0 + threadIdx.x;
            int32_t seg = -1;
            int64_t off = 0;
            if (r < n_rows && a.map[r]) {
                seg = 0;
                while (r >= a.seg_off[seg + 1]) ++seg;
                off = l * a.s_layer + h * a.s_head + (r - a.seg_off[seg]) * a.s_token;
            }
            s_seg[threadIdx.x] = seg;
            s_off[threadIdx.x] = off;
        }
        __syncthreads();
        // 4 pieces per thread in flight: all loads before the stores
        for (int e0 = threadIdx.x; e0 < total; e0 += 4 * kThreads) {
            uint4 v[4];
            uint8_t* dst[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                dst[i] = nullptr;
                const int e = e0 + i * kThreads;
                if (e < total) {
                    const int row = e / a.chunks, c = e - row * a.chunks;
                    const int rr = row % kRows;
                    const int seg = s_seg[rr];
                    if (seg >= 0) {
                        const bool is_v = row >= kRows;
                        const int64_t o = s_off[rr] + c * 16;
                        v[i] = ld_nc((is_v ? a.src_v[seg] : a.src_k[seg]) + o);
                        dst[i] = (is_v ? a.dst_v[seg] : a.dst_k[seg]) + o;
                    }
                }
            }
#pragma unroll
            for (int i = 0; i < 4; ++i)
                if (dst[i]) *reinterpret_cast<uint4*>(dst[i]) = v[i];
        }
        __syncthreads();  // the next item rewrites the row table
    }
}

bool stride_ok(int64_t s, int64_t elem) { return s >= 0 && ((s * elem) % 16) == 0; }

}  // namespace
}  // namespace semshare

namespace {
size_t round256(size_t x) { return ((x + 255) / 256) * 256; }
}  // namespace

extern "C" size_t semshare_fetch_workspace_size(int64_t n_rows) {
    using namespace semshare;
    if (n_rows <= 0) return 0;
    const size_t rblocks = (static_cast<size_t>(n_rows) + kRows - 1) / kRows;
    return round256(static_cast<size_t>(n_rows)) + round256(rblocks);
}

extern "C" semshare_status semshare_fetch_rows(const void* const* ref_k, const void* const* ref_v,
                                               void* const* dev_k, void* const* dev_v, const int64_t* seg_offsets,
                                               int32_t n_seg, semshare_kv_layout layout, const int32_t* idx,
                                               int64_t n_idx, void* workspace, size_t workspace_bytes,
                                               uint32_t* err_flag, void* stream) {
    using namespace semshare;
    if (n_seg < 1 || n_seg > kMaxSeg || !ref_k || !ref_v || !dev_k || !dev_v || !seg_offsets || n_idx < 0)
        return SEMSHARE_EINVAL;
    if (layout.n_layers < 1 || layout.n_heads < 1 || layout.head_dim < 1) return SEMSHARE_EINVAL;
    if (layout.elem_bytes != 1 && layout.elem_bytes != 2 && layout.elem_bytes != 4 && layout.elem_bytes != 8)
        return SEMSHARE_EINVAL;
    const int64_t eb = layout.elem_bytes;
    const int64_t row_bytes = static_cast<int64_t>(layout.head_dim) * eb;
    if (row_bytes % 16 != 0 || !stride_ok(layout.stride_layer, eb) || !stride_ok(layout.stride_head, eb) ||
        !stride_ok(layout.stride_token, eb))
        return SEMSHARE_EINVAL;
    if (seg_offsets[0] != 0) return SEMSHARE_EINVAL;
    for (int s = 0; s < n_seg; ++s) {
        if (seg_offsets[s + 1] < seg_offsets[s]) return SEMSHARE_EINVAL;
        if (seg_offsets[s + 1] > seg_offsets[s]) {
            for (const void* p : {ref_k[s], ref_v[s], static_cast<const void*>(dev_k[s]), static_cast<const void*>(dev_v[s])})
                if (!p || !aligned(p, 16)) return SEMSHARE_EINVAL;
        }
    }
    const int64_t n_rows = seg_offsets[n_seg];
    if (n_rows >= (int64_t(1) << 31)) return SEMSHARE_EUNSUPPORTED;
    if (n_idx == 0 || n_rows == 0) return SEMSHARE_OK;
    if (!idx || !aligned(idx, 4) || !workspace || workspace_bytes < semshare_fetch_workspace_size(n_rows) ||
        (err_flag && !aligned(err_flag, 4)))
        return SEMSHARE_EINVAL;
    int sms = 0;
    if (current_sm_count(&sms, nullptr) != SEMSHARE_OK) return SEMSHARE_ECUDA;
    cudaStream_t s = as_stream(stream);
    // workspace: the row map, then (256-byte aligned) the row-block map; both cleared here
    auto* map = static_cast<uint8_t*>(workspace);
    const int64_t rblocks = (n_rows + kRows - 1) / kRows;
    const int64_t map_bytes = static_cast<int64_t>(round256(static_cast<size_t>(n_rows)));
    uint8_t* block_map = map + map_bytes;
    const int64_t clear_bytes = map_bytes + rblocks;
    const int64_t gm = (clear_bytes + 255) / 256, gi = (n_idx + 255) / 256;
    if (launch_pdl(clear_map_kernel, dim3(static_cast<unsigned>(gm < sms * 8 ? gm : sms * 8)), dim3(256), 0, s, map,
                   clear_bytes) != cudaSuccess ||
        launch_pdl(mark_rows_kernel, dim3(static_cast<unsigned>(gi < sms * 8 ? gi : sms * 8)), dim3(256), 0, s, idx, n_idx,
                   n_rows, map, block_map, err_flag) != cudaSuccess)
        return SEMSHARE_ECUDA;
    FetchArgs a{};
    for (int i = 0; i < n_seg; ++i) {
        a.src_k[i] = static_cast<const uint8_t*>(ref_k[i]);
        a.src_v[i] = static_cast<const uint8_t*>(ref_v[i]);
        a.dst_k[i] = static_cast<uint8_t*>(dev_k[i]);
        a.dst_v[i] = static_cast<uint8_t*>(dev_v[i]);
    }
    for (int i = 0; i <= n_seg; ++i) a.seg_off[i] = seg_offsets[i];
    a.n_seg = n_seg;
    a.n_layers = layout.n_layers;
    a.n_heads = layout.n_heads;
    a.chunks = static_cast<int32_t>(row_bytes / 16);
    a.s_layer = layout.stride_layer * eb;
    a.s_head = layout.stride_head * eb;
    a.s_token = layout.stride_token * eb;
    a.map = map;
    a.block_map = block_map;
    const int64_t planes = static_cast<int64_t>(layout.n_layers) * layout.n_heads;
    const int64_t n_items = planes * rblocks;
    const int64_t cap = static_cast<int64_t>(kCtasPerSm) * sms;
    const unsigned grid = static_cast<unsigned>(n_items < cap ? n_items : cap);
    if (launch_pdl(fetch_rows_kernel, dim3(grid), dim3(kThreads), 0, s, a, n_rows, rblocks, n_items) != cudaSuccess)
        return SEMSHARE_ECUDA;
    return launch_status();
}
