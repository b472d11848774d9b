// api.cu -- status helpers and semshare_rope_table (the per-pair rotation frequencies of
// Eq. 1 in fixed point, consumed by the hash kernel).
#include "common.cuh"

namespace semshare {
namespace {

// Rotation table of Eq. 1 (App. A.1), theta_k = base^(-2k/d), k < d/2:
//   table[k]           frac(theta_k / (2*pi)) * 2^64 rounded: the turns per position modulo one
//                      full turn, an unsigned 0.64 fixed-point fraction (scaling by 2^64 is exact)
//   table[d/2 + k]     cos(32*theta_k) and sin(32*theta_k) as two floats (low word: cos): the
//                      rotation between positions 32 apart, for stepping from one row to another
__global__ void rope_table_kernel(int32_t d, double base, uint64_t* __restrict__ table) {
    pdl_prologue();
    const int32_t k = blockIdx.x * blockDim.x + threadIdx.x;
    if (k >= d / 2) return;
    const double theta = pow(base, -2.0 * static_cast<double>(k) / static_cast<double>(d));
    double turns = theta / 6.283185307179586476925286766559;
    turns -= floor(turns);
    const double q = ldexp(turns, 64);
    table[k] = q >= 18446744073709551616.0 ? 0ull : __double2ull_rn(q);
    const double a32 = 6.283185307179586476925286766559 * (32.0 * turns - floor(32.0 * turns));
    const float c = static_cast<float>(cos(a32)), s = static_cast<float>(sin(a32));
    table[d / 2 + k] = static_cast<uint64_t>(__float_as_uint(c)) | (static_cast<uint64_t>(__float_as_uint(s)) << 32);
}

}  // namespace
}  // namespace semshare

extern "C" const char* semshare_status_string(semshare_status s) {
    switch (s) {
        case SEMSHARE_OK: return "ok";
        case SEMSHARE_EINVAL: return "invalid argument";
        case SEMSHARE_EUNSUPPORTED: return "unsupported argument";
        case SEMSHARE_ECUDA: return "CUDA error";
        case SEMSHARE_EINDEX: return "index out of range";
        case SEMSHARE_ETIMEOUT: return "kernel wait timed out";
        case SEMSHARE_ETOOLARGE: return "size exceeds the fixed scratch capacity";
    }
    return "unknown status";
}

extern "C" semshare_status semshare_flag_status(uint32_t flags) {
    if (flags & SEMSHARE_FLAG_TIMEOUT) return SEMSHARE_ETIMEOUT;
    if (flags & SEMSHARE_FLAG_INDEX) return SEMSHARE_EINDEX;
    return SEMSHARE_OK;
}

extern "C" int32_t semshare_abi_version(void) { return SEMSHARE_ABI_VERSION; }

extern "C" semshare_status semshare_rope_table(int32_t d, double rope_base, uint64_t* table, void* stream) {
    using namespace semshare;
    if (d < 2 || d > 65536 || (d & 1)) return SEMSHARE_EINVAL;
    if (!(rope_base > 0.0) || !(rope_base < 1e300)) return SEMSHARE_EINVAL;
    if (table == nullptr || !aligned(table, 16)) return SEMSHARE_EINVAL;
    const int32_t pairs = d / 2;
    if (launch_pdl(rope_table_kernel, dim3(static_cast<unsigned>((pairs + 255) / 256)), dim3(256), 0, as_stream(stream),
                   d, rope_base, table) != cudaSuccess)
        return SEMSHARE_ECUDA;
    return launch_status();
}
