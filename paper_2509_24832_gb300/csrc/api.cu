// api.cu -- status helpers and semshare_rope_table (the per-pair rotation frequencies of
// Eq. 1 in fixed point, consumed by the hash kernel).
#include "common.cuh"

namespace semshare {
namespace {

// table[k] = frac(theta_k / (2*pi)) * 2^64 rounded, theta_k = base^(-2k/d)  (Eq. 1, App. A.1):
// the turns per position modulo one full turn, as an unsigned 0.64 fixed-point fraction.
// Whole turns do not change the rotation, so only the fraction is kept; scaling by 2^64 is exact.
__global__ void rope_table_kernel(int32_t d, double base, uint64_t* __restrict__ table) {
    const int32_t k = blockIdx.x * blockDim.x + threadIdx.x;
    if (k >= d / 2) return;
    const double theta = pow(base, -2.0 * static_cast<double>(k) / static_cast<double>(d));
    double turns = theta / 6.283185307179586476925286766559;
    turns -= floor(turns);
    const double q = ldexp(turns, 64);
    table[k] = q >= 18446744073709551616.0 ? 0ull : __double2ull_rn(q);
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
    if (table == nullptr || !aligned(table, 8)) return SEMSHARE_EINVAL;
    const int32_t pairs = d / 2;
    rope_table_kernel<<<(pairs + 255) / 256, 256, 0, as_stream(stream)>>>(d, rope_base, table);
    return launch_status();
}
