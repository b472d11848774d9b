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

// A check that fails on purpose (checked build): confirms how failures reach err_flag.
__global__ void check_selftest_kernel(uint32_t* err) {
    pdl_prologue();
    if (threadIdx.x == 0) SEMSHARE_CHECK(false, err, SEMSHARE_KERNEL_SELFTEST);
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
        case SEMSHARE_ECHECK: return "checked build: a pipeline bookkeeping check failed";
    }
    return "unknown status";
}

extern "C" semshare_status semshare_flag_status(uint32_t flags) {
    if (flags & SEMSHARE_FLAG_TIMEOUT) return SEMSHARE_ETIMEOUT;
    if (flags & SEMSHARE_FLAG_CHECK) return SEMSHARE_ECHECK;
    if (flags & SEMSHARE_FLAG_INDEX) return SEMSHARE_EINDEX;
    return SEMSHARE_OK;
}

extern "C" int32_t semshare_checked_build(void) { return semshare::kChecked ? 1 : 0; }

extern "C" semshare_status semshare_check_selftest(uint32_t* err_flag, void* stream) {
    using namespace semshare;
    if (!kChecked) return SEMSHARE_EUNSUPPORTED;
    if (err_flag == nullptr || !aligned(err_flag, 4)) return SEMSHARE_EINVAL;
    if (launch_pdl(check_selftest_kernel, dim3(1), dim3(32), 0, as_stream(stream), err_flag) != cudaSuccess)
        return SEMSHARE_ECUDA;
    return launch_status();
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

// ---- host-side counts of the method (no device work) --------------------------------------

extern "C" int64_t semshare_hd_count(int64_t n_tok, int32_t percent) {
    if (n_tok < 0 || n_tok >= (int64_t(1) << 40) || percent < 0 || percent > 100) return -1;
    // ceil(n_tok * percent / 100) in integers
    return (n_tok * percent + 99) / 100;
}

namespace semshare {
namespace {

// Unsigned integer of up to kLimbs 32-bit limbs (least significant first): just the two
// operations Retain[i] needs, multiply and divide by a 32-bit value.
constexpr int kRetainLimbs = 160;  // 31 bits of n_tok + 31 bits per layer for 128 layers, with room

struct BigUint {
    uint32_t limb[kRetainLimbs];
    int n;  // limbs in use (the top one non-zero, or n == 0 for zero)
};

void big_set(BigUint& x, uint64_t v) {
    x.n = 0;
    while (v) {
        x.limb[x.n++] = static_cast<uint32_t>(v);
        v >>= 32;
    }
}

bool big_mul(BigUint& x, uint32_t m) {
    uint64_t carry = 0;
    for (int i = 0; i < x.n; ++i) {
        const uint64_t t = static_cast<uint64_t>(x.limb[i]) * m + carry;
        x.limb[i] = static_cast<uint32_t>(t);
        carry = t >> 32;
    }
    if (carry) {
        if (x.n == kRetainLimbs) return false;
        x.limb[x.n++] = static_cast<uint32_t>(carry);
    }
    while (x.n > 0 && x.limb[x.n - 1] == 0) --x.n;
    return true;
}

void big_div(BigUint& x, uint32_t d) {  // x = floor(x / d)
    uint64_t rem = 0;
    for (int i = x.n - 1; i >= 0; --i) {
        const uint64_t cur = (rem << 32) | x.limb[i];
        x.limb[i] = static_cast<uint32_t>(cur / d);
        rem = cur % d;
    }
    while (x.n > 0 && x.limb[x.n - 1] == 0) --x.n;
}

}  // namespace
}  // namespace semshare

extern "C" semshare_status semshare_retain_counts(int64_t n_tok, const int32_t* alpha_num, int32_t alpha_den,
                                                  int32_t n_layers, int64_t* counts) {
    using namespace semshare;
    if (n_tok < 0 || n_tok >= (int64_t(1) << 31) || alpha_den < 1 || n_layers < 0 || n_layers > 128)
        return SEMSHARE_EINVAL;
    if (n_layers > 0 && (alpha_num == nullptr || counts == nullptr)) return SEMSHARE_EINVAL;
    for (int32_t i = 0; i < n_layers; ++i)
        if (alpha_num[i] < 0 || alpha_num[i] > alpha_den) return SEMSHARE_EINVAL;
    // Retain[i] = floor(n_tok * prod_{j<=i} num_j / den^(i+1)), exact: the numerator as a big
    // integer, then i+1 divisions by den (floor(floor(x/a)/b) = floor(x/(a*b)) for integers).
    BigUint num;
    big_set(num, static_cast<uint64_t>(n_tok));
    for (int32_t i = 0; i < n_layers; ++i) {
        if (!big_mul(num, static_cast<uint32_t>(alpha_num[i]))) return SEMSHARE_EUNSUPPORTED;
        BigUint q = num;
        for (int32_t j = 0; j <= i && q.n > 0; ++j) big_div(q, static_cast<uint32_t>(alpha_den));
        uint64_t v = 0;
        for (int k = q.n - 1; k >= 0; --k) v = (v << 32) | q.limb[k];  // <= n_tok < 2^31
        counts[i] = static_cast<int64_t>(v);
    }
    return SEMSHARE_OK;
}
