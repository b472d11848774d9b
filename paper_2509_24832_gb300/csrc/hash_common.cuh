// hash_common.cuh -- device helpers shared by the two LSH hash kernels (hash.cu, hash_2sm.cu):
// the stream-K range split, the rotation of Eq. 1 from the fixed-point turn table, and the
// sign-packing epilogue stores.
#pragma once

#include <cuda_bf16.h>

#include <cstdint>

namespace semshare {
namespace hashk {

// Rotation variants of a hash kernel, fixed at compile time so that the plain rotary kernel
// carries no test for the others: every row rotated; no row rotated (SEMSHARE_ROPE_NONE); a pair
// call, which hashes every row twice -- logical tiles below pair_rows as they are, the tiles from
// pair_rows on (the same rows again) rotated.
enum RotVariant { kRotAll = 0, kRotNone = 1, kRotPair = 2 };

// First iteration of CTA b's range (b = gridDim.x gives the end).
__device__ __forceinline__ int64_t range_begin(int64_t b, int64_t total, int64_t G) { return (b * total) / G; }

// The CTA whose range holds iteration i.
__device__ __forceinline__ int64_t range_owner(int64_t i, int64_t total, int64_t G) {
    int64_t b = (i * G) / total;
    while (b + 1 < G && range_begin(b + 1, total, G) <= i) ++b;
    while (b > 0 && range_begin(b, total, G) > i) --b;
    return b;
}

// cos and sin of the rotation angle m * theta_k (Eq. 1).  turns_q64 = frac(theta_k/(2*pi)) as
// a 0.64 fixed-point fraction, so bits 32..63 of m * turns_q64 (mod 2^64) are the angle's
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

// Sign bits of 32 fp32 values given as bit patterns: bit j = [v_j > 0].
__device__ __forceinline__ uint32_t sign_word(const uint32_t (&v)[32]) {
    uint32_t bits = 0u;
#pragma unroll
    for (int j = 0; j < 32; ++j) bits |= (static_cast<int32_t>(v[j]) > 0 ? 1u : 0u) << j;
    return bits;
}

__device__ __forceinline__ void store_proj(float* proj, int64_t row, int nbits, int q, const uint32_t (&v)[32]) {
    float4* pp = reinterpret_cast<float4*>(proj + row * nbits + q * 32);
#pragma unroll
    for (int j = 0; j < 8; ++j)
        pp[j] = make_float4(__uint_as_float(v[4 * j]), __uint_as_float(v[4 * j + 1]), __uint_as_float(v[4 * j + 2]),
                            __uint_as_float(v[4 * j + 3]));
}

// 32 code bits as the operand bytes of the tensor-core match: e4m3 +1 (0x38) for a set bit, -1
// (0xB8) for a clear one (byte = 0xB8 ^ bit << 7), bit j at byte j of dst (16-byte aligned).  Four
// bits m spread to bit 7 of four bytes by one multiply: m * 0x10204080 puts bit i of m at bit
// 8i+7 (the shifted copies of m do not overlap).
__device__ __forceinline__ void store_sign_bytes(uint8_t* dst, uint32_t bits) {
    uint32_t w[8];
#pragma unroll
    for (int q = 0; q < 8; ++q) w[q] = 0xB8B8B8B8u ^ ((((bits >> (4 * q)) & 0xFu) * 0x10204080u) & 0x80808080u);
    uint4* d = reinterpret_cast<uint4*>(dst);
    d[0] = make_uint4(w[0], w[1], w[2], w[3]);
    d[1] = make_uint4(w[4], w[5], w[6], w[7]);
}

// The zero bytes that pad a sign row to its pitch.
__device__ __forceinline__ void store_sign_pad(uint8_t* dst) {
    uint4* d = reinterpret_cast<uint4*>(dst);
    d[0] = make_uint4(0u, 0u, 0u, 0u);
    d[1] = make_uint4(0u, 0u, 0u, 0u);
}

// A whole sign row: the W code words as bytes, then zeros up to pitch (a multiple of 32, <= 256).
__device__ __forceinline__ void store_sign_row(uint8_t* signs, int64_t row, int pitch, int W, const uint32_t (&words)[8]) {
    uint8_t* d = signs + row * pitch;
#pragma unroll
    for (int q = 0; q < 8; ++q) {
        if (q < W)
            store_sign_bytes(d + 32 * q, words[q]);
        else if (32 * q < pitch)
            store_sign_pad(d + 32 * q);
    }
}

__device__ __forceinline__ void store_codes(uint32_t* codes, int64_t row, int W, const uint32_t (&words)[8]) {
    uint32_t* cp = codes + row * W;
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

}  // namespace hashk
}  // namespace semshare
