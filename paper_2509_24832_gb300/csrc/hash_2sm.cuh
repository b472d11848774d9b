// hash_2sm.cuh -- host-side entry of the CTA-pair hash kernel (hash_2sm.cu), called by hash.cu's
// entry points for bf16 rows with the interleaved pairing or no rotation.
#pragma once

#include <cstddef>
#include <cstdint>

#include "semshare.h"

namespace semshare {

struct Hash2smCall {
    const void* emb;          // bf16 [n][row_stride]
    int64_t n;
    int32_t d;
    int64_t row_stride;       // elements
    const int32_t* positions; // nullable: row index
    const uint64_t* rope_table;
    const uint16_t* hyperplanes;
    int32_t nbits;
    bool none;                // no rotation (SEMSHARE_ROPE_NONE)
    bool pair;                // semshare_hash_pair: rows as they are into codes, rotated into codes2
    int64_t pair_rows;        // pair: n rounded up to 256 rows
    uint32_t* codes;
    uint32_t* codes2;
    float* proj;
    uint8_t* signs;           // nullable: the codes as e4m3 +-1 rows of signs_pitch bytes
    int32_t signs_pitch;
    uint32_t* err_flag;
    void* partials;           // workspace partial-slot region
    size_t partial_bytes;
    uint32_t* tile_count;     // workspace counters (zero between calls)
    size_t count_bytes;
    void* stream;
};

// Validated arguments in, one cluster launch out (ECUDA on a launch failure).
semshare_status launch_hash_2sm(const Hash2smCall& c);

}  // namespace semshare
