/*
 * semshare_probe.h -- measurement support for the GB300 fuzzy token-matching library.
 *
 * The exhaustive Hamming search of semshare_match (Sec. 3.3: each target token's nearest
 * reference token by code distance) spends its time in one word operation: xor two 32-bit code
 * words, count the set bits, add the count to a running distance.  Its roofline is therefore
 * the device's sustained rate of that operation, which no vendor table states for this chip.
 * This probe measures it: independent xor/popc/add chains in registers, no memory traffic.
 * Not part of the matching path; bench.py uses it for the denominator of the xor/popc
 * matcher's roofline.  A second probe times the hash kernel's operand stream on its own.
 */
#ifndef SEMSHARE_PROBE_H
#define SEMSHARE_PROBE_H

#include <stdint.h>

#include "semshare.h"

#ifdef __cplusplus
extern "C" {
#endif

/* Independent chains per thread: one launch performs threads * iters * SEMSHARE_PROBE_CHAINS
 * word operations. */
#define SEMSHARE_PROBE_CHAINS 8

/* Threads the probe launches on the current device (fully occupied SMs), or -1 if the
 * device cannot be queried. */
int64_t semshare_probe_hamming_threads(void);

/*
 * semshare_probe_hamming_rate -- enqueue one launch of the word-operation probe.
 *
 *   iters       iterations per thread, 1 .. 2^24; each does SEMSHARE_PROBE_CHAINS word ops
 *   sink        device uint32[sink_words]: one word per thread receives its chains' combined
 *               result (keeps the work observable); contents are meaningless
 *   sink_words  >= semshare_probe_hamming_threads()
 *   stream      cudaStream_t; time the launch with events on it
 * Returns EINVAL for bad arguments, ECUDA if the device query or the launch fails.
 */
semshare_status semshare_probe_hamming_rate(int64_t iters, uint32_t* sink, int64_t sink_words, void* stream);

/*
 * semshare_probe_operand_stream -- enqueue one launch that moves the LSH projection's operands
 * the way semshare_hash's pipeline moves them, and nothing else.
 *
 * semshare_hash (Sec. 3.3.1 and App. A.2: rotate each embedding row, project it on nbits random
 * hyperplanes, keep the signs) streams, per 128-row tile and 64-wide K block, one 128 x 64 bf16
 * embedding block and one nbits x 64 bf16 hyperplane block into shared memory with 128-byte
 * swizzled TMA boxes, one persistent CTA per SM taking an equal contiguous share of the
 * (tile, K block) iterations.  This probe does exactly that with no rotation and no MMA: a slot
 * is released as soon as its copy lands.  Its launch time is the floor the operand traffic sets
 * for the hash kernel under the same cache state.  Not part of the matching path.
 *
 *   emb          device bf16 [n][d], rows d*2 bytes apart, 16-byte aligned; n a positive
 *                multiple of 128 (< 2^31), d a positive multiple of 64
 *   hyperplanes  device bf16 [nbits][d] (16-byte aligned), or NULL to stream the embedding
 *                blocks only
 *   nbits        32..256, a multiple of 32 (read only with hyperplanes)
 *   slots        shared-memory ring slots, 1..12; each holds one embedding block and, with
 *                hyperplanes, one hyperplane block (EUNSUPPORTED if they do not fit)
 *   prefetch     L2 prefetch distance of the embedding blocks in iterations, 0..64 (0: none)
 *   err_flag     device uint32 or NULL; SEMSHARE_FLAG_TIMEOUT is OR-ed in if a wait exceeds
 *                its limit (the launch then ends early)
 *   stream       cudaStream_t; time the launch with events on it
 * Returns EINVAL / EUNSUPPORTED for bad arguments, ECUDA if the device query, the tensor-map
 * encoding or the launch fails.
 */
semshare_status semshare_probe_operand_stream(const uint16_t* emb, int64_t n, int32_t d, const uint16_t* hyperplanes,
                                              int32_t nbits, int32_t slots, int32_t prefetch, uint32_t* err_flag,
                                              void* stream);

#ifdef __cplusplus
}
#endif

#endif /* SEMSHARE_PROBE_H */
