/*
 * semshare_probe.h -- measurement support for the GB300 fuzzy token-matching library.
 *
 * The exhaustive Hamming search of semshare_match (Sec. 3.3: each target token's nearest
 * reference token by code distance) spends its time in one word operation: xor two 32-bit code
 * words, count the set bits, add the count to a running distance.  Its roofline is therefore
 * the device's sustained rate of that operation, which no vendor table states for this chip.
 * This probe measures it: independent xor/popc/add chains in registers, no memory traffic.
 * Not part of the matching path: it is built into its own library, libsemshare_probe.so, which
 * bench.py loads for the denominator of the xor/popc matcher's roofline.
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

#ifdef __cplusplus
}
#endif

#endif /* SEMSHARE_PROBE_H */
