/*
 * semshare.h -- C ABI of the GB300 (sm_103a) fuzzy token-matching library.
 *
 * SemShareKV (arXiv 2509.24832) lets a target prompt reuse the KV cache of a semantically
 * similar reference prompt.  Its matching path (Sec. 3.2, Sec. 3.3) has four steps:
 * rotary position encoding of both prompts' embedding rows (Sec. 3.3.1, Eq. 1), locality
 * sensitive hashing of the rotated rows (Sec. 3.3, App. A.2), a per-token nearest-neighbour
 * match of every target token to a reference token (Sec. 3.3), and a rearrangement of the
 * reference K/V cache to the target's token order (Sec. 3.3, Sec. 3.3.2).  This library
 * exposes them as three calls, semshare_hash (steps 1-2), semshare_match (step 3) and
 * semshare_gather_kv (step 4), plus semshare_rope_table, which precomputes the per-pair
 * rotation frequencies that semshare_hash consumes.  Around them: semshare_match_tc (step 3 on
 * the tensor cores), semshare_retrieve (which stored prompt to reuse, Sec. 3.2) and
 * semshare_match_tc_selected (step 3 against the retrieved prompt, chosen on the device),
 * semshare_fetch_rows (the selected rows of a host-resident cache, brought in once each),
 * semshare_gather_kv_retained (step 4 for each layer's retained tokens, Sec. 3.3.4) and
 * semshare_kv_deviation / semshare_select_hd (the high-deviation tokens, App. A.4).
 *
 * Conventions shared by every call:
 *   - Buffers are owned by the caller.  Pointers marked "device" point to memory of the
 *     current CUDA device; "host" marks host memory read during the call only.  No call
 *     allocates or frees memory.  Scratch memory is passed in by the caller (the
 *     workspace arguments); apart from semshare_match_static the library keeps no state
 *     between calls.
 *   - `stream` is a cudaStream_t (NULL = the legacy default stream).  Work is enqueued on it
 *     and runs asynchronously; a call returns once the work is enqueued.
 *   - Argument errors are detected on the host before anything is enqueued and returned as
 *     SEMSHARE_EINVAL / SEMSHARE_EUNSUPPORTED; nothing is launched in that case.  A failed
 *     launch returns SEMSHARE_ECUDA.
 *   - Errors found by a kernel while it runs are OR-ed into an optional device word
 *     `err_flag` (SEMSHARE_FLAG_*); the caller reads it after synchronising and may turn it
 *     into a status with semshare_flag_status().  Kernels never trap.
 *   - Every wait inside a pipelined kernel is bounded (2 s by default; the environment
 *     variable SEMSHARE_WAIT_LIMIT_NS, read at each call, overrides it for diagnostics).  A
 *     wait that runs out raises SEMSHARE_FLAG_TIMEOUT; the kernel then lets its copies in
 *     flight land, frees its tensor memory and returns, and the CUDA context stays usable.
 *   - Results are deterministic: the same inputs give the same bits on every run.
 */
#ifndef SEMSHARE_H
#define SEMSHARE_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define SEMSHARE_ABI_VERSION 1

typedef enum {
    SEMSHARE_OK = 0,
    SEMSHARE_EINVAL = 1,        /* null / misaligned pointer, bad size or stride */
    SEMSHARE_EUNSUPPORTED = 2,  /* valid request outside what the kernels implement */
    SEMSHARE_ECUDA = 3,         /* a CUDA runtime or driver call failed */
    SEMSHARE_EINDEX = 4,        /* a kernel met an index outside its table (from err_flag) */
    SEMSHARE_ETIMEOUT = 5,      /* a kernel pipeline wait hit its time limit (from err_flag) */
    SEMSHARE_ETOOLARGE = 6,     /* a size exceeds semshare_match_static's fixed scratch capacity */
    SEMSHARE_ECHECK = 7         /* checked build: a pipeline bookkeeping check failed (from err_flag) */
} semshare_status;

typedef enum { SEMSHARE_BF16 = 0, SEMSHARE_F32 = 1 } semshare_dtype;

/* Bits a kernel ORs into `err_flag`. */
#define SEMSHARE_FLAG_INDEX 1u
#define SEMSHARE_FLAG_TIMEOUT 2u
/* Checked build only (see semshare_checked_build): a bookkeeping check failed.  The first failed
 * check also stores its kernel id in bits 8..15 of err_flag and its source line in bits 16..31. */
#define SEMSHARE_FLAG_CHECK 4u
#define SEMSHARE_CHECK_KERNEL(flags) (((flags) >> 8) & 0xFFu)
#define SEMSHARE_CHECK_LINE(flags) ((flags) >> 16)
/* Kernel ids of SEMSHARE_CHECK_KERNEL. */
#define SEMSHARE_KERNEL_HASH_2SM 1u      /* bf16 rows on SM pairs (hash_2sm.cu) */
#define SEMSHARE_KERNEL_HASH 2u          /* fp32 rows, rotate-half (hash.cu) */
#define SEMSHARE_KERNEL_HAMMING_TC 3u    /* tensor-core search (match_tc.cu) */
#define SEMSHARE_KERNEL_SELFTEST 15u     /* semshare_check_selftest */

/* Human-readable name of a status. */
const char* semshare_status_string(semshare_status s);

/* Maps the err_flag bits read back by the caller to a status (TIMEOUT wins over CHECK, CHECK over
 * INDEX). */
semshare_status semshare_flag_status(uint32_t flags);

/*
 * The checked build: the same library compiled with -DSEMSHARE_CHECKED (libsemshare_checked.so,
 * built beside libsemshare.so; a stand-in for a race/synchronisation sanitizer, which this
 * project does not rely on).  Its pipelined kernels also verify their barrier bookkeeping while
 * they run: every ring slot a consumer acquires was filled exactly once since its last use and
 * every slot a producer refills was released by all of its consumers; at the end every role has
 * handled as many stages and segments as its range implies; the tensor-memory allocation starts
 * at column 0; every stream-K tile is closed after exactly its expected number of arrivals.  A
 * failed check ORs SEMSHARE_FLAG_CHECK into err_flag (when err_flag is non-NULL) and the kernel
 * carries on; results are the same as the plain build's.  This is not part of the paper; it
 * exists to test the library.
 *
 * semshare_checked_build: 1 in the checked build, 0 in the plain one.
 * semshare_check_selftest: checked build only (SEMSHARE_EUNSUPPORTED otherwise): enqueues a
 * one-thread kernel whose check fails on purpose, so that a caller can confirm how failures
 * reach err_flag (kernel id SEMSHARE_KERNEL_SELFTEST).  err_flag: device, 4-byte aligned.
 */
int32_t semshare_checked_build(void);
semshare_status semshare_check_selftest(uint32_t* err_flag, void* stream);

/* SEMSHARE_ABI_VERSION of the loaded library. */
int32_t semshare_abi_version(void);

/*
 * semshare_rope_table -- rotation frequencies of Eq. 1 (App. A.1) in fixed point.
 *
 * Pair k of a d-wide embedding row turns by theta_k = rope_base^(-2k/d) radians per position
 * (Eq. 1; the angle at position m is m * theta_k, Sec. 3.3.1).  For k < d/2, table[k] receives
 * frac(theta_k / (2*pi)) * 2^64 rounded: the turns per position modulo one turn as an
 * unsigned 0.64 fixed-point fraction, so a kernel gets the angle of position m modulo a full
 * turn from the low 64 bits of m * table[k] with integer arithmetic; table[d/2 + k] receives
 * cos(32*theta_k) (low 32 bits) and sin(32*theta_k) (high 32 bits) as floats, the rotation
 * between two positions 32 apart.  Computed on the device in double precision.
 *
 *   d          embedding dimension, even, 2 <= d <= 65536
 *   rope_base  the RoPE base (10000 in Eq. 1), finite and > 0
 *   table      device, d uint64 words, 16-byte aligned; written
 * Returns EINVAL for a bad d, base or pointer.  The table depends only on (d, rope_base):
 * compute it once and reuse it for every semshare_hash call.
 */
semshare_status semshare_rope_table(int32_t d, double rope_base, uint64_t* table, void* stream);

/*
 * semshare_hash -- steps 1-2: rotary encoding + random-hyperplane LSH codes.
 *
 * For each row i (Sec. 3.3.1: RoPE is applied to the E cache of both prompts, then LSH):
 *   y = RoPE(emb[i], positions[i])       Eq. 1, pairs (2k, 2k+1), angle positions[i]*theta_k
 *   p_j = <hyperplanes[j], bf16(y)>      fp32 accumulation on the tensor cores
 *   bit j of codes[i] = [p_j > 0]         sign random projection (App. A.2, App. D: LSH)
 * y is computed in fp32 and rounded to bf16 (nearest even) before the products.  The K range
 * of a 128-row tile may be split across SMs; the partial sums are then added in K order, so
 * the codes are the same on every run on a given device.
 *
 *   emb         device, n rows of d elements of `dtype`, row i at element offset i*row_stride;
 *               16-byte aligned base, row_stride*element_size a multiple of 16 bytes
 *   dtype       SEMSHARE_BF16 or SEMSHARE_F32
 *   n           rows (0 is allowed: nothing is launched); n < 2^31
 *   d           embedding dimension, a multiple of 64, 64 <= d <= 65536
 *   row_stride  elements between consecutive rows, >= d
 *   positions   device, n int32 token positions >= 0, or NULL for positions 0..n-1.  Each
 *               prompt uses its own 0-based positions; rows of several prompts may be hashed
 *               in one call by passing each row's position.
 *   rope_table  device, the d words written by semshare_rope_table(d, base, ...)
 *   hyperplanes device, [nbits][d] bf16 bit patterns, row-major, 16-byte aligned
 *   nbits       code length: 32, 64, ..., 256
 *   codes       device, [n][nbits/32] uint32, bit j of row i in word j/32 at bit j%32; written
 *   proj_out    device or NULL; if given, [n][nbits] float32 projections p_j are written too
 *   workspace   device scratch of at least semshare_hash_workspace_size(n, d, nbits) bytes,
 *               256-byte aligned.  It must be zero-filled before its first use; every call
 *               that completes without an error flag leaves the part that must be zero
 *               zero-filled again, so one workspace (sized for the largest call) serves any
 *               number of calls of any sizes made one after another on the same device.
 *               Calls that may run concurrently need separate workspaces.
 *   err_flag    device or NULL; SEMSHARE_FLAG_TIMEOUT is OR-ed in if a pipeline wait of the
 *               kernel exceeds its limit (the kernel then stops, leaves codes incomplete and
 *               the workspace in an unknown state: zero it before the next call)
 * Returns EINVAL / EUNSUPPORTED for bad arguments (EINVAL for a short workspace), ECUDA if the
 * launch fails.  semshare_hash_workspace_size returns 0 for arguments semshare_hash rejects;
 * it depends on the current device (its SM count).
 */
size_t semshare_hash_workspace_size(int64_t n, int32_t d, int32_t nbits);

/*
 * semshare_hash_ex -- semshare_hash with a choice of rotary pairing.
 *
 * rope_layout SEMSHARE_ROPE_INTERLEAVED: pairs (2k, 2k+1), as Eq. 1 prints them (semshare_hash);
 *             SEMSHARE_ROPE_HALF: pairs (k, k + d/2) ("rotate-half", the arrangement of many
 *             model implementations), each turned by the same angle m * theta_k and rounded to
 *             bf16 the same way.  The rotation table is the same for both.
 *             SEMSHARE_ROPE_NONE: no rotation -- the rows are hashed as they are (rounded to bf16
 *             when fp32), the codes of y = x; positions and rope_table are ignored and may be
 *             NULL.  (Used for the retrieval codes of Sec. 3.2, which compare whole prompts; it
 *             equals SEMSHARE_ROPE_INTERLEAVED with every position 0, at which RoPE is the
 *             identity, and skips the rotation work.)
 * SEMSHARE_ROPE_HALF takes bf16 rows and d a multiple of 128 (else EUNSUPPORTED).  Every other
 * argument, and the result for SEMSHARE_ROPE_INTERLEAVED, as for semshare_hash.
 */
#define SEMSHARE_ROPE_INTERLEAVED 0u
#define SEMSHARE_ROPE_HALF 1u
#define SEMSHARE_ROPE_NONE 2u
semshare_status semshare_hash_ex(const void* emb, semshare_dtype dtype, int64_t n, int32_t d, int64_t row_stride,
                                 const int32_t* positions, const uint64_t* rope_table, const uint16_t* hyperplanes,
                                 int32_t nbits, uint32_t rope_layout, uint32_t* codes, float* proj_out,
                                 void* workspace, size_t workspace_bytes, uint32_t* err_flag, void* stream);
/*
 * semshare_hash_pair -- the codes of the same rows without and with rotation, in one launch.
 *
 * Reference retrieval (Sec. 3.2) compares prompts by the codes of their rows as they are; the
 * token matching that follows (Sec. 3.3.1) uses the codes of the rows after RoPE.  For a target
 * prompt both are needed; this call computes
 *     codes_plain  = semshare_hash_ex(..., SEMSHARE_ROPE_NONE, ...)
 *     codes_rotary = semshare_hash(..., positions, rope_table, ...)
 * bit for bit, in one launch over twice the row tiles (one pipeline fill and one split of the
 * work over the SMs instead of two).
 *
 *   emb, dtype, n (< 2^30), d, row_stride, positions, rope_table, hyperplanes, nbits, err_flag,
 *   stream        as for semshare_hash
 *   codes_plain, codes_rotary   device, [n][nbits/32] uint32 each, 16-byte aligned; written
 *   workspace     as for semshare_hash, at least semshare_hash_pair_workspace_size(n, d, nbits)
 *                 bytes (zero-filled before first use; left zero-filled by every call)
 * No projections are written.  Returns as semshare_hash.
 */
size_t semshare_hash_pair_workspace_size(int64_t n, int32_t d, int32_t nbits);
semshare_status semshare_hash_pair(const void* emb, semshare_dtype dtype, int64_t n, int32_t d, int64_t row_stride,
                                   const int32_t* positions, const uint64_t* rope_table, const uint16_t* hyperplanes,
                                   int32_t nbits, uint32_t* codes_plain, uint32_t* codes_rotary, void* workspace,
                                   size_t workspace_bytes, uint32_t* err_flag, void* stream);
semshare_status semshare_hash(const void* emb, semshare_dtype dtype, int64_t n, int32_t d, int64_t row_stride,
                              const int32_t* positions, const uint64_t* rope_table, const uint16_t* hyperplanes,
                              int32_t nbits, uint32_t* codes, float* proj_out, void* workspace,
                              size_t workspace_bytes, uint32_t* err_flag, void* stream);

/*
 * semshare_hash_signs -- semshare_hash_ex that also writes the codes as the +-1 operand rows of
 * the tensor-core match (semshare_match_tc_signs).
 *
 * The tensor-core search of Sec. 3.3's nearest token computes popcount(a XOR b) as
 * (nbits - <s_a, s_b>) / 2 with s = 2*bit - 1; its operands are the codes as rows of e4m3 bytes.
 * The hash epilogue holds the sign bits already, so it writes those rows beside the packed codes
 * and the match needs no expansion pass.
 *
 *   every argument as for semshare_hash_ex, plus
 *   signs   device, [n][semshare_signs_pitch(nbits)] bytes, 16-byte aligned; written: byte j of
 *           row i is 0x38 (e4m3 +1) if bit j of codes[i] is set, else 0xB8 (e4m3 -1); bytes
 *           nbits .. pitch-1 of every row are 0
 * Returns as semshare_hash_ex (EINVAL for a NULL or misaligned signs when n > 0).
 */
int32_t semshare_signs_pitch(int32_t nbits); /* 128 * ceil(nbits / 128); 0 for an unsupported nbits */
semshare_status semshare_hash_signs(const void* emb, semshare_dtype dtype, int64_t n, int32_t d, int64_t row_stride,
                                    const int32_t* positions, const uint64_t* rope_table, const uint16_t* hyperplanes,
                                    int32_t nbits, uint32_t rope_layout, uint32_t* codes, uint8_t* signs,
                                    float* proj_out, void* workspace, size_t workspace_bytes, uint32_t* err_flag,
                                    void* stream);

/*
 * semshare_match -- step 3: Hamming nearest reference token of every target token.
 *
 * Sec. 3.3: "for each token in the target prompt, the most similar token in the reference
 * prompt".  idx[t] = the lowest j minimising popcount(tgt_codes[t] XOR ref_codes[j]) over
 * 0 <= j < n_ref; dist[t] = that minimum.  Ties go to the lowest reference index, so the
 * result does not depend on how the search is split across the GPU.  A pool of reference
 * prompts is searched by concatenating their codes; idx is then the global pool row.
 *
 *   tgt_codes  device, [n_tgt][nbits/32] uint32, 16-byte aligned
 *   n_tgt      target rows, 0 <= n_tgt < 2^31 (0: nothing is launched)
 *   ref_codes  device, [n_ref][nbits/32] uint32, 16-byte aligned
 *   n_ref      reference rows, 1 <= n_ref < 2^31
 *   nbits      32, 64, ..., 256
 *   idx        device, [n_tgt] int32; written
 *   dist       device, [n_tgt] int32, or NULL; written
 *   workspace  device scratch of at least semshare_match_workspace_size(n_tgt) bytes,
 *              8-byte aligned; its contents on entry do not matter and are overwritten
 * Returns EINVAL / EUNSUPPORTED for bad arguments, ECUDA if a launch fails.
 */
size_t semshare_match_workspace_size(int64_t n_tgt);
semshare_status semshare_match(const uint32_t* tgt_codes, int64_t n_tgt, const uint32_t* ref_codes, int64_t n_ref,
                               int32_t nbits, int32_t* idx, int32_t* dist, void* workspace, size_t workspace_bytes,
                               void* stream);

/*
 * semshare_match_tc -- step 3 on the tensor cores: exactly semshare_match's result.
 *
 * Same problem and tie rule as semshare_match (Sec. 3.3: the most similar reference token of
 * each target token).  With s = 2*bit - 1, popcount(a XOR b) = (nbits - <s_a, s_b>) / 2, so
 * the all-pairs distances are one dense contraction: the codes are expanded to fp8 +-1 rows
 * and multiplied on the tcgen05 tensor cores (fp32 accumulation, exact for these integers),
 * and each row of the product is reduced to its best reference on the fly.
 *
 *   arguments as for semshare_match, plus
 *   workspace  device scratch of at least semshare_match_tc_workspace_size(n_tgt, n_ref, nbits)
 *              bytes, 256-byte aligned; contents on entry do not matter, overwritten
 *   err_flag   device or NULL; SEMSHARE_FLAG_TIMEOUT is OR-ed in if a pipeline wait of the
 *              kernel exceeds its limit (idx/dist are then incomplete)
 * tgt_codes and ref_codes need only 4-byte alignment here.  Returns as semshare_match.
 */
size_t semshare_match_tc_workspace_size(int64_t n_tgt, int64_t n_ref, int32_t nbits);
semshare_status semshare_match_tc(const uint32_t* tgt_codes, int64_t n_tgt, const uint32_t* ref_codes, int64_t n_ref,
                                  int32_t nbits, int32_t* idx, int32_t* dist, void* workspace, size_t workspace_bytes,
                                  uint32_t* err_flag, void* stream);

/*
 * semshare_match_tc_signs -- semshare_match_tc on sign rows written by semshare_hash_signs, in
 * one launch.
 *
 * Same problem, tie rule and result as semshare_match (Sec. 3.3: the most similar reference token
 * of each target token, ties to the lowest index).  The operands are already +-1 rows, so there is
 * no expansion pass, and the search's last CTA to finish turns the per-target keys into idx and
 * dist (for up to 16384 targets; larger calls add one small launch that does it).
 *
 *   tgt_signs  device, [n_tgt][semshare_signs_pitch(nbits)] bytes as semshare_hash_signs writes
 *              them, 16-byte aligned
 *   ref_signs  device, [n_ref][semshare_signs_pitch(nbits)] bytes, 16-byte aligned
 *   n_tgt, n_ref, nbits, idx, dist, err_flag, stream   as for semshare_match_tc
 *   workspace  device scratch of at least semshare_match_tc_signs_workspace_size(n_tgt) bytes,
 *              256-byte aligned.  Every byte must be 0xFF before its first use (e.g.
 *              cudaMemsetAsync(workspace, 0xFF, bytes)); every call leaves it that way again, also
 *              when a pipeline wait gives up, so one workspace (sized for the largest call) serves
 *              any number of calls made one after another on the same device.  Calls that may
 *              run concurrently need separate workspaces.
 * Returns EINVAL / EUNSUPPORTED for bad arguments, ECUDA if a launch fails.
 */
size_t semshare_match_tc_signs_workspace_size(int64_t n_tgt);
semshare_status semshare_match_tc_signs(const uint8_t* tgt_signs, int64_t n_tgt, const uint8_t* ref_signs,
                                        int64_t n_ref, int32_t nbits, int32_t* idx, int32_t* dist, void* workspace,
                                        size_t workspace_bytes, uint32_t* err_flag, void* stream);

/*
 * semshare_retrieve -- reference retrieval: which stored prompt the target should reuse.
 *
 * Sec. 3.2: the stored prompt with the highest LSH-distance-based similarity to the target is
 * the reference.  App. A.3: Similarity = clip(1 - d_norm, 0, 1) with d_norm = LSH_dist / max_dist
 * (the paper's min(dist) = 0, max(dist) = 30).  Sec. 4.4: reuse applies only when that
 * similarity exceeds 0.8.  The paper does not spell out LSH_dist for two prompts; here it is the
 * mean, over the target's tokens, of each token's Hamming distance to its nearest token of the
 * candidate (the per-token distance of Sec. 3.3 averaged over the target).
 *
 *   tgt_codes     device, [n_tgt][nbits/32] packed codes of the target prompt (4-byte aligned)
 *   pool_codes    device, the codes of all candidates concatenated, [n_pool][nbits/32]
 *   cand_offsets  HOST, n_cand + 1 values: candidate c is pool rows
 *                 [cand_offsets[c], cand_offsets[c+1]); cand_offsets[0] = 0, strictly
 *                 increasing (no empty candidate), n_pool = cand_offsets[n_cand]; read before
 *                 the call returns
 *   n_cand        1 <= n_cand <= SEMSHARE_RETRIEVE_MAX_CANDIDATES (more returns EUNSUPPORTED)
 *   nbits         32..256, a multiple of 32
 *   max_dist      the normaliser of d_norm (> 0); threshold: reuse applies when the best
 *                 similarity is strictly above it
 *   mean_dist     device double[n_cand] or NULL: LSH_dist of every candidate (exact: the integer
 *                 sum of nearest distances divided by n_tgt in fp64)
 *   similarity    device double[n_cand] or NULL: clip(1 - mean_dist/max_dist, 0, 1) in fp64
 *   best          device int32: the candidate of greatest similarity, lowest index on ties
 *   applies       device int32 or NULL: 1 if similarity[best] > threshold, else 0
 *   idx, dist     device int32[n_tgt] or NULL: each target token's nearest row of the best
 *                 candidate (a global pool row; ties to the lowest row) and its distance --
 *                 semshare_match against that candidate's rows, shifted by its offset
 *   workspace     device scratch of at least semshare_retrieve_workspace_size(n_tgt, n_pool,
 *                 n_cand, nbits) bytes, 256-byte aligned; contents on entry do not matter
 *   err_flag      as for semshare_match_tc (SEMSHARE_FLAG_TIMEOUT: the outputs are invalid)
 * n_tgt must be >= 1 (the mean of no distances is undefined).  Returns EINVAL / EUNSUPPORTED
 * for bad arguments before anything is enqueued, ECUDA if a launch fails.  Outputs are written
 * in stream order; read them after synchronising the stream.
 */
#define SEMSHARE_RETRIEVE_MAX_CANDIDATES 256
size_t semshare_retrieve_workspace_size(int64_t n_tgt, int64_t n_pool, int32_t n_cand, int32_t nbits);
semshare_status semshare_retrieve(const uint32_t* tgt_codes, int64_t n_tgt, const uint32_t* pool_codes,
                                  const int64_t* cand_offsets, int32_t n_cand, int32_t nbits, double max_dist,
                                  double threshold, double* mean_dist, double* similarity, int32_t* best,
                                  int32_t* applies, int32_t* idx, int32_t* dist, void* workspace,
                                  size_t workspace_bytes, uint32_t* err_flag, void* stream);

/*
 * semshare_match_tc_selected -- token matching (Sec. 3.3) against the candidate that a device
 * value names, with no host round trip.
 *
 * After retrieval (semshare_retrieve, Sec. 3.2) the target's tokens are matched against the
 * chosen reference prompt.  This entry point reads the choice (`best`, e.g. semshare_retrieve's
 * output) on the device, so retrieval, matching and the gather can be enqueued back to back (and
 * captured in one CUDA graph) without the host learning the winner first.  For every target
 * token t, with c = *best:
 *     idx[t]  = cand_offsets[c] + the nearest row of candidate c (ties to the lowest row)
 *     dist[t] = its Hamming distance
 * -- semshare_match_tc against candidate c's rows, shifted to pool rows, so that
 * semshare_gather_kv over the pool's segments (one per candidate) gathers the right rows.
 *
 *   tgt_codes, nbits  as for semshare_match_tc
 *   pool_codes        device, [n_pool][nbits/32], every candidate's codes back to back
 *   cand_offsets      HOST, as for semshare_retrieve (strictly increasing, from 0)
 *   best              device int32: the candidate; outside [0, n_cand) sets SEMSHARE_FLAG_INDEX
 *                     and every idx/dist to -1
 *   idx, dist         device int32[n_tgt] (dist may be NULL)
 *   workspace         device scratch of at least semshare_match_tc_selected_workspace_size(
 *                     n_tgt, cand_offsets, n_cand, nbits) bytes, 256-byte aligned
 *   err_flag          as for semshare_match_tc
 * The search is sized for the longest candidate; a shorter one leaves its tail columns masked.
 * Returns EINVAL / EUNSUPPORTED for bad arguments, ECUDA if a launch fails.
 */
size_t semshare_match_tc_selected_workspace_size(int64_t n_tgt, const int64_t* cand_offsets, int32_t n_cand,
                                                 int32_t nbits);
semshare_status semshare_match_tc_selected(const uint32_t* tgt_codes, int64_t n_tgt, const uint32_t* pool_codes,
                                           const int64_t* cand_offsets, int32_t n_cand, const int32_t* best,
                                           int32_t nbits, int32_t* idx, int32_t* dist, void* workspace,
                                           size_t workspace_bytes, uint32_t* err_flag, void* stream);

/*
 * semshare_match_static -- semshare_match without a caller-provided workspace.
 *
 * The paper has no counterpart: this entry point exists for callers that cannot allocate
 * device memory (for example code embedded in a host framework that owns the whole device
 * memory pool and forbids allocations, or a serving loop that must not allocate on its hot
 * path).  It computes exactly what semshare_match computes, with the same arguments minus the
 * workspace, and allocates nothing: its scratch (one 64-bit key per target) is a fixed array
 * inside the library, SEMSHARE_MATCH_STATIC_MAX_TARGETS keys (2 MiB), which every device that
 * loads the library holds until the process exits.
 *
 *   n_tgt      0 <= n_tgt <= SEMSHARE_MATCH_STATIC_MAX_TARGETS; larger requests return
 *              SEMSHARE_ETOOLARGE before anything is enqueued
 *   other arguments as for semshare_match
 * The first call on a device looks up that device's address of the array (with the device
 * current), and looks it up again on the first call after the device's current context has
 * changed (cudaDeviceReset, or a context the caller made current); make the first call on a
 * device, and the first after such a change, before any stream capture.  All calls on a
 * device share the one array and it keeps the previous call's contents; each call resets the
 * keys it uses before its search.  Calls whose work overlaps on the GPU (other streams, other
 * host threads on the same device) race on the array and give wrong results: serialise them.
 * Unlike the other entry points this one keeps state: the array and the per-device address.
 */
#define SEMSHARE_MATCH_STATIC_MAX_TARGETS 262144
semshare_status semshare_match_static(const uint32_t* tgt_codes, int64_t n_tgt, const uint32_t* ref_codes,
                                      int64_t n_ref, int32_t nbits, int32_t* idx, int32_t* dist, void* stream);

/*
 * Layout of a K or V cache: element (b, l, h, t, e) of a cache with this layout lives at
 * element offset b*stride_batch + l*stride_layer + h*stride_head + t*stride_token + e.
 * A row (fixed b, l, h, t) holds head_dim contiguous elements of elem_bytes bytes.
 */
typedef struct {
    int32_t n_layers;     /* L */
    int32_t n_heads;      /* KV heads H */
    int32_t head_dim;     /* elements per row */
    int32_t elem_bytes;   /* 2 for bf16/fp16, 4 for fp32 */
    int64_t stride_batch; /* elements; ignored for the reference cache */
    int64_t stride_layer;
    int64_t stride_head;
    int64_t stride_token;
} semshare_kv_layout;

/*
 * semshare_gather_kv -- step 4: rearrange the reference K/V cache to the target's order.
 *
 * Sec. 3.3: the reordered cache matches the target prompt's length and its key-value pairs
 * all come from the reference cache; Sec. 3.3.2: K/V are stored after RoPE, so rows are
 * copied bit for bit with no re-encoding.  For every target prompt b < n_batch, layer l,
 * KV head h and target token t < n_tgt:
 *     out_k[b][l][h][t][:] = ref_k[l][h][idx[b*n_tgt + t]][:]      (same for V)
 *
 *   ref_k, ref_v   host arrays of n_seg base pointers, one reference prompt each: device memory,
 *                  or page-locked host memory the device can address (the kernel then reads the
 *                  selected rows across the host link, and only those rows cross it).
 *                  Global reference row r belongs to the segment s with
 *                  seg_offsets[s] <= r < seg_offsets[s+1] and is its local row
 *                  r - seg_offsets[s].  Every segment uses the strides of `src`.
 *   seg_offsets    host, n_seg+1 ascending int64 values, seg_offsets[0] = 0
 *   n_seg          1 <= n_seg <= 64
 *   src            layout of every reference segment (stride_batch ignored)
 *   idx            device, [n_batch][n_tgt] int32 global reference rows (from semshare_match)
 *   n_tgt, n_batch target tokens per prompt and prompts; 0 of either launches nothing
 *   out_k, out_v   device destination caches with layout `dst`
 *   dst            layout of the destination (same n_layers, n_heads, head_dim, elem_bytes)
 *   err_flag       device or NULL; a row whose idx lies outside [0, seg_offsets[n_seg]) is
 *                  not written and SEMSHARE_FLAG_INDEX is OR-ed in
 * Every base pointer and every stride (in bytes) must be a multiple of 16, and
 * head_dim*elem_bytes a multiple of 16: rows move as 16-byte vectors.
 * Returns EINVAL for bad arguments, ECUDA if the launch fails.
 */
semshare_status semshare_gather_kv(const void* const* ref_k, const void* const* ref_v, const int64_t* seg_offsets,
                                   int32_t n_seg, semshare_kv_layout src, const int32_t* idx, int64_t n_tgt,
                                   int32_t n_batch, void* out_k, void* out_v, semshare_kv_layout dst,
                                   uint32_t* err_flag, void* stream);

/*
 * semshare_hd_count -- how many tokens of a layer are high-deviation (HD) tokens.
 *
 * Insight 1 (App. A.4) names the tokens with the highest KV deviation, 40% of them, HD tokens.
 * Returns ceil(n_tok * percent / 100) computed in integers (percent = 40 for the paper's
 * figure), the k that semshare_select_hd takes.  Host-only, no device work.
 *   n_tok     0 <= n_tok < 2^40
 *   percent   0..100
 * Returns -1 for arguments outside those ranges.
 */
int64_t semshare_hd_count(int64_t n_tok, int32_t percent);

/*
 * semshare_retain_counts -- retained tokens per layer, Retain[i] = T * prod_{j<=i} alpha[j].
 *
 * App. A gives the number of tokens layer i keeps as the product of T (the target's length)
 * and the retention ratios of layers 0..i; Sec. 3.3.4 sets them.  The ratios are rationals
 * alpha[j] = alpha_num[j] / alpha_den, and the count is rounded down exactly (integer
 * arithmetic on the exact product, no floating point): counts[i] = floor(T * prod num / den^(i+1)).
 * Host-only, no device work.
 *   n_tok       T, 0 <= T < 2^31
 *   alpha_num   host int32[n_layers], 0 <= alpha_num[j] <= alpha_den
 *   alpha_den   >= 1 (e.g. 1000 for ratios given to three decimals)
 *   n_layers    0..128
 *   counts      host int64[n_layers], written
 * Returns EINVAL for arguments outside those ranges.
 */
semshare_status semshare_retain_counts(int64_t n_tok, const int32_t* alpha_num, int32_t alpha_den,
                                       int32_t n_layers, int64_t* counts);

/*
 * semshare_gather_kv_retained -- step 4 with retention: each layer keeps only its retained tokens.
 *
 * Sec. 3.3.4 and App. A: layer i retains Retain[i] = T * prod_{j<=i} alpha_retain[j] of the T
 * target tokens and evicts the rest.  Given each layer's retained target tokens (chosen from
 * attention scores by the caller), the layer's rearranged cache holds only their rows, packed in
 * list order, for one target prompt:
 *     out_k[l][h][r][:] = ref_k[l][h][idx[retained[ret_offsets[l] + r]]][:]    (same for V)
 * for r < ret_offsets[l+1] - ret_offsets[l].  Evicted tokens are neither read nor written.
 *
 *   ref_k, ref_v, seg_offsets, n_seg, src   as for semshare_gather_kv
 *   idx          device int32[n_tgt]: the target prompt's global reference rows
 *   retained     device int32: the layers' retained target tokens back to back (values in
 *                [0, n_tgt); conventionally ascending within a layer)
 *   ret_offsets  HOST int64[n_layers + 1], ret_offsets[0] = 0, non-decreasing; read before the
 *                call returns.  n_layers <= SEMSHARE_RETAIN_MAX_LAYERS
 *   out_k, out_v device destination, layout `dst` (stride_batch ignored); its token dimension must
 *                hold the longest list; rows past a layer's count are left untouched
 *   err_flag     device or NULL; a retained token outside [0, n_tgt) or an idx outside the
 *                reference leaves its row untouched and sets SEMSHARE_FLAG_INDEX
 * Alignment rules as for semshare_gather_kv.  Returns EINVAL / EUNSUPPORTED for bad arguments,
 * ECUDA if the launch fails.
 */
#define SEMSHARE_RETAIN_MAX_LAYERS 128
semshare_status semshare_gather_kv_retained(const void* const* ref_k, const void* const* ref_v,
                                            const int64_t* seg_offsets, int32_t n_seg, semshare_kv_layout src,
                                            const int32_t* idx, int64_t n_tgt, const int32_t* retained,
                                            const int64_t* ret_offsets, void* out_k, void* out_v,
                                            semshare_kv_layout dst, uint32_t* err_flag, void* stream);

/*
 * semshare_fetch_rows -- bring the reference rows a match selects into device memory, each once.
 *
 * Sec. 3.2 loads the retrieved reference prompt onto the GPU with its KV cache before the
 * rearrangement of Sec. 3.3, which reads only the rows the match selects -- and several target
 * tokens often select the same row.  For every layer l, KV head h and global reference row r
 * that some idx[i] (i < n_idx) names:
 *     dev_k[s][l][h][r - seg_offsets[s]][:] = ref_k[s][l][h][r - seg_offsets[s]][:]  (same for V)
 * with s the segment of r.  Rows that no idx names are neither read nor written, so a row
 * selected by many targets crosses the host link once; semshare_gather_kv (or _retained) with
 * ref_k/ref_v replaced by dev_k/dev_v and the same idx then gives the same result as on the
 * original cache.  Copies are bitwise.
 *
 *   ref_k, ref_v     host arrays of n_seg source base pointers: device memory or page-locked
 *                    host memory the device can address
 *   dev_k, dev_v     host arrays of n_seg device base pointers, each segment laid out like its
 *                    source (same strides, `layout`); may not overlap the sources
 *   seg_offsets, n_seg, layout   as seg_offsets, n_seg and src of semshare_gather_kv
 *   idx              device int32[n_idx]: global reference rows (any order, repeats allowed)
 *   workspace        device scratch of at least semshare_fetch_workspace_size(n_rows) bytes,
 *                    n_rows = seg_offsets[n_seg]; the call rewrites all of it
 *   err_flag         device or NULL; an idx outside [0, n_rows) is skipped and sets
 *                    SEMSHARE_FLAG_INDEX
 * Alignment rules as for semshare_gather_kv.  n_idx = 0 or n_rows = 0 launches nothing.
 * Returns EINVAL for bad arguments, EUNSUPPORTED for n_rows >= 2^31, ECUDA if a launch fails.
 */
size_t semshare_fetch_workspace_size(int64_t n_rows);
semshare_status semshare_fetch_rows(const void* const* ref_k, const void* const* ref_v, void* const* dev_k,
                                    void* const* dev_v, const int64_t* seg_offsets, int32_t n_seg,
                                    semshare_kv_layout layout, const int32_t* idx, int64_t n_idx, void* workspace,
                                    size_t workspace_bytes, uint32_t* err_flag, void* stream);

/*
 * semshare_kv_deviation -- Key-Value deviation of the reused cache (App. A.4).
 *
 * sigma_K = ||K_reused - K_recomputed||_2, sigma_V likewise, sigma_KV = sigma_K + sigma_V
 * (App. A.4), computed for every layer l < n_layers and token t < n_tok, the norm running over
 * all n_heads x head_dim values of that token:
 *     sigma_k[l][t] = sqrt(sum_h sum_e (k_reused[l][h][t][e] - k_recomp[l][h][t][e])^2)
 * On the first layer every token is recomputed and this comparison picks the tokens for
 * recomputation (Sec. 3.2); pass one layer (n_layers = 1) for that, more for per-layer analysis.
 *
 *   k_reused, v_reused  device, the rearranged cache (e.g. semshare_gather_kv's output for one
 *                       target prompt), layout `reused` (stride_batch ignored)
 *   k_recomp, v_recomp  device, the recomputed cache, layout `recomp`; n_layers, n_heads,
 *                       head_dim and elem_bytes equal to `reused`'s
 *   dtype               SEMSHARE_BF16 (elem_bytes 2) or SEMSHARE_F32 (elem_bytes 4)
 *   n_tok               tokens; 0 launches nothing
 *   sigma_k, sigma_v    device float[n_layers][n_tok] or NULL
 *   sigma_kv            device float[n_layers][n_tok]
 * Differences are squared and summed in fp32 in a fixed order (the same bits on every call);
 * sqrt is correctly rounded.  Base pointers, strides (in bytes) and head_dim*elem_bytes must be
 * multiples of 16.  Returns EINVAL for bad arguments, ECUDA if the launch fails.
 */
semshare_status semshare_kv_deviation(const void* k_reused, const void* v_reused, semshare_kv_layout reused,
                                      const void* k_recomp, const void* v_recomp, semshare_kv_layout recomp,
                                      semshare_dtype dtype, int64_t n_tok, float* sigma_k, float* sigma_v,
                                      float* sigma_kv, void* stream);

/*
 * semshare_select_hd -- the high-deviation (HD) tokens of every layer.
 *
 * Insight 1 calls the tokens of highest KV deviation (40% of them) HD tokens; Sec. 3.2 hands
 * the ones found on the first layer to recomputation.  For each layer l < n_layers: the k tokens
 * with the largest sigma[l][t], ties at the k-th value going to the lower token index, listed in
 * ascending token order.  The order is total: every NaN (either sign, any payload) counts as
 * larger than every number, including +inf, and NaNs tie with each other (lower token first);
 * -0 and +0 are the same value.
 *
 *   sigma     device float[n_layers][n_tok] (e.g. semshare_kv_deviation's sigma_kv)
 *   k         0 <= k <= n_tok (the paper's 40%: k = ceil(0.4 * n_tok))
 *   hd_idx    device int32[n_layers][k]
 *   hd_mask   device uint8[n_layers][n_tok] or NULL: 1 for an HD token, else 0
 * n_tok < 2^31, n_layers <= 65535.  Returns EINVAL for bad arguments, ECUDA if the launch fails.
 */
semshare_status semshare_select_hd(const float* sigma, int32_t n_layers, int64_t n_tok, int64_t k, int32_t* hd_idx,
                                   uint8_t* hd_mask, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* SEMSHARE_H */
