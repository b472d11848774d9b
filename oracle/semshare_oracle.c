/*
 * semshare_oracle.c -- CPU oracle for SemShareKV's fuzzy token-matching path.
 *
 * TEST INFRASTRUCTURE ONLY.  The tests, the smoke check and the bench's CPU-baseline leg
 * are the only callers.  The product path (the CUDA library) never calls, links or loads
 * this file, and this file shares no code, header, table or helper with it.
 *
 * It is a plain, slow restatement of what the path computes, in fp64, one step at a time,
 * in the paper's order (SemShareKV, arXiv 2509.24832):
 *
 *   1. rope    Rotary position encoding of every embedding row (Sec. 3.3.1: RoPE is applied
 *              to the E cache of both the reference and the target prompt; formula Eq. 1,
 *              App. A.1).  Pair (x[2k], x[2k+1]) of the row at position m is rotated by the
 *              angle m * theta_k, theta_k = base^(-2k/d), d = the embedding dimension.
 *              A second pairing, (k, k + d/2) ("rotate-half"), is available as an option.
 *   2. hash    Random-hyperplane LSH (Sec. 3.3 "we use LSH", App. A.2, App. D "LSH from
 *              FAISS"): p_j = <r_j, y> for each of nbits hyperplanes r_j, code bit j = [p_j > 0],
 *              packed LSB-first into 32-bit words (bit j -> word j/32, bit j%32).
 *              Operand contract: y is rounded to bf16 (nearest, ties to even) before the
 *              products, the hyperplanes are bf16; the dot product is accumulated in fp64.
 *   3. match   For each target token the reference token with the smallest Hamming distance
 *              between codes (Sec. 3.3: "for each token in the target prompt, the most similar
 *              token in the reference prompt"); an exhaustive scan in ascending reference
 *              order that keeps the first minimum, so ties go to the lowest index.
 *   4. gather  The reordered cache has the target's length and every row comes from the
 *              reference cache (Sec. 3.3): out[b][l][h][t] = ref[l][h][idx[b][t]] for every
 *              layer l and KV head h, copied bit for bit (Sec. 3.3.2: KV is stored after RoPE,
 *              so nothing is re-encoded).
 *   5. retrieve  Reference retrieval (Sec. 3.2, App. A.3, Sec. 4.4): each stored candidate
 *              prompt's LSH distance to the target -- read as the mean over target tokens of the
 *              nearest Hamming distance -- is normalised by 30 and turned into a similarity in
 *              [0, 1]; the most similar candidate wins and is reused if above 0.8.
 *   6. kv_deviation / select_hd  Key-Value deviation (App. A.4): per layer and token,
 *              ||K_reused - K_recomputed||_2 + ||V_reused - V_recomputed||_2 over all heads; the
 *              tokens of highest deviation (40% in the paper, Insight 1) are the HD tokens that
 *              the first layer's comparison hands to recomputation (Sec. 3.2).
 *   7. gather_kv_retained  Retention (Sec. 3.3.4, App. A): each layer keeps only its retained
 *              target tokens; its rearranged cache holds just their rows, packed in list order.
 *
 * Build: gcc -O2 -fopenmp -ffp-contract=off -shared -fPIC (no fused multiply-add, so x86 and
 * Arm hosts produce the same bits).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#ifdef _OPENMP
#include <omp.h>
#endif

int oracle_num_threads(void) {
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

/* Threads of the following calls' parallel loops (n >= 1); returns the previous setting.  Only
 * the timing of the CPU baseline uses it: results do not depend on the thread count. */
int oracle_set_threads(int n) {
#ifdef _OPENMP
    const int prev = omp_get_max_threads();
    if (n >= 1) omp_set_num_threads(n);
    return prev;
#else
    (void)n;
    return 1;
#endif
}

/* ---- bf16 <-> fp64 --------------------------------------------------------------------- */

/* Value of a bf16 bit pattern (exact). */
double oracle_bf16_value(uint16_t h) {
    uint32_t u = (uint32_t)h << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

/* Nearest bf16 to v, ties to even, rounded once from the fp64 value.
 * (float)v is rounded first; that second rounding can only differ from the direct one when
 * (float)v lands exactly on a bf16 midpoint while v itself does not, and then the side v
 * lies on decides. */
uint16_t oracle_bf16_round(double v) {
    if (v != v) return (uint16_t)0x7FC0u;
    float f = (float)v;
    uint32_t u;
    memcpy(&u, &f, sizeof u);
    if ((u & 0xFFFFu) == 0x8000u && (double)f != v && !isinf(f))
        return (uint16_t)((u >> 16) + (fabs(v) > fabs((double)f) ? 1u : 0u));
    u += 0x7FFFu + ((u >> 16) & 1u);
    return (uint16_t)(u >> 16);
}

/* ---- step 1: rotary position encoding (Eq. 1) ----------------------------------------- */

/* theta_k = base^(-2k/d), the rotation frequency of pair k (Eq. 1, App. A.1). */
double oracle_theta(int32_t k, int32_t d, double base) {
    return pow(base, -2.0 * (double)k / (double)d);
}

/* Pair k of a row is (2k, 2k+1) as Eq. 1 prints it (half = 0), or (k, k + d/2), the
 * "rotate-half" arrangement of common implementations (half = 1); either way it turns by
 * m * theta_k. */
static void rope_row(const double* x, int32_t d, double m, const double* theta, double* y, int32_t half) {
    for (int32_t k = 0; k < d / 2; ++k) {
        const double a = m * theta[k];
        const double c = cos(a), s = sin(a);
        const int32_t i0 = half ? k : 2 * k, i1 = half ? k + d / 2 : 2 * k + 1;
        const double x0 = x[i0], x1 = x[i1];
        y[i0] = x0 * c - x1 * s;
        y[i1] = x0 * s + x1 * c;
    }
}

/* y[i] = RoPE(x[i], pos[i]) for n rows of width d (row-major, fp64); half selects the pairing. */
void oracle_rope_layout(const double* x, int64_t n, int32_t d, const int32_t* pos, double base, double* y,
                        int32_t half) {
    double* theta = (double*)malloc(sizeof(double) * (size_t)(d / 2));
    for (int32_t k = 0; k < d / 2; ++k) theta[k] = oracle_theta(k, d, base);
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < n; ++i)
        rope_row(x + i * d, d, (double)pos[i], theta, y + i * d, half);
    free(theta);
}

void oracle_rope(const double* x, int64_t n, int32_t d, const int32_t* pos, double base, double* y) {
    oracle_rope_layout(x, n, d, pos, base, y, 0);
}

/* ---- step 2: random-hyperplane LSH codes ----------------------------------------------- */

/* emb: n rows of d values, row i starting at element i*row_stride; emb_f32 = 1 for float32
 * rows, 0 for bf16 bit patterns.  positions: n token positions (NULL -> 0..n-1).
 * hyperplanes: [nbits][d] bf16 bit patterns.  codes: [n][nbits/32] words.
 * proj (nullable): [n][nbits] float projections (the fp64 sum rounded to float).
 * round_operand = 1 applies the bf16 operand contract to y; 0 keeps y in fp64 (diagnostic). */
void oracle_hash_layout(const void* emb, int32_t emb_f32, int64_t n, int32_t d, int64_t row_stride,
                        const int32_t* positions, double base, const uint16_t* hyperplanes, int32_t nbits,
                        uint32_t* codes, float* proj, int32_t round_operand, int32_t half) {
    const int32_t w = nbits / 32;
    double* theta = (double*)malloc(sizeof(double) * (size_t)(d / 2));
    double* r = (double*)malloc(sizeof(double) * (size_t)nbits * (size_t)d);
    for (int32_t k = 0; k < d / 2; ++k) theta[k] = oracle_theta(k, d, base);
    for (int64_t e = 0; e < (int64_t)nbits * d; ++e) r[e] = oracle_bf16_value(hyperplanes[e]);

#pragma omp parallel
    {
        double* x = (double*)malloc(sizeof(double) * (size_t)d);
        double* y = (double*)malloc(sizeof(double) * (size_t)d);
#pragma omp for schedule(dynamic, 16)
        for (int64_t i = 0; i < n; ++i) {
            for (int32_t c = 0; c < d; ++c)
                x[c] = emb_f32 ? (double)((const float*)emb)[i * row_stride + c]
                               : oracle_bf16_value(((const uint16_t*)emb)[i * row_stride + c]);
            const double m = positions ? (double)positions[i] : (double)i;
            rope_row(x, d, m, theta, y, half);
            if (round_operand)
                for (int32_t c = 0; c < d; ++c) y[c] = oracle_bf16_value(oracle_bf16_round(y[c]));
            for (int32_t q = 0; q < w; ++q) codes[i * w + q] = 0u;
            for (int32_t j = 0; j < nbits; ++j) {
                double p = 0.0;
                for (int32_t c = 0; c < d; ++c) p += r[(int64_t)j * d + c] * y[c];
                if (p > 0.0) codes[i * w + j / 32] |= 1u << (j % 32);
                if (proj) proj[i * nbits + j] = (float)p;
            }
        }
        free(x);
        free(y);
    }
    free(theta);
    free(r);
}

void oracle_hash(const void* emb, int32_t emb_f32, int64_t n, int32_t d, int64_t row_stride,
                 const int32_t* positions, double base, const uint16_t* hyperplanes, int32_t nbits,
                 uint32_t* codes, float* proj, int32_t round_operand) {
    oracle_hash_layout(emb, emb_f32, n, d, row_stride, positions, base, hyperplanes, nbits, codes, proj,
                       round_operand, 0);
}

/* ---- step 3: Hamming nearest neighbour ------------------------------------------------- */

/* Hamming distance between two packed codes of w words. */
int32_t oracle_hamming(const uint32_t* a, const uint32_t* b, int32_t w) {
    int32_t s = 0;
    for (int32_t q = 0; q < w; ++q) s += __builtin_popcount(a[q] ^ b[q]);
    return s;
}

/* idx[t] = the lowest j minimising hamming(tgt[t], ref[j]); dist[t] = that minimum. */
void oracle_match(const uint32_t* tgt, int64_t n_tgt, const uint32_t* ref, int64_t n_ref, int32_t nbits,
                  int32_t* idx, int32_t* dist) {
    const int32_t w = nbits / 32;
#pragma omp parallel for schedule(dynamic, 64)
    for (int64_t t = 0; t < n_tgt; ++t) {
        int32_t best = nbits + 1;
        int64_t best_j = -1;
        for (int64_t j = 0; j < n_ref; ++j) {
            const int32_t h = oracle_hamming(tgt + t * w, ref + j * w, w);
            if (h < best) {
                best = h;
                best_j = j;
            }
        }
        idx[t] = (int32_t)best_j;
        dist[t] = best;
    }
}

/* ---- step 4: KV rearrangement ---------------------------------------------------------- */

/* Reference cache: n_seg segments (one per reference prompt); segment s holds the global rows
 * seg_offsets[s] <= r < seg_offsets[s+1] as its local rows r - seg_offsets[s], laid out
 * [L][H][n_s][row_bytes] with n_s = seg_offsets[s+1] - seg_offsets[s].
 * idx: [n_batch][n_tgt] global rows.  out_k/out_v: [n_batch][L][H][n_tgt][row_bytes].
 * A row whose idx is outside [0, seg_offsets[n_seg]) is left untouched and counted.
 * Returns the number of such rows (per batch and target token). */
int64_t oracle_gather_kv(const uint8_t* const* seg_k, const uint8_t* const* seg_v, const int64_t* seg_offsets,
                         int32_t n_seg, int32_t L, int32_t H, int64_t row_bytes, const int32_t* idx, int64_t n_tgt,
                         int32_t n_batch, uint8_t* out_k, uint8_t* out_v) {
    const int64_t total = seg_offsets[n_seg];
    int64_t bad = 0;
    for (int64_t e = 0; e < (int64_t)n_batch * n_tgt; ++e)
        if (idx[e] < 0 || idx[e] >= total) ++bad;
#pragma omp parallel for collapse(2) schedule(static)
    for (int32_t b = 0; b < n_batch; ++b)
        for (int32_t l = 0; l < L; ++l)
            for (int32_t h = 0; h < H; ++h)
                for (int64_t t = 0; t < n_tgt; ++t) {
                    const int64_t r = idx[(int64_t)b * n_tgt + t];
                    if (r < 0 || r >= total) continue;
                    int32_t s = 0;
                    while (!(seg_offsets[s] <= r && r < seg_offsets[s + 1])) ++s;
                    const int64_t n_s = seg_offsets[s + 1] - seg_offsets[s];
                    const int64_t src_row = ((int64_t)l * H + h) * n_s + (r - seg_offsets[s]);
                    const int64_t dst_row = (((int64_t)b * L + l) * H + h) * n_tgt + t;
                    memcpy(out_k + dst_row * row_bytes, seg_k[s] + src_row * row_bytes, (size_t)row_bytes);
                    memcpy(out_v + dst_row * row_bytes, seg_v[s] + src_row * row_bytes, (size_t)row_bytes);
                }
    return bad;
}

/* ---- reference retrieval: LSH-distance similarity of whole prompts ------------------------ */

/* Reference retrieval (Sec. 3.2: the stored prompt with the highest LSH-distance-based
 * similarity to the target is retrieved; App. A.3: Similarity = clip(1 - (LSH_dist - 0)/(30 - 0),
 * 0, 1); Sec. 4.4: reuse applies when the similarity is above 0.8).  LSH_dist of a candidate
 * prompt is read here as the mean over the target tokens of each token's Hamming distance to
 * its nearest token of the candidate.  The pool is one code array; candidate s holds rows
 * seg_offsets[s] <= j < seg_offsets[s+1] (each non-empty).
 * Outputs: mean_dist[s], similarity[s] (n_seg doubles), *best = the lowest s of greatest
 * similarity, *applies = similarity[*best] > threshold. */
void oracle_retrieve(const uint32_t* tgt, int64_t n_tgt, const uint32_t* pool, const int64_t* seg_offsets,
                     int32_t n_seg, int32_t nbits, double dmax, double threshold, double* mean_dist,
                     double* similarity, int32_t* best, int32_t* applies) {
    const int32_t w = nbits / 32;
    for (int32_t s = 0; s < n_seg; ++s) {
        int64_t sum = 0;
#pragma omp parallel for reduction(+ : sum) schedule(dynamic, 64)
        for (int64_t t = 0; t < n_tgt; ++t) {
            int32_t m = nbits + 1;
            for (int64_t j = seg_offsets[s]; j < seg_offsets[s + 1]; ++j) {
                const int32_t h = oracle_hamming(tgt + t * w, pool + j * w, w);
                if (h < m) m = h;
            }
            sum += m;
        }
        mean_dist[s] = (double)sum / (double)n_tgt;
        double sim = 1.0 - mean_dist[s] / dmax;
        if (sim < 0.0) sim = 0.0;
        if (sim > 1.0) sim = 1.0;
        similarity[s] = sim;
    }
    int32_t b = 0;
    for (int32_t s = 1; s < n_seg; ++s)
        if (similarity[s] > similarity[b]) b = s;
    *best = b;
    *applies = similarity[b] > threshold ? 1 : 0;
}

/* ---- KV deviation and high-deviation tokens -------------------------------------------- */

/* Value of element e of a K/V array: bf16 bit patterns (is_f32 = 0) or float32. */
static double kv_elem(const void* base, int32_t is_f32, int64_t e) {
    return is_f32 ? (double)((const float*)base)[e] : oracle_bf16_value(((const uint16_t*)base)[e]);
}

/* Key-Value deviation (App. A.4): sigma_K = ||K_reused - K_recomputed||_2, sigma_V likewise,
 * sigma_KV = sigma_K + sigma_V.  Read per layer l and token t, the norm running over all heads
 * and head dimensions of that token's K (V) rows.  Arrays are [L][H][T][hd] contiguous.
 * Outputs [L][T] (sigma_k, sigma_v nullable). */
void oracle_kv_deviation(const void* k_re, const void* v_re, const void* k_rc, const void* v_rc, int32_t is_f32,
                         int32_t L, int32_t H, int64_t T, int32_t hd, double* sigma_k, double* sigma_v,
                         double* sigma_kv) {
#pragma omp parallel for collapse(2) schedule(static)
    for (int32_t l = 0; l < L; ++l)
        for (int64_t t = 0; t < T; ++t) {
            double sk = 0.0, sv = 0.0;
            for (int32_t h = 0; h < H; ++h)
                for (int32_t e = 0; e < hd; ++e) {
                    const int64_t i = (((int64_t)l * H + h) * T + t) * hd + e;
                    const double dk = kv_elem(k_re, is_f32, i) - kv_elem(k_rc, is_f32, i);
                    const double dv = kv_elem(v_re, is_f32, i) - kv_elem(v_rc, is_f32, i);
                    sk += dk * dk;
                    sv += dv * dv;
                }
            const double a = sqrt(sk), b = sqrt(sv);
            if (sigma_k) sigma_k[(int64_t)l * T + t] = a;
            if (sigma_v) sigma_v[(int64_t)l * T + t] = b;
            sigma_kv[(int64_t)l * T + t] = a + b;
        }
}

/* High-deviation tokens (Insight 1: the tokens of highest deviation, 40% of them in the paper):
 * for each layer, the k tokens of largest sigma (ties to the lower token index), listed in
 * ascending token order in hd_idx[l][0..k).  A plain sort of (-sigma, t) under a total order:
 * every NaN (either sign, any payload) ranks above +inf and NaNs tie with each other; -0 and +0
 * are the same number; equal values go to the lower token.  The comparator is therefore
 * transitive, so qsort's result is defined even when sigma holds NaNs. */
static const double* g_sort_sigma;
static int cmp_desc_sigma(const void* a, const void* b) {
    const int64_t i = *(const int64_t*)a, j = *(const int64_t*)b;
    const double x = g_sort_sigma[i], y = g_sort_sigma[j];
    const int nx = isnan(x) != 0, ny = isnan(y) != 0;
    if (nx != ny) return nx ? -1 : 1;     /* a NaN comes before every number */
    if (!nx) {                            /* two numbers (-0 == +0 here) */
        if (x > y) return -1;
        if (x < y) return 1;
    }
    return i < j ? -1 : (i > j ? 1 : 0);
}
static int cmp_i64(const void* a, const void* b) {
    const int64_t i = *(const int64_t*)a, j = *(const int64_t*)b;
    return i < j ? -1 : (i > j ? 1 : 0);
}

void oracle_select_hd(const double* sigma, int32_t L, int64_t T, int64_t k, int32_t* hd_idx) {
    int64_t* order = (int64_t*)malloc(sizeof(int64_t) * (size_t)(T > 0 ? T : 1));
    for (int32_t l = 0; l < L; ++l) {
        for (int64_t t = 0; t < T; ++t) order[t] = t;
        g_sort_sigma = sigma + (int64_t)l * T;
        qsort(order, (size_t)T, sizeof(int64_t), cmp_desc_sigma);
        qsort(order, (size_t)k, sizeof(int64_t), cmp_i64);
        for (int64_t i = 0; i < k; ++i) hd_idx[(int64_t)l * k + i] = (int32_t)order[i];
    }
    free(order);
}

/* ---- retention-aware rearrangement --------------------------------------------------------- */

/* Retention (Sec. 3.3.4; App. A: Retain[i] = T * prod_{j<=i} alpha_retain[j], tokens not retained
 * are evicted): layer l keeps only the target tokens ret[ret_off[l] .. ret_off[l+1]) and its
 * rearranged cache holds just those rows, packed in list order:
 *     out[l][h][r] = ref[l][h][idx[ret[ret_off[l] + r]]]
 * One reference prompt [L][H][N][row_bytes], idx [n_tgt], out [L][H][cap][row_bytes] (cap >= the
 * longest list; rows past a layer's count are left as they were).  A retained token outside
 * [0, n_tgt) or an idx outside [0, N) leaves its row untouched and is counted; returns the count. */
int64_t oracle_gather_kv_retained(const uint8_t* ref_k, const uint8_t* ref_v, int32_t L, int32_t H, int64_t N,
                                  int64_t row_bytes, const int32_t* idx, int64_t n_tgt, const int32_t* ret,
                                  const int64_t* ret_off, int64_t cap, uint8_t* out_k, uint8_t* out_v) {
    int64_t bad = 0;
    for (int32_t l = 0; l < L; ++l)
        for (int64_t r = 0; r < ret_off[l + 1] - ret_off[l]; ++r) {
            const int64_t t = ret[ret_off[l] + r];
            if (t < 0 || t >= n_tgt || idx[t] < 0 || idx[t] >= N) {
                ++bad;
                continue;
            }
            for (int32_t h = 0; h < H; ++h) {
                const int64_t src = (((int64_t)l * H + h) * N + idx[t]) * row_bytes;
                const int64_t dst = (((int64_t)l * H + h) * cap + r) * row_bytes;
                memcpy(out_k + dst, ref_k + src, (size_t)row_bytes);
                memcpy(out_v + dst, ref_v + src, (size_t)row_bytes);
            }
        }
    return bad;
}

/* ---- loading the selected reference rows ---------------------------------------------------- */

/* Sec. 3.2 loads the retrieved reference prompt's KV cache onto the GPU before the rearrangement
 * of Sec. 3.3, which reads only the rows the match selects.  This copies, for every layer l and
 * head h, each reference row r named by some idx[i] (i < n_idx) from seg_k/seg_v to dev_k/dev_v
 * (both laid out per segment as [L][H][n_s][row_bytes], as in oracle_gather_kv); every other row
 * of dev_k/dev_v is left as it was.  An idx outside [0, seg_offsets[n_seg]) is skipped and
 * counted; returns the count. */
int64_t oracle_fetch_rows(const uint8_t* const* seg_k, const uint8_t* const* seg_v, uint8_t* const* dev_k,
                          uint8_t* const* dev_v, const int64_t* seg_offsets, int32_t n_seg, int32_t L, int32_t H,
                          int64_t row_bytes, const int32_t* idx, int64_t n_idx) {
    const int64_t total = seg_offsets[n_seg];
    int64_t bad = 0;
    for (int64_t i = 0; i < n_idx; ++i) {
        const int64_t r = idx[i];
        if (r < 0 || r >= total) {
            ++bad;
            continue;
        }
        int32_t s = 0;
        while (!(seg_offsets[s] <= r && r < seg_offsets[s + 1])) ++s;
        const int64_t n_s = seg_offsets[s + 1] - seg_offsets[s];
        for (int32_t l = 0; l < L; ++l)
            for (int32_t h = 0; h < H; ++h) {
                const int64_t off = (((int64_t)l * H + h) * n_s + (r - seg_offsets[s])) * row_bytes;
                memcpy(dev_k[s] + off, seg_k[s] + off, (size_t)row_bytes);
                memcpy(dev_v[s] + off, seg_v[s] + off, (size_t)row_bytes);
            }
    }
    return bad;
}
