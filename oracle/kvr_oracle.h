/*
 * kvr_oracle.h -- plain fp64 CPU oracle of the evicted-KV decode step.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product path may call this code:
 * only the tests, the smoke check and the CPU-baseline leg of the benchmark use
 * it.  It shares no code, header, table or constant with the CUDA library.
 *
 * What it computes (KV-Rescue, arXiv 2608.15797):
 *   - Attn(q_t, C_t^B) of Eq. 1 (Sec. 2.1) for the G query heads that share one
 *     KV head (grouped-query attention), softmax scale 1/sqrt(d) unless given;
 *   - the accumulated-attention importance s_i named in Sec. 2.1 (the example
 *     score of Eq. 1), updated every step by the mean over the G query heads of
 *     that step's attention probability;
 *   - TopB of Eq. 1 with the protected recent window of Sec. 4.1 / App. D
 *     (physical bound B' = B + w): the W most recent tokens are always kept,
 *     the B best of the rest are kept, ties go to the lower position;
 *   - eviction fires every step once the live length exceeds B' (App. D,
 *     "Decode compute").
 *
 * Layout: a "unit" is one (sequence, layer, KV head).  Every array is
 * unit-major; rows of a unit are kept compacted in slots [0, len) in entry
 * order.  Positions are int32.  All arithmetic is double.
 */
#ifndef KVR_ORACLE_H
#define KVR_ORACLE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Attention of G query heads over n rows of one KV head (Eq. 1, Attn).
 * K, V: [n][d]; q: [G][d]; out: [G][d]; prob: [G][n] (may be NULL).
 * Returns 0, or -1 if n < 1. */
int kvro_attend_unit(int n, int d, int G, double scale, const double *K,
                     const double *V, const double *q, double *out,
                     double *prob);

/* TopB selection with a protected window (Eq. 1 + Sec. 4.1).
 * keep[i] is set to 1 for retained rows, 0 for evicted ones.
 * Returns the number of evicted rows (0 when n <= B + W), -1 on bad input. */
int kvro_select_unit(int n, const double *score, const int32_t *pos, int B,
                     int W, uint8_t *keep);

/* One decode step for n_units units (append, attend, accumulate, optionally
 * evict).  K, V: [n_units][cap][d]; score: [n_units][cap]; pos:
 * [n_units][cap]; len: [n_units]; q: [n_units][G][d]; k_new, v_new:
 * [n_units][d]; new_pos: [n_units]; out: [n_units][G][d].
 * If evict != 0 the unit is cut back to B + W rows after the step.
 * Returns 0, or -1 if a unit has no room for the appended row. */
int kvro_step(int n_units, int cap, int d, int G, double scale, double *K,
              double *V, double *score, int32_t *pos, int32_t *len,
              const double *q, const double *k_new, const double *v_new,
              const int32_t *new_pos, int B, int W, int evict, double *out);

/* Evict every unit to B + W rows with kvro_select_unit, compacting stably. */
int kvro_evict(int n_units, int cap, int d, double *K, double *V,
               double *score, int32_t *pos, int32_t *len, int B, int W);

/* Keep exactly the rows with keep[u][i] != 0 (slots [0, len[u])) and compact
 * stably; used to adopt a retained set chosen elsewhere. */
int kvro_keep_rows(int n_units, int cap, int d, double *K, double *V,
                   double *score, int32_t *pos, int32_t *len,
                   const uint8_t *keep);

#ifdef __cplusplus
}
#endif
#endif
