/*
 * kvr_oracle.c -- plain fp64 CPU oracle of the evicted-KV decode step.
 *
 * TEST INFRASTRUCTURE ONLY (see kvr_oracle.h).  Written for clarity, not
 * speed: every quantity is computed directly from its definition, one unit
 * (sequence, layer, KV head) at a time, single-threaded.
 */
#include "kvr_oracle.h"

#include <math.h>
#include <stdlib.h>
#include <string.h>

/* Eq. 1, Attn(q_t, C): for each of the G query heads g,
 *   l_{g,i} = scale * <q_g, k_i>,  p_{g,i} = exp(l_{g,i} - max_j l_{g,j}) / sum,
 *   out_g   = sum_i p_{g,i} v_i.                                              */
int kvro_attend_unit(int n, int d, int G, double scale, const double *K,
                     const double *V, const double *q, double *out,
                     double *prob) {
  if (n < 1 || d < 1 || G < 1) return -1;
  double *p = (double *)malloc(sizeof(double) * (size_t)n);
  if (!p) return -1;
  for (int g = 0; g < G; ++g) {
    const double *qg = q + (size_t)g * d;
    double m = -INFINITY;
    for (int i = 0; i < n; ++i) {
      double dot = 0.0;
      for (int c = 0; c < d; ++c) dot += qg[c] * K[(size_t)i * d + c];
      p[i] = scale * dot;
      if (p[i] > m) m = p[i];
    }
    double z = 0.0;
    for (int i = 0; i < n; ++i) {
      p[i] = exp(p[i] - m);
      z += p[i];
    }
    for (int i = 0; i < n; ++i) p[i] /= z;
    double *og = out + (size_t)g * d;
    for (int c = 0; c < d; ++c) og[c] = 0.0;
    for (int i = 0; i < n; ++i)
      for (int c = 0; c < d; ++c) og[c] += p[i] * V[(size_t)i * d + c];
    if (prob)
      for (int i = 0; i < n; ++i) prob[(size_t)g * n + i] = p[i];
  }
  free(p);
  return 0;
}

typedef struct {
  double score;
  int32_t pos;
  int slot;
} kvro_row;

/* Newest position first: the protected window is the W largest positions. */
static int by_pos_desc(const void *a, const void *b) {
  const kvro_row *x = (const kvro_row *)a, *y = (const kvro_row *)b;
  return (x->pos < y->pos) - (x->pos > y->pos);
}

/* TopB order: higher accumulated score first; equal scores keep the earlier
 * (lower) position first. */
static int by_score_then_pos(const void *a, const void *b) {
  const kvro_row *x = (const kvro_row *)a, *y = (const kvro_row *)b;
  if (x->score > y->score) return -1;
  if (x->score < y->score) return 1;
  return (x->pos > y->pos) - (x->pos < y->pos);
}

int kvro_select_unit(int n, const double *score, const int32_t *pos, int B,
                     int W, uint8_t *keep) {
  if (n < 0 || B < 0 || W < 0) return -1;
  if (n <= B + W) {
    for (int i = 0; i < n; ++i) keep[i] = 1;
    return 0;
  }
  kvro_row *r = (kvro_row *)malloc(sizeof(kvro_row) * (size_t)n);
  if (!r) return -1;
  for (int i = 0; i < n; ++i) {
    r[i].score = score[i];
    r[i].pos = pos[i];
    r[i].slot = i;
    keep[i] = 0;
  }
  /* Protected recent window: the W most recent positions. */
  qsort(r, (size_t)n, sizeof(kvro_row), by_pos_desc);
  for (int i = 0; i < W; ++i) keep[r[i].slot] = 1;
  /* TopB over the remaining rows. */
  qsort(r + W, (size_t)(n - W), sizeof(kvro_row), by_score_then_pos);
  for (int i = 0; i < B; ++i) keep[r[W + i].slot] = 1;
  free(r);
  return n - (B + W);
}

/* Stable in-place compaction of one unit to the rows with keep != 0. */
static int compact_unit(int n, int d, double *K, double *V, double *score,
                        int32_t *pos, const uint8_t *keep) {
  int w = 0;
  for (int i = 0; i < n; ++i) {
    if (!keep[i]) continue;
    if (w != i) {
      memmove(K + (size_t)w * d, K + (size_t)i * d, sizeof(double) * d);
      memmove(V + (size_t)w * d, V + (size_t)i * d, sizeof(double) * d);
      score[w] = score[i];
      pos[w] = pos[i];
    }
    ++w;
  }
  return w;
}

int kvro_step(int n_units, int cap, int d, int G, double scale, double *K,
              double *V, double *score, int32_t *pos, int32_t *len,
              const double *q, const double *k_new, const double *v_new,
              const int32_t *new_pos, int B, int W, int evict, double *out) {
  double *prob = (double *)malloc(sizeof(double) * (size_t)G * cap);
  uint8_t *keep = (uint8_t *)malloc((size_t)cap);
  if (!prob || !keep) {
    free(prob);
    free(keep);
    return -1;
  }
  int rc = 0;
  for (int u = 0; u < n_units && rc == 0; ++u) {
    double *Ku = K + (size_t)u * cap * d, *Vu = V + (size_t)u * cap * d;
    double *su = score + (size_t)u * cap;
    int32_t *pu = pos + (size_t)u * cap;
    int n0 = len[u];
    if (n0 + 1 > cap) {
      rc = -1;
      break;
    }
    /* Append the step's key/value; its score starts at zero. */
    memcpy(Ku + (size_t)n0 * d, k_new + (size_t)u * d, sizeof(double) * d);
    memcpy(Vu + (size_t)n0 * d, v_new + (size_t)u * d, sizeof(double) * d);
    su[n0] = 0.0;
    pu[n0] = new_pos[u];
    int n = n0 + 1;
    /* Attend over every live row, the new one included. */
    kvro_attend_unit(n, d, G, scale, Ku, Vu, q + (size_t)u * G * d,
                     out + (size_t)u * G * d, prob);
    /* Accumulated attention: add the mean over the G query heads. */
    for (int i = 0; i < n; ++i) {
      double acc = 0.0;
      for (int g = 0; g < G; ++g) acc += prob[(size_t)g * n + i];
      su[i] += acc / G;
    }
    len[u] = n;
    if (evict && kvro_select_unit(n, su, pu, B, W, keep) > 0)
      len[u] = compact_unit(n, d, Ku, Vu, su, pu, keep);
  }
  free(prob);
  free(keep);
  return rc;
}

int kvro_evict(int n_units, int cap, int d, double *K, double *V,
               double *score, int32_t *pos, int32_t *len, int B, int W) {
  uint8_t *keep = (uint8_t *)malloc((size_t)cap);
  if (!keep) return -1;
  for (int u = 0; u < n_units; ++u) {
    double *Ku = K + (size_t)u * cap * d, *Vu = V + (size_t)u * cap * d;
    double *su = score + (size_t)u * cap;
    int32_t *pu = pos + (size_t)u * cap;
    if (kvro_select_unit(len[u], su, pu, B, W, keep) > 0)
      len[u] = compact_unit(len[u], d, Ku, Vu, su, pu, keep);
  }
  free(keep);
  return 0;
}

int kvro_keep_rows(int n_units, int cap, int d, double *K, double *V,
                   double *score, int32_t *pos, int32_t *len,
                   const uint8_t *keep) {
  for (int u = 0; u < n_units; ++u)
    len[u] = compact_unit(len[u], d, K + (size_t)u * cap * d,
                          V + (size_t)u * cap * d, score + (size_t)u * cap,
                          pos + (size_t)u * cap, keep + (size_t)u * cap);
  return 0;
}
