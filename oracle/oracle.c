/*
 * Plain CPU oracle for smashed-KV decode attention (HAMburger, arXiv 2505.20438).
 *
 * TEST INFRASTRUCTURE ONLY (see oracle.h).  Slow and direct on purpose: fp64
 * everywhere, one (sequence, head) at a time, loops in the order of the definition.
 *
 * What it computes, and where the paper fixes it:
 *  - A macro-step is one forward of the base model that stores ONE key/value set
 *    for the whole group of tokens it fused (Sec. 3.1; Sec. 3.7 "Token Fusion").
 *    The cache is therefore a list of slots, each standing for 1..4 tokens, and
 *    the attention of a decode step is ordinary softmax attention over that list:
 *    nothing in the paper weights a slot by its token count.
 *  - With a single token per slot the computation is the base model's own
 *    (Sec. 3.4; Sec. 3.7 "Minimal Overhead"), i.e. standard causal decode.
 *  - The base model is Llama-3.2-1B-Instruct (Sec. 4.1): rotate-half RoPE,
 *    grouped-query attention, softmax scale 1/sqrt(head_dim).
 *  - The merged embedding is sent to the base model with an offset position that
 *    reflects the fused token count (Sec. 3.2); the position of each new slot is
 *    an input here (slot index, or tokens so far).
 */
#include "oracle.h"

#include <math.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

double oracle_bf16_to_f64(uint16_t bits) {
  uint32_t u = (uint32_t)bits << 16;
  float f;
  memcpy(&f, &u, sizeof f);
  return (double)f;
}

uint16_t oracle_f64_to_bf16(double x) {
  uint16_t sign = signbit(x) ? 0x8000u : 0u;
  if (isnan(x)) return (uint16_t)(sign | 0x7FC0u);
  double ax = fabs(x);
  if (ax == 0.0) return sign;
  if (isinf(ax)) return (uint16_t)(sign | 0x7F80u);
  /* ax in [2^(e-1), 2^e).  bf16 keeps 8 significant bits, so its spacing there is
   * 2^(e-8); below 2^-126 (subnormal bf16) the spacing is fixed at 2^-133. */
  int e;
  (void)frexp(ax, &e);
  int qexp = e - 8;
  if (qexp < -133) qexp = -133;
  double r = ldexp(nearbyint(ldexp(ax, -qexp)), qexp); /* ties to even */
  if (r >= 0x1p128) return (uint16_t)(sign | 0x7F80u);
  float f = (float)r; /* exact: at most 8 significant bits, inside float range */
  uint32_t u;
  memcpy(&u, &f, sizeof u);
  return (uint16_t)(sign | (uint16_t)(u >> 16));
}

void oracle_rope_f64(const uint16_t *x, double *y, int32_t d, int64_t pos, double base) {
  int32_t half = d / 2;
  for (int32_t i = 0; i < half; ++i) {
    double inv_freq = pow(base, -(2.0 * (double)i) / (double)d);
    double theta = (double)pos * inv_freq;
    double c = cos(theta);
    double s = sin(theta);
    double x0 = oracle_bf16_to_f64(x[i]);
    double x1 = oracle_bf16_to_f64(x[i + half]);
    double x0c = x0 * c, x1s = x1 * s;
    double x1c = x1 * c, x0s = x0 * s;
    y[i] = x0c - x1s;
    y[i + half] = x1c + x0s;
  }
}

void oracle_rope_bf16(const uint16_t *x, uint16_t *y, int32_t rows, int32_t d, int64_t pos,
                      double base) {
  double *tmp = (double *)malloc(sizeof(double) * (size_t)d);
  for (int32_t r = 0; r < rows; ++r) {
    oracle_rope_f64(x + (size_t)r * d, tmp, d, pos, base);
    for (int32_t i = 0; i < d; ++i) y[(size_t)r * d + i] = oracle_f64_to_bf16(tmp[i]);
  }
  free(tmp);
}

/* Element offset of (slot n of sequence b, KV head g) in a pool, or -1 if the page id
 * is outside the pool. */
static int64_t slot_row(const oracle_cache *c, int32_t b, int64_t n, int32_t g) {
  int64_t page = c->page_table[(int64_t)b * c->max_pages + n / c->page_slots];
  if (page < 0 || page >= c->pool_pages) return -1;
  int64_t row = (page * c->n_kv_heads + g) * c->page_slots + n % c->page_slots;
  return row * c->head_dim;
}

static int64_t slot_meta(const oracle_cache *c, int32_t b, int64_t n) {
  int64_t page = c->page_table[(int64_t)b * c->max_pages + n / c->page_slots];
  if (page < 0 || page >= c->pool_pages) return -1;
  return page * c->page_slots + n % c->page_slots;
}

static int check_cache(const oracle_cache *c) {
  if (!c || c->batch < 0 || c->n_kv_heads <= 0 || c->n_q_heads <= 0 || c->head_dim <= 0 ||
      c->head_dim % 2 || c->page_slots <= 0 || c->n_q_heads % c->n_kv_heads)
    return ORACLE_EINVAL;
  return 0;
}

int oracle_gather(const oracle_cache *c, int32_t b, int32_t g, double *k_out, double *v_out) {
  if (check_cache(c) || b < 0 || b >= c->batch || g < 0 || g >= c->n_kv_heads)
    return ORACLE_EINVAL;
  int64_t L = c->num_slots[b];
  if (L < 0 || L > (int64_t)c->max_pages * c->page_slots) return ORACLE_EINVAL;
  for (int64_t j = 0; j < L; ++j) {
    int64_t off = slot_row(c, b, j, g);
    if (off < 0) return ORACLE_EPAGE;
    for (int32_t i = 0; i < c->head_dim; ++i) {
      k_out[j * c->head_dim + i] = oracle_bf16_to_f64(c->k_pool[off + i]);
      v_out[j * c->head_dim + i] = oracle_bf16_to_f64(c->v_pool[off + i]);
    }
  }
  return 0;
}

int oracle_fill(oracle_cache *c, const uint16_t *k_log, const uint16_t *v_log,
                const int32_t *pos, const int32_t *ntok, const int32_t *counts, int32_t lmax) {
  if (check_cache(c)) return ORACLE_EINVAL;
  const int64_t row = (int64_t)c->n_kv_heads * c->head_dim;
  for (int32_t b = 0; b < c->batch; ++b) {
    if (counts[b] < 0 || counts[b] > lmax || counts[b] > c->max_slots) return ORACLE_EINVAL;
    int64_t tokens = 0;
    for (int64_t j = 0; j < counts[b]; ++j) {
      const int64_t src = ((int64_t)b * lmax + j) * row;
      for (int32_t g = 0; g < c->n_kv_heads; ++g) {
        int64_t off = slot_row(c, b, j, g);
        if (off < 0) return ORACLE_EPAGE;
        memcpy(c->k_pool + off, k_log + src + (int64_t)g * c->head_dim,
               sizeof(uint16_t) * (size_t)c->head_dim);
        memcpy(c->v_pool + off, v_log + src + (int64_t)g * c->head_dim,
               sizeof(uint16_t) * (size_t)c->head_dim);
      }
      int64_t m = slot_meta(c, b, j);
      c->slot_pos[m] = pos[(int64_t)b * lmax + j];
      c->slot_ntok[m] = ntok[(int64_t)b * lmax + j];
      tokens += ntok[(int64_t)b * lmax + j];
    }
    c->num_slots[b] = counts[b];
    c->num_tokens[b] = tokens;
  }
  return 0;
}

/* Attention of one query row qh [d] (bf16 bits) over slots 0..count-1 of sequence b, KV
 * head g: weights w[count] and output out[d]. */
static int attend_prefix(const oracle_cache *c, const uint16_t *qh, int32_t b, int32_t g,
                         int64_t count, double *w, double *out) {
  const int32_t d = c->head_dim;
  const double scale = 1.0 / sqrt((double)d);
  for (int32_t i = 0; i < d; ++i) out[i] = 0.0;
  if (count <= 0) return 0; /* empty sequence: output 0 */
  double m = -INFINITY;
  for (int64_t j = 0; j < count; ++j) {
    int64_t off = slot_row(c, b, j, g);
    if (off < 0) return ORACLE_EPAGE;
    double s = 0.0;
    for (int32_t i = 0; i < d; ++i)
      s += oracle_bf16_to_f64(qh[i]) * oracle_bf16_to_f64(c->k_pool[off + i]);
    w[j] = s * scale;
    if (w[j] > m) m = w[j];
  }
  double l = 0.0;
  for (int64_t j = 0; j < count; ++j) {
    w[j] = exp(w[j] - m);
    l += w[j];
  }
  for (int64_t j = 0; j < count; ++j) {
    w[j] /= l;
    int64_t off = slot_row(c, b, j, g);
    for (int32_t i = 0; i < d; ++i) out[i] += w[j] * oracle_bf16_to_f64(c->v_pool[off + i]);
  }
  return 0;
}

/* Attention of one query head over one sequence: weights w[L] and output out[d]. */
static int attend_one(const oracle_cache *c, const uint16_t *q, int32_t b, int32_t h,
                      double *w, double *out) {
  const int32_t d = c->head_dim;
  const int32_t group = c->n_q_heads / c->n_kv_heads;
  const uint16_t *qh = q + ((int64_t)b * c->n_q_heads + h) * d;
  return attend_prefix(c, qh, b, h / group, c->num_slots[b], w, out);
}

int oracle_decode_attn(const oracle_cache *c, const uint16_t *q, double *out,
                       int32_t n_threads) {
  if (check_cache(c) || !q || !out) return ORACLE_EINVAL;
  for (int32_t b = 0; b < c->batch; ++b)
    if (c->num_slots[b] < 0 || c->num_slots[b] > (int64_t)c->max_pages * c->page_slots)
      return ORACLE_EINVAL;
  const int64_t pairs = (int64_t)c->batch * c->n_q_heads;
  int status = 0;
#ifdef _OPENMP
  int nt = n_threads > 0 ? n_threads : omp_get_max_threads();
#pragma omp parallel for schedule(dynamic, 1) num_threads(nt) reduction(min : status)
#endif
  for (int64_t bh = 0; bh < pairs; ++bh) {
    int32_t b = (int32_t)(bh / c->n_q_heads), h = (int32_t)(bh % c->n_q_heads);
    int64_t L = c->num_slots[b];
    double *w = (double *)malloc(sizeof(double) * (size_t)(L > 0 ? L : 1));
    int rc = attend_one(c, q, b, h, w, out + bh * c->head_dim);
    free(w);
    if (rc < status) status = rc;
  }
  (void)n_threads;
  return status;
}

int oracle_attn_weights(const oracle_cache *c, const uint16_t *q, int32_t b, int32_t h,
                        double *w) {
  if (check_cache(c) || b < 0 || b >= c->batch || h < 0 || h >= c->n_q_heads)
    return ORACLE_EINVAL;
  double *out = (double *)malloc(sizeof(double) * (size_t)c->head_dim);
  int rc = attend_one(c, q, b, h, w, out);
  free(out);
  return rc;
}

int oracle_append(oracle_cache *c, const uint16_t *k_new, const uint16_t *v_new,
                  uint16_t *q_inout, const int32_t *pos, const int32_t *ntok,
                  int32_t pos_mode, double rope_base) {
  if (check_cache(c) || !k_new || !v_new || !ntok || pos_mode < 0 || pos_mode > 1)
    return ORACLE_EINVAL;
  const int32_t d = c->head_dim;
  int status = 0;
  for (int32_t b = 0; b < c->batch; ++b) {
    int64_t n = c->num_slots[b];
    if (ntok[b] < 1) { status = ORACLE_EINVAL; continue; }
    if (n >= c->max_slots) { status = ORACLE_ECAPACITY; continue; }
    int64_t p = pos ? pos[b] : (pos_mode == 0 ? n : c->num_tokens[b]);
    int64_t m = slot_meta(c, b, n);
    if (m < 0) { status = ORACLE_EPAGE; continue; }
    for (int32_t g = 0; g < c->n_kv_heads; ++g) {
      int64_t off = slot_row(c, b, n, g);
      const uint16_t *kg = k_new + ((int64_t)b * c->n_kv_heads + g) * d;
      oracle_rope_bf16(kg, c->k_pool + off, 1, d, p, rope_base);
      memcpy(c->v_pool + off, v_new + ((int64_t)b * c->n_kv_heads + g) * d,
             sizeof(uint16_t) * (size_t)d);
    }
    if (q_inout) {
      uint16_t *qb = q_inout + (int64_t)b * c->n_q_heads * d;
      oracle_rope_bf16(qb, qb, c->n_q_heads, d, p, rope_base);
    }
    c->slot_pos[m] = (int32_t)p;
    c->slot_ntok[m] = ntok[b];
    c->num_slots[b] = (int32_t)(n + 1);
    c->num_tokens[b] += ntok[b];
  }
  return status;
}

/* Chunked prefill.  A prompt's tokens are not fused (the paper fuses only response tokens:
 * Figure 2, training, item 2), so every new row becomes its own slot.  Sequence b's new rows
 * are offsets[b] .. offsets[b+1]-1, in order; with L = num_slots[b] before the call, row
 * r = offsets[b] + j becomes slot L + j exactly as oracle_append would append it (position
 * pos[r], or the slot index / the tokens so far), and its query heads then attend over slots
 * 0 .. L + j of the sequence: the causal attention of the chunk over the cache and over
 * itself.  want (nullable, [T]) restricts the attention to the rows it marks (the others get
 * 0; every row is still appended), for sampled checks of large chunks.  A sequence whose rows do not all fit (a token count < 1, no room, a bad page) is
 * left untouched and its out rows are 0.  q [T][n_q_heads][d] is rotated in place; out
 * [T][n_q_heads][d] doubles. */
int oracle_prefill(oracle_cache *c, uint16_t *q, const uint16_t *k_new, const uint16_t *v_new,
                   const int32_t *offsets, const int32_t *pos, const int32_t *ntok,
                   int32_t pos_mode, double rope_base, double *out, const uint8_t *want,
                   int32_t n_threads) {
  if (check_cache(c) || !q || !k_new || !v_new || !offsets || !ntok || !out || pos_mode < 0 ||
      pos_mode > 1 || offsets[0] != 0)
    return ORACLE_EINVAL;
  for (int32_t b = 0; b < c->batch; ++b)
    if (offsets[b + 1] < offsets[b]) return ORACLE_EINVAL;
  const int32_t d = c->head_dim, hq = c->n_q_heads, hkv = c->n_kv_heads;
  const int64_t T = offsets[c->batch];
  int64_t *row_slot = (int64_t *)malloc(sizeof(int64_t) * (size_t)(T > 0 ? T : 1));
  int status = 0;
  for (int32_t b = 0; b < c->batch; ++b) {
    const int64_t L = c->num_slots[b], n = offsets[b + 1] - offsets[b];
    int rc = 0;
    for (int64_t j = 0; j < n && !rc; ++j)
      if (ntok[offsets[b] + j] < 1) rc = ORACLE_EINVAL;
    if (!rc && L + n > c->max_slots) rc = ORACLE_ECAPACITY;
    for (int64_t j = 0; j < n && !rc; ++j)
      if (slot_meta(c, b, L + j) < 0) rc = ORACLE_EPAGE;
    if (rc) {
      if (rc < status) status = rc;
      for (int64_t j = 0; j < n; ++j) row_slot[offsets[b] + j] = -1;
      continue;
    }
    for (int64_t j = 0; j < n; ++j) {
      const int64_t r = offsets[b] + j, slot = L + j;
      const int64_t p = pos ? pos[r] : (pos_mode == 0 ? slot : c->num_tokens[b]);
      for (int32_t g = 0; g < hkv; ++g) {
        int64_t off = slot_row(c, b, slot, g);
        oracle_rope_bf16(k_new + (r * hkv + g) * d, c->k_pool + off, 1, d, p, rope_base);
        memcpy(c->v_pool + off, v_new + (r * hkv + g) * d, sizeof(uint16_t) * (size_t)d);
      }
      oracle_rope_bf16(q + r * hq * d, q + r * hq * d, hq, d, p, rope_base);
      int64_t m = slot_meta(c, b, slot);
      c->slot_pos[m] = (int32_t)p;
      c->slot_ntok[m] = ntok[r];
      c->num_slots[b] = (int32_t)(slot + 1);
      c->num_tokens[b] += ntok[r];
      row_slot[r] = slot;
    }
  }
  /* row r, head h: slots 0 .. row_slot[r] of its sequence (b found from the offsets) */
  const int64_t pairs = T * hq;
  int astatus = 0;
#ifdef _OPENMP
  int nt = n_threads > 0 ? n_threads : omp_get_max_threads();
#pragma omp parallel for schedule(dynamic, 16) num_threads(nt) reduction(min : astatus)
#endif
  for (int64_t rh = 0; rh < pairs; ++rh) {
    const int64_t r = rh / hq;
    const int32_t h = (int32_t)(rh % hq);
    int32_t b = 0;
    while (offsets[b + 1] <= r) ++b;
    double *o = out + rh * d;
    if (row_slot[r] < 0 || (want && !want[r])) {
      for (int32_t i = 0; i < d; ++i) o[i] = 0.0;
      continue;
    }
    double *w = (double *)malloc(sizeof(double) * (size_t)(row_slot[r] + 1));
    int rc = attend_prefix(c, q + rh * d, b, h / (hq / hkv), row_slot[r] + 1, w, o);
    free(w);
    if (rc < astatus) astatus = rc;
  }
  (void)n_threads;
  free(row_slot);
  return status < astatus ? status : astatus;
}

int oracle_max_threads(void) {
#ifdef _OPENMP
  return omp_get_max_threads();
#else
  return 1;
#endif
}
