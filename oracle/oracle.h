/*
 * Plain CPU oracle for smashed-KV decode attention (HAMburger, arXiv 2505.20438).
 *
 * TEST INFRASTRUCTURE ONLY.  Only the tests, the smoke check and the bench's CPU
 * baseline may load this library.  It shares no code with the CUDA path: its own
 * page gather, its own RoPE, its own bf16 rounding, fp64 arithmetic throughout.
 *
 * Paged cache layout (the format the CUDA library documents for its pool, restated
 * and implemented here independently):
 *   K and V pools  [pool_pages][n_kv_heads][page_slots][head_dim]   bf16 bits (uint16)
 *   slot_pos/ntok  [pool_pages][page_slots]                          int32
 *   page_table     [batch][max_pages]                                int32
 *   slot n of sequence b lives in page page_table[b][n / page_slots], row n % page_slots.
 *
 * Return codes: 0 ok, ORACLE_EINVAL bad argument, ORACLE_EPAGE page id outside the
 * pool, ORACLE_ECAPACITY no room for a new slot.
 */
#ifndef HAM_ORACLE_H
#define HAM_ORACLE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define ORACLE_EINVAL (-1)
#define ORACLE_EPAGE (-2)
#define ORACLE_ECAPACITY (-3)

typedef struct {
  int32_t batch;
  int32_t n_q_heads;
  int32_t n_kv_heads;
  int32_t head_dim;
  int32_t page_slots;
  int32_t max_pages;        /* page-table row length */
  int64_t pool_pages;
  int64_t max_slots;        /* capacity of one sequence, in slots */
  uint16_t *k_pool;
  uint16_t *v_pool;
  int32_t *slot_pos;
  int32_t *slot_ntok;
  int32_t *page_table;
  int32_t *num_slots;       /* [batch] */
  int64_t *num_tokens;      /* [batch] */
} oracle_cache;

/* bf16 bits -> exact double.  (The paper fixes no rounding; the base model's tensors are bf16,
 * Sec. 4.1, and a stored element is decoded exactly.) */
double oracle_bf16_to_f64(uint16_t bits);
/* double -> bf16 bits, round to nearest, ties to even (overflow gives infinity): the one rounding
 * of a stored key and of an output, by the IEEE rule (reading c6; the paper fixes none). */
uint16_t oracle_f64_to_bf16(double x);

/* RoPE, rotate-half pairing (i, i + d/2), theta_i = pos * base^(-2i/d), all in fp64: the base
 * model's rotary embedding (Llama, Sec. 4.1) at the slot's offset position (Sec. 3.2). */
void oracle_rope_f64(const uint16_t *x, double *y, int32_t d, int64_t pos, double base);
/* Same rotation of `rows` vectors, each rounded to bf16. In-place use (x == y) is allowed. */
void oracle_rope_bf16(const uint16_t *x, uint16_t *y, int32_t rows, int32_t d, int64_t pos,
                      double base);

/* Logical view of sequence b, KV head g: k_out/v_out [num_slots[b]][head_dim] doubles.  The
 * cache is the list of slots, one key/value set per macro-step (Sec. 3.1); the pages are only
 * where the list is stored. */
int oracle_gather(const oracle_cache *c, int32_t b, int32_t g, double *k_out, double *v_out);

/* Scatter a logical cache [batch][lmax][n_kv_heads][head_dim] into the pages and set
 * num_slots = counts, slot metadata from pos/ntok [batch][lmax], num_tokens = sum ntok
 * (the slot list of Sec. 3.1, each slot standing for ntok tokens, Sec. 3.7 "Token Fusion"). */
int oracle_fill(oracle_cache *c, const uint16_t *k_log, const uint16_t *v_log,
                const int32_t *pos, const int32_t *ntok, const int32_t *counts, int32_t lmax);

/* Softmax attention of every query head over the slots of its sequence (one decode step):
 * the base model's attention, unchanged, over one key/value set per slot (Sec. 3.1, Sec. 3.7
 * "Token Fusion"; with one token a slot it is the base model's own decode, Sec. 3.7 "Minimal
 * Overhead"), grouped-query heads and scale 1/sqrt(head_dim) as in Llama (Sec. 4.1).
 * q [batch][n_q_heads][head_dim] bf16 bits; out [batch][n_q_heads][head_dim] doubles.
 * Query head h reads KV head h / (n_q_heads / n_kv_heads).  n_threads <= 0: default. */
int oracle_decode_attn(const oracle_cache *c, const uint16_t *q, double *out,
                       int32_t n_threads);

/* Attention weights of one (b, h) over the slots of sequence b: w [num_slots[b]] (the softmax
 * of oracle_decode_attn, same passages). */
int oracle_attn_weights(const oracle_cache *c, const uint16_t *q, int32_t b, int32_t h,
                        double *w);

/* Append one slot per sequence: RoPE(k_new) and v_new go to slot num_slots[b]; q_inout
 * (nullable) is rotated in place at the same position.  pos == NULL takes the position
 * from pos_mode: 0 = slot index, 1 = tokens already in the sequence.  One macro-step stores
 * one key/value set for the tokens it fused (Sec. 3.1) at an offset position (Sec. 3.2). */
int oracle_append(oracle_cache *c, const uint16_t *k_new, const uint16_t *v_new,
                  uint16_t *q_inout, const int32_t *pos, const int32_t *ntok,
                  int32_t pos_mode, double rope_base);

/* Chunked prefill (prompt tokens are not fused: Figure 2, training, item 2): sequence b's new
 * rows offsets[b] .. offsets[b+1]-1 (offsets [batch+1],
 * offsets[0] = 0) each become one slot, appended in order as oracle_append appends (pos [T]
 * nullable, ntok [T]), and each row's query heads attend over the slots of its sequence up
 * to and including its own.  q [T][n_q_heads][head_dim] rotated in place; out
 * [T][n_q_heads][head_dim] doubles; want (nullable [T]): attend only the marked rows (others
 * 0).  A sequence whose rows do not all fit is left untouched (out rows 0) and the error is
 * returned. */
int oracle_prefill(oracle_cache *c, uint16_t *q, const uint16_t *k_new, const uint16_t *v_new,
                   const int32_t *offsets, const int32_t *pos, const int32_t *ntok,
                   int32_t pos_mode, double rope_base, double *out, const uint8_t *want,
                   int32_t n_threads);

/* Threads an OpenMP region of this library uses by default (1 without OpenMP). */
int oracle_max_threads(void);

#ifdef __cplusplus
}
#endif
#endif
