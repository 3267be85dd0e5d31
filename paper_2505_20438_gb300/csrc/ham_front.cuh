// Internal declarations of the macro-step layer front (ham_qkv_append) of libham.so.
#pragma once

#include "ham_internal.cuh"

namespace ham {

// Sequences one front CTA row (blockIdx.y) covers; the grid has ceil(batch / 32) rows.
constexpr int kFrontBatchTile = 32;
// Arrival counters the front keeps in the handle's scratch, one per CTA row.
constexpr int kFrontMaxRows = (kMaxBatch + kFrontBatchTile - 1) / kFrontBatchTile;

// q/k/v projection of the layer input, RoPE at the new slot's position and the append, in one
// kernel.  Output row o of the fused weight is query head o / d for o < Hq d, then key heads,
// then value heads; element o % d of its head.
struct FrontView {
  const uint16_t *x;           // [batch][hidden]
  const uint16_t *w;           // [(n_q_heads + 2 n_kv_heads) head_dim][hidden]
  uint16_t *q_rot;             // [batch][n_q_heads][head_dim]
  uint16_t *k_pool, *v_pool;   // this layer
  int32_t *slot_pos, *slot_ntok;
  const int32_t *page_table;
  int32_t *num_slots;          // [batch] of this layer
  int64_t *num_tokens;         // [batch] of this layer
  const double *inv_freq;      // [head_dim / 2]
  const double2 *rope_table;   // [rope_positions][head_dim / 2]: (cos, sin)(p * inv_freq[i])
  int64_t rope_positions;
  const int32_t *pos;          // nullable [batch]
  const int32_t *ntok;         // [batch]
  int32_t *arrive;             // scratch [ceil(batch / 32)]: CTAs of a row done with the
                               // counters (0 between launches; the last to arrive resets it)
  // FP8 (e4m3) pools (head_dim 128): the layer's exponents, and scratch for the new slot's key
  // (rotated) and value rows as bf16, [batch][n_kv_heads][2][head_dim], which the row's last CTA
  // encodes (else both null)
  int8_t *kv_exp;
  uint16_t *stage;
  int32_t *enc_arrive;         // FP8 pools: [ceil(batch / 32)][2 n_kv_heads] arrivals of a head's
                               // CTAs (0 between launches; the last to arrive resets it)
  int32_t *err;
  int64_t pool_pages;
  int32_t batch, hidden, n_q_heads, n_kv_heads, head_dim, page_slots, max_pages, max_slots;
  int32_t pos_mode;
};

cudaError_t launch_front(const FrontView &v, cudaStream_t stream);
// hidden sizes the front kernel takes: multiples of 256
constexpr int kFrontHiddenQuantum = 256;

}  // namespace ham
