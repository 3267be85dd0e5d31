// Internal declarations of the micro-step attention (ham_micro_step) of libham.so.
#pragma once

#include "ham_internal.cuh"

namespace ham {

// Largest per-sequence cache the micro-step kernel covers: one 16-slot chunk.
constexpr int kMicroMaxSlots = 16;
// KV heads of one sequence form a thread-block cluster (portable size).
constexpr int kMicroMaxKvHeads = 8;

// One step of a decoder whose per-sequence cache holds at most 16 slots (the micro-step
// decoder's local context), as one kernel: RoPE of q and k at the new slot's position, the
// append, and attention over the slots including the new one.
struct MicroView {
  const uint16_t *q;           // [batch][n_q_heads][head_dim], unrotated
  uint16_t *q_rot;             // nullable, same shape: RoPE(q) where the append happens
  const uint16_t *k_new, *v_new;  // [batch][n_kv_heads][head_dim]
  const int32_t *pos;          // nullable [batch]
  const int32_t *ntok;         // [batch]
  void *out;                   // [batch][n_q_heads][head_dim], bf16 or f32
  uint16_t *k_pool, *v_pool;   // this layer
  int32_t *slot_pos, *slot_ntok;
  const int32_t *page_table;
  int32_t *num_slots;          // [batch] of this layer
  int64_t *num_tokens;         // [batch] of this layer
  const double *inv_freq;      // [head_dim / 2]
  const double2 *rope_table;   // [rope_positions][head_dim / 2]
  int64_t rope_positions;
  int32_t *err;
  int64_t pool_pages;
  int32_t batch, n_q_heads, n_kv_heads, head_dim, page_slots, max_pages, max_slots, pos_mode;
  int32_t out_f32;
};

cudaError_t launch_micro(const MicroView &v, cudaStream_t stream);

}  // namespace ham
