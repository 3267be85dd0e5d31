// Internal declarations of the chunked prefill (ham_prefill) of libham.so.
#pragma once

#include "ham_internal.cuh"

namespace ham {

// Chunked prefill (ham_prefill): sequence b's new rows offsets[b] .. offsets[b+1]-1.
struct PrefillView {
  uint16_t *k_pool, *v_pool;   // this layer
  int32_t *slot_pos, *slot_ntok;
  const int32_t *page_table;
  int32_t *num_slots;          // [batch] of this layer
  int64_t *num_tokens;         // [batch] of this layer
  const float4 *rope_table_ff; // [rope_positions][head_dim / 2]: (cos, sin) of the fp64 table,
                               // each as an fp32 pair (hi, lo) with hi + lo = the fp64 value to
                               // about 48 bits
  const double *inv_freq;      // [head_dim / 2] (positions past the table)
  int64_t rope_positions;
  uint16_t *q;                 // [rows][n_q_heads][head_dim], rotated in place
  const uint16_t *k_new, *v_new;
  const int32_t *offsets, *pos, *ntok;  // pos, ntok nullable
  void *out;                   // [rows][n_q_heads][head_dim], bf16 or f32
  int4 *seq_info;              // scratch [batch]: (first new slot or -1, rows, query-block
                               // start, 0)
  int32_t *row_pos;            // scratch [rows]: position of each new row
  int32_t *err;
  int64_t pool_pages;
  int32_t batch, rows, n_q_heads, n_kv_heads, head_dim, page_slots, max_pages, max_slots;
  int32_t pos_mode;
  uint64_t wait_ns;            // limit of the attention's data waits (0: the default 2 s)
};
cudaError_t launch_prefill(const CUtensorMap &tk, const CUtensorMap &tv, const PrefillView &v,
                           int out_dtype, cudaStream_t stream);
bool prefill_supported(int head_dim, int group);
// Query rows of one sequence that one prefill attention CTA covers (128 / group).
int prefill_query_rows(int group);

}  // namespace ham
