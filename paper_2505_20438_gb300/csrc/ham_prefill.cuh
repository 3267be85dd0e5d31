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
                               // start, 1 when the call's offsets are valid, else 0)
  int2 *row_info;              // scratch [rows]: (position, pool row page * page_slots + row
                               // in page, or -1 when the row is not stored) of each new row
  int32_t *err;
  int64_t pool_pages;
  int32_t batch, rows, n_q_heads, n_kv_heads, head_dim, page_slots, max_pages, max_slots;
  int32_t pos_mode;
  uint64_t wait_ns;            // limit of the attention's data waits (0: the default 2 s)
  // Split over slots (a short chunk over a long cache): the attention grid's z dimension.  A
  // sequence of L cached slots uses prefill_splits(L, splits) of them; a split that is not alone
  // leaves its rows' unnormalised partials (output, running maximum and sum) here, and the merge
  // kernel combines them: part_o [splits][rows][n_q_heads][head_dim], part_ml [same without d].
  float *part_o;
  float2 *part_ml;
  int32_t splits;
};
// Slots a prefill split covers at least (whole 64-slot tiles of the cached part), and the most
// splits a launch uses.
constexpr int kPrefillSplitMinTiles = 8, kPrefillMaxSplits = 32;
// Splits of a sequence holding L cached slots, at most Z: each takes at least
// kPrefillSplitMinTiles tiles of the cached part, the last one also the chunk's own slots.
__host__ __device__ inline int prefill_splits(int L, int Z) {
  const int by_len = (L / 64) / kPrefillSplitMinTiles;
  return by_len < 1 ? 1 : (by_len < Z ? by_len : Z);
}
// Scratch floats the split partials may use: SMs x 256 (row, head) pairs x head_dim (a launch
// splits only while its CTAs, 256 pairs each, fit the SMs).
inline size_t prefill_part_floats(int sms, int head_dim) {
  return (size_t)sms * 256 * (size_t)head_dim;
}
cudaError_t launch_prefill(const CUtensorMap &tk, const CUtensorMap &tv, const PrefillView &v,
                           int out_dtype, cudaStream_t stream);
bool prefill_supported(int head_dim, int group);
// Query rows of one sequence that one prefill attention CTA covers (128 / group).
int prefill_query_rows(int group);

}  // namespace ham
