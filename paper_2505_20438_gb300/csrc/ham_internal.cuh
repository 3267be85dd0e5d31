// Internal declarations of libham.so (not installed; the public ABI is include/ham.h).
#pragma once

#include <cuda.h>
#include <cuda_fp8.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <vector>

#include <nvtx3/nvToolsExt.h>

#include "ham.h"

namespace ham {

// A chunk is the unit of the split plan and of one TMA stage: 16 consecutive slots of one
// (sequence, KV head) pair.  Pages hold a multiple of 16 slots, so a chunk never straddles
// two pages and its K (or V) rows are one contiguous 16 * head_dim * 2-byte block.
constexpr int kChunkSlots = 16;
constexpr int kMaxBatch = 4096;

// FP8 (e4m3) pools (ham.h, "FP8 (e4m3) pools"): head_dim 128; per layer the K codes
// [pages][Hkv][P][128], the V codes [pages][Hkv][128][P] (a page's value rows transposed) and
// the exponents [pages][Hkv][P/16][2][16] (per chunk: 16 keys', then 16 values'), one block
// after the other in the pool allocation.
constexpr int kFp8HeadDim = 128;
constexpr int kFp8ExpMin = -124, kFp8ExpMax = 119;
// Byte of slot s (0..15) of a chunk within its transposed value rows: the slots are kept in the
// order 0, 1, 8, 9, 2, 3, 10, 11, 4, 5, 12, 13, 6, 7, 14, 15 (the attention kernel's e4m3
// products meet four consecutive bytes of a row with the scores of slots 2t, 2t + 1, 8 + 2t,
// 9 + 2t).
__host__ __device__ inline int fp8_v_slot_byte(int s) {
  return ((s & 7) >> 1) * 4 + (s >> 3) * 2 + (s & 1);
}
struct Fp8Layer {
  uint8_t *k, *v;
  int8_t *e;
};
// Bytes of one layer's FP8 block: rows = pool_pages * n_kv_heads * page_slots.
inline size_t fp8_layer_bytes(int64_t rows) {
  return (size_t)rows * kFp8HeadDim * 2 + (((size_t)rows * 2 + 1023) / 1024) * 1024;
}
inline Fp8Layer fp8_layer(void *pool, int64_t rows, int layer) {
  uint8_t *base = static_cast<uint8_t *>(pool) + (size_t)layer * fp8_layer_bytes(rows);
  return {base, base + (size_t)rows * kFp8HeadDim,
          reinterpret_cast<int8_t *>(base + (size_t)rows * kFp8HeadDim * 2)};
}

// ---------------------------------------------------------------------------------------
// Split plan.  The chunks of all (sequence b, KV head g) segments are numbered b-major,
// then g, then chunk index; W is their total.  Of the launched CTAs, C = min(launched,
// ceil(W / kMinChunksPerCta)) take part (a small problem spread over every CTA would leave
// each a chunk or two and every segment dozens of partials to merge) and CTA c < C takes
// chunks [floor(c W / C), floor((c+1) W / C)), never empty because W >= C.  So the CTAs touching a segment are exactly owner(first chunk) ..
// owner(last chunk).  A CTA writes one partial per segment it touches, at index c + s,
// which is unique because (c, s) only ever grows along the chunk order.
// ---------------------------------------------------------------------------------------
constexpr int kMinChunksPerCta = 4;
__host__ __device__ inline int32_t plan_ctas(int64_t W, int32_t launched) {
  const int64_t want = (W + kMinChunksPerCta - 1) / kMinChunksPerCta;
  return (int32_t)(want < (int64_t)launched ? want : (int64_t)launched);
}
__host__ __device__ inline int64_t plan_cta_begin(int64_t W, int32_t C, int64_t c) {
  return (W * c) / C;
}
// CTA that owns chunk x (0 <= x < W): the largest c with floor(c W / C) <= x.
__host__ __device__ inline int32_t plan_owner(int64_t W, int32_t C, int64_t x) {
  return (int32_t)(((x + 1) * (int64_t)C - 1) / W);
}
__host__ __device__ inline int32_t chunks_of(int32_t slots) {
  return (slots + kChunkSlots - 1) / kChunkSlots;
}

// Default attention grid: at most 4 CTAs per SM even where more would fit.  Four 32 KiB
// rings per SM keep ~19 MB of copies in flight on 152 SMs, above what HBM needs to stay
// busy; a fifth CTA per SM measured slower on every workload (more partials, more queueing),
// and the spare slot lets the combine kernel, scheduled early under programmatic dependent
// launch, sit beside the next attention grid without pushing one of its CTAs into a second
// wave (a CTA that starts late doubles the launch: the split plan gives every CTA an equal
// share).
constexpr int kDefaultCtasPerSm = 4;
// FP8 pools: two CTAs an SM, each with a ring of three 32 KiB tiles (ham_attn_fp8.cu).
constexpr int kDefaultCtasPerSmFp8 = 2;
inline int32_t default_attention_ctas(int32_t num_sms, int32_t resident_per_sm,
                                      bool fp8 = false) {
  const int32_t cap = fp8 ? kDefaultCtasPerSmFp8 : kDefaultCtasPerSm;
  const int32_t per = resident_per_sm < cap ? resident_per_sm : cap;
  return num_sms * (per < 1 ? 1 : per);
}

// Everything one attention launch needs; all pointers are device pointers.
// Extra inputs when the attention launch also performs this macro-step's append (the
// fused decode step): the attention pass turns q in registers and covers the stored slots;
// the combine kernel adds the new slot and commits it, q_rot and the counters.
struct StepArgs {
  const uint16_t *k_new, *v_new;   // [batch][n_kv_heads][head_dim]
  uint16_t *q_rot;                 // nullable [batch][n_q_heads][head_dim]: RoPE(q), fp64-exact
  const int32_t *pos;              // nullable [batch]
  const int32_t *ntok;             // [batch]
  int32_t *num_slots;              // [batch] of this layer (advanced by the combine kernel)
  int64_t *num_tokens;             // [batch] of this layer
  int32_t *slot_pos, *slot_ntok;
  uint16_t *k_pool, *v_pool;       // this layer (the new slot's rows, written by combine)
  int8_t *kv_exp;                  // FP8 pools: the layer's exponents (else null)
  const double *inv_freq;          // [head_dim / 2]
  const double2 *rope_table;       // [rope_positions][head_dim / 2] (cos, sin)
  const float2 *rope_table_f;      // same, fp32
  int64_t rope_positions;
  int4 *stash;                     // scratch [batch]: (slot n, 0 or HAM_DEVERR_*, position, ntok)
  int32_t *arrive;                 // scratch: combine CTAs done reading the counters (0 between
                                   // launches; the last one to arrive resets it)
  int32_t pos_mode;
};

struct AttnView {
  const uint16_t *k_pool;      // this layer: [pool_pages][n_kv_heads][page_slots][head_dim]
  const uint16_t *v_pool;      // (FP8 pools: the code blocks, through their TMA maps)
  const int8_t *kv_exp;        // FP8 pools: the layer's exponents (else null)
  const int32_t *page_table;   // [batch][max_pages]
  const int32_t *num_slots;    // [batch] of this layer
  const uint16_t *q;           // [batch][n_q_heads][head_dim]
  void *out;                   // [batch][n_q_heads][head_dim], bf16 or f32
  float *part_acc;             // scratch [(ctas + batch*n_kv_heads)][group][head_dim]
  float2 *part_ml;             // scratch [(ctas + batch*n_kv_heads)][group]: (max, sum)
  int2 *seg_range;             // scratch [batch*n_kv_heads]: CTAs first..last of a segment
                               // whose partials the combine kernel merges (-1: nothing)
  int32_t *err;                // device error word
  int64_t pool_pages;
  int32_t batch, n_kv_heads, group, page_slots, max_pages, max_slots;
  int32_t ctas;
  int32_t sms;                 // SMs of the device (the combine's choice of mode)
  // 1: the previous launch on the stream wrote nothing of this layer's counters, page table or
  // pools, so the kernel may read them before its programmatic-dependency wait (the host
  // decides; 0 is always correct)
  int32_t early;
  uint64_t wait_ns;            // limit of the ring and data waits (0: the default 2 s)
  StepArgs step;               // used by launch_decode_step only
};

struct AppendView {
  uint16_t *k_pool, *v_pool;   // this layer (FP8 pools: uint8 codes, V transposed per page)
  int8_t *kv_exp;              // FP8 pools: the layer's exponents (else null)
  int32_t *slot_pos, *slot_ntok;
  const int32_t *page_table;
  int32_t *num_slots;          // [batch] of this layer
  int64_t *num_tokens;         // [batch] of this layer
  const double *inv_freq;      // [head_dim / 2]: base^(-2i/d)
  const double2 *rope_table;   // [rope_positions][head_dim / 2]: (cos, sin)(p * inv_freq[i])
  int64_t rope_positions;      // positions covered by rope_table (others use sincos)
  uint16_t *q;                 // nullable
  const uint16_t *k_new, *v_new;
  const int32_t *pos;          // nullable
  const int32_t *ntok;
  int32_t *err;
  int64_t pool_pages;
  int32_t batch, n_q_heads, n_kv_heads, head_dim, page_slots, max_pages, max_slots, pos_mode;
  int32_t kv_per_block;        // KV heads per append block (append_kv_per_block)
};

struct FillView {
  uint16_t *k_pool, *v_pool;   // (FP8 pools: uint8 codes, V transposed per page)
  int8_t *kv_exp;              // FP8 pools: the layer's exponents (else null)
  int32_t *slot_pos, *slot_ntok;
  const int32_t *page_table;
  int32_t *num_slots;
  int64_t *num_tokens;
  const uint16_t *k_log, *v_log;
  const int32_t *pos, *ntok, *counts;
  int32_t *err;
  int64_t pool_pages;
  int32_t batch, n_kv_heads, head_dim, page_slots, max_pages, max_slots, lmax;
};

// Launchers (return cudaError_t of the launch; argument checks are done by the callers).
// tk / tv: TMA maps of the layer's K and V pools (make_pool_tensor_map).
cudaError_t launch_attention(const CUtensorMap &tk, const CUtensorMap &tv, const AttnView &v,
                             int head_dim, int out_dtype, cudaStream_t stream);
// Fused decode step: attention with the append of v.step folded in, then combine + counters.
cudaError_t launch_decode_step(const CUtensorMap &tk, const CUtensorMap &tv, const AttnView &v,
                               int head_dim, int out_dtype, cudaStream_t stream);
// The attention pass over FP8 pools (ham_attn_fp8.cu: tcgen05 products of e4m3 operands over
// 128-slot tiles), without the combine kernel that follows it; step: the fused decode step's
// pass.  Same plan, partials and errors as the bf16 pass.
cudaError_t launch_fp8_attention_pass(const CUtensorMap &tk, const CUtensorMap &tv,
                                      const AttnView &v, int out_dtype, bool step,
                                      cudaStream_t stream);
int fp8_attention_ctas_per_sm(int group, int batch, bool step, int out_dtype);
// CTAs of one SM for the attention kernel of this shape and output type (0 if the shape is not
// compiled).
int attention_ctas_per_sm(int head_dim, int group, int batch, bool step,
                          int out_dtype = HAM_DTYPE_BF16, bool fp8 = false);
// Set the shared-memory attribute of every compiled attention instance of the plain (non-step)
// kernel, for the current device: bf16 and fp32 output at head_dim 64 and 128.  Later launches
// of those instances then make no attribute call.
cudaError_t configure_attention_instances();
bool attention_supported(int head_dim, int group);
// TMA map of one pool [pool_pages][n_kv_heads][page_slots][head_dim] bf16 viewed as
// {64 elements, head_dim / 64, rows} with a box of {64, head_dim / 64, 16 rows} (half_box:
// {64, 1, 16 rows}, one 64-column half of a chunk) and the 128-byte swizzle.  Returns a
// CUresult (0 on success).
// TMA map of a row-major [rows][cols] bf16 matrix with a box of {64 columns, box_rows rows} (128
// bytes of each row) and the 128-byte swizzle: one K-major operand tile of a tcgen05 product.
// cols must be a multiple of 8; boxes past the last row or column read zeros.  Returns a CUresult.
int make_matrix_tensor_map(CUtensorMap *map, const void *base, int64_t rows, int64_t cols,
                           int box_rows);
// TMA map of fp32 split parts [splits][rows][ld] (columns 0..cols-1 used) with a box of {32
// columns, 32 rows, 1 part} and the 128-byte swizzle: the store of one epilogue warp.  ld a
// multiple of 4 and base 16-byte aligned.  Returns a CUresult.
int make_parts_tensor_map(CUtensorMap *map, void *base, int splits, int64_t rows, int64_t cols,
                          int64_t ld);
// Y[s][rows][ldy] (fp32, columns 0..F-1) = X[rows][K_s] . W[F][K_s]^T, the K columns split in
// `splits` ranges K_s of whole 64-column tiles, as even as the tile count allows (the caller sums
// the parts): tcgen05 products of 128 output features by up to 256 rows.  W is either pre-tiled
// (wt, from tile_weights) or given by tw (a tensor map of make_matrix_tensor_map with box_rows
// 128); X by tx (box_rows = gemm_row_tile(rows)).  splits <= ceil(K / 64).  With `pdl` the
// launch may start before the previous kernel on the stream ends: it loads W tiles before its
// dependency wait and X only after.
int gemm_row_tile(int rows);
int gemm_splits(int F, int K, int rows, int max_splits);
// W [F][K] row-major bf16 -> wt: each 128 x 64 tile one contiguous 16 KiB block in the 128-byte
// swizzle layout, tiles [ceil(F/128)][ceil(K/64)], zeros past the matrix (one launch).
size_t tiled_weight_bytes(int F, int K);
cudaError_t tile_weights(const void *W, int F, int K, void *wt, cudaStream_t stream);
cudaError_t launch_gemm_xwt(const CUtensorMap *tw, const void *wt, const CUtensorMap &tx,
                            float *Y, int64_t ldy, int32_t *err, int rows, int F, int K,
                            int splits, bool pdl, cudaStream_t stream);
// TMA map of a row-major [rows][heads][head_dim] bf16 tensor viewed as {64 elements,
// head_dim / 64, heads, rows} with a box of {64, 1, box_heads, box_rows} (one 64-column half of
// box_heads x box_rows head rows) and the 128-byte swizzle.  Boxes past the last row read zeros.
// Returns a CUresult (0 on success).
int make_rows_tensor_map(CUtensorMap *map, const void *base, int64_t rows, int heads,
                         int head_dim, int box_heads, int box_rows);
int make_pool_tensor_map(CUtensorMap *map, const void *pool, int64_t rows, int head_dim,
                         bool half_box);
cudaError_t launch_append(const AppendView &v, cudaStream_t stream);
// KV heads per append block (0 if the shape does not fit the append kernel).
int append_kv_per_block(int n_q_heads, int n_kv_heads, int head_dim);
cudaError_t launch_fill(const FillView &v, cudaStream_t stream);

// TMA maps of one layer's FP8 code blocks: K [rows][128] uint8 with a box of {128, 16 rows}
// and the 128-byte swizzle; V [rows_d = pages * Hkv * 128][page_slots] uint8 with a box of
// {16 slots, 128 rows} (one chunk's value rows, transposed), no swizzle.  Return a CUresult.
int make_fp8_k_tensor_map(CUtensorMap *map, const void *k_codes, int64_t rows);
int make_fp8_v_tensor_map(CUtensorMap *map, const void *v_codes, int64_t rows_d, int page_slots);

// One row of 128 values (element 4 * lane + i in x[i] of lane `lane`, every lane of the warp
// taking part) encoded as e4m3 codes with a power-of-two scale 2^e: e = E - 8 for the row's
// largest magnitude m 2^E (0.5 <= m < 1), clamped to [-124, 119], 0 for a zero row; each element
// x 2^-e (exact) rounded to nearest even with saturation at +-448 by the hardware conversion.
// Returns e; `codes` gets the lane's four codes, element 4 * lane + i in byte i.
__device__ inline int encode_e4m3_row(const float (&x)[4], uint32_t &codes) {
  float a = fmaxf(fmaxf(fabsf(x[0]), fabsf(x[1])), fmaxf(fabsf(x[2]), fabsf(x[3])));
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) a = fmaxf(a, __shfl_xor_sync(0xffffffffu, a, o));
  int e = 0;
  if (a > 0.f) {
    int E = 0;
    frexpf(a, &E);
    e = min(max(E - 8, kFp8ExpMin), kFp8ExpMax);
  }
  const __nv_fp8x2_storage_t lo = __nv_cvt_float2_to_fp8x2(
      make_float2(ldexpf(x[0], -e), ldexpf(x[1], -e)), __NV_SATFINITE, __NV_E4M3);
  const __nv_fp8x2_storage_t hi = __nv_cvt_float2_to_fp8x2(
      make_float2(ldexpf(x[2], -e), ldexpf(x[3], -e)), __NV_SATFINITE, __NV_E4M3);
  codes = (uint32_t)lo | ((uint32_t)hi << 16);
  return e;
}

// An NVTX range named after a C-ABI call, for the duration of the call (host side: the call's
// launches and checks).  NVTX v3 is header-only; without a profiler attached a push and a pop
// cost a load and a branch each.
struct ApiRange {
  explicit ApiRange(const char *name) { nvtxRangePushA(name); }
  ~ApiRange() { nvtxRangePop(); }
  ApiRange(const ApiRange &) = delete;
  ApiRange &operator=(const ApiRange &) = delete;
};
// Record `msg` as this thread's ham_last_error() and return `status`.
int set_last_error(int status, const char *msg);

// Device error word: keep the first error.
__device__ inline void record_error(int32_t *err, int32_t code) {
  if (err) atomicCAS(err, 0, code);
}

}  // namespace ham

// Library-internal handle (opaque to users).
struct ham_kv {
  ham_config cfg;
  int device = 0;
  int num_sms = 0;
  int32_t max_pages = 0;
  int32_t attn_ctas = 0;        // 0: default
  uint64_t wait_ns = 0;         // attention / prefill data-wait limit (0: the default 2 s)
  int32_t default_ctas = 0;     // SMs x resident attention CTAs per SM (set at allocation)
  int32_t default_step_ctas = 0;  // same for the fused decode step
  int32_t max_ctas = 0;         // scratch is sized for this many CTAs
  int64_t pool_elems = 0;       // elements of ONE pool (K or V) of one layer
  int32_t fp8 = 0;              // 1: FP8 (e4m3) pools (kv_dtype HAM_KV_E4M3)
  uint16_t *pool = nullptr;     // bf16: [layers][2][pool_elems]; FP8: [layers] x fp8_layer_bytes
  uint8_t *meta = nullptr;      // everything else, carved below
  int32_t *slot_pos = nullptr, *slot_ntok = nullptr, *page_table = nullptr;
  int32_t *num_slots = nullptr; // [layers][batch]
  int64_t *num_tokens = nullptr;
  double *inv_freq = nullptr;
  double2 *rope_table = nullptr;  // own allocation
  float2 *rope_table_f = nullptr;  // own allocation
  float4 *rope_table_ff = nullptr;  // own allocation: fp32 (hi, lo) pairs of the fp64 table
  int64_t rope_positions = 0;
  int32_t *err = nullptr;
  int4 *stash = nullptr;           // fused step: per-sequence append record
  int32_t *arrive = nullptr;       // fused step: the combine's arrival counter
  float *part_acc = nullptr;
  float2 *part_ml = nullptr;
  int2 *seg_range = nullptr;
  int4 *prefill_seq = nullptr;     // ham_prefill: per-sequence plan [batch]
  int2 *prefill_rows = nullptr;    // ham_prefill: per-row (position, pool row) [batch * max_slots]
  float *prefill_part = nullptr;   // ham_prefill: split partials (bf16 caches)
  float2 *prefill_part_ml = nullptr;
  int64_t scratch_bytes = 0;
  std::vector<CUtensorMap> tmaps;  // [layers][2]: TMA maps of the K and V pools
  std::vector<CUtensorMap> tmaps_half;  // [layers][2]: the same, one 64-column half per box
  void *host_stage = nullptr;   // pinned: counters and error word read-back
};
