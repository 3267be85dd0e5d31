/*
 * ham.h -- C ABI of the GB300 (sm_103a) smashed-KV decode-attention library, libham.so.
 *
 * Method: HAMburger (Liu & Zhang, arXiv 2505.20438).  A macro-step is one forward of the
 * base model that stores ONE key/value set for the whole group of 1..4 tokens it fused
 * (Sec. 3.1; Sec. 3.7 "Token Fusion"); the cache therefore holds one "slot" per macro-step,
 * and each decode step attends over the slots and appends the slot just produced.  The
 * merged embedding enters the base model at an offset position reflecting the fused token
 * count (Sec. 3.2).  With one token per slot everything reduces to the base model's own
 * decode (Sec. 3.4).  Decoding reads the whole cache every step and is bound by memory
 * bandwidth (Sec. 2.3, KV-cache compression).
 *
 * Conventions
 *  - Every call returns an int status (ham_status).  No exception or abort crosses the ABI.
 *    On failure ham_last_error() gives a message (thread-local, valid until the next call
 *    on the same thread).
 *  - `stream` is a cudaStream_t passed as void* (NULL = the legacy default stream).  Calls
 *    taking a stream are asynchronous unless stated otherwise.
 *  - bf16 tensors are raw 16-bit bfloat16 values, row-major, 16-byte aligned device memory
 *    owned by the caller.  The library owns the KV pool, page tables, counters and its
 *    scratch; ham_kv_free releases them.
 *  - Kernels never trap.  A bad value that can only be seen on the device (a page id outside
 *    the pool, a full sequence, a token count < 1, a bounded wait that ran out) is recorded
 *    in a device error word and the offending write is skipped; ham_kv_status or
 *    ham_slot_lengths report it as HAM_EDEVICE.
 */
#ifndef HAM_H
#define HAM_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define HAM_ABI_VERSION 1

typedef enum ham_status {
  HAM_OK = 0,
  HAM_EINVAL = 1,       /* bad argument seen on the host; nothing was launched */
  HAM_ENOMEM = 2,       /* device or pinned-host allocation failed */
  HAM_ECAPACITY = 3,    /* configuration does not fit (pool smaller than the page tables) */
  HAM_ECUDA = 4,        /* a CUDA runtime call failed (message has the CUDA error) */
  HAM_EDEVICE = 5,      /* a kernel recorded an error in the device error word */
  HAM_EUNSUPPORTED = 6  /* shape outside the compiled kernels (head_dim, group size) */
} ham_status;

/* Device error word values (ham_kv_status). The first error recorded wins. */
enum {
  HAM_DEVERR_NONE = 0,
  HAM_DEVERR_CAPACITY = 1,  /* append into a sequence already holding max_slots_per_seq */
  HAM_DEVERR_NTOK = 2,      /* token count < 1 for a new slot */
  HAM_DEVERR_PAGE = 3,      /* page-table entry outside [0, pool_pages) */
  HAM_DEVERR_SLOTS = 4,     /* slot counter outside [0, max_slots_per_seq] */
  HAM_DEVERR_TIMEOUT = 5    /* a bounded wait inside a kernel ran out */
};

/* Position given to a new slot when ham_kv_append gets pos == NULL (Sec. 3.2). */
enum {
  HAM_POS_SLOT = 0,   /* the slot index, i.e. the macro-step number */
  HAM_POS_TOKEN = 1   /* tokens already in the sequence: the position of the group's first token */
};

enum { HAM_DTYPE_BF16 = 0, HAM_DTYPE_F32 = 1 };

/* Storage type of the KV pools (ham_config.kv_dtype); see "FP8 (e4m3) pools" below. */
enum { HAM_KV_BF16 = 0, HAM_KV_E4M3 = 1 };

typedef struct ham_kv ham_kv; /* opaque handle: one paged smashed-KV cache, all layers */

typedef struct ham_config {
  int32_t layers;            /* >= 1 */
  int32_t batch;             /* sequences, 1..4096 */
  int32_t n_q_heads;         /* query heads */
  int32_t n_kv_heads;        /* KV heads; n_q_heads / n_kv_heads in {1, 2, 4, 8} */
  int32_t head_dim;          /* 64 or 128 */
  int32_t page_slots;        /* slots per page, a multiple of 16 */
  int32_t max_slots_per_seq; /* capacity of one sequence, in slots */
  int32_t pos_mode;          /* HAM_POS_SLOT or HAM_POS_TOKEN */
  int64_t pool_pages;        /* pages in the pool; 0 = batch * ceil(max_slots_per_seq / page_slots) */
  double rope_base;          /* RoPE base (10000 for Llama-style models) */
  uint64_t page_seed;        /* 0: sequence b gets pages [b*P, (b+1)*P); else a seeded shuffle */
  int32_t kv_dtype;          /* HAM_KV_BF16 (0) or HAM_KV_E4M3 (8-bit rows, head_dim 128) */
} ham_config;

typedef struct ham_kv_info {
  ham_config cfg;            /* with pool_pages resolved */
  int32_t max_pages_per_seq; /* page-table row length = ceil(max_slots_per_seq / page_slots) */
  int32_t attn_ctas;         /* CTAs of one attention launch */
  int32_t num_sms;           /* SMs of the device the handle lives on */
  int32_t device;            /* CUDA device ordinal */
  int64_t pool_bytes;        /* K+V bytes of ONE layer's pool (FP8: codes and exponents) */
  int64_t scratch_bytes;     /* split-attention partials and per-segment CTA ranges */
} ham_kv_info;

/* ------------------------------------------------------------------------------------
 * The four calls of a macro-step
 * ------------------------------------------------------------------------------------ */

/* Allocate a paged smashed-KV cache on the current CUDA device (synchronous).
 *
 * Device layout (one allocation; every pointer below lives inside it):
 *   K pool, V pool of layer l  [pool_pages][n_kv_heads][page_slots][head_dim] bf16
 *   slot_pos, slot_ntok        [pool_pages][page_slots] int32   (shared by all layers)
 *   page table                 [batch][max_pages_per_seq] int32
 *   num_slots                  [layers][batch] int32,  num_tokens [layers][batch] int64
 * Slot n of sequence b is row n % page_slots of page page_table[b][n / page_slots].
 * Every sequence starts empty.  Pages are reserved at allocation (page_seed), so appends
 * never need the host.  Errors: HAM_EINVAL (bad config), HAM_ECAPACITY (pool_pages <
 * batch * max_pages_per_seq), HAM_EUNSUPPORTED, HAM_ENOMEM, HAM_ECUDA.  *out is NULL on
 * failure. */
int ham_kv_alloc(const ham_config *cfg, ham_kv **out);

/* Free everything the handle owns (synchronizes the device first).  NULL is a no-op. */
int ham_kv_free(ham_kv *kv);

/* Append the slot of this macro-step to every sequence of one layer (Sec. 3.1: one KV set
 * per macro-step; Sec. 3.2: its position).  One fused kernel: for each sequence b, with
 * n = num_slots[layer][b] and position p = pos[b] (or, if pos == NULL, n for HAM_POS_SLOT
 * and num_tokens[layer][b] for HAM_POS_TOKEN):
 *   K row of slot n  <- RoPE(k_new[b], p)   (rotate-half, theta_i = p * base^(-2i/d),
 *                                            computed in fp64, stored bf16 round-to-nearest-even)
 *   V row of slot n  <- v_new[b]             (bit copy)
 *   q_inout[b]       <- RoPE(q_inout[b], p)  (if q_inout != NULL, in place)
 *   slot_pos = p, slot_ntok = ntok[b], num_slots += 1, num_tokens += ntok[b]
 * q_inout  nullable, device bf16 [batch][n_q_heads][head_dim]
 * k_new, v_new      device bf16 [batch][n_kv_heads][head_dim]
 * pos      nullable, device int32 [batch];  ntok  device int32 [batch], each >= 1
 * A full sequence or ntok < 1 skips that sequence and sets the device error word.
 * Host errors: HAM_EINVAL (NULL / unaligned pointer, layer out of range), HAM_ECUDA. */
int ham_kv_append(ham_kv *kv, int32_t layer, void *q_inout, const void *k_new,
                  const void *v_new, const int32_t *pos, const int32_t *ntok, void *stream);

/* One decode step of one layer: every query head attends over all slots of its sequence
 * (softmax(q K^T / sqrt(head_dim)) V over the slot list; no weighting by token count).
 * Query head h reads KV head h / (n_q_heads / n_kv_heads).  Split-KV: the slots of all
 * (sequence, KV head) pairs are cut into equal contiguous ranges, one per CTA, and a second
 * kernel merges the partial softmax states of pairs that span several CTAs (two launches on
 * `stream`, the second with programmatic dependent launch).  Sequences with no slots give 0.
 * Slot counts are read on the device (no host sync).
 * q    device bf16 [batch][n_q_heads][head_dim], already rotated (e.g. by ham_kv_append)
 * out  device bf16 [batch][n_q_heads][head_dim]
 * Host errors: HAM_EINVAL, HAM_ECUDA.  Calls on one handle must not overlap in time (they
 * share the handle's scratch); serialize them on one stream. */
int ham_decode_attn(ham_kv *kv, int32_t layer, const void *q, void *out, void *stream);

/* ham_kv_append followed by ham_decode_attn in one pass over the cache (Sec. 3.1 + Sec. 3.4:
 * the macro-step's slot is stored and every query head then attends over the slot list
 * that includes it).  q is the UNROTATED query; the step turns it by the new slot's
 * position internally and never writes it.  On return the cache and the counters hold
 * exactly what ham_kv_append leaves (fp64 RoPE, bf16 round-to-nearest-even), and out holds
 * the attention of RoPE(q) over the n + 1 slots.  Inside the attention pass q and the new
 * key are turned in fp32 from a float cos/sin table, so a rotated element can differ from
 * the stored one by one bf16 ulp; out stays within the ham_decode_attn tolerance of the
 * two-call result.  q_rot (nullable) receives the fp64-exact RoPE(q), the bits
 * ham_kv_append would leave in q_inout, for the sequences whose append happens (other rows
 * are not written).
 * A sequence whose append fails (full, ntok < 1, bad counter) is not appended, attends with
 * its unrotated q over its old slots and sets the device error word, as the two calls
 * would.  Two launches on `stream` (the second with programmatic dependent launch).
 * q        device bf16 [batch][n_q_heads][head_dim];  q_rot nullable, same shape
 * k_new, v_new, pos, ntok as for ham_kv_append
 * out      device [batch][n_q_heads][head_dim], bf16 or f32 (out_dtype)
 * q, q_rot and out must not overlap; k_new and v_new must not overlap the cache.
 * Host errors: HAM_EINVAL (NULL / unaligned / overlapping pointers, layer out of range,
 * out_dtype), HAM_ECUDA.  Same serialization rule as ham_decode_attn. */
int ham_decode_step(ham_kv *kv, int32_t layer, const void *q, void *q_rot, const void *k_new,
                    const void *v_new, const int32_t *pos, const int32_t *ntok, void *out,
                    int32_t out_dtype, void *stream);

/* The layer front of a macro-step: the q/k/v projection of the layer's input, RoPE at the new
 * slot's position and the append, in one kernel (Sec. 3.1: one forward of the base model per
 * macro-step stores one key/value set; Sec. 3.2: at an offset position; Sec. 4.1: the Llama
 * base model, whose attention projects its normalised input with bias-free linear maps).
 * For sequence b, with n = num_slots[layer][b] and p chosen as for ham_kv_append:
 *   y = W x[b]  (fp32 accumulation on the tensor cores of the bf16 products), W = w_qkv
 *   q_rot[b][h]   <- RoPE(y[h d .. h d + d), p)                          h < n_q_heads
 *   K row of slot n, KV head g <- RoPE(y[(n_q_heads + g) d ..), p)
 *   V row of slot n, KV head g <- y[(n_q_heads + n_kv_heads + g) d ..)
 *   slot_pos = p, slot_ntok = ntok[b], num_slots += 1, num_tokens += ntok[b]
 * The rotation takes the fp32 projection, is evaluated in fp64 and rounded once to bf16 (nearest,
 * ties to even); values are the fp32 projection rounded once.  ham_decode_attn(kv, layer, q_rot,
 * ...) then attends over the slots including the new one.
 * x      device bf16 [batch][hidden], the layer's normalised input
 * w_qkv  device bf16 [(n_q_heads + 2 n_kv_heads) head_dim][hidden], row-major ([out][in]): the
 *        rows of W_q, then W_k, then W_v (a fused projection weight); caller-owned, not copied
 * hidden a multiple of 256 (at most 2^20); head_dim 64 or 128
 * pos    nullable device int32 [batch];  ntok  device int32 [batch], each >= 1
 * q_rot  device bf16 [batch][n_q_heads][head_dim] (output)
 * A sequence whose append cannot happen (full, ntok < 1, bad page or counter) gets no slot, sets
 * the device error word and receives its unrotated projection in q_rot.  One launch on `stream`
 * (programmatic dependent launch: the kernel may prefetch w_qkv into L2 before the previous
 * kernel on the stream has finished; it reads x and the counters only after).  q_rot must not
 * overlap x, w_qkv or the cache.  Host errors: HAM_EINVAL (NULL / unaligned / overlapping
 * pointers, layer or hidden out of range), HAM_EUNSUPPORTED (head_dim), HAM_ECUDA.  Same
 * serialization rule as ham_decode_attn. */
int ham_qkv_append(ham_kv *kv, int32_t layer, const void *x, const void *w_qkv, int32_t hidden,
                   const int32_t *pos, const int32_t *ntok, void *q_rot, void *stream);

/* One step of the micro-step decoder's attention (Sec. 3.3: the decoder that emits a
 * macro-step's tokens one by one, conditioned on hidden states of several middle layers of the
 * base model; Sec. 4.1: four layers with the base model's configuration).  Its cache is local to
 * the macro-step: the context entries and the micro-tokens so far, a handful of slots, so the
 * step costs the same at any sequence length (Sec. 3.7, the constant c).  Same operation and
 * results as ham_decode_step (append of the new slot with RoPE at its position, attention over
 * all slots including it, counters advanced; q_rot and out as there), for handles whose
 * sequences hold at most 16 slots, in one kernel launch instead of two: one CTA per (sequence,
 * KV head), the query is rotated in fp64 like the stored key (q_rot holds exactly the bits
 * ham_kv_append leaves in q_inout), softmax and sums in fp32.  Typical use: a handle with
 * layers = the decoder's layers, max_slots_per_seq = context entries + micro-tokens (<= 16),
 * page_slots 16; each macro-step fills the context entries (ham_kv_fill or ham_prefill) and
 * each micro-step calls this once per layer; ham_kv_set_lengths or ham_kv_reset clears the
 * local cache for the next macro-step.
 * Arguments, errors and serialization as for ham_decode_step; HAM_EUNSUPPORTED if the handle's
 * max_slots_per_seq exceeds 16, n_kv_heads exceeds 8 or head_dim is not 64 or 128. */
int ham_micro_step(ham_kv *kv, int32_t layer, const void *q, void *q_rot, const void *k_new,
                   const void *v_new, const int32_t *pos, const int32_t *ntok, void *out,
                   int32_t out_dtype, void *stream);

/* Slot and token counts of every sequence after the last layer's appends (synchronous:
 * copies on `stream`, then waits for it).  num_slots_host [batch], num_tokens_host [batch]
 * (either may be NULL).  Returns HAM_EDEVICE if the device error word is set. */
int ham_slot_lengths(ham_kv *kv, int32_t *num_slots_host, int64_t *num_tokens_host,
                     void *stream);

/* Chunked prefill of one layer: prompt ingestion over the smashed cache.  The paper fuses
 * only response tokens (Figure 2, training), so each prompt token becomes its own slot;
 * the chunk's queries attend causally over the cache and over the chunk itself.  Sequence
 * b's new rows are rows offsets[b] .. offsets[b+1]-1 of q/k_new/v_new, in order (a sequence
 * may have none).  With L = num_slots[layer][b] before the call, row r = offsets[b] + j:
 *   becomes slot L + j as ham_kv_append would store it: position pos[r], or (pos == NULL)
 *     L + j for HAM_POS_SLOT and the tokens before it (num_tokens[layer][b] plus the ntok of
 *     the sequence's earlier rows) for HAM_POS_TOKEN; K row RoPE(k_new[r]), V row v_new[r],
 *     slot_pos, slot_ntok = ntok[r]; num_slots += rows, num_tokens += their ntok;
 *   q_inout[r] <- RoPE(q_inout[r]) at the same position, in place;
 *   out[r][h] = softmax(q[r][h] K^T / sqrt(head_dim)) V over slots 0 .. L + j of the
 *     sequence, KV head h / (n_q_heads / n_kv_heads).
 * The rotations are evaluated to about 48 bits in fp32 pairs from the fp64 cos/sin table
 * and rounded once to bf16: the bits ham_kv_append stores, unless the exact rotation lies
 * within about 2^-40 (relative) of a bf16 rounding boundary.  The attention runs on the
 * tensor cores (bf16 in, fp32 accumulation and softmax, probabilities rounded to bf16).
 * q_inout  device bf16 [total_rows][n_q_heads][head_dim]
 * k_new, v_new  device bf16 [total_rows][n_kv_heads][head_dim]
 * offsets  device int32 [batch + 1]: offsets[0] = 0, non-decreasing, offsets[batch] =
 *          total_rows
 * pos      nullable device int32 [total_rows];  ntok  nullable device int32 [total_rows]
 *          (NULL: 1 token per row)
 * out      device [total_rows][n_q_heads][head_dim], bf16 or f32 (out_dtype)
 * A sequence whose rows cannot all be stored (a token count < 1, no room for them, a bad
 * page, offsets that leave the call's rows) gets no slot, keeps q unrotated and 0 out
 * rows, and sets the device error word.  total_rows == 0 launches nothing (the buffers may
 * then be NULL).  Three launches
 * on `stream` (plan, RoPE + append, attention), four when a short chunk lets the attention
 * split over the cached slots (a merge of the splits' partials, kept in the handle's scratch;
 * the result does not depend on the split).  q_inout, out, k_new and v_new must not
 * overlap each other or the cache.  Host errors: HAM_EINVAL (NULL / unaligned / overlapping
 * pointers, layer or out_dtype out of range, total_rows above batch * max_slots_per_seq),
 * HAM_ECUDA.  Same serialization rule as ham_decode_attn. */
int ham_prefill(ham_kv *kv, int32_t layer, void *q_inout, const void *k_new, const void *v_new,
                const int32_t *offsets, const int32_t *pos, const int32_t *ntok,
                int32_t total_rows, void *out, int32_t out_dtype, void *stream);

/* ------------------------------------------------------------------------------------
 * Helpers: inspection, test set-up, tuning
 * ------------------------------------------------------------------------------------ */

/* Message of the last failed call on this thread ("" if none). */
const char *ham_last_error(void);

/* Sizes and resolved settings of a handle. */
int ham_kv_get_info(const ham_kv *kv, ham_kv_info *info);

/* Same as ham_decode_attn with the output type chosen: HAM_DTYPE_BF16 or HAM_DTYPE_F32
 * (fp32 output, for tight comparisons). */
int ham_decode_attn_ex(ham_kv *kv, int32_t layer, const void *q, void *out,
                       int32_t out_dtype, void *stream);

/* Per-layer counters (synchronous, like ham_slot_lengths). */
int ham_kv_layer_lengths(ham_kv *kv, int32_t layer, int32_t *num_slots_host,
                         int64_t *num_tokens_host, void *stream);

/* Read and clear the device error word (synchronizes `stream`).  *device_code (nullable)
 * gets the HAM_DEVERR_* value.  Returns HAM_EDEVICE if it was set. */
int ham_kv_status(ham_kv *kv, void *stream, int32_t *device_code);

/* Replace the page table with host_pt [batch][max_pages_per_seq] (synchronous).  Entries
 * must lie in [0, pool_pages) and no page may appear twice; else HAM_EINVAL and nothing
 * changes.  Existing slot contents are NOT moved. */
int ham_kv_set_page_table(ham_kv *kv, const int32_t *host_pt);

/* Copy the page table to host_pt [batch][max_pages_per_seq] (synchronous). */
int ham_kv_get_page_table(const ham_kv *kv, int32_t *host_pt);

/* Load a logical cache into one layer: slot j < counts[b] of sequence b gets
 * k_log/v_log[b][j] (bit copy, no RoPE: keys are taken as already rotated; an FP8 pool
 * stores the rows encoded as described under "FP8 (e4m3) pools") and, if given,
 * slot_pos = pos[b][j], slot_ntok = ntok[b][j] (defaults: j and 1).  Sets
 * num_slots[layer][b] = counts[b] and num_tokens[layer][b] = sum of the ntok.
 * k_log, v_log  device bf16 [batch][lmax][n_kv_heads][head_dim]
 * pos, ntok     nullable device int32 [batch][lmax];  counts  device int32 [batch]
 * A count outside [0, min(lmax, max_slots_per_seq)] sets the device error word. */
int ham_kv_fill(ham_kv *kv, int32_t layer, const void *k_log, const void *v_log,
                const int32_t *pos, const int32_t *ntok, const int32_t *counts, int32_t lmax,
                void *stream);

/* Copy one layer's raw pools and the slot metadata out (device or pinned host destinations,
 * cudaMemcpyDefault).  k_dst, v_dst: one pool each, pool_pages * n_kv_heads * page_slots *
 * head_dim elements (bf16, or FP8 codes in the layouts below); pos_dst, ntok_dst:
 * pool_pages * page_slots int32 each.  Any destination may be NULL. */
int ham_kv_export(ham_kv *kv, int32_t layer, void *k_dst, void *v_dst, int32_t *pos_dst,
                  int32_t *ntok_dst, void *stream);

/* ------------------------------------------------------------------------------------
 * FP8 (e4m3) pools: kv_dtype = HAM_KV_E4M3, head_dim 128
 * ------------------------------------------------------------------------------------
 * Decoding re-reads every stored key and value each step and is bound by memory bandwidth
 * (Sec. 2.3; Sec. 3.7: the KV cache is what the method shrinks), so the rows of a slot may be
 * stored in 8 bits: 2 x (128 + 1) bytes per (slot, KV head) instead of 2 x 256.  The paper
 * keeps the base model's precision; this storage format is the library's own:
 *  - elements: e4m3 codes (1 sign, 4 exponent bits of bias 7, 3 mantissa bits; no
 *    infinities; largest finite 448); each element scaled exactly and rounded once, to
 *    nearest with ties to even, saturating at +-448, the sign kept (also on zero);
 *  - one scale per stored row (one slot of one KV head), a power of two 2^e, e an int8:
 *    e = E - 8 for the row's largest magnitude m 2^E (0.5 <= m < 1), clamped to [-124, 119]
 *    so that every decoded value is a finite bf16 value; a row of zeros has e = 0;
 *  - the key is rotated first (the bf16 row a bf16 cache would hold), then encoded; the value
 *    is encoded as given.  A decoded element code * 2^e has at most 4 significant bits and
 *    is an exact bf16 value: attention over an FP8 pool is attention over the decoded rows.
 * Layout of one layer's pools:
 *   K codes    [pool_pages][n_kv_heads][page_slots][128] uint8
 *   V codes    [pool_pages][n_kv_heads][128][page_slots] uint8  (a page's value rows
 *              transposed: element d of slot s at [d][16 (s / 16) + b(s % 16)], the 16 slots
 *              of a chunk in the order 0, 1, 8, 9, 2, 3, 10, 11, 4, 5, 12, 13, 6, 7, 14, 15,
 *              i.e. b(s) = 4 ((s % 8) / 2) + 2 (s / 8) + s % 2)
 *   exponents  [pool_pages][n_kv_heads][page_slots / 16][2][16] int8  (per 16-slot chunk:
 *              the 16 keys' exponents, then the 16 values')
 * FP8 caches work with ham_kv_fill (it encodes the bf16 rows it is given), ham_kv_export,
 * ham_kv_export_scales, ham_kv_append, ham_decode_attn, ham_decode_attn_ex, ham_decode_step
 * (its new slot is encoded as ham_kv_append encodes it, and attended as the cache then holds
 * it), ham_qkv_append (the projected rows, the key rotated, rounded to bf16 as for a bf16 cache
 * and then encoded by the same rule) and the counter calls; ham_prefill and ham_micro_step
 * return HAM_EUNSUPPORTED for them. */

/* Copy one layer's exponent array out (layout above): pool_pages * n_kv_heads * page_slots *
 * 2 bytes.  HAM_EINVAL for a bf16 cache. */
int ham_kv_export_scales(ham_kv *kv, int32_t layer, void *e_dst, void *stream);

/* Set the slot and token counters of one layer from device arrays (e.g. to roll back the
 * slots of a rejected macro-step): num_slots [batch] int32, num_tokens [batch] int64
 * (nullable: tokens unchanged).  Slots at or past the new count are free and the next
 * append overwrites them.  A count outside [0, max_slots_per_seq] sets the device error
 * word and leaves that sequence unchanged.  One small kernel; can be captured in a graph. */
int ham_kv_set_lengths(ham_kv *kv, int32_t layer, const int32_t *num_slots,
                       const int64_t *num_tokens, void *stream);

/* Set every sequence of every layer back to 0 slots / 0 tokens (pages stay reserved). */
int ham_kv_reset(ham_kv *kv, void *stream);

/* Number of CTAs one attention launch uses (0 = default: SMs x min(4, resident CTAs per
 * SM)).  Range 1 .. 8 x SMs.  Any value gives the same result up to fp32 summation order. */
int ham_kv_set_attn_ctas(ham_kv *kv, int32_t ctas);

/* Limit, in nanoseconds, of the data waits of this handle's attention and prefill kernels: the
 * waits of the shared-memory ring for copies to land and for stages to be freed.  0 restores the
 * default, 2 s (the largest value accepted).  A wait that runs out records HAM_DEVERR_TIMEOUT
 * (read by ham_kv_status), stops its CTA's work and leaves that launch's output undefined; the
 * copies a CTA already issued are still waited for, with the default bound, before it exits.  This
 * is a testing aid for the failure path (a limit of a few nanoseconds makes the waits run out on
 * an otherwise healthy GPU); production callers leave the default. */
int ham_kv_set_wait_limit_ns(ham_kv *kv, uint64_t ns);

/* Host evaluation of the split plan the attention kernel uses (no GPU needed).  Chunks are
 * 16 slots; the chunks of (sequence b, KV head g), b-major, are numbered contiguously (W in
 * all).  The first min(ctas, ceil(W / 4)) CTAs get equal non-empty ranges (a small problem
 * gets ranges of about 4 chunks instead of being spread over every CTA), CTA c the chunks
 * [cta_begin[c], cta_begin[c+1]); the others stay idle.  For each segment
 * s = b*n_kv_heads+g, seg_first_cta[s] .. seg_last_cta[s] are exactly the CTAs that touch
 * it (-1, -1 if empty).
 * cta_begin [ctas+1] int64; seg_first_cta, seg_last_cta [batch*n_kv_heads] int32. */
int ham_split_plan(int32_t batch, int32_t n_kv_heads, const int32_t *num_slots_host,
                   int32_t ctas, int64_t *cta_begin, int32_t *seg_first_cta,
                   int32_t *seg_last_cta);

/* ------------------------------------------------------------------------------------
 * Decode attention without any allocation
 * ------------------------------------------------------------------------------------
 * No counterpart in the paper: this entry point exists for callers that cannot allocate
 * device memory themselves -- code whose device memory is owned by a host framework or a
 * fixed-size arena (an inference-server plugin, for instance), or code that must not call
 * cudaMalloc at the point where attention runs.  They own the cache in their own layout-
 * compatible buffers and pass every input and output; the split-attention scratch comes
 * from an 8 MiB array compiled into libham.so, which every GPU that loads the library keeps
 * until the process exits.  The call itself allocates nothing (no cudaMalloc, cudaFree or
 * allocating library routine).
 *  - The first call on each device looks up that array's device address and sets the kernel
 *    attributes of every output type and head_dim it supports (not only the first call's);
 *    make that first call before any stream capture on the device.
 *  - All calls share the one array: calls that overlap on the GPU (other streams, other
 *    threads) race on it and give wrong results.  Serialize them.
 *  - A configuration whose scratch would exceed the array ((ctas + batch*n_kv_heads) *
 *    group * (head_dim + 2) * 4 bytes, about) is rejected with HAM_EINVAL; nothing runs.
 * The computation is that of ham_decode_attn_ex over the given pool and page table.        */
typedef struct ham_attn_args {
  const void *k_pool, *v_pool;  /* device bf16 [pool_pages][n_kv_heads][page_slots][head_dim] */
  const int32_t *page_table;    /* device [batch][max_pages]: slot n of sequence b is row
                                   n % page_slots of page page_table[b][n / page_slots] */
  const int32_t *num_slots;     /* device [batch]: slots to attend over, each <= max_slots */
  const void *q;                /* device bf16 [batch][n_q_heads][head_dim], already rotated */
  void *out;                    /* device [batch][n_q_heads][head_dim], bf16 or f32 */
  int32_t *err;                 /* nullable device int32: first HAM_DEVERR_* seen, else kept */
  int64_t pool_pages;
  int32_t batch, n_q_heads, n_kv_heads, head_dim, page_slots, max_pages, max_slots;
  int32_t ctas;                 /* 0: SMs x resident CTAs per SM */
  int32_t out_dtype;            /* HAM_DTYPE_BF16 or HAM_DTYPE_F32 */
} ham_attn_args;

int ham_decode_attn_noalloc(const ham_attn_args *args, void *stream);

/* ------------------------------------------------------------------------------------
 * Compositional embedder (Sec. 3.2, Sec. 3.4, Sec. 4.1)
 * ------------------------------------------------------------------------------------
 * Before a macro-step's forward, the 1..max_patch tokens each sequence produced in the last
 * one are fused into a single hidden state of the model width H: a multi-head cross-attention
 * whose query is the mean of the token embeddings and whose keys and values come from the
 * embeddings plus a learned embedding of each token's place in the patch, then a linear layer.
 * A sequence with one token skips the module: its hidden state is the token's embedding, bit
 * for bit.  For sequence b with n >= 2 tokens x_0..x_{n-1}:
 *   q = W_q mean(x),  k_i = W_k (x_i + P[i]),  v_i = W_v (x_i + P[i]),
 *   per head h: o_h = sum_i softmax_i(q_h . k_{i,h} / sqrt(head_dim)) v_{i,h},   out_b = W_o o.
 * Weights are bf16 [out][in] row-major (y = W x); accumulation is fp32, o and out are
 * rounded to bf16 (o reaches the output projection as a hi + lo pair of bf16 values, about
 * 16 bits).  The handle owns copies of the weights (pre-tiled for the projection kernel) and
 * all workspace; the dense projections (tcgen05 tensor-core products that stream the weights)
 * and the fusion (mean query, position terms, softmax, bypass) run in this library's kernels. */
typedef struct ham_embedder ham_embedder; /* opaque handle: weights and workspace */

typedef struct ham_embed_config {
  int32_t hidden;     /* H, the model width: a multiple of n_heads and of 8 */
  int32_t n_heads;    /* heads; head_dim = hidden / n_heads must be 32, 64 or 128 */
  int32_t max_batch;  /* sequences per ham_embed call, at most */
  int32_t max_patch;  /* tokens per sequence, at most (1..8; the paper's macro-steps emit 4) */
} ham_embed_config;

/* Allocate an embedder and copy its weights (device bf16): wq, wk, wv, wo [H][H]; pos
 * [max_patch][H].  Host errors: HAM_EINVAL (bad config, NULL or unaligned pointer),
 * HAM_ENOMEM, HAM_ECUDA. */
int ham_embedder_alloc(const ham_embed_config *cfg, const void *wq, const void *wk,
                       const void *wv, const void *wo, const void *pos, ham_embedder **out);
int ham_embedder_free(ham_embedder *e);

/* Fuse the tokens of `batch` sequences.  x: device bf16 [total_tokens][H], sequence b owning
 * rows offsets[b] .. offsets[b+1]-1; offsets: device int32 [batch + 1], offsets[0] = 0 and
 * offsets[batch] = total_tokens; out: device bf16 [batch][H].  A sequence whose token count
 * is outside 1..max_patch gets zeros and sets the device error word (HAM_DEVERR_NTOK).
 * Asynchronous on `stream`.  Host errors: HAM_EINVAL (NULL/unaligned pointers, batch or
 * total_tokens out of range), HAM_ECUDA.  Calls on one handle must not overlap in time. */
int ham_embed(ham_embedder *e, const void *x, const int32_t *offsets, int32_t batch,
              int32_t total_tokens, void *out, void *stream);

/* Read and clear the embedder's device error word (synchronizes `stream`).  Returns
 * HAM_EDEVICE if it was set, with the code in *device_code. */
int ham_embedder_status(ham_embedder *e, void *stream, int32_t *device_code);

/* Give the embedder the vocabulary's token-embedding table (device bf16 [vocab][H], copied) for
 * ham_embed_tokens.  The tokens' projections [W_q; W_k; W_v] E[v] are tabulated once, in fp32
 * ([vocab][3H], 12 H bytes per entry: 3.2 GB for 128k entries at H = 2048), so that a call
 * gathers rows instead of multiplying by the weights; the result is the same function as
 * ham_embed of the gathered embeddings.  Synchronous.  Host errors: HAM_EINVAL, HAM_ENOMEM,
 * HAM_ECUDA. */
int ham_embedder_set_vocab(ham_embedder *e, const void *table, int32_t vocab);

/* ham_embed of the embeddings E[ids[t]]: ids device int32 [total_tokens], grouped by sequence
 * through offsets as for ham_embed.  A token id outside [0, vocab) gives its sequence zeros and
 * sets the device error word (HAM_DEVERR_NTOK).  Host errors as for ham_embed, and HAM_EINVAL
 * if no vocabulary was set. */
int ham_embed_tokens(ham_embedder *e, const int32_t *ids, const int32_t *offsets,
                     int32_t batch, int32_t total_tokens, void *out, void *stream);

#ifdef __cplusplus
}
#endif
#endif /* HAM_H */
