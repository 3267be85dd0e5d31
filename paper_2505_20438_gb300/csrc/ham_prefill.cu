// Chunked prefill over the paged smashed-KV cache (sm_103a): prompt ingestion.
//
// What it computes (HAMburger, arXiv 2505.20438): only response tokens are fused into
// multi-token slots (Figure 2, training), so a prompt's tokens each become one slot, stored
// exactly as the decode path's append stores a slot (RoPE at the slot's position, Sec. 3.2;
// one KV set per slot, Sec. 3.1).  The chunk's queries then attend causally: new row j of a
// sequence holding L slots attends over slots 0 .. L + j (Llama-3.2 base model, Sec. 4.1:
// softmax scale 1/sqrt(d), query head h reads KV head h / G).  Unlike decode this is a dense
// contraction: every K/V tile serves 128 query rows, so it runs on the tensor cores.
//
// Three launches (four when the attention splits over the cached slots):
//  1. prefill_plan_kernel, one block per sequence: checks that the sequence's rows fit
//     (counts, capacity, pages), gives each row its position (slot index, running token count
//     or the caller's) and pool row (or -1: not stored), numbers the query blocks, and advances
//     the counters.
//  2. prefill_rope_kernel, one block per row: turns q and k at the row's position and stores
//     k and v into the row's slot.  The rotation x0 c - x1 s is evaluated from the fp64 cos/sin
//     table in pairs of fp32 values (error-free products and sums, about 48 bits) and rounded
//     once to bf16, which gives the bits of the fp64 evaluation except when the exact value
//     lies within ~2^-44 (relative) of a rounding boundary.  This GPU's fp64 pipe would take
//     about half a millisecond for a 16k-row chunk of a Llama-8B layer; the fp32 pairs take
//     microseconds.
//  3. prefill_attn_kernel, one CTA per (KV head, two Q tiles of 128 (query row, head) rows of
//     one sequence), one CTA an SM: S = Q K^T and O += P V on the 5th-generation tensor cores
//     (tcgen05.mma kind::f16, M = 128, bf16 operands, fp32 accumulators in tensor memory).
//     Q, K and V reach shared memory by TMA (64-slot K/V tiles of four 16-slot chunks, each
//     64-column half one box in the 128-byte swizzle; K and V in rings of their own, filled by
//     two producer warps whose lanes issue the copies and look the pages up 32 chunks ahead).
//     Two warps issue the S products of the two Q tiles and two the O products (one thread
//     issues a tcgen05.mma only about every 125 cycles); eight softmax warps, one thread a row,
//     read S from tensor memory, keep the online softmax in fp32 (exp2 domain, running maximum
//     raised only past 2^8), write the bf16 probabilities to tensor memory columns of their own
//     (the A operand of O += P V, so the next S is computed meanwhile) and rescale O there when
//     the maximum moves.  The causal mask applies to the tiles that reach past a row's own slot;
//     CTAs are scheduled latest query tiles first, the longest rows of the causal triangle.
//     When the grid would leave SMs idle (a short chunk: few query blocks) it gets a third
//     dimension, the split over slots: a sequence with L cached slots is cut into up to
//     floor(L / 512) contiguous ranges of 64-slot tiles (the last range also takes the chunk's
//     own slots), each CTA streams one range, and a split that is not alone leaves its rows'
//     unnormalised output, running maximum and sum as a partial.
//  4. prefill_merge_kernel (split launches only), one warp per (row, head): the split-softmax
//     merge of the partials in split order (as the decode combine merges its CTAs').
//
// Every wait is bounded (about 2 s); a wait that runs out records HAM_DEVERR_TIMEOUT, lets the
// CTA's copies land and returns.  No trap, no unbounded spin.
#include <cuda.h>
#include <cuda_bf16.h>

#include <cmath>
#include <type_traits>

#include "ham_internal.cuh"
#include "ham_prefill.cuh"
#include "ham_ptx.cuh"

namespace ham {
namespace {

constexpr int kPlanThreads = 256;
constexpr int kPlanRun = 8;  // consecutive rows a plan thread takes per tile
constexpr float kRescaleSlack = 8.0f;  // log2 units: the running max lags by at most 2^8
constexpr int kRopeThreads = 256;

// ------------------------------------------------------------------------------------
// 1. plan
// ------------------------------------------------------------------------------------
__device__ __forceinline__ int block_sum(int x, int *red) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(kFull, x, o);
  __syncthreads();  // red may still be read from a previous call
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = x;
  __syncthreads();
  int total = 0;
  for (int w = 0; w < (int)(blockDim.x >> 5); ++w) total += red[w];
  return total;
}

// Inclusive prefix sum over the block (thread order); *total gets the block's sum.
__device__ __forceinline__ int block_scan(int x, int *red, int *total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(kFull, x, o);
    if (lane >= o) x += y;
  }
  __syncthreads();
  if (lane == 31) red[warp] = x;
  __syncthreads();
  int before = 0, all = 0;
  for (int w = 0; w < (int)(blockDim.x >> 5); ++w) {
    if (w < warp) before += red[w];
    all += red[w];
  }
  *total = all;
  return x + before;
}

__global__ void __launch_bounds__(kPlanThreads) prefill_plan_kernel(PrefillView v, int qb_rows) {
  __shared__ int red[kPlanThreads / 32];
  const int b = blockIdx.x, tid = threadIdx.x, B = v.batch;
  // The offsets must describe the call's rows: every block checks all of them, so that all
  // agree, and counts the query blocks of the sequences before its own.
  int bad_off = 0, qb = 0;
  for (int i = tid; i < B; i += kPlanThreads) {
    const int a = v.offsets[i], e = v.offsets[i + 1];
    bad_off |= e < a;
    if (i < b && e > a) qb += (e - a + qb_rows - 1) / qb_rows;
  }
  if (tid == 0) bad_off |= v.offsets[0] != 0 || v.offsets[B] != v.rows;
  bad_off = __syncthreads_or(bad_off);
  qb = block_sum(qb, red);
  if (bad_off) {
    if (tid == 0) {
      v.seq_info[b] = make_int4(-1, 0, 0, 0);
      if (b == 0) record_error(v.err, HAM_DEVERR_NTOK);
    }
    return;
  }
  const int a = v.offsets[b], n = v.offsets[b + 1] - a;
  const int L = v.num_slots[b];
  int err = 0;
  if (L < 0 || L > v.max_slots) err = HAM_DEVERR_SLOTS;
  else if ((int64_t)L + n > v.max_slots) err = HAM_DEVERR_CAPACITY;
  int bad_tok = 0, bad_page = 0;
  if (!err && n > 0) {
    if (v.ntok)
      for (int j = tid; j < n; j += kPlanThreads) bad_tok |= v.ntok[a + j] < 1;
    const int p0 = L / v.page_slots, p1 = (L + n - 1) / v.page_slots;
    for (int pg = p0 + tid; pg <= p1; pg += kPlanThreads) {
      const int page = v.page_table[(int64_t)b * v.max_pages + pg];
      bad_page |= page < 0 || page >= v.pool_pages;
    }
  }
  bad_tok = __syncthreads_or(bad_tok);
  bad_page = __syncthreads_or(bad_page);
  if (!err && bad_tok) err = HAM_DEVERR_NTOK;
  if (!err && bad_page) err = HAM_DEVERR_PAGE;
  if (err) {  // none of the rows is stored
    for (int j = tid; j < n; j += kPlanThreads) v.row_info[a + j] = make_int2(0, -1);
    if (tid == 0) {
      record_error(v.err, err);
      v.seq_info[b] = make_int4(-1, n, qb, 1);
    }
    return;
  }
  // positions (the caller's, the slot index, or the tokens before the row) and pool rows.  A
  // thread takes kPlanRun consecutive rows of each tile of kPlanThreads * kPlanRun rows: their
  // token counts, positions and page-table entries are loaded together, and one block scan of
  // the threads' sums a tile gives every row its tokens before it.
  const int64_t t0 = v.num_tokens[b];
  int64_t carry = 0;
  for (int j0 = 0; j0 < n; j0 += kPlanThreads * kPlanRun) {
    const int jb = j0 + tid * kPlanRun;
    int t[kPlanRun], run = 0;
#pragma unroll
    for (int k = 0; k < kPlanRun; ++k) {
      t[k] = jb + k < n ? (v.ntok ? v.ntok[a + jb + k] : 1) : 0;
      run += t[k];
    }
    int total = 0;
    int64_t before = t0 + carry + (block_scan(run, red, &total) - run);
#pragma unroll
    for (int k = 0; k < kPlanRun; ++k) {
      const int j = jb + k;
      if (j < n) {
        int64_t p;
        if (v.pos) p = v.pos[a + j];
        else if (v.pos_mode == HAM_POS_SLOT) p = (int64_t)L + j;
        else p = before;
        const int slot = L + j, pg = slot / v.page_slots;
        const int page = v.page_table[(int64_t)b * v.max_pages + pg];
        v.row_info[a + j] = make_int2((int32_t)p, page * v.page_slots + (slot - pg * v.page_slots));
      }
      before += t[k];
    }
    carry += total;
  }
  if (tid == 0) {
    v.seq_info[b] = make_int4(L, n, qb, 1);
    v.num_slots[b] = L + n;
    v.num_tokens[b] = t0 + carry;
  }
}

// ------------------------------------------------------------------------------------
// 2. RoPE + append
// ------------------------------------------------------------------------------------
// bf16 bits of hi + lo (|lo| <= half an fp32 ulp of hi), rounded to nearest, ties to even:
// the rounding of hi alone, except where hi sits exactly halfway between two bf16 values and
// lo says on which side the sum lies.
__device__ __forceinline__ uint16_t bf16_of_pair(float hi, float lo) {
  const uint32_t u = __float_as_uint(hi);
  if ((u & 0xFFFFu) == 0x8000u && lo != 0.f && (u & 0x7F800000u) != 0x7F800000u) {
    const bool away = (lo > 0.f) == (hi > 0.f);
    return (uint16_t)((u >> 16) + (away ? 1u : 0u));
  }
  return __bfloat16_as_ushort(__float2bfloat16_rn(hi));
}

// Fast evaluation of a c - b s, with c = ch + cl and s = sh + sl given as fp32 pairs and a, b
// exact (bf16 values): y = a ch - b sh in plain fp32 lies within 3 * 2^-24 (|a| + |b|) < e / 2
// of the exact value, e = (|a| + |b|) 2^-21.  When no bf16 rounding boundary is within e of y
// (the nearest one is the midpoint sharing y's upper 16 bits; the others are a quarter of a
// bf16 spacing away, more than e once e < 2^-11 |y|), the exact value rounds as y does and
// *sure is set; otherwise rotate_exact gives the rounding.
__device__ __forceinline__ float rotate_fast(float a, float b, float ch, float sh, float e,
                                             bool *sure) {
  const float y = __fmaf_rn(a, ch, -__fmul_rn(b, sh));
  const float mid = __uint_as_float((__float_as_uint(y) & 0xFFFF0000u) | 0x8000u);
  *sure = fabsf(__fsub_rn(y, mid)) > e && e < __fmul_rn(fabsf(y), 0x1p-11f);
  return y;
}

// a c - b s rounded once to bf16 near a rounding boundary: products by FMA error terms and sums
// by two-sum are exact, only the small terms are rounded, so the pair carries about 48 bits of
// the exact value.
__device__ __noinline__ uint16_t rotate_exact(float a, float b, float ch, float cl, float sh,
                                              float sl) {
  const float p1 = __fmul_rn(a, ch), e1 = __fmaf_rn(a, ch, -p1);
  const float p2 = __fmul_rn(b, sh), e2 = __fmaf_rn(b, sh, -p2);
  const float s = __fsub_rn(p1, p2);  // two-sum of p1 and -p2: s + t = p1 - p2
  const float bp = __fsub_rn(s, p1);
  const float t = __fadd_rn(__fsub_rn(p1, __fsub_rn(s, bp)), __fsub_rn(-p2, bp));
  const float low =
      __fmaf_rn(a, cl, __fmaf_rn(-b, sl, __fadd_rn(t, __fsub_rn(e1, e2))));
  if (low == 0.f) return __bfloat16_as_ushort(__float2bfloat16_rn(s));  // keeps s's zero sign
  const float hi = __fadd_rn(s, low);  // two-sum of s and low
  const float hb = __fsub_rn(hi, s);
  const float lo = __fadd_rn(__fsub_rn(s, __fsub_rn(hi, hb)), __fsub_rn(low, hb));
  return bf16_of_pair(hi, lo);
}

__device__ __forceinline__ float bf16_value(uint16_t b) {
  return __uint_as_float((uint32_t)b << 16);
}

__device__ __forceinline__ void split_double(double x, float &hi, float &lo) {
  hi = __double2float_rn(x);
  lo = __double2float_rn(x - (double)hi);  // x - hi is exact in fp64
}

// Shared-memory index of frequency i of the (cos, sin) row: the eight frequencies a thread
// reads, 8 (i / 8) .. + 7, rotated by i / 8 within their group of eight, so that the eight
// threads of a head (distinct i / 8, same step) read eight distinct 16-byte bank groups.
__device__ __forceinline__ int cs_index(int i) { return (i & ~7) | ((i + (i >> 3)) & 7); }

// One block per row.  Thread t owns the eight pairs (i, i + d/2), i = 8 (t % (d/16)) .. + 7, of
// heads t / (d/16), t / (d/16) + 256 / (d/16), ... (query heads, then key heads): a 16-byte load
// and store of each half.  The plan left the row's position and pool row in row_info, so every
// load the block makes needs only the row index, and is issued at once: the first two heads'
// halves, a 16-byte piece of the value row, and then the (cos, sin) row of the position, which
// goes to shared memory, read by the threads of every head.
template <int D, typename OutT>
__global__ void __launch_bounds__(kRopeThreads) prefill_rope_kernel(PrefillView v) {
  constexpr int kHalf = D / 2, kOcts = kHalf / 8, kHeadsPass = kRopeThreads / kOcts;
  constexpr int kVPieces = D / 8;  // 16-byte pieces of one head's value row
  static_assert(kHalf <= kRopeThreads, "one thread a frequency");
  __shared__ float4 cs_s[kHalf];   // (c_hi, c_lo, s_hi, s_lo) of frequency i at cs_index(i)
  const int64_t r = blockIdx.x;
  const int tid = threadIdx.x, j = tid % kOcts, h0 = tid / kOcts, h1 = h0 + kHeadsPass;
  const int Hq = v.n_q_heads, Hkv = v.n_kv_heads, H = Hq + Hkv, nv = Hkv * kVPieces;
  uint16_t *const qrow = v.q + r * Hq * D;
  const uint16_t *const krow = v.k_new + r * Hkv * D;
  const uint4 *const vrow = reinterpret_cast<const uint4 *>(v.v_new + r * Hkv * D);
  auto half_of = [&](int h, int upper) {  // 16-byte piece j of head h's lower or upper half
    const uint16_t *src = h < Hq ? qrow + h * D : krow + (h - Hq) * D;
    return *reinterpret_cast<const uint4 *>(src + upper * kHalf + 8 * j);
  };
  // 1. the loads (the row's pool row is -1 when it is not stored; the call's offsets are valid
  //    when sequence 0's plan entry says so)
  const int2 ri = v.row_info[r];
  const int offsets_ok = v.seq_info[0].w;
  uint4 x0l{}, x0h{}, x1l{}, x1h{}, vv{};
  if (h0 < H) { x0l = half_of(h0, 0); x0h = half_of(h0, 1); }
  if (h1 < H) { x1l = half_of(h1, 0); x1h = half_of(h1, 1); }
  if (tid < nv) vv = vrow[tid];
  const int p = ri.x;
  const bool in_table = p >= 0 && p < v.rope_positions;
  float4 c4{};
  if (tid < kHalf && in_table) c4 = v.rope_table_ff[(int64_t)p * kHalf + tid];
  if (!offsets_ok || ri.y < 0) {  // not stored: its output rows are 0
    OutT *o = static_cast<OutT *>(v.out) + r * Hq * D;
    for (int e = tid; e < Hq * D; e += kRopeThreads) o[e] = OutT(0.f);
    return;
  }
  // 2. the (cos, sin) row in shared memory (past the table: from fp64 sincos) and the slot's
  //    page and row in it
  __shared__ int2 where;  // (page, row in page)
  if (tid < kHalf) {
    if (!in_table) {
      double c, sn;
      sincos((double)p * v.inv_freq[tid], &sn, &c);
      split_double(c, c4.x, c4.y);
      split_double(sn, c4.z, c4.w);
    }
    cs_s[cs_index(tid)] = c4;
  }
  if (tid == 0) {
    where = make_int2(ri.y / v.page_slots, ri.y % v.page_slots);
    v.slot_pos[ri.y] = p;
    v.slot_ntok[ri.y] = v.ntok ? v.ntok[r] : 1;
  }
  __syncthreads();
  const int64_t page = where.x;
  const int prow = where.y;
  auto pool_row = [&](uint16_t *pool, int g) {
    return pool + ((page * Hkv + g) * v.page_slots + prow) * D;
  };
  // 3. the value row (a bit copy)
  if (tid < nv) reinterpret_cast<uint4 *>(pool_row(v.v_pool, tid / kVPieces))[tid % kVPieces] = vv;
  for (int e = tid + kRopeThreads; e < nv; e += kRopeThreads)
    reinterpret_cast<uint4 *>(pool_row(v.v_pool, e / kVPieces))[e % kVPieces] = vrow[e];
  // 4. query heads in place, key heads into the slot
  // Every output by the fast path, two to a conversion; the rare outputs whose rounding the
  // fast path leaves open (bit 2 m + u of `open`: pair m, lower (u = 0) or upper half) are
  // redone exactly in a loop of their own, so the exact path costs nothing where it is not used.
  auto rotate_store = [&](int h, const uint4 &xl, const uint4 &xh) {
    uint16_t *dst = h < Hq ? qrow + h * D : pool_row(v.k_pool, h - Hq);
    uint32_t wl[4] = {xl.x, xl.y, xl.z, xl.w}, wh[4] = {xh.x, xh.y, xh.z, xh.w};
    uint32_t open = 0;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      float yl[2], yh[2];
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        const float4 c = cs_s[cs_index(8 * j + 2 * k + e)];
        const float x0 = bf16_value((uint16_t)(wl[k] >> (16 * e)));
        const float x1 = bf16_value((uint16_t)(wh[k] >> (16 * e)));
        const float err = __fmul_rn(__fadd_rn(fabsf(x0), fabsf(x1)), 0x1p-21f);
        bool sure_l, sure_h;
        yl[e] = rotate_fast(x0, x1, c.x, c.z, err, &sure_l);   // x0 c - x1 s
        yh[e] = rotate_fast(x1, x0, c.x, -c.z, err, &sure_h);  // x1 c + x0 s
        open |= (sure_l ? 0u : 1u) << (2 * (2 * k + e));
        open |= (sure_h ? 0u : 2u) << (2 * (2 * k + e));
      }
      const __nv_bfloat162 ol = __floats2bfloat162_rn(yl[0], yl[1]);
      const __nv_bfloat162 oh = __floats2bfloat162_rn(yh[0], yh[1]);
      const uint32_t uol = *reinterpret_cast<const uint32_t *>(&ol);
      const uint32_t uoh = *reinterpret_cast<const uint32_t *>(&oh);
      wl[k] = uol;  // wl/wh now hold outputs; the exact path reads the inputs from xl/xh
      wh[k] = uoh;
    }
    while (open) {
      const int bit = __ffs(open) - 1;
      open &= open - 1;
      const int m = bit >> 1, k = m >> 1, e = m & 1, upper = bit & 1;
      const uint32_t in_l = k == 0 ? xl.x : k == 1 ? xl.y : k == 2 ? xl.z : xl.w;
      const uint32_t in_h = k == 0 ? xh.x : k == 1 ? xh.y : k == 2 ? xh.z : xh.w;
      const float4 c = cs_s[cs_index(8 * j + m)];
      const float x0 = bf16_value((uint16_t)(in_l >> (16 * e)));
      const float x1 = bf16_value((uint16_t)(in_h >> (16 * e)));
      const uint32_t y = upper ? rotate_exact(x1, x0, c.x, c.y, -c.z, -c.w)
                               : rotate_exact(x0, x1, c.x, c.y, c.z, c.w);
      const uint32_t keep = e ? 0x0000FFFFu : 0xFFFF0000u, put = y << (16 * e);
#pragma unroll
      for (int kk = 0; kk < 4; ++kk) {
        if (kk != k) continue;
        if (upper) wh[kk] = (wh[kk] & keep) | put;
        else wl[kk] = (wl[kk] & keep) | put;
      }
    }
    *reinterpret_cast<uint4 *>(dst + 8 * j) = make_uint4(wl[0], wl[1], wl[2], wl[3]);
    *reinterpret_cast<uint4 *>(dst + kHalf + 8 * j) = make_uint4(wh[0], wh[1], wh[2], wh[3]);
  };
  if (h0 < H) rotate_store(h0, x0l, x0h);
  if (h1 < H) rotate_store(h1, x1l, x1h);
  for (int h = h1 + kHeadsPass; h < H; h += kHeadsPass)
    rotate_store(h, half_of(h, 0), half_of(h, 1));
}

// ------------------------------------------------------------------------------------
// 3. causal attention of the chunk, on the 5th-generation tensor cores (tcgen05)
// ------------------------------------------------------------------------------------
// A CTA covers one KV head and two Q tiles of 128 rows each; a row is a (query row, head)
// pair, m = (row - first row of the tile) * G + head within the group, and sits in TMEM lane m.
// Tensor-memory columns per Q tile q: S_q (64 fp32 scores of the current 64-slot K tile), P_q
// (the bf16 probabilities of the tile as pairs: the A operand of O += P V) and O_q (head_dim
// fp32).  The products of a Q tile are issued by two warps, one for S = Q K^T and one for
// O += P V: one thread issues a tcgen05.mma only about every 125 cycles (measured on GB300),
// so a single issuer would keep the tensor cores half idle.  Because P has columns of its own,
// S_q(t + 1) is computed while the softmax group still works on tile t.
template <int D>
struct TcShape {
  static constexpr int kTile = 64;                           // slots per K/V tile
  static constexpr int kChunks = kTile / kChunkSlots;        // 16-slot TMA chunks per tile
  static constexpr int kHalves = D / 64;                     // 64-column halves of a row
  static constexpr int kHalfTileBytes = kTile * 128;         // one half of a K or V tile
  static constexpr int kKVBytes = kHalves * kHalfTileBytes;  // a K (or V) tile
  static constexpr int kKStages = D == 128 ? 4 : 8;          // K tiles in flight
  static constexpr int kVStages = D == 128 ? 5 : 8;          // V tiles in flight
  static constexpr int kQHalfBytes = 128 * 128;              // one half of a Q tile
  static constexpr int kQBytes = kHalves * kQHalfBytes;
  static constexpr int kOffK = 2 * kQBytes;                  // Q tiles at 0
  static constexpr int kOffV = kOffK + kKStages * kKVBytes;
  static constexpr int kOffBar = kOffV + kVStages * kKVBytes;
  // k_full, k_empty [kKStages]; v_full, v_empty [kVStages]; q_full; s_full, s_free, p_full,
  // pv_done [2]; mma_done
  static constexpr int kBars = 2 * kKStages + 2 * kVStages + 10;
  static constexpr int kSmem = 1024 + kOffBar + kBars * 8 + 16;
  static constexpr uint32_t kTmemCols = 512;
  static constexpr int kOffP = 2 * kTile;                    // TMEM column of P_0 (S_0 at 0)
  static constexpr int kOffO = kOffP + kTile;                // TMEM column of O_0
  // softmax: warps 0-3 (Q tile 0) and 4-7 (Q tile 1); TMA producers of Q and K (8) and of V
  // (10); MMA issue of S_0 (9), S_1 (11), O_0 (12), O_1 (13).
  static constexpr int kProducerWarp = 8, kVProducerWarp = 10;
  static constexpr int kSWarp0 = 9, kSWarp1 = 11, kOWarp0 = 12, kOWarp1 = 13;
  static constexpr int kThreads = 14 * 32;
  static_assert(D == 64 || D == 128, "head_dim 64 or 128");
  static_assert(kOffO + 2 * D <= (int)kTmemCols, "TMEM columns");
  static_assert(kSmem <= 227 * 1024, "shared memory");
};

template <typename OutT>
__device__ __forceinline__ void store_row32(OutT *dst, const uint32_t (&o)[32], float scale) {
  if constexpr (std::is_same<OutT, float>::value) {
#pragma unroll
    for (int e = 0; e < 32; e += 4)
      *reinterpret_cast<float4 *>(dst + e) =
          make_float4(__uint_as_float(o[e]) * scale, __uint_as_float(o[e + 1]) * scale,
                      __uint_as_float(o[e + 2]) * scale, __uint_as_float(o[e + 3]) * scale);
  } else {
#pragma unroll
    for (int e = 0; e < 32; e += 8)
      *reinterpret_cast<uint4 *>(dst + e) = make_uint4(
          pack_bf16x2(__uint_as_float(o[e]) * scale, __uint_as_float(o[e + 1]) * scale),
          pack_bf16x2(__uint_as_float(o[e + 2]) * scale, __uint_as_float(o[e + 3]) * scale),
          pack_bf16x2(__uint_as_float(o[e + 4]) * scale, __uint_as_float(o[e + 5]) * scale),
          pack_bf16x2(__uint_as_float(o[e + 6]) * scale, __uint_as_float(o[e + 7]) * scale));
  }
}

// One CTA per SM (shared memory and 512 TMEM columns).
template <int D, typename OutT>
__global__ void __launch_bounds__(TcShape<D>::kThreads, 1)
    prefill_attn_kernel(const __grid_constant__ CUtensorMap tmap_q,
                        const __grid_constant__ CUtensorMap tmap_k,
                        const __grid_constant__ CUtensorMap tmap_v, const PrefillView v) {
  using S = TcShape<D>;
  const int Hq = v.n_q_heads, Hkv = v.n_kv_heads, G = Hq / Hkv, R = 128 / G, QB = 2 * R;
  const int g = blockIdx.x;
  const int64_t xq = (int64_t)gridDim.y - 1 - blockIdx.y;  // latest query blocks first
  int lo = 0, hi = v.batch - 1;                            // the sequence of query block xq
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (v.seq_info[mid].z <= xq) lo = mid; else hi = mid - 1;
  }
  const int4 si = v.seq_info[lo];
  if (si.x < 0 || xq < si.z || xq >= (int64_t)si.z + (si.y + QB - 1) / QB) return;
  const int b = lo, L = si.x, n = si.y;
  const int qb0 = (int)(xq - si.z) * QB;
  const int64_t row0 = v.offsets[b];
  // rows of each Q tile and the K/V tiles they reach (slots 0 .. L + last row)
  const int rows_q0 = min(R, n - qb0), rows_q1 = max(0, min(R, n - qb0 - R));
  int ntile[2];
  ntile[0] = (L + qb0 + rows_q0 + S::kTile - 1) / S::kTile;
  ntile[1] = rows_q1 > 0 ? (L + qb0 + R + rows_q1 + S::kTile - 1) / S::kTile : 0;
  const int ntiles = max(ntile[0], ntile[1]);
  const int kv_end = L + qb0 + (rows_q1 > 0 ? R + rows_q1 : rows_q0);  // no slot >= is attended
  // Split z of the sequence's zs takes tiles t0 .. t1 - 1: the cached part's whole tiles cut
  // evenly, the last split also the rest (the chunk's own slots, the causal edge).  Every split
  // starts at or before slot L - 64, which every row attends, so no row of a split is empty.
  const int zs = prefill_splits(L, (int)gridDim.z), z = (int)blockIdx.z;
  if (z >= zs) return;
  const int Lt = L / S::kTile;
  const int t0 = (int)((int64_t)z * Lt / zs);
  const int t1 = z + 1 == zs ? ntiles : (int)((int64_t)(z + 1) * Lt / zs);
  const int ntq[2] = {max(0, min(t1, ntile[0]) - t0), max(0, min(t1, ntile[1]) - t0)};
  const int nts = max(ntq[0], ntq[1]);  // tiles this CTA streams

  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = reinterpret_cast<uint8_t *>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t *k_full = reinterpret_cast<uint64_t *>(smem + S::kOffBar);
  uint64_t *k_empty = k_full + S::kKStages, *v_full = k_empty + S::kKStages;
  uint64_t *v_empty = v_full + S::kVStages, *q_full = v_empty + S::kVStages;
  uint64_t *s_full = q_full + 1, *s_free = q_full + 3, *p_full = q_full + 5;
  uint64_t *pv_done = q_full + 7, *mma_done = q_full + 9;
  uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(k_full + S::kBars);
  volatile int *abort_flag = reinterpret_cast<volatile int *>(tmem_slot + 1);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  if (tid == 0) {
    // a stage is free once the products of both Q tiles that read it have completed
    for (int s = 0; s < S::kKStages; ++s) {
      mbar_init(&k_full[s], 1);
      mbar_init(&k_empty[s], 2);
    }
    for (int s = 0; s < S::kVStages; ++s) {
      mbar_init(&v_full[s], 1);
      mbar_init(&v_empty[s], 2);
    }
    mbar_init(q_full, 1);
    for (int q = 0; q < 2; ++q) {
      mbar_init(&s_full[q], 1);
      mbar_init(&s_free[q], 4);  // the softmax group has read S_q (one arrival per warp)
      mbar_init(&p_full[q], 4);  // ... and written P_q
      mbar_init(&pv_done[q], 1);
    }
    mbar_init(mma_done, 4);      // the four MMA warps
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == S::kProducerWarp && lane == 0) {
    prefetch_tensormap(&tmap_q);
    prefetch_tensormap(&tmap_k);
    prefetch_tensormap(&tmap_v);
  }
  if (warp == S::kSWarp0) tmem_alloc<S::kTmemCols>(tmem_slot);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  // ring and data waits: the launch's limit; draining in-flight work keeps the default 2 s
  const uint64_t wait_lim = data_wait_limit(v.wait_ns);

  if (warp == S::kProducerWarp || warp == S::kVProducerWarp) {
    // ------------------------------------------------------------ producers: TMA copies
    // One warp streams Q and the K tiles, another the V tiles, each as far ahead as its ring
    // allows (K tiles are needed a tile before V tiles and are released earlier).  A chunk at or
    // past kv_end is not copied: its rows are masked (K) or zeroed (V).
    const bool is_v = warp == S::kVProducerWarp;
    const uint64_t pol_kv = policy_evict_last();   // every query block of the sequence reads them
    if (!is_v && lane == 0) {
      const uint64_t pol_q = policy_evict_first();
      const int nq = rows_q1 > 0 ? 2 : 1;
      mbar_arrive_tx(q_full, (uint32_t)(nq * S::kQBytes));
      for (int q = 0; q < nq; ++q)
        for (int hh = 0; hh < S::kHalves; ++hh)
          tma_load_4d(smem + q * S::kQBytes + hh * S::kQHalfBytes, &tmap_q, 0, hh, g * G,
                      (int)(row0 + qb0 + q * R), q_full, pol_q);
    }
    const int stages = is_v ? S::kVStages : S::kKStages;
    uint8_t *ring = smem + (is_v ? S::kOffV : S::kOffK);
    uint64_t *full = is_v ? v_full : k_full, *empty = is_v ? v_empty : k_empty;
    const CUtensorMap *map = is_v ? &tmap_v : &tmap_k;
    // Page-table entries of 32 chunks (4 tiles) at a time, one per lane, requested a batch
    // ahead: lane l holds the pool row of chunk base + l (-1: at or past kv_end; -2: a page
    // outside the pool).
    const int nchunks = (kv_end + kChunkSlots - 1) / kChunkSlots;
    auto lookup = [&](int base) {
      int row = -1;
      if (base + lane < nchunks) {
        const int slot0 = (base + lane) * kChunkSlots;
        const int page = v.page_table[(int64_t)b * v.max_pages + slot0 / v.page_slots];
        row = page < 0 || page >= v.pool_pages
                  ? -2
                  : (int)(((int64_t)page * Hkv + g) * v.page_slots + slot0 % v.page_slots);
      }
      return row;
    };
    constexpr int kTilesPerBatch = 32 / S::kChunks;
    const int cbase = t0 * S::kChunks;  // the split's first chunk
    int row = lookup(cbase), row_next = lookup(cbase + 32);
    int issued = 0;
    for (int i = 0; i < nts; ++i) {  // tile t0 + i, the i-th of this CTA's ring
      if (i > 0 && i % kTilesPerBatch == 0) {
        row = row_next;
        row_next = lookup(cbase + (i / kTilesPerBatch + 1) * 32);
      }
      int my_row = __shfl_sync(kFull, row, ((i % kTilesPerBatch) * S::kChunks + lane) & 31);
      if (lane >= S::kChunks) my_row = -1;
      if (__any_sync(kFull, my_row == -2)) {  // the plan validated the table: this ends the CTA
        if (lane == 0) {
          record_error(v.err, HAM_DEVERR_PAGE);
          *abort_flag = 1;
        }
        break;
      }
      const int st = i % stages;
      int ok_wait = 1;
      if (lane == 0 && i >= stages)
        ok_wait = thread_wait(&empty[st], (uint32_t)((i / stages) - 1) & 1u, abort_flag, true,
                              wait_lim);
      if (!__shfl_sync(kFull, ok_wait, 0)) {
        if (lane == 0 && !*abort_flag) {
          record_error(v.err, HAM_DEVERR_TIMEOUT);
          *abort_flag = 1;
        }
        break;
      }
      // lane 0 posts the byte count, then lane c issues chunk c's boxes, so that the warp has
      // the tile's copies in flight at once
      const uint32_t nck = __popc(__ballot_sync(kFull, my_row >= 0));
      if (lane == 0) mbar_arrive_tx(&full[st], nck * (uint32_t)(kChunkSlots * D * 2));
      __syncwarp();
      if (my_row >= 0) {
#pragma unroll
        for (int hh = 0; hh < S::kHalves; ++hh)
          tma_load_3d(ring + st * S::kKVBytes + hh * S::kHalfTileBytes + lane * kChunkSlots * 128,
                      map, 0, hh, my_row, &full[st], pol_kv);
      }
      issued = i + 1;
    }
    if (lane == 0) {
      // every copy this warp issued lands before the CTA can exit
      if (!is_v) thread_wait(q_full, 0u, abort_flag, false);
      for (int t = max(0, issued - stages); t < issued; ++t)
        thread_wait(&full[t % stages], (uint32_t)(t / stages) & 1u, abort_flag, false);
    }
  } else if (warp == S::kSWarp0 || warp == S::kSWarp1 || warp == S::kOWarp0 ||
             warp == S::kOWarp1) {
    // ------------------------------------------------------------ MMA issue (lane 0)
    // S warp of Q tile q: S_q(t) = Q_q K_t^T once the softmax group has read S_q(t - 1) into
    // registers (s_free) and K_t has landed.  O warp: O_q += P_q(t) V_t once the group has
    // written P_q(t) (p_full) and V_t has landed; the group waits for pv_done before it writes
    // the next P or rescales O.  A K or V stage is released by a commit for each Q tile that
    // reads it; a tile that only one Q tile reaches is released twice by that tile's warp.
    const bool is_o = warp == S::kOWarp0 || warp == S::kOWarp1;
    const int q = (warp == S::kSWarp0 || warp == S::kOWarp0) ? 0 : 1;
    const int nt = ntq[q], other = ntile[q ^ 1];  // (tile t0 + i; other: absolute)
    bool ok = true;
    if (!is_o) {
      constexpr uint32_t id_s = idesc_bf16(128, S::kTile, false);  // K-major Q and K
      const uint32_t q_base = smem_u32(smem) + q * S::kQBytes;
      if (nt > 0) ok = warp_wait(q_full, 0u, abort_flag, wait_lim);
      for (int i = 0; ok && i < nt; ++i) {
        const int t = t0 + i, ks = i % S::kKStages;
        if ((i > 0 && !warp_wait(&s_free[q], (uint32_t)(i - 1) & 1u, abort_flag, wait_lim)) ||
            !warp_wait(&k_full[ks], (uint32_t)(i / S::kKStages) & 1u, abort_flag, wait_lim)) {
          ok = false;
          break;
        }
        if (lane == 0) {
          tc_fence_after();
          const uint32_t kt = smem_u32(smem + S::kOffK + ks * S::kKVBytes);
#pragma unroll
          for (int k = 0; k < D / 16; ++k) {
            const uint64_t a =
                smem_desc_sw128(q_base + (k >> 2) * S::kQHalfBytes + (k & 3) * 32, 16, 1024);
            const uint64_t bk =
                smem_desc_sw128(kt + (k >> 2) * S::kHalfTileBytes + (k & 3) * 32, 16, 1024);
            tc_mma(tmem + q * S::kTile, a, bk, id_s, k > 0);
          }
          tc_commit(&s_full[q]);
          tc_commit(&k_empty[ks]);
          if (t >= other) tc_commit(&k_empty[ks]);
        }
        __syncwarp();
      }
    } else {
      constexpr uint32_t id_o = idesc_bf16(128, D, true);  // P from TMEM, MN-major V
      for (int i = 0; ok && i < nt; ++i) {
        const int t = t0 + i, vs = i % S::kVStages;
        if (!warp_wait(&v_full[vs], (uint32_t)(i / S::kVStages) & 1u, abort_flag, wait_lim)) {
          ok = false;
          break;
        }
        if (t == ntiles - 1 && kv_end < (t + 1) * S::kTile) {
          // slots >= kv_end get p = 0; zero their value rows so that stale bits never reach O
          // (both O warps may write the same zeros)
          const int z0 = kv_end - t * S::kTile, per_half = (S::kTile - z0) * 8;
          uint8_t *vt = smem + S::kOffV + vs * S::kKVBytes;
          for (int e = lane; e < S::kHalves * per_half; e += 32) {
            const int hh = e / per_half, r = e % per_half;
            *reinterpret_cast<uint4 *>(vt + hh * S::kHalfTileBytes + z0 * 128 + r * 16) =
                make_uint4(0u, 0u, 0u, 0u);
          }
          fence_proxy_async_smem();
          __syncwarp();
        }
        if (!warp_wait(&p_full[q], (uint32_t)i & 1u, abort_flag, wait_lim)) {
          ok = false;
          break;
        }
        if (lane == 0) {
          tc_fence_after();
          const uint32_t vt = smem_u32(smem + S::kOffV + vs * S::kKVBytes);
#pragma unroll
          for (int k = 0; k < S::kTile / 16; ++k) {
            const uint64_t bv = smem_desc_sw128(vt + k * 2048, S::kHalfTileBytes, 1024);
            tc_mma_tmem_a(tmem + S::kOffO + q * D, tmem + S::kOffP + q * (S::kTile / 2) + k * 8,
                          bv, id_o, i > 0 || k > 0);
          }
          tc_commit(&pv_done[q]);
          tc_commit(&v_empty[vs]);
          if (t >= other) tc_commit(&v_empty[vs]);
        }
        __syncwarp();
      }
    }
    if (!ok && lane == 0 && !*abort_flag) {
      record_error(v.err, HAM_DEVERR_TIMEOUT);
      *abort_flag = 1;
    }
    // every MMA issued completes before the tensor memory is freed
    if (lane == 0) {
      tc_commit(mma_done);
      thread_wait(mma_done, 0u, abort_flag, false);
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------ softmax groups
    // Thread = TMEM lane = row m of Q tile q.  Each row's scores arrive whole in its own thread,
    // so the row maximum and sum need no shuffles.
    const int q = warp >> 2, m = tid & 127;
    const uint32_t lane_base = (uint32_t)((warp & 3) * 32) << 16;
    const uint32_t t_s = tmem + lane_base + q * S::kTile;
    const uint32_t t_p = tmem + lane_base + S::kOffP + q * (S::kTile / 2);
    const uint32_t t_o = tmem + lane_base + S::kOffO + q * D;
    const int j = qb0 + q * R + m / G;          // the row's index in the sequence's chunk
    const int lim = L + min(j, n - 1);          // last slot it attends (rows past n: not stored)
    const int lim_min = L + qb0 + q * R;        // smallest limit of the tile's stored rows
    const float sl2 = (float)(1.4426950408889634 / sqrt((double)D));  // 1/sqrt(d), log2(e)
    float m_run = -INFINITY, l_run = 0.f;
    bool ok = true;
    for (int i = 0; i < ntq[q]; ++i) {
      const int t = t0 + i;
      if (!warp_wait(&s_full[q], (uint32_t)i & 1u, abort_flag, wait_lim)) {
        ok = false;
        break;
      }
      tc_fence_after();
      float s[S::kTile];
#pragma unroll
      for (int c0 = 0; c0 < S::kTile; c0 += 32) {
        uint32_t r[32];
        tmem_ld32(t_s + c0, r);
#pragma unroll
        for (int c = 0; c < 32; ++c) s[c0 + c] = __uint_as_float(r[c]);
      }
      tmem_wait_ld();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&s_free[q]);  // the next scores may overwrite S_q
      const int tbase = t * S::kTile;
      if (tbase + S::kTile - 1 > lim_min) {  // the causal edge (and the chunk's end) in this tile
#pragma unroll
        for (int c = 0; c < S::kTile; ++c)
          if (tbase + c > lim) s[c] = -INFINITY;
      }
      float mx;
      {  // tree maximum
        float r[16];
#pragma unroll
        for (int c = 0; c < 16; ++c)
          r[c] = fmaxf(fmaxf(s[c], s[c + 16]), fmaxf(s[c + 32], s[c + 48]));
#pragma unroll
        for (int w = 8; w > 0; w >>= 1)
#pragma unroll
          for (int c = 0; c < w; ++c) r[c] = fmaxf(r[c], r[c + w]);
        mx = r[0] * sl2;
      }
      // Running maximum in the exp2 domain, raised lazily: only when a score passes it by more
      // than kRescaleSlack (p then stays below 2^kRescaleSlack), so O is rarely rescaled.  The
      // split's first tile always raises it (its first slot is attended by every row).
      float alpha = 1.f;
      if (mx > m_run + kRescaleSlack) {
        alpha = ex2(m_run - mx);
        m_run = mx;
      }
      uint32_t pk[S::kTile / 2];
      float rs0 = 0.f, rs1 = 0.f, rs2 = 0.f, rs3 = 0.f;
#pragma unroll
      for (int c = 0; c < S::kTile; c += 4) {
        const float p0 = ex2(fmaf(s[c], sl2, -m_run));
        const float p1 = ex2(fmaf(s[c + 1], sl2, -m_run));
        const float p2 = ex2(fmaf(s[c + 2], sl2, -m_run));
        const float p3 = ex2(fmaf(s[c + 3], sl2, -m_run));
        rs0 += p0;
        rs1 += p1;
        rs2 += p2;
        rs3 += p3;
        pk[c / 2] = pack_bf16x2(p0, p1);
        pk[c / 2 + 1] = pack_bf16x2(p2, p3);
      }
      l_run = l_run * alpha + ((rs0 + rs1) + (rs2 + rs3));
      // O_q and P_q are free once the previous product has completed
      if (i > 0) {
        if (!warp_wait(&pv_done[q], (uint32_t)(i - 1) & 1u, abort_flag, wait_lim)) {
          ok = false;
          break;
        }
        tc_fence_after();
        if (__any_sync(kFull, alpha != 1.f)) {  // rescale O (some row of the warp raised its max)
#pragma unroll
          for (int c0 = 0; c0 < D; c0 += 32) {
            uint32_t o[32];
            tmem_ld32(t_o + c0, o);
            tmem_wait_ld();
#pragma unroll
            for (int e = 0; e < 32; ++e) o[e] = __float_as_uint(__uint_as_float(o[e]) * alpha);
            tmem_st32(t_o + c0, o);
          }
        }
      }
      tmem_st32(t_p, pk);  // P_q: the tile's 64 probabilities as 32 bf16 pairs
      tmem_wait_st();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&p_full[q]);
    }
    if (ok && ntq[q] > 0) {
      if (!warp_wait(&pv_done[q], (uint32_t)(ntq[q] - 1) & 1u, abort_flag, wait_lim)) {
        ok = false;
      } else {
        tc_fence_after();
        const int64_t rh = (row0 + j) * Hq + g * G + m % G;  // (row, head) of the call
        if (zs == 1) {  // the whole row: normalised output
          const float inv = l_run > 0.f ? 1.f / l_run : 0.f;
          OutT *orow = static_cast<OutT *>(v.out) + rh * (int64_t)D;
#pragma unroll
          for (int c0 = 0; c0 < D; c0 += 32) {
            uint32_t o[32];
            tmem_ld32(t_o + c0, o);
            tmem_wait_ld();
            if (j < n) store_row32<OutT>(orow + c0, o, inv);
          }
        } else {  // this split's partial: O in units of 2^m_run, the running max and sum
          const int64_t pr = (int64_t)z * v.rows * Hq + rh;
          float *prow = v.part_o + pr * D;
#pragma unroll
          for (int c0 = 0; c0 < D; c0 += 32) {
            uint32_t o[32];
            tmem_ld32(t_o + c0, o);
            tmem_wait_ld();
            if (j < n) store_row32<float>(prow + c0, o, 1.f);
          }
          if (j < n) v.part_ml[pr] = make_float2(m_run, l_run);
        }
      }
    }
    if (!ok && lane == 0 && !*abort_flag) {
      record_error(v.err, HAM_DEVERR_TIMEOUT);
      *abort_flag = 1;
    }
  }
  // all tensor-memory reads and MMAs are done: free the columns
  tc_fence_before();
  __syncthreads();
  if (warp == S::kSWarp0) {
    tc_fence_after();
    tmem_dealloc<S::kTmemCols>(tmem);
  }
}

// ------------------------------------------------------------------------------------
// 4. merge of the split partials (only when the attention grid has splits)
// ------------------------------------------------------------------------------------
// out = sum_z 2^(m_z - M) O_z / sum_z 2^(m_z - M) l_z over the splits z of the row's sequence, in
// split order (M = max_z m_z; the split-softmax merge of the decode combine).  One warp per
// (row, head), D / 32 elements a lane; rows of sequences that were not split (written by the
// attention itself) or that the plan refused are left alone.
constexpr int kMergeWarps = 8;
template <typename OutT>
__global__ void __launch_bounds__(kMergeWarps * 32) prefill_merge_kernel(const PrefillView v) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int Hq = v.n_q_heads, D = v.head_dim;
  const int64_t rh = (int64_t)blockIdx.x * kMergeWarps + warp;  // (row, head)
  if (rh >= (int64_t)v.rows * Hq) return;
  const int r = (int)(rh / Hq);
  int lo = 0, hi = v.batch - 1;  // the row's sequence: the last b with offsets[b] <= r
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (v.offsets[mid] <= r) lo = mid; else hi = mid - 1;
  }
  const int4 si = v.seq_info[lo];
  if (si.x < 0) return;
  const int zs = prefill_splits(si.x, v.splits);
  if (zs <= 1) return;
  const int64_t zstride = (int64_t)v.rows * Hq;
  float M = -INFINITY;
  for (int z = 0; z < zs; ++z) M = fmaxf(M, v.part_ml[z * zstride + rh].x);
  const int per = D / 32;  // 4 or 2
  float num[4] = {0.f, 0.f, 0.f, 0.f}, den = 0.f;
  for (int z = 0; z < zs; ++z) {
    const float2 ml = v.part_ml[z * zstride + rh];
    const float w = ml.x == -INFINITY ? 0.f : ex2(ml.x - M);
    den += w * ml.y;
    const float *po = v.part_o + (z * zstride + rh) * D + lane * per;
    for (int e = 0; e < per; ++e) num[e] += w * po[e];
  }
  const float inv = den > 0.f ? 1.f / den : 0.f;
  OutT *dst = static_cast<OutT *>(v.out) + rh * D + lane * per;
  for (int e = 0; e < per; ++e) {
    if constexpr (std::is_same<OutT, float>::value)
      dst[e] = num[e] * inv;
    else
      dst[e] = __float2bfloat16_rn(num[e] * inv);
  }
}

template <int D, typename OutT>
cudaError_t launch_attn(const CUtensorMap &tq, const CUtensorMap &tk, const CUtensorMap &tv,
                        const PrefillView &v, cudaStream_t stream) {
  using S = TcShape<D>;
  cudaError_t e = cudaFuncSetAttribute(prefill_attn_kernel<D, OutT>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, S::kSmem);
  if (e != cudaSuccess) return e;
  const int QB = prefill_query_rows(v.n_q_heads / v.n_kv_heads);
  const int Z = v.splits < 1 ? 1 : v.splits;
  const dim3 grid((unsigned)v.n_kv_heads, (unsigned)(v.rows / QB + v.batch), (unsigned)Z);
  prefill_attn_kernel<D, OutT><<<grid, S::kThreads, S::kSmem, stream>>>(tq, tk, tv, v);
  e = cudaGetLastError();
  if (e != cudaSuccess || Z == 1) return e;
  const int64_t pairs = (int64_t)v.rows * v.n_q_heads;
  prefill_merge_kernel<OutT><<<(unsigned)((pairs + kMergeWarps - 1) / kMergeWarps),
                               kMergeWarps * 32, 0, stream>>>(v);
  return cudaGetLastError();
}

template <typename OutT>
cudaError_t launch_all(const CUtensorMap &tk, const CUtensorMap &tv, const PrefillView &v,
                       cudaStream_t stream) {
  const int G = v.n_q_heads / v.n_kv_heads;
  CUtensorMap tq;  // the chunk's queries, rotated in place by the RoPE kernel
  if (make_rows_tensor_map(&tq, v.q, v.rows, v.n_q_heads, v.head_dim, G, 128 / G) != 0)
    return cudaErrorInvalidValue;
  prefill_plan_kernel<<<(unsigned)v.batch, kPlanThreads, 0, stream>>>(v, prefill_query_rows(G));
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  if (v.head_dim == 128)
    prefill_rope_kernel<128, OutT><<<(unsigned)v.rows, kRopeThreads, 0, stream>>>(v);
  else
    prefill_rope_kernel<64, OutT><<<(unsigned)v.rows, kRopeThreads, 0, stream>>>(v);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  return v.head_dim == 128 ? launch_attn<128, OutT>(tq, tk, tv, v, stream)
                           : launch_attn<64, OutT>(tq, tk, tv, v, stream);
}

}  // namespace

bool prefill_supported(int head_dim, int group) {
  return (head_dim == 64 || head_dim == 128) &&
         (group == 1 || group == 2 || group == 4 || group == 8);
}

// Two Q tiles of 128 (row, head) pairs per CTA.
int prefill_query_rows(int group) { return 256 / group; }

cudaError_t launch_prefill(const CUtensorMap &tk, const CUtensorMap &tv, const PrefillView &v,
                           int out_dtype, cudaStream_t stream) {
  return out_dtype == HAM_DTYPE_F32 ? launch_all<float>(tk, tv, v, stream)
                                    : launch_all<__nv_bfloat16>(tk, tv, v, stream);
}

}  // namespace ham
