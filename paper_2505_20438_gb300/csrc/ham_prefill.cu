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
// Three launches:
//  1. prefill_plan_kernel, one block per sequence: checks that the sequence's rows fit
//     (counts, capacity, pages), gives each row its position (slot index, running token count
//     or the caller's), numbers the query blocks, and advances the counters.
//  2. prefill_rope_kernel, one block per row: turns q and k at the row's position and stores
//     k and v into the row's slot.  The rotation x0 c - x1 s is evaluated from the fp64 cos/sin
//     table in pairs of fp32 values (error-free products and sums, about 48 bits) and rounded
//     once to bf16, which gives the bits of the fp64 evaluation except when the exact value
//     lies within ~2^-44 (relative) of a rounding boundary.  This GPU's fp64 pipe would take
//     about half a millisecond for a 16k-row chunk of a Llama-8B layer; the fp32 pairs take
//     microseconds.
//  3. prefill_attn_kernel, one CTA per (KV head, block of 128 / G query rows of one sequence):
//     eight consumer warps, each one 16-row m-tile of one query head, and a producer warp that
//     streams 64-slot K/V tiles (four 16-slot chunks, each 64-column half of a chunk one TMA
//     copy with the 128-byte swizzle, so that ldmatrix reads are free of bank conflicts)
//     through a shared-memory ring.  S = Q K^T and O += P V are mma.sync m16n8k16 (bf16 in, fp32
//     accumulate); the softmax is online, fp32, in the exp2 domain; the causal mask applies to
//     the tiles that reach past a row's own slot, and tiles past a warp's last row are skipped.
//     CTAs are scheduled latest query block first, the longest rows of the causal triangle.
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
  if (err) {
    if (tid == 0) {
      record_error(v.err, err);
      v.seq_info[b] = make_int4(-1, n, qb, 0);
    }
    return;
  }
  // positions: the caller's, the slot index, or the tokens before the row
  const int64_t t0 = v.num_tokens[b];
  int64_t carry = 0;
  for (int j0 = 0; j0 < n; j0 += kPlanThreads) {
    const int j = j0 + tid;
    const int t = j < n ? (v.ntok ? v.ntok[a + j] : 1) : 0;
    int total = 0;
    const int excl = block_scan(t, red, &total) - t;
    if (j < n) {
      int64_t p;
      if (v.pos) p = v.pos[a + j];
      else if (v.pos_mode == HAM_POS_SLOT) p = (int64_t)L + j;
      else p = t0 + carry + excl;
      v.row_pos[a + j] = (int32_t)p;
    }
    carry += total;
  }
  if (tid == 0) {
    v.seq_info[b] = make_int4(L, n, qb, 0);
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

// a c - b s rounded once to bf16, with c = ch + cl and s = sh + sl given as fp32 pairs and a, b
// exact (bf16 values).  Near a rounding boundary: products by FMA error terms and sums by
// two-sum are exact, only the small terms are rounded, so the pair carries about 48 bits of
// the exact value.
__device__ __forceinline__ uint16_t rotate_dd(float a, float b, float ch, float cl, float sh,
                                              float sl) {
  // Fast path: y = a ch - b sh in plain fp32 lies within 3 * 2^-24 (|a| + |b|) < e / 2 of the
  // exact a c - b s.  When no bf16 rounding boundary is within e of y (the nearest one is the
  // midpoint sharing y's upper 16 bits; the others are a quarter of a bf16 spacing away, more
  // than e once e < 2^-11 |y|), the exact value rounds as y does.
  const float y = __fmaf_rn(a, ch, -__fmul_rn(b, sh));
  const float e = __fmul_rn(__fadd_rn(fabsf(a), fabsf(b)), 0x1p-21f);
  const float mid = __uint_as_float((__float_as_uint(y) & 0xFFFF0000u) | 0x8000u);
  if (fabsf(__fsub_rn(y, mid)) > e && e < __fmul_rn(fabsf(y), 0x1p-11f))
    return __bfloat16_as_ushort(__float2bfloat16_rn(y));
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

// One block per row; a thread owns four consecutive pairs (i, i + d/2), i = 4 (tid % (d/8)) ..,
// of one head at a time (8-byte loads and stores of each half).
template <typename OutT>
__global__ void __launch_bounds__(kRopeThreads) prefill_rope_kernel(PrefillView v) {
  const int64_t r = blockIdx.x;
  const int D = v.head_dim, half = D / 2, Hq = v.n_q_heads, Hkv = v.n_kv_heads;
  int lo = 0, hi = v.batch - 1;  // the sequence of row r
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (v.offsets[mid] <= r) lo = mid; else hi = mid - 1;
  }
  const int b = lo;
  const int4 si = v.seq_info[b];
  const int a = v.offsets[b];
  if (si.x < 0 || r < a || r >= (int64_t)a + si.y) {  // not stored: its output rows are 0
    OutT *o = static_cast<OutT *>(v.out) + r * Hq * D;
    for (int e = threadIdx.x; e < Hq * D; e += kRopeThreads) o[e] = OutT(0.f);
    return;
  }
  const int slot = si.x + (int)(r - a);
  const int p = v.row_pos[r];
  const int64_t page = v.page_table[(int64_t)b * v.max_pages + slot / v.page_slots];
  const int prow = slot % v.page_slots;
  if (threadIdx.x == 0) {
    v.slot_pos[page * v.page_slots + prow] = p;
    v.slot_ntok[page * v.page_slots + prow] = v.ntok ? v.ntok[r] : 1;
  }
  for (int e = threadIdx.x; e < Hkv * D / 8; e += kRopeThreads) {  // values: bit copy
    const int gg = e / (D / 8), k = e % (D / 8);
    reinterpret_cast<uint4 *>(v.v_pool + ((page * Hkv + gg) * v.page_slots + prow) * D)[k] =
        reinterpret_cast<const uint4 *>(v.v_new + (r * Hkv + gg) * D)[k];
  }
  const int quads = half / 4, i0 = 4 * (threadIdx.x % quads);
  float4 cs[4];  // (c_hi, c_lo, s_hi, s_lo) of frequencies i0 .. i0 + 3
  if (p >= 0 && p < v.rope_positions) {
#pragma unroll
    for (int e = 0; e < 4; ++e) cs[e] = v.rope_table_ff[(int64_t)p * half + i0 + e];
  } else {
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      double c, sn;
      sincos((double)p * v.inv_freq[i0 + e], &sn, &c);
      split_double(c, cs[e].x, cs[e].y);
      split_double(sn, cs[e].z, cs[e].w);
    }
  }
  // query heads in place, then the key heads into the slot
  for (int hh = threadIdx.x / quads; hh < Hq + Hkv; hh += kRopeThreads / quads) {
    const uint16_t *src;
    uint16_t *dst;
    if (hh < Hq) {
      src = dst = v.q + (r * Hq + hh) * D;
    } else {
      const int gg = hh - Hq;
      src = v.k_new + (r * Hkv + gg) * D;
      dst = v.k_pool + ((page * Hkv + gg) * v.page_slots + prow) * D;
    }
    const uint2 xl = *reinterpret_cast<const uint2 *>(src + i0);
    const uint2 xh = *reinterpret_cast<const uint2 *>(src + i0 + half);
    const uint32_t wl[2] = {xl.x, xl.y}, wh[2] = {xh.x, xh.y};
    uint32_t yl[2], yh[2];
#pragma unroll
    for (int k = 0; k < 2; ++k) {
      uint32_t ol = 0, oh = 0;
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        const float4 c4 = cs[2 * k + e];
        const float x0 = bf16_value((uint16_t)(wl[k] >> (16 * e)));
        const float x1 = bf16_value((uint16_t)(wh[k] >> (16 * e)));
        ol |= (uint32_t)rotate_dd(x0, x1, c4.x, c4.y, c4.z, c4.w) << (16 * e);   // x0 c - x1 s
        oh |= (uint32_t)rotate_dd(x1, x0, c4.x, c4.y, -c4.z, -c4.w) << (16 * e); // x1 c + x0 s
      }
      yl[k] = ol;
      yh[k] = oh;
    }
    *reinterpret_cast<uint2 *>(dst + i0) = make_uint2(yl[0], yl[1]);
    *reinterpret_cast<uint2 *>(dst + i0 + half) = make_uint2(yh[0], yh[1]);
  }
}

// ------------------------------------------------------------------------------------
// 3. causal attention of the chunk
// ------------------------------------------------------------------------------------
template <int D>
struct PShape {
  static constexpr int kWarps = 8;                         // consumer warps, one m-tile each
  static constexpr int kThreads = (kWarps + 1) * 32;       // and the producer warp
  static constexpr int kRows = kWarps * 16;                // (query row, head) pairs per CTA
  static constexpr int kTile = 64;                         // slots per K/V tile
  static constexpr int kChunks = kTile / kChunkSlots;      // 16-slot TMA chunks per tile
  static constexpr int kChunkBytes = kChunkSlots * D * 2;
  static constexpr int kStageBytes = 2 * kChunks * kChunkBytes;  // K chunks, then V chunks
  static constexpr int kStages = 98304 / kStageBytes;      // 96 KiB ring: 3 (d 128), 6 (d 64)
  static constexpr int kKSteps = D / 16;                   // k-steps of q.k
  static constexpr int kONBlocks = D / 8;                  // n-blocks of o
  static constexpr int kOffBar = kStages * kStageBytes;    // from a 1024-byte aligned base
  static constexpr int kSmem = 1024 + kOffBar + 2 * kStages * 8 + kStages * 4 + 16;
  static_assert(D == 64 || D == 128, "head_dim 64 or 128");
  static_assert(kStages >= 2, "ring depth");
};

// A chunk tile in shared memory: its 64-column halves one after the other, each 16 slot rows
// of 128 bytes written by its own TMA copy with the 128-byte swizzle.  Byte offset of the
// 16-byte piece c (elements 8c .. 8c+7) of slot row `row`: the piece index inside the line is
// XORed with the row, so the eight rows of an ldmatrix matrix hit eight different bank groups.
constexpr int kHalfBytes = kChunkSlots * 128;
__device__ __forceinline__ uint32_t half_tile_offset(int row, int c) {
  return (uint32_t)((c >> 3) * kHalfBytes + row * 128 + (((c & 7) ^ (row & 7)) << 4));
}

template <typename OutT>
__device__ __forceinline__ void store_pair(void *out, int64_t i, float x, float y) {
  if constexpr (std::is_same<OutT, float>::value) {
    *reinterpret_cast<float2 *>(static_cast<float *>(out) + i) = make_float2(x, y);
  } else {
    *reinterpret_cast<uint32_t *>(static_cast<__nv_bfloat16 *>(out) + i) = pack_bf16x2(x, y);
  }
}

// One CTA per SM.  Registers are granted to a block in groups of four warps, so the nine warps
// (twelve as allocated) may use at most 170 registers a thread: 168, with a few bytes spilled
// at head_dim 128.
template <int D, typename OutT>
__global__ void __launch_bounds__(PShape<D>::kThreads, 1)
    prefill_attn_kernel(const __grid_constant__ CUtensorMap tmap_k,
                        const __grid_constant__ CUtensorMap tmap_v, const PrefillView v) {
  using S = PShape<D>;
  const int Hq = v.n_q_heads, Hkv = v.n_kv_heads, G = Hq / Hkv, QB = S::kRows / G;
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
  const int kv_end = L + min(qb0 + QB, n);  // the CTA's rows attend over slots 0 .. kv_end-1
  const int ntiles = (kv_end + S::kTile - 1) / S::kTile;
  const int64_t row0 = v.offsets[b];

  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = reinterpret_cast<uint8_t *>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t *full = reinterpret_cast<uint64_t *>(smem + S::kOffBar);
  uint64_t *empty = full + S::kStages;
  int *chunk_ok = reinterpret_cast<int *>(empty + S::kStages);  // bit c: chunk c was copied
  volatile int *abort_flag = chunk_ok + S::kStages;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  if (tid == 0) {
    for (int s = 0; s < S::kStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], S::kWarps);
    }
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (tid == S::kWarps * 32) {
    prefetch_tensormap(&tmap_k);
    prefetch_tensormap(&tmap_v);
  }
  __syncthreads();

  // ring and data waits: the launch's limit; the final drain of in-flight copies keeps 2 s
  const uint64_t wait_lim = data_wait_limit(v.wait_ns);
  if (warp == S::kWarps) {
    // Producer: one lane streams the tiles.  A chunk past the last attended slot or on a page
    // outside the pool is not copied (its bit stays clear and the consumers mask it).
    if (lane != 0) return;
    const uint64_t pol = policy_evict_last();  // every query block of the sequence reads them
    int issued = 0;
    for (int t = 0; t < ntiles; ++t) {
      const int s = t % S::kStages;
      if (t >= S::kStages &&
          !thread_wait(&empty[s], (uint32_t)((t / S::kStages) - 1) & 1u, abort_flag, true,
                       wait_lim)) {
        if (!*abort_flag) {
          record_error(v.err, HAM_DEVERR_TIMEOUT);
          *abort_flag = 1;
        }
        break;
      }
      int mask = 0, rows[S::kChunks];
#pragma unroll
      for (int c = 0; c < S::kChunks; ++c) {
        const int slot0 = t * S::kTile + c * kChunkSlots;
        rows[c] = 0;
        if (slot0 >= kv_end) continue;
        const int page = v.page_table[(int64_t)b * v.max_pages + slot0 / v.page_slots];
        if (page < 0 || page >= v.pool_pages) {
          record_error(v.err, HAM_DEVERR_PAGE);
          continue;
        }
        rows[c] = (page * Hkv + g) * v.page_slots + slot0 % v.page_slots;
        mask |= 1 << c;
      }
      chunk_ok[s] = mask;
      mbar_arrive_tx(&full[s], (uint32_t)(__popc(mask) * 2 * S::kChunkBytes));
      uint8_t *dst = smem + s * S::kStageBytes;
#pragma unroll
      for (int c = 0; c < S::kChunks; ++c) {
        if (!(mask & (1 << c))) continue;
#pragma unroll
        for (int hh = 0; hh < D / 64; ++hh) {  // one 64-column half of the chunk per copy
          tma_load_3d(dst + c * S::kChunkBytes + hh * kHalfBytes, &tmap_k, 0, hh, rows[c],
                      &full[s], pol);
          tma_load_3d(dst + (S::kChunks + c) * S::kChunkBytes + hh * kHalfBytes, &tmap_v, 0, hh,
                      rows[c], &full[s], pol);
        }
      }
      issued = t + 1;
    }
    // copies still in flight land before the CTA exits
    for (int t = max(0, issued - S::kStages); t < issued; ++t)
      thread_wait(&full[t % S::kStages], (uint32_t)(t / S::kStages) & 1u, abort_flag, false);
    return;
  }

  // Consumer warp: the m-tile of query head h = g G + (warp % G), sequence-local rows
  // j0 .. j0 + 15.  Lane rows ra = j0 + lane / 4 and rb = ra + 8.
  const int h = g * G + warp % G;
  const int j0 = qb0 + (warp / G) * 16;
  const int ra = j0 + (lane >> 2), rb = ra + 8;
  const int warp_end = j0 < n ? L + min(j0 + 15, n - 1) + 1 : 0;  // slots < warp_end
  const int lim_a = min(L + ra, warp_end - 1), lim_b = min(L + rb, warp_end - 1);
  uint32_t qf[S::kKSteps][4];  // A operand: rows ra / rb, k-columns 2 (lane % 4) (+ 8)
  {
    const int c0 = 2 * (lane & 3);
    const uint32_t *qa = reinterpret_cast<const uint32_t *>(v.q + ((row0 + ra) * Hq + h) * D);
    const uint32_t *qb = reinterpret_cast<const uint32_t *>(v.q + ((row0 + rb) * Hq + h) * D);
#pragma unroll
    for (int ks = 0; ks < S::kKSteps; ++ks) {
      qf[ks][0] = ra < n ? qa[(ks * 16 + c0) / 2] : 0u;
      qf[ks][1] = rb < n ? qb[(ks * 16 + c0) / 2] : 0u;
      qf[ks][2] = ra < n ? qa[(ks * 16 + c0 + 8) / 2] : 0u;
      qf[ks][3] = rb < n ? qb[(ks * 16 + c0 + 8) / 2] : 0u;
    }
  }
  // softmax scale and log2(e): scores in the exp2 domain
  const float sl2 = (float)(1.4426950408889634 / sqrt((double)D));
  float o[S::kONBlocks][4];
#pragma unroll
  for (int on = 0; on < S::kONBlocks; ++on) o[on][0] = o[on][1] = o[on][2] = o[on][3] = 0.f;
  float m_a = -INFINITY, m_b = -INFINITY, l_a = 0.f, l_b = 0.f;
  const int mi = lane >> 3, mr = lane & 7;  // ldmatrix: this lane's matrix and row
  bool ok = true;
  for (int t = 0; t < ntiles; ++t) {
    const int s = t % S::kStages;
    if (!warp_wait(&full[s], (uint32_t)(t / S::kStages) & 1u, abort_flag, wait_lim)) {
      if (lane == 0 && !*abort_flag) {
        record_error(v.err, HAM_DEVERR_TIMEOUT);
        *abort_flag = 1;
      }
      ok = false;
      break;
    }
    const int tbase = t * S::kTile;
    if (tbase < warp_end) {
      const int mask = chunk_ok[s];
      const uint8_t *kt = smem + s * S::kStageBytes;
      const uint8_t *vt = kt + S::kChunks * S::kChunkBytes;
      float sc[2 * S::kChunks][4];
#pragma unroll
      for (int nb = 0; nb < 2 * S::kChunks; ++nb) sc[nb][0] = sc[nb][1] = sc[nb][2] = sc[nb][3] = 0.f;
      // S = Q K^T: per chunk, ldmatrix matrices (slots 0-7 | 8-15) x (d lo | hi) give the
      // B fragments of the chunk's two 8-slot n-blocks.  k-steps outside, chunks inside: the
      // eight accumulators take turns instead of chaining on one.
#pragma unroll
      for (int ks = 0; ks < S::kKSteps; ++ks) {
#pragma unroll
        for (int c = 0; c < S::kChunks; ++c) {
          if (tbase + c * kChunkSlots >= warp_end) continue;
          uint32_t kf[4];
          ldmatrix_x4(kf, smem_u32(kt + c * S::kChunkBytes +
                                   half_tile_offset((mi >> 1) * 8 + mr, 2 * ks + (mi & 1))));
          mma_16816(sc[2 * c], qf[ks], kf[0], kf[1]);
          mma_16816(sc[2 * c + 1], qf[ks], kf[2], kf[3]);
        }
      }
      // causal mask and copied chunks (only on tiles that reach past the m-tile's first row or
      // miss a chunk); row maxima of the raw scores over the quad
      if (tbase + S::kTile - 1 > L + j0 || mask != (1 << S::kChunks) - 1) {
#pragma unroll
        for (int nb = 0; nb < 2 * S::kChunks; ++nb) {
          const bool cok = (mask >> (nb >> 1)) & 1;
          const int slot = tbase + nb * 8 + 2 * (lane & 3);
          if (!(cok && slot <= lim_a)) sc[nb][0] = -INFINITY;
          if (!(cok && slot + 1 <= lim_a)) sc[nb][1] = -INFINITY;
          if (!(cok && slot <= lim_b)) sc[nb][2] = -INFINITY;
          if (!(cok && slot + 1 <= lim_b)) sc[nb][3] = -INFINITY;
        }
      }
      float mx_a = -INFINITY, mx_b = -INFINITY;
#pragma unroll
      for (int nb = 0; nb < 2 * S::kChunks; ++nb) {
        mx_a = fmaxf(mx_a, fmaxf(sc[nb][0], sc[nb][1]));
        mx_b = fmaxf(mx_b, fmaxf(sc[nb][2], sc[nb][3]));
      }
#pragma unroll
      for (int off = 1; off < 4; off <<= 1) {
        mx_a = fmaxf(mx_a, __shfl_xor_sync(kFull, mx_a, off));
        mx_b = fmaxf(mx_b, __shfl_xor_sync(kFull, mx_b, off));
      }
      // Running maxima in the exp2 domain, raised lazily: only when a score passes them by more
      // than kRescaleSlack (p then stays below 2^kRescaleSlack), so most tiles skip rescaling O.
      mx_a *= sl2;
      mx_b *= sl2;
      float al_a = 1.f, al_b = 1.f;
      if (mx_a > m_a + kRescaleSlack) {
        al_a = ex2(m_a - mx_a);
        m_a = mx_a;
      }
      if (mx_b > m_b + kRescaleSlack) {
        al_b = ex2(m_b - mx_b);
        m_b = mx_b;
      }
      const float ref_a = m_a == -INFINITY ? 0.f : m_a;  // nothing attended yet
      const float ref_b = m_b == -INFINITY ? 0.f : m_b;
      float rs_a = 0.f, rs_b = 0.f;
#pragma unroll
      for (int nb = 0; nb < 2 * S::kChunks; ++nb) {
        sc[nb][0] = ex2(fmaf(sc[nb][0], sl2, -ref_a));
        sc[nb][1] = ex2(fmaf(sc[nb][1], sl2, -ref_a));
        sc[nb][2] = ex2(fmaf(sc[nb][2], sl2, -ref_b));
        sc[nb][3] = ex2(fmaf(sc[nb][3], sl2, -ref_b));
        rs_a += sc[nb][0] + sc[nb][1];
        rs_b += sc[nb][2] + sc[nb][3];
      }
      l_a = l_a * al_a + rs_a;  // per-lane partial sums, reduced over the quad at the end
      l_b = l_b * al_b + rs_b;
      if (__any_sync(kFull, al_a != 1.f || al_b != 1.f)) {
#pragma unroll
        for (int on = 0; on < S::kONBlocks; ++on) {
          o[on][0] *= al_a;
          o[on][1] *= al_a;
          o[on][2] *= al_b;
          o[on][3] *= al_b;
        }
      }
      // O += P V: P of chunk kk is the A fragment of k-step kk; V by transposing ldmatrix
      // (matrices (slots 0-7 | 8-15) x (d lo | hi))
#pragma unroll
      for (int kk = 0; kk < S::kChunks; ++kk) {
        if (tbase + kk * kChunkSlots >= warp_end || !((mask >> kk) & 1)) continue;
        const uint32_t pa[4] = {pack_bf16x2(sc[2 * kk][0], sc[2 * kk][1]),
                                pack_bf16x2(sc[2 * kk][2], sc[2 * kk][3]),
                                pack_bf16x2(sc[2 * kk + 1][0], sc[2 * kk + 1][1]),
                                pack_bf16x2(sc[2 * kk + 1][2], sc[2 * kk + 1][3])};
        const uint8_t *vc = vt + kk * S::kChunkBytes;
#pragma unroll
        for (int np = 0; np < D / 16; ++np) {
          uint32_t vf[4];
          ldmatrix_x4_trans(vf, smem_u32(vc + half_tile_offset((mi & 1) * 8 + mr,
                                                               2 * np + (mi >> 1))));
          mma_16816(o[2 * np], pa, vf[0], vf[1]);
          mma_16816(o[2 * np + 1], pa, vf[2], vf[3]);
        }
      }
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(&empty[s]);
  }
  if (!ok) return;
#pragma unroll
  for (int off = 1; off < 4; off <<= 1) {
    l_a += __shfl_xor_sync(kFull, l_a, off);
    l_b += __shfl_xor_sync(kFull, l_b, off);
  }
  const float inv_a = l_a > 0.f ? 1.f / l_a : 0.f, inv_b = l_b > 0.f ? 1.f / l_b : 0.f;
  const int64_t oa = ((row0 + ra) * Hq + h) * D, ob = ((row0 + rb) * Hq + h) * D;
#pragma unroll
  for (int on = 0; on < S::kONBlocks; ++on) {
    const int d = on * 8 + 2 * (lane & 3);
    if (ra < n) store_pair<OutT>(v.out, oa + d, o[on][0] * inv_a, o[on][1] * inv_a);
    if (rb < n) store_pair<OutT>(v.out, ob + d, o[on][2] * inv_b, o[on][3] * inv_b);
  }
}

template <int D, typename OutT>
cudaError_t launch_attn(const CUtensorMap &tk, const CUtensorMap &tv, const PrefillView &v,
                        cudaStream_t stream) {
  using S = PShape<D>;
  cudaError_t e = cudaFuncSetAttribute(prefill_attn_kernel<D, OutT>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, S::kSmem);
  if (e != cudaSuccess) return e;
  const int QB = S::kRows / (v.n_q_heads / v.n_kv_heads);
  const dim3 grid((unsigned)v.n_kv_heads, (unsigned)(v.rows / QB + v.batch));
  prefill_attn_kernel<D, OutT><<<grid, S::kThreads, S::kSmem, stream>>>(tk, tv, v);
  return cudaGetLastError();
}

template <typename OutT>
cudaError_t launch_all(const CUtensorMap &tk, const CUtensorMap &tv, const PrefillView &v,
                       cudaStream_t stream) {
  const int QB = PShape<128>::kRows / (v.n_q_heads / v.n_kv_heads);
  prefill_plan_kernel<<<(unsigned)v.batch, kPlanThreads, 0, stream>>>(v, QB);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  prefill_rope_kernel<OutT><<<(unsigned)v.rows, kRopeThreads, 0, stream>>>(v);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  return v.head_dim == 128 ? launch_attn<128, OutT>(tk, tv, v, stream)
                           : launch_attn<64, OutT>(tk, tv, v, stream);
}

}  // namespace

bool prefill_supported(int head_dim, int group) {
  return (head_dim == 64 || head_dim == 128) &&
         (group == 1 || group == 2 || group == 4 || group == 8);
}

int prefill_query_rows(int group) { return PShape<128>::kRows / group; }

cudaError_t launch_prefill(const CUtensorMap &tk, const CUtensorMap &tv, const PrefillView &v,
                           int out_dtype, cudaStream_t stream) {
  return out_dtype == HAM_DTYPE_F32 ? launch_all<float>(tk, tv, v, stream)
                                    : launch_all<__nv_bfloat16>(tk, tv, v, stream);
}

}  // namespace ham
