// Split-KV GQA decode attention over FP8 (e4m3) pools on the tcgen05 tensor cores (sm_103a).
//
// What it computes is what the bf16 pass computes (ham_attn.cu; HAMburger, arXiv 2505.20438,
// Sec. 3.1 and Sec. 3.7: softmax attention of each query head over the slots of its sequence,
// scale 1/sqrt(d), query head h reading KV head h / G), over caches whose rows are e4m3 codes
// with one power-of-two scale each (ham.h, "FP8 (e4m3) pools").  The split plan, the partials
// and the combine kernel are the bf16 pass's; the pass itself is built for 8-bit rows, which
// the tensor cores read as they are:
//
//  * A tile is 128 slots: up to 8 consecutive chunks of one segment (fewer at the end of the
//    segment or of the CTA's range), the M of two tcgen05 products of kind::f8f6f4 (e4m3 x e4m3,
//    fp32 accumulators in tensor memory) that one thread issues:
//      S^T = K Q8^T  (128 slots x N): K as the TMA copy leaves it (128-byte swizzle);
//      O^T = V^T P^T (128 head dims x N): the pool's transposed value rows, whose 16-slot
//            chunks are exactly the no-swizzle operand layout (8 rows of 16 bytes a core
//            matrix), so no code is ever converted by a thread.
//  * The B operands hold each head as three e4m3 pieces (x ~ hi + mid / 2^4 + lo / 2^8, about 12
//    significant bits): N = 16 columns for groups of up to 5 heads, 32 up to 8.  q enters as
//    q 2^-f per head (its largest element in [2^7, 2^8)): bf16 values and the fp32 rotation of
//    the fused step are then held exactly.  The key exponents scale the scores in fp32.  The
//    weights enter as p 2^(e_v - Gv + 7) <= 2^7, Gv being the tile's largest score + e_v of the
//    head (log2): a tile's largest term is 2^7 whatever the rows' scales, and the tile's O^T,
//    read back into fp32 registers (one thread per head dim), is added times 2^(Gv - 7 - m).
//  * Warps 0-3 own TMEM lanes 0-127: slot t of a tile for the scores, head dim t for the
//    output.  They take the scores, the tile's per-head maxima (warp redux, then one bounded
//    mbarrier round among the four warps), the weights and their pieces into shared memory, and
//    the output accumulation.  Warp 4 issues the TMA copies (per chunk a K box, a V box and 32
//    exponent bytes); warp 5 allocates tensor memory and issues the products, S of the next tile
//    while the softmax of this one runs.  S, P and O are double buffered in tensor / shared
//    memory; the ring holds three tiles (two CTAs an SM).
//  * Sequences with no slots attend to nothing (output 0); a chunk whose page id is out of range
//    is skipped and HAM_DEVERR_PAGE recorded, as in the bf16 pass.
//
// Every wait is bounded (the launch's data-wait limit, 2 s by default); a wait that runs out
// records HAM_DEVERR_TIMEOUT, every warp of the CTA gives up, copies and products in flight are
// waited for, tensor memory is freed and the CTA returns.  No trap, no unbounded spin.
#include <cuda.h>
#include <cuda_bf16.h>

#include <algorithm>
#include <climits>
#include <mutex>

#include "ham_attn.cuh"
#include "ham_internal.cuh"
#include "ham_ptx.cuh"

namespace ham {
namespace {

constexpr int kD8 = kFp8HeadDim;                        // 128
constexpr int kTileChunks = 8;
constexpr int kTileSlots = kTileChunks * kChunkSlots;   // 128: the products' M
constexpr int kBox8 = kChunkSlots * kD8;                // a chunk's K (or V) codes: 2 KiB
constexpr int kHalf8 = kTileChunks * kBox8;             // a tile's K (or V) codes: 16 KiB
constexpr int kStage8 = 2 * kHalf8;                     // K, then V
constexpr int kChunkExp = 2 * kChunkSlots;              // a chunk's exponents (16 K, 16 V)
constexpr int kChunkTx = 2 * kBox8 + kChunkExp;         // bytes one chunk's copies bring
constexpr int kStages8 = 3;
constexpr int kSoftWarps = 4, kSoftThreads = 32 * kSoftWarps;
constexpr int kProducerWarp = 4, kIssuerWarp = 5;
constexpr int kThreads8 = 32 * 6;
constexpr int kEnd = 8;                                 // tile flag: the CTA's last tile
constexpr int kPreTiles = 1;  // tiles whose copies `early` issues before the dependency wait
static_assert(kTileSlots == kSoftThreads && kD8 == kSoftThreads, "one TMEM lane per thread");

template <int kCols>
struct Fp8Cfg {
  static constexpr int kMaxG = kCols == 16 ? 5 : 8;     // heads: 3 pieces each in kCols columns
  static constexpr int kOperand = kCols * 128;          // one B operand (Q8 or P), kCols rows
  static constexpr uint32_t kTmemCols = 4 * kCols;      // S x 2, O x 2
  static constexpr int kOffQ8 = kStages8 * kStage8;
  static constexpr int kOffP = kOffQ8 + 2 * kOperand;
  static constexpr int kOffExp = kOffP + 2 * kOperand;
  // per-tile maxima [2][4 warps][2 kMaxG], segment sums [4][kMaxG], q maxima [4][kMaxG]
  static constexpr int kRedTile = kSoftWarps * 2 * kMaxG;
  static constexpr int kOffRed = kOffExp + kStages8 * kTileChunks * kChunkExp;
  static constexpr int kRedFloats = 2 * kRedTile + 2 * kSoftWarps * kMaxG;
  static constexpr int kOffBar = kOffRed + align_up(kRedFloats * 4, 16);
  // full[S], empty[S]; s_full, p_full, o_full, o_free, q8_full [2] each; done; soft
  static constexpr int kBars = 2 * kStages8 + 5 * 2 + 2;
  static constexpr int kOffInfo = kOffBar + align_up(kBars * 8, 16);
  static constexpr int kOffMisc = kOffInfo + kStages8 * 16;  // TMEM base, abort flag
  static constexpr int kOffQ = align_up(kOffMisc + 16, 128);
  // A segment's q buffer is reused three segment openings later, by which time the CTA's
  // products have released the stage of the tile that read it.
  static constexpr int kQBufs = kStages8;
  static_assert(kOffQ8 % 1024 == 0 && kOperand % 1024 == 0, "swizzled operands: 1024 B");
};

// Shared memory after the fixed part: q buffers (bf16 heads, and for the fused step the fp32
// (cos, sin) row of the new slot's position), then cum [B+1], lens [B] and, for the fused step,
// the new slot's position and append flag [B] each.
template <int kCols>
struct Fp8Layout {
  int q_stride, off_cum, total;
  __host__ __device__ Fp8Layout(int group, bool step, int batch) {
    using Cf = Fp8Cfg<kCols>;
    q_stride = align_up(group * kD8 * 2 + (step ? (kD8 / 2) * 8 : 0), 128);
    off_cum = Cf::kOffQ + Cf::kQBufs * q_stride;
    total = off_cum + 4 * (batch + 1) + 4 * batch * (step ? 3 : 1);
  }
};

// Byte (row, k) of an operand tile of 128-byte rows in the 128-byte swizzle (1024-byte aligned).
__device__ __forceinline__ uint32_t sw128_byte(int row, int k) {
  return (uint32_t)(row * 128 + ((((k >> 4) ^ row) & 7) << 4) + (k & 15));
}
__device__ __forceinline__ uint8_t e4m3_code(float x) {
  return (uint8_t)__nv_cvt_float_to_fp8(x, __NV_SATFINITE, __NV_E4M3);
}
__device__ __forceinline__ float e4m3_value(uint8_t c) {
  return __half2float(__half(__nv_cvt_fp8_to_halfraw((__nv_fp8_storage_t)c, __NV_E4M3)));
}
// x (|x| < 2^8) as three e4m3 pieces: x ~ v(c0) + v(c1) 2^-4 + v(c2) 2^-8.  Each residual is
// exact in fp32 and below half a step of the piece before, so each piece adds about 4 bits.
__device__ __forceinline__ void e4m3_pieces(float x, uint8_t &c0, uint8_t &c1, uint8_t &c2) {
  c0 = e4m3_code(x);
  const float r1 = (x - e4m3_value(c0)) * 16.f;
  c1 = e4m3_code(r1);
  const float r2 = (r1 - e4m3_value(c1)) * 16.f;
  c2 = e4m3_code(r2);
}
__device__ __forceinline__ float bf16_value(uint16_t b) { return __uint_as_float((uint32_t)b << 16); }
__device__ __forceinline__ float round_bf16(float x) {
  return __bfloat162float(__float2bfloat16_rn(x));
}
template <int kCols>
__device__ __forceinline__ void tmem_ld_cols(uint32_t taddr, uint32_t (&r)[kCols]) {
  if constexpr (kCols == 16) tmem_ld16(taddr, r);
  else tmem_ld32(taddr, r);
}
// One head's value from its three piece columns of a product.
__device__ __forceinline__ float join_pieces(uint32_t hi, uint32_t mid, uint32_t lo) {
  return __uint_as_float(hi) + __uint_as_float(mid) * 0.0625f + __uint_as_float(lo) * 0.00390625f;
}

template <typename OutT, bool kStep, int kCols>
__global__ void __launch_bounds__(kThreads8, 2)
    decode_attn_fp8_kernel(const __grid_constant__ CUtensorMap tmap_k,
                           const __grid_constant__ CUtensorMap tmap_v, const AttnView v) {
  using Cf = Fp8Cfg<kCols>;
  constexpr int kMaxG = Cf::kMaxG;
  const int B = v.batch, Hkv = v.n_kv_heads, G = v.group;
  const Fp8Layout<kCols> lay(G, kStep, B);
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = reinterpret_cast<uint8_t *>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t *ring = smem;
  uint8_t *q8 = smem + Cf::kOffQ8;  // [2] B operand of S: the heads' q pieces
  uint8_t *pw = smem + Cf::kOffP;   // [2] B operand of O: the weights' pieces
  int8_t *exps = reinterpret_cast<int8_t *>(smem + Cf::kOffExp);
  float *red_tile = reinterpret_cast<float *>(smem + Cf::kOffRed);
  float *red_seg = red_tile + 2 * Cf::kRedTile;
  float *red_q = red_seg + kSoftWarps * kMaxG;
  uint64_t *full = reinterpret_cast<uint64_t *>(smem + Cf::kOffBar);
  uint64_t *empty = full + kStages8;
  uint64_t *s_full = empty + kStages8, *p_full = s_full + 2, *o_full = p_full + 2;
  uint64_t *o_free = o_full + 2, *q8_full = o_free + 2, *done = q8_full + 2, *soft = done + 1;
  int4 *info = reinterpret_cast<int4 *>(smem + Cf::kOffInfo);
  uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(smem + Cf::kOffMisc);
  volatile int *flags = reinterpret_cast<volatile int *>(smem + Cf::kOffMisc + 4);  // abort
  uint8_t *qbufs = smem + Cf::kOffQ;
  int32_t *cum = reinterpret_cast<int32_t *>(smem + lay.off_cum);  // [B+1] chunk prefix
  int32_t *lens = cum + B + 1;                                      // [B] slots attended
  int32_t *posb = lens + B;                                         // [B] new slot position
  int32_t *appb = posb + B;                                         // [B] 1: append happens

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const bool early = v.early != 0;

  if (tid == 0) {
    for (int s = 0; s < kStages8; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int j = 0; j < 2; ++j) {
      mbar_init(&s_full[j], 1);
      mbar_init(&p_full[j], kSoftThreads);
      mbar_init(&o_full[j], 1);
      mbar_init(&o_free[j], kSoftThreads);
      mbar_init(&q8_full[j], kSoftThreads);
    }
    mbar_init(done, 1);
    mbar_init(soft, kSoftThreads);
    flags[0] = 0;
    fence_mbar_init();
  }
  if (tid == kProducerWarp * 32) {
    prefetch_tensormap(&tmap_k);
    prefetch_tensormap(&tmap_v);
  }
  if (warp == kIssuerWarp) tmem_alloc<Cf::kTmemCols>(tmem_slot);
  // The value halves of the ring start zeroed: a tile's chunks past its end keep the codes an
  // earlier tile left (finite, multiplied by zero weights), never bytes no copy wrote.
  if (warp < kSoftWarps) {
    for (int s = 0; s < kStages8; ++s) {
      uint4 *p = reinterpret_cast<uint4 *>(ring + s * kStage8 + kHalf8);
      for (int j = tid; j < kHalf8 / 16; j += kSoftThreads) p[j] = make_uint4(0u, 0u, 0u, 0u);
    }
    fence_proxy_async_smem();
  }
  // Programmatic dependent launch, as in the bf16 pass: with `early` the counters and the plan
  // are read before the dependency wait (this layer's library state, which no running kernel
  // writes); caller inputs and the shared scratch only after it.
  if (!early) {
    grid_dependency_wait();
    grid_launch_dependents();
  }
  if (warp == 0) {  // chunks per sequence and their prefix sums
    int run = 0;
    for (int b0 = 0; b0 < B; b0 += 32) {
      const int b = b0 + lane;
      int n = 0;
      if (b < B) {
        int L = v.num_slots[b];
        const bool bad = L < 0 || L > v.max_slots;
        if (bad) {
          record_error(v.err, HAM_DEVERR_SLOTS);
          L = L < 0 ? 0 : v.max_slots;
        }
        if constexpr (kStep) {
          if (!v.step.pos) posb[b] = (int32_t)step_position(v.step, b, L);
        }
        lens[b] = L;
        n = chunks_of(L);
      }
      int x = n;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(kFull, x, o);
        if (lane >= o) x += y;
      }
      if (b < B) cum[b + 1] = run + x;
      run += __shfl_sync(kFull, x, 31);
    }
    if (lane == 0) cum[0] = 0;
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  const int64_t W = (int64_t)Hkv * cum[B];
  const int C = plan_ctas(W, gridDim.x);
  const bool active_cta = (int)blockIdx.x < C;
  const int64_t x0 = active_cta ? plan_cta_begin(W, C, blockIdx.x) : 0;
  const int64_t x1 = active_cta ? plan_cta_begin(W, C, (int64_t)blockIdx.x + 1) : 0;
  const int nchunks = (int)(x1 - x0);

  // ---- the producer's first 32 chunks, decoded before the dependency wait (their counters and
  // page-table entries are this layer's state).  With `early`, the K / V / exponent copies of
  // the first tile are issued then too, and the first segment's q is prefetched into L2 (a
  // prefetch reads nothing into the CTA; the copy of q after the wait takes it as the previous
  // kernel left it).  (Three tiles before the wait measured slower: their 72 copies take ~2.5 us
  // to issue and held back the first tile's q when the wait returned sooner.)
  auto decode = [&](int64_t x, int &seg, int &valid, int &fl, int &row0, int &ph, int &c) {
    int lo = 0, hi = B - 1;
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if ((int64_t)Hkv * cum[mid] <= x) lo = mid; else hi = mid - 1;
    }
    const int b = lo;
    const int nch = cum[b + 1] - cum[b];
    const int r = (int)(x - (int64_t)Hkv * cum[b]);
    const int g = r / nch;
    c = r - g * nch;
    seg = b * Hkv + g;
    valid = min(kChunkSlots, lens[b] - c * kChunkSlots);
    const int slot0 = c * kChunkSlots;
    const int page = v.page_table[(int64_t)b * v.max_pages + slot0 / v.page_slots];
    const bool page_ok = page >= 0 && page < v.pool_pages;
    ph = (page_ok ? page : 0) * Hkv + g;
    row0 = ph * v.page_slots + slot0 % v.page_slots;
    fl = (page_ok ? kPageOk : 0) | ((c == 0 || x == x0) ? kFirst : 0) |
         ((c == nch - 1 || x == x1 - 1) ? kLast : 0);
  };
  const uint64_t pol = policy_evict_first();
  const uint32_t q_bytes = (uint32_t)(G * kD8 * 2);
  // 16-slot pages: a chunk's transposed value rows are one contiguous 2 KiB block
  const bool v_block = v.page_slots == kChunkSlots;
  const uint8_t *v_codes = reinterpret_cast<const uint8_t *>(v.v_pool);
  // this lane's chunk's copies into position `pos` of a stage's tile
  auto issue_chunk = [&](int stage, int pos, int row0, int ph) {
    uint8_t *dst = ring + stage * kStage8 + pos * kBox8;
    tma_load_2d(dst, &tmap_k, 0, row0, &full[stage], pol);
    if (v_block)
      bulk_load(dst + kHalf8, v_codes + (int64_t)ph * kD8 * kChunkSlots, (uint32_t)kBox8,
                &full[stage]);
    else
      tma_load_2d(dst + kHalf8, &tmap_v, row0 - ph * v.page_slots, ph * kD8, &full[stage], pol);
    bulk_load(exps + (stage * kTileChunks + pos) * kChunkExp,
              v.kv_exp + (int64_t)row0 * (kChunkExp / kChunkSlots), (uint32_t)kChunkExp,
              &full[stage]);
  };
  int d_seg = 0, d_valid = 0, d_fl = 0, d_row0 = 0, d_ph = 0, d_c = 0;  // lane: chunk x0 + lane
  int pre = 0;  // tiles whose K / V copies are under way before the wait
  if (active_cta && warp == kProducerWarp) {
    const int nb = min(32, nchunks);
    if (lane < nb) decode(x0 + lane, d_seg, d_valid, d_fl, d_row0, d_ph, d_c);
    if (early) {
      const uint32_t closes =
          __ballot_sync(kFull, lane < nb && ((d_fl & kLast) || (d_c & 7) == 7));
      const uint32_t okm = __ballot_sync(kFull, lane < nb && (d_fl & kPageOk));
      const int last = 31 - __clz(closes);
      if (lane == 0) bulk_prefetch_l2(v.q + (int64_t)d_seg * G * kD8, q_bytes);  // chunk x0's
      for (int ts = 0; ts <= last && pre < kPreTiles;) {
        const int te = ts + __ffs(closes >> ts) - 1;
        const uint32_t tm = (okm >> ts) & ((1u << (te - ts + 1)) - 1u);
        if (lane == 0) mbar_expect_tx(&full[pre], (uint32_t)__popc(tm) * (uint32_t)kChunkTx);
        __syncwarp();
        if (lane >= ts && lane <= te && (d_fl & kPageOk)) issue_chunk(pre, lane - ts, d_row0, d_ph);
        ++pre;
        ts = te + 1;
      }
    }
  }

  if (early) {
    grid_dependency_wait();
    grid_launch_dependents();
  }
  if constexpr (kStep) {  // caller inputs of the append: explicit positions and append flags
    if (warp == 0) {
      if (v.step.pos)
        for (int b = lane; b < B; b += 32) posb[b] = v.step.pos[b];
      for (int b = lane; b < B; b += 32) {
        int L = v.num_slots[b];
        const bool bad = L < 0 || L > v.max_slots;
        L = L < 0 ? 0 : (bad ? v.max_slots : L);
        const int t = v.step.ntok[b];
        const int why = t < 1 ? HAM_DEVERR_NTOK
                        : bad ? HAM_DEVERR_SLOTS
                        : L == v.max_slots ? HAM_DEVERR_CAPACITY : 0;
        appb[b] = why == 0;
        if (blockIdx.x == 0) v.step.stash[b] = make_int4(L, why, posb[b], t);
      }
    }
  }
  // Sequences with no slots attend to nothing: their output is 0 (segment s zeroed by CTA
  // s % gridDim.x).
  for (int s = blockIdx.x; s < B * Hkv; s += gridDim.x) {
    const int b = s / Hkv;
    if (cum[b + 1] != cum[b]) continue;
    for (int idx = tid; idx < G * kD8; idx += blockDim.x)
      store_out<OutT>(v.out, (int64_t)s * G * kD8 + idx, 0.f);
    if (tid == 0) v.seg_range[s] = make_int2(-1, -1);
  }
  __syncthreads();
  const uint64_t wait_lim = data_wait_limit(v.wait_ns);

  if (active_cta && warp == kProducerWarp) {
    // ------------------------------------------------------------------ producer warp
    // Tiles: a segment's chunks in groups of 8 aligned to its start (chunk index c with the
    // same c / 8), cut at the ends of the CTA's range.  A chunk opens a tile if it is the range's
    // first or c % 8 == 0 and closes one if it is the range's last, its segment's last or
    // c % 8 == 7, so that every lane places its own chunk.  Lanes decode 32 chunks at a time
    // (whole tiles of them); per tile lane 0 waits for the stage and posts the bytes to expect,
    // the tile's lanes issue the copies of their chunks together (the K box, the V block, the
    // 32 exponent bytes), and lane 0 records the tile and arrives.
    int tiles = 0, nseg = 0;
    bool stop = false;
    for (int base = 0; base < nchunks && !stop;) {
      const int nb = min(32, nchunks - base);
      const bool in = lane < nb;
      const int64_t x = x0 + base + lane;
      int seg = d_seg, valid = d_valid, fl = d_fl, row0 = d_row0, ph = d_ph, c = d_c;
      if (base > 0 && in) decode(x, seg, valid, fl, row0, ph, c);
      const uint32_t closes = __ballot_sync(kFull, in && ((fl & kLast) || (c & 7) == 7));
      const uint32_t okm = __ballot_sync(kFull, in && (fl & kPageOk));
      // (the batch's last chunk closes a tile when nb < 32, and 32 chunks hold closes)
      const int last = 31 - __clz(closes);
      for (int ts = 0; ts <= last;) {
        const int te = ts + __ffs(closes >> ts) - 1;  // the tile's lanes: ts .. te
        const int n = te - ts + 1;
        const int stage = tiles % kStages8;
        const int f0 = __shfl_sync(kFull, fl, ts), f1 = __shfl_sync(kFull, fl, te);
        const int t_seg = __shfl_sync(kFull, seg, ts);
        const int vlast = __shfl_sync(kFull, valid, te);
        const uint32_t tm = (okm >> ts) & ((1u << n) - 1u);  // chunks whose page is valid
        const bool kv_issued = tiles < pre;                   // (before the wait)
        int failed = 0, qb = 0;
        if (lane == 0) {
          const uint32_t par = ((uint32_t)(tiles / kStages8) & 1u) ^ 1u;
          if (tiles >= kStages8 && !thread_wait(&empty[stage], par, flags, true, wait_lim)) {
            record_error(v.err, HAM_DEVERR_TIMEOUT);
            flags[0] = 1;
            failed = 1;
          } else {
            uint32_t bytes = kv_issued ? 0u : (uint32_t)__popc(tm) * (uint32_t)kChunkTx;
            bool tabled = false;
            int64_t p = 0;
            if (f0 & kFirst) {
              if constexpr (kStep) {
                p = posb[t_seg / Hkv];
                tabled = p >= 0 && p < v.step.rope_positions;
              }
              bytes += q_bytes + (tabled ? (uint32_t)(kD8 / 2) * 8 : 0u);
            }
            mbar_expect_tx(&full[stage], bytes);
            if (f0 & kFirst) {  // the segment's q (and the step's (cos, sin) row)
              qb = nseg++ % Cf::kQBufs;
              uint8_t *qdst = qbufs + qb * lay.q_stride;
              bulk_load(qdst, v.q + (int64_t)t_seg * G * kD8, q_bytes, &full[stage]);
              if (tabled)
                bulk_load(qdst + q_bytes, v.step.rope_table_f + p * (kD8 / 2),
                          (uint32_t)(kD8 / 2) * 8, &full[stage]);
            }
            if (tm != (1u << n) - 1u) record_error(v.err, HAM_DEVERR_PAGE);
          }
        }
        if (__shfl_sync(kFull, failed, 0)) {
          stop = true;
          break;
        }
        __syncwarp();
        if (!kv_issued && lane >= ts && lane <= te && (fl & kPageOk))
          issue_chunk(stage, lane - ts, row0, ph);
        __syncwarp();
        if (lane == 0) {
          const bool end = x0 + base + te == x1 - 1;
          info[stage] = make_int4(t_seg, (n - 1) * kChunkSlots + vlast,
                                  (f0 & kFirst) | (f1 & kLast) | (end ? kEnd : 0) | (int)(tm << 8),
                                  qb);
          mbar_arrive(&full[stage]);
        }
        ++tiles;
        ts = te + 1;
      }
      base += last + 1;
    }
    // Let every copy this CTA issued land before the CTA can exit.
    if (lane == 0) {
      for (int i = max(0, tiles - kStages8); i < tiles; ++i)
        thread_wait(&full[i % kStages8], (uint32_t)(i / kStages8) & 1u, flags, false);
    }
  } else if (active_cta && warp == kIssuerWarp) {
    // ------------------------------------------------------------------ product issuer
    // S of tile nS once its copies (and, opening a segment, its q pieces) are in and S's buffer
    // is free (nS <= nO + 1: the softmax of tile nS - 2 has read it); O of tile nO once its
    // weights are written and O's buffer has been read back.  O's completion frees the stage.
    if (lane == 0) {
      constexpr uint32_t kId = idesc_e4m3(kTileSlots, kCols);
      int nS = 0, nO = 0, segS = -1, nT = INT_MAX;
      uint64_t t0 = global_timer_ns();
      uint32_t idle = 0;
      while (nO < nT) {
        bool prog = false;
        if (nS < nT && nS <= nO + 1) {
          const int st = nS % kStages8;
          if (mbar_poll(&full[st], (uint32_t)(nS / kStages8) & 1u)) {
            const int4 inf = info[st];
            const bool first = (inf.z & kFirst) != 0;
            const int qk = first ? segS + 1 : segS;
            if (!first || mbar_poll(&q8_full[qk & 1], (uint32_t)(qk >> 1) & 1u)) {
              segS = qk;
              tc_fence_after();
              const uint32_t ka = smem_u32(ring + st * kStage8);
              const uint32_t qa = smem_u32(q8 + (segS & 1) * Cf::kOperand);
              const uint32_t d = tmem + (uint32_t)((nS & 1) * kCols);
#pragma unroll
              for (int k = 0; k < kD8 / 32; ++k)
                tc_mma_e4m3(d, smem_desc_sw128(ka + 32 * k, 16, 1024),
                            smem_desc_sw128(qa + 32 * k, 16, 1024), kId, k > 0);
              tc_commit(&s_full[nS & 1]);
              if (inf.z & kEnd) nT = nS + 1;
              ++nS;
              prog = true;
            }
          }
        }
        if (nO < nS && mbar_poll(&p_full[nO & 1], (uint32_t)(nO >> 1) & 1u) &&
            (nO < 2 || mbar_poll(&o_free[nO & 1], (uint32_t)((nO >> 1) - 1) & 1u))) {
          tc_fence_after();
          const int st = nO % kStages8;
          const uint32_t va = smem_u32(ring + st * kStage8 + kHalf8);
          const uint32_t pa = smem_u32(pw + (nO & 1) * Cf::kOperand);
          const uint32_t d = tmem + (uint32_t)(2 * kCols + (nO & 1) * kCols);
#pragma unroll
          for (int k = 0; k < kTileSlots / 32; ++k)  // 32 slots = two chunks a product
            tc_mma_e4m3(d, smem_desc_plain(va + 2 * kBox8 * k, kBox8, 128),
                        smem_desc_sw128(pa + 32 * k, 16, 1024), kId, k > 0);
          tc_commit(&o_full[nO & 1]);
          tc_commit(&empty[st]);
          ++nO;
          prog = true;
        }
        if (prog) {
          idle = 0;
          t0 = global_timer_ns();
        } else if ((++idle & 63u) == 0) {
          if (*flags) break;
          if (global_timer_ns() - t0 > wait_lim) {
            record_error(v.err, HAM_DEVERR_TIMEOUT);
            flags[0] = 1;
            break;
          }
        }
      }
      // every product issued has completed before tensor memory is freed
      tc_commit(done);
      thread_wait(done, 0u, flags, false);
    }
  } else if (active_cta && warp < kSoftWarps) {
    // ------------------------------------------------------------------ softmax / output warps
    const int t = tid;                       // slot t of a tile; head dim t of the output
    const int c = t >> 4, s = t & 15;        // its chunk and slot within the chunk
    const int kcol = c * kChunkSlots + fp8_v_slot_byte(s);  // its column of P (V^T's order)
    const uint32_t lane_base = tmem + ((uint32_t)(warp * 32) << 16);
    const float qscale = rsqrtf((float)kD8) * 1.4426950408889634f;  // 1/sqrt(d) * log2(e)
    float m[kMaxG], l[kMaxG], acc[kMaxG], qs[kMaxG], md[kMaxG], ld[kMaxG], fa[kMaxG], fc[kMaxG];
#pragma unroll
    for (int h = 0; h < kMaxG; ++h) {
      m[h] = -INFINITY;
      l[h] = 0.f;
      acc[h] = 0.f;
      qs[h] = 0.f;
      md[h] = -INFINITY;
      ld[h] = 0.f;
      fa[h] = 1.f;
      fc[h] = 0.f;
    }
    uint32_t sph = 0;  // rounds of the four warps' barrier so far
    // All four warps meet (bounded; false once the CTA gives up).
    auto soft_sync = [&]() -> bool {
      mbar_arrive(soft);
      const bool ok = warp_wait(soft, sph & 1u, flags, wait_lim);
      ++sph;
      return ok;
    };
    // The pieces of the segment's q (rotated by the new slot's position in the fused step) into
    // Q8 buffer k & 1, and each head's scale.
    auto build_q8 = [&](const int4 &inf, int k) -> bool {
      uint8_t *qraw = qbufs + inf.w * lay.q_stride;
      const uint16_t *q = reinterpret_cast<const uint16_t *>(qraw);
      float xq[kMaxG];
#pragma unroll
      for (int h = 0; h < kMaxG; ++h) xq[h] = h < G ? bf16_value(q[h * kD8 + t]) : 0.f;
      if constexpr (kStep) {
        // turned in fp32 and rounded to bf16, as the bf16 pass and the combine kernel do
        const int bq = inf.x / Hkv;
        if (appb[bq]) {
          float2 *cs = reinterpret_cast<float2 *>(qraw + G * kD8 * 2);
          const int64_t p = posb[bq];
          if (!(p >= 0 && p < v.step.rope_positions)) {
            if (warp == 0) fill_cs_row(cs, p, v.step.inv_freq, kD8 / 2, lane);
            if (!soft_sync()) return false;
          }
          const float2 cv = cs[t & (kD8 / 2 - 1)];
#pragma unroll
          for (int h = 0; h < kMaxG; ++h) {
            if (h < G) {
              const float o = bf16_value(q[h * kD8 + (t ^ (kD8 / 2))]);
              xq[h] = t < kD8 / 2 ? round_bf16(xq[h] * cv.x - o * cv.y)
                                  : round_bf16(xq[h] * cv.x + o * cv.y);
            }
          }
        }
      }
      float *rq = red_q + warp * kMaxG;
#pragma unroll
      for (int h = 0; h < kMaxG; ++h) {
        if (h < G) {
          const float a = warp_max_f32(fabsf(xq[h]));
          if (lane == 0) rq[h] = a;
        }
      }
      if (!soft_sync()) return false;
      uint8_t *qb = q8 + (k & 1) * Cf::kOperand;
#pragma unroll
      for (int h = 0; h < kMaxG; ++h) {
        if (h < G) {
          const float A = fmaxf(fmaxf(red_q[h], red_q[kMaxG + h]),
                                fmaxf(red_q[2 * kMaxG + h], red_q[3 * kMaxG + h]));
          int f = 0;
          if (A > 0.f) {
            int E = 0;
            frexpf(A, &E);
            // (clamped so that 2^+-f stays a normal float: a head whose largest element lies
            // below 2^-92 keeps fewer bits of its smallest elements)
            f = min(max(E - 8, -100), 100);
          }
          qs[h] = qscale * pow2i(f);
          uint8_t c0, c1, c2;
          e4m3_pieces(xq[h] * pow2i(-f), c0, c1, c2);
          qb[sw128_byte(h, t)] = c0;
          qb[sw128_byte(kMaxG + h, t)] = c1;
          qb[sw128_byte(2 * kMaxG + h, t)] = c2;
        }
      }
      fence_proxy_async_smem();
      mbar_arrive(&q8_full[k & 1]);
      return true;
    };
    // Tile j's O^T into the registers: acc = acc * alpha + O 2^(Gv - 7 - m) (factors fa, fc).
    auto accumulate = [&](int j) -> bool {
      if (!warp_wait(&o_full[j & 1], (uint32_t)(j >> 1) & 1u, flags, wait_lim)) return false;
      tc_fence_after();
      uint32_t o[kCols];
      tmem_ld_cols<kCols>(lane_base + (uint32_t)(2 * kCols + (j & 1) * kCols), o);
      tmem_wait_ld();
      tc_fence_before();
      mbar_arrive(&o_free[j & 1]);
#pragma unroll
      for (int h = 0; h < kMaxG; ++h)
        acc[h] = acc[h] * fa[h] + join_pieces(o[h], o[kMaxG + h], o[2 * kMaxG + h]) * fc[h];
      return true;
    };
    // End of a segment in this CTA: the output, or the partial (max md, sum, acc) that the
    // combine kernel merges.
    auto finalize = [&](const int4 &inf) -> bool {
      float Ls[kMaxG];
#pragma unroll
      for (int h = 0; h < kMaxG; ++h) {
        float x = h < G ? ld[h] : 0.f;
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) x += __shfl_xor_sync(kFull, x, off);
        Ls[h] = x;
        if (lane == 0) red_seg[warp * kMaxG + h] = x;
      }
      if (!soft_sync()) return false;
#pragma unroll
      for (int h = 0; h < kMaxG; ++h)
        Ls[h] = (red_seg[h] + red_seg[kMaxG + h]) + (red_seg[2 * kMaxG + h] + red_seg[3 * kMaxG + h]);
      const int seg = inf.x;
      const int b = seg / Hkv, gk = seg - b * Hkv;
      const int nch = cum[b + 1] - cum[b];
      const int64_t X0 = (int64_t)Hkv * cum[b] + (int64_t)gk * nch;
      const int first = plan_owner(W, C, X0), last = plan_owner(W, C, X0 + nch - 1);
      const int64_t obase = (int64_t)seg * G * kD8;
      // (fused step: the combine kernel still adds the appended slot, so always the partials)
      if (!kStep && first == last) {
#pragma unroll
        for (int h = 0; h < kMaxG; ++h)
          if (h < G)
            store_out<OutT>(v.out, obase + (int64_t)h * kD8 + t, Ls[h] > 0.f ? acc[h] / Ls[h] : 0.f);
      } else {
        const int64_t pidx = (int64_t)blockIdx.x + seg;
        float *pacc = v.part_acc + pidx * G * kD8;
#pragma unroll
        for (int h = 0; h < kMaxG; ++h) {
          if (h < G) {
            pacc[h * kD8 + t] = acc[h];
            if (t == h) v.part_ml[pidx * G + h] = make_float2(md[h], Ls[h]);
          }
        }
      }
      if (t == 0 && (int)blockIdx.x == first) v.seg_range[seg] = make_int2(first, last);
#pragma unroll
      for (int h = 0; h < kMaxG; ++h) acc[h] = 0.f;
      return true;
    };

    int segq = -1;
    int4 prev = make_int4(0, 0, 0, 0);
    bool ok = true;
    for (int i = 0; ok; ++i) {
      const int st = i % kStages8, bb = i & 1;
      if (!warp_wait(&full[st], (uint32_t)(i / kStages8) & 1u, flags, wait_lim)) {
        ok = false;
        break;
      }
      const int4 inf = info[st];
      const int fl = inf.z;
      if (fl & kFirst) {  // a new segment: keep the finished one's state for its output
#pragma unroll
        for (int h = 0; h < kMaxG; ++h) {
          md[h] = m[h];
          ld[h] = l[h];
          m[h] = -INFINITY;
          l[h] = 0.f;
        }
        if (!build_q8(inf, ++segq)) {
          ok = false;
          break;
        }
      }
      if (!warp_wait(&s_full[bb], (uint32_t)(i >> 1) & 1u, flags, wait_lim)) {
        ok = false;
        break;
      }
      tc_fence_after();
      uint32_t r[kCols];
      tmem_ld_cols<kCols>(lane_base + (uint32_t)(bb * kCols), r);
      tmem_wait_ld();
      // scores (log2 units) of this thread's slot; -inf where masked
      const int mask = (fl >> 8) & 0xFF;
      const bool valid = t < inf.y && ((mask >> c) & 1);
      const int8_t *ex = exps + (st * kTileChunks + c) * kChunkExp;
      const float ks = pow2i(ex[s]);
      const float ev = (float)ex[kChunkSlots + s];
      float x[kMaxG], y[kMaxG];
      float *rt = red_tile + bb * Cf::kRedTile + warp * 2 * kMaxG;
#pragma unroll
      for (int h = 0; h < kMaxG; ++h) {
        x[h] = (valid && h < G) ? join_pieces(r[h], r[kMaxG + h], r[2 * kMaxG + h]) * ks * qs[h]
                                : -INFINITY;
        y[h] = x[h] + ev;
        if (h < G) {
          const float a = warp_max_f32(x[h]), e = warp_max_f32(y[h]);
          if (lane == 0) {
            rt[h] = a;
            rt[kMaxG + h] = e;
          }
        }
      }
      if (!soft_sync()) {
        ok = false;
        break;
      }
      const float *rr = red_tile + bb * Cf::kRedTile;
      uint8_t *pb = pw + bb * Cf::kOperand;
      float nfa[kMaxG], nfc[kMaxG];
#pragma unroll
      for (int h = 0; h < kMaxG; ++h) {
        nfa[h] = 1.f;
        nfc[h] = 0.f;
        if (h < G) {
          float M = rr[h], Gv = rr[kMaxG + h];
#pragma unroll
          for (int w = 1; w < kSoftWarps; ++w) {
            M = fmaxf(M, rr[w * 2 * kMaxG + h]);
            Gv = fmaxf(Gv, rr[w * 2 * kMaxG + kMaxG + h]);
          }
          const float mn = fmaxf(m[h], M);
          nfa[h] = mn == m[h] ? 1.f : ex2(m[h] - mn);
          nfc[h] = Gv == -INFINITY ? 0.f : ex2(Gv - 7.f - mn);
          const float p = x[h] == -INFINITY ? 0.f : ex2(x[h] - mn);
          l[h] = l[h] * nfa[h] + p;
          m[h] = mn;
          const float w = y[h] == -INFINITY ? 0.f : ex2(y[h] - Gv + 7.f);
          uint8_t c0, c1, c2;
          e4m3_pieces(w, c0, c1, c2);
          pb[sw128_byte(h, kcol)] = c0;
          pb[sw128_byte(kMaxG + h, kcol)] = c1;
          pb[sw128_byte(2 * kMaxG + h, kcol)] = c2;
        }
      }
      fence_proxy_async_smem();
      tc_fence_before();
      mbar_arrive(&p_full[bb]);
      if (i > 0) {  // the previous tile's output, and its segment's if that ended there
        if (!accumulate(i - 1) || ((prev.z & kLast) && !finalize(prev))) {
          ok = false;
          break;
        }
      }
#pragma unroll
      for (int h = 0; h < kMaxG; ++h) {
        fa[h] = nfa[h];
        fc[h] = nfc[h];
      }
      prev = inf;
      if (fl & kEnd) {
#pragma unroll
        for (int h = 0; h < kMaxG; ++h) {
          md[h] = m[h];
          ld[h] = l[h];
        }
        ok = accumulate(i) && finalize(inf);
        break;
      }
    }
    if (!ok && lane == 0) {
      record_error(v.err, HAM_DEVERR_TIMEOUT);
      flags[0] = 1;
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == kIssuerWarp) {
    tc_fence_after();
    tmem_dealloc<Cf::kTmemCols>(tmem);
  }
}

template <typename OutT, bool kStep, int kCols>
struct Fp8Instance {
  static auto fn() { return &decode_attn_fp8_kernel<OutT, kStep, kCols>; }
  static size_t smem_bytes(int group, int batch) {
    return 1024 + (size_t)Fp8Layout<kCols>(group, kStep, batch).total;
  }
  // Allow the largest dynamic shared memory any group and batch need, once per device.
  static cudaError_t configure() {
    static std::mutex mu;
    static bool done[64] = {};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    std::lock_guard<std::mutex> lock(mu);
    if (dev >= 0 && dev < 64 && done[dev]) return cudaSuccess;
    e = cudaFuncSetAttribute(fn(), cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)smem_bytes(Fp8Cfg<kCols>::kMaxG, kMaxBatch));
    // all of the unified L1 / shared memory as shared memory: two CTAs (two 96 KiB rings) an
    // SM, which the occupancy query reports only with this preference
    if (e == cudaSuccess)
      e = cudaFuncSetAttribute(fn(), cudaFuncAttributePreferredSharedMemoryCarveout,
                               (int)cudaSharedmemCarveoutMaxShared);
    if (e == cudaSuccess && dev >= 0 && dev < 64) done[dev] = true;
    return e;
  }
  static cudaError_t launch(const CUtensorMap &tk, const CUtensorMap &tv, const AttnView &v,
                            cudaStream_t stream) {
    cudaError_t e = configure();
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)v.ctas);
    cfg.blockDim = dim3(kThreads8);
    cfg.dynamicSmemBytes = smem_bytes(v.group, v.batch);
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, decode_attn_fp8_kernel<OutT, kStep, kCols>, tk, tv, v);
  }
  // CTAs of this instance an SM can hold.  (The occupancy query answers one for every kernel
  // that allocates tensor memory, whatever its needs; two of these CTAs do run side by side.)
  // The smallest of the limits of shared memory (with the runtime's reserve a CTA), registers
  // (allocated 256 a warp), threads and tensor-memory columns.
  static int ctas_per_sm(int group, int batch) {
    if (configure() != cudaSuccess) return 0;
    int dev = 0, smem_sm = 0, reserve = 0, regs_sm = 0, threads_sm = 0;
    cudaFuncAttributes a;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&smem_sm, cudaDevAttrMaxSharedMemoryPerMultiprocessor, dev) !=
            cudaSuccess ||
        cudaDeviceGetAttribute(&reserve, cudaDevAttrReservedSharedMemoryPerBlock, dev) !=
            cudaSuccess ||
        cudaDeviceGetAttribute(&regs_sm, cudaDevAttrMaxRegistersPerMultiprocessor, dev) !=
            cudaSuccess ||
        cudaDeviceGetAttribute(&threads_sm, cudaDevAttrMaxThreadsPerMultiProcessor, dev) !=
            cudaSuccess ||
        cudaFuncGetAttributes(&a, fn()) != cudaSuccess)
      return 0;
    int n = smem_sm / (int)(smem_bytes(group, batch) + (size_t)reserve + a.sharedSizeBytes);
    const int regs_warp = (a.numRegs * 32 + 255) / 256 * 256;
    n = std::min(n, regs_sm / (regs_warp * (kThreads8 / 32)));
    n = std::min(n, threads_sm / kThreads8);
    n = std::min(n, (int)(512 / Fp8Cfg<kCols>::kTmemCols));
    return std::max(n, 0);
  }
};

template <typename F>
cudaError_t fp8_dispatch(int group, int out_dtype, bool step, F &&f) {
  const bool f32 = out_dtype == HAM_DTYPE_F32;
  if (group <= Fp8Cfg<16>::kMaxG) {
    if (step)
      return f32 ? f(Fp8Instance<float, true, 16>()) : f(Fp8Instance<__nv_bfloat16, true, 16>());
    return f32 ? f(Fp8Instance<float, false, 16>()) : f(Fp8Instance<__nv_bfloat16, false, 16>());
  }
  if (step)
    return f32 ? f(Fp8Instance<float, true, 32>()) : f(Fp8Instance<__nv_bfloat16, true, 32>());
  return f32 ? f(Fp8Instance<float, false, 32>()) : f(Fp8Instance<__nv_bfloat16, false, 32>());
}

}  // namespace

cudaError_t launch_fp8_attention_pass(const CUtensorMap &tk, const CUtensorMap &tv,
                                      const AttnView &v, int out_dtype, bool step,
                                      cudaStream_t stream) {
  if (v.ctas < 1 || v.group < 1 || v.group > kMaxGroup) return cudaErrorInvalidConfiguration;
  return fp8_dispatch(v.group, out_dtype, step,
                      [&](auto inst) { return decltype(inst)::launch(tk, tv, v, stream); });
}

int fp8_attention_ctas_per_sm(int group, int batch, bool step, int out_dtype) {
  if (group < 1 || group > kMaxGroup) return 0;
  int n = 0;
  fp8_dispatch(group, out_dtype, step, [&](auto inst) {
    n = decltype(inst)::ctas_per_sm(group, batch);
    return cudaSuccess;
  });
  return n;
}

}  // namespace ham
