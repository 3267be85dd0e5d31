// Split-KV GQA decode attention over the paged smashed-KV cache (sm_103a).
//
// What it computes (HAMburger, arXiv 2505.20438): one KV set per macro-step (Sec. 3.1,
// Sec. 3.6 "Token Fusion"), so a decode step is plain softmax attention of each query head
// over the slot list of its sequence, scale 1/sqrt(d), query head h reading KV head h / G
// (Llama-3.2 base model, Sec. 4.1).  Decoding re-reads the whole cache every step and is
// bound by memory bandwidth (Sec. 2.3), so the kernel is built around moving every K/V
// byte from HBM exactly once per (sequence, KV head):
//
//  * Split plan: the 16-slot chunks of all (sequence, KV head) segments are numbered
//    contiguously and cut into gridDim.x equal ranges, one per CTA (ham_internal.cuh).
//    Ragged batches balance for free; the plan is computed on the device from the slot
//    counters, so the launch never waits on the host.
//  * Producer warp: one lane issues 1-D bulk copies (cp.async.bulk, the TMA engine) of a
//    chunk's K rows and V rows (each one contiguous block inside a page) into a ring of
//    shared-memory stages, completing on an mbarrier, with an L2 evict-first hint.  The
//    query heads of a segment ride on the first stage of the segment.
//  * Consumer warps: a chunk's 16 slots are split over the consumer warps; a slot's
//    head_dim values are spread over kLanesPerSlot lanes (16-byte conflict-free shared
//    loads).  q.k partials of the G heads use packed fp32 FMAs (__ffma2_rn), then a
//    reduce-scatter over the slot's lanes leaves each lane one head's score, with no
//    selects because every lane keeps its heads in the order (i XOR its own head).  The
//    online softmax is fp32 in the exp2 domain with a lazy running max (rescale only when
//    a score exceeds the running max by more than 2^8).
//  * Combine: at the end of a segment the consumer warps merge their states in shared
//    memory; a segment covered by one CTA is written directly, otherwise the CTA writes a
//    partial (max, sum, acc) and the last CTA to finish the segment (atomic ticket) merges
//    the partials in CTA order, so the result does not depend on timing or page ids.
//
// Every wait is bounded (about 2 s); a wait that runs out records HAM_DEVERR_TIMEOUT,
// lets the CTA's copies land and returns.  No trap, no unbounded spin.
#include <cuda_bf16.h>

#include <mutex>
#include <type_traits>

#include "ham_internal.cuh"

namespace ham {
namespace {

constexpr uint32_t kFull = 0xffffffffu;
constexpr float kRescaleSlack = 8.0f;              // log2 units
constexpr uint64_t kWaitLimitNs = 2000000000ull;   // bounded waits: 2 s
constexpr int kFirst = 1, kLast = 2, kPageOk = 4;  // stage flags

// ------------------------------------------------------------------------------------
// PTX wrappers
// ------------------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_u32(const void *p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ uint64_t global_timer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
__device__ __forceinline__ void mbar_init(uint64_t *bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count)
               : "memory");
}
__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void mbar_arrive(uint64_t *bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}
__device__ __forceinline__ void mbar_arrive_tx(uint64_t *bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(bytes)
               : "memory");
}
__device__ __forceinline__ bool mbar_test(uint64_t *bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
      " selp.u32 %0, 1, 0, p;\n}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}
__device__ __forceinline__ uint64_t policy_evict_first() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}
// 1-D bulk copy global -> shared through the TMA engine; 16-byte aligned, size % 16 == 0.
__device__ __forceinline__ void bulk_load(void *dst, const void *src, uint32_t bytes,
                                          uint64_t *bar, uint64_t policy) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1], %2, [%3], %4;" ::"r"(smem_u32(dst)),
      "l"(src), "r"(bytes), "r"(smem_u32(bar)), "l"(policy)
      : "memory");
}
__device__ __forceinline__ void bulk_load(void *dst, const void *src, uint32_t bytes,
                                          uint64_t *bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1], %2, [%3];" ::"r"(smem_u32(dst)),
      "l"(src), "r"(bytes), "r"(smem_u32(bar))
      : "memory");
}
__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
// Two bf16 packed in a 32-bit word (element 2j low, 2j+1 high) -> exact fp32 pair.
__device__ __forceinline__ float2 bf16x2_to_float2(uint32_t w) {
  return make_float2(__uint_as_float(w << 16), __uint_as_float(w & 0xFFFF0000u));
}
__device__ __forceinline__ uint32_t word_of(const uint4 &v, int j) {
  return j == 0 ? v.x : j == 1 ? v.y : j == 2 ? v.z : v.w;
}

// One thread waits on an mbarrier phase, bounded.  honor_abort: give up early once another
// warp has aborted (not used while draining in-flight copies).
__device__ bool thread_wait(uint64_t *bar, uint32_t parity, volatile int *abort_flag,
                            bool honor_abort) {
  if (mbar_test(bar, parity)) return true;
  const uint64_t t0 = global_timer_ns();
  for (uint32_t n = 1;; ++n) {
    if (mbar_test(bar, parity)) return true;
    if ((n & 15u) == 0) {
      if (honor_abort && *abort_flag) return false;
      if (global_timer_ns() - t0 > kWaitLimitNs) return false;
    }
  }
}

// The whole warp waits on an mbarrier phase, bounded; the result is warp-uniform.
__device__ bool warp_wait(uint64_t *bar, uint32_t parity, volatile int *abort_flag) {
  if (__all_sync(kFull, mbar_test(bar, parity))) return true;
  const uint64_t t0 = global_timer_ns();
  for (uint32_t n = 1;; ++n) {
    if (__all_sync(kFull, mbar_test(bar, parity))) return true;
    if ((n & 15u) == 0) {
      int stop = 0;
      if ((threadIdx.x & 31) == 0)
        stop = (*abort_flag != 0) || (global_timer_ns() - t0 > kWaitLimitNs);
      if (__shfl_sync(kFull, stop, 0)) return false;
    }
  }
}

// ------------------------------------------------------------------------------------
// Shape of one kernel instance
// ------------------------------------------------------------------------------------
constexpr int align_up(int x, int a) { return (x + a - 1) / a * a; }

template <int D, int G, int E>
struct Shape {
  static constexpr int kLanesPerSlot = D / E;                  // lanes sharing one slot row
  static constexpr int kSlotsPerWarp = 32 / kLanesPerSlot;
  static constexpr int kConsumerWarps = kChunkSlots / kSlotsPerWarp;
  static constexpr int kPieces = E / 8;                        // 16-byte pieces per lane
  static constexpr int kHeadLanes = kLanesPerSlot / G;         // lanes left holding one head
  static constexpr int kChunkBytes = kChunkSlots * D * 2;      // K (or V) rows of a chunk
  static constexpr int kStageBytes = 2 * kChunkBytes;
  static constexpr int kStages = D == 128 ? 8 : 12;
  static constexpr int kQBufs = kStages + 1;
  static constexpr int kQBytes = G * D * 2;
  static constexpr int kThreads = 32 * (kConsumerWarps + 1);
  static constexpr int kConsumerThreads = 32 * kConsumerWarps;
  // q and acc take 4*G*E/2 registers; two CTAs per SM while that leaves room (~200/thread)
  static constexpr int kMinBlocks = kThreads * (2 * G * E + 48) <= 32768 ? 2 : 1;
  // shared memory map
  static constexpr int kOffQ = kStages * kStageBytes;
  static constexpr int kOffBar = kOffQ + kQBufs * kQBytes;
  static constexpr int kOffInfo = align_up(kOffBar + (2 * kStages + 1) * 8, 16);
  static constexpr int kOffMergeAcc = kOffInfo + kStages * 16;
  static constexpr int kOffMergeML = kOffMergeAcc + kConsumerWarps * G * D * 4;
  static constexpr int kOffFlags = kOffMergeML + kConsumerWarps * G * 8;
  static constexpr int kOffCum = kOffFlags + 16;
  static size_t smem_bytes(int batch) { return (size_t)kOffCum + 4u * (2u * batch + 1u); }

  static_assert(D % E == 0 && E % 8 == 0, "lane slice must be whole 16-byte pieces");
  static_assert(32 % kLanesPerSlot == 0 && kChunkSlots % kSlotsPerWarp == 0, "lane layout");
  static_assert(G >= 1 && G <= kLanesPerSlot && kLanesPerSlot % G == 0, "group vs lanes");
};

template <typename OutT>
__device__ __forceinline__ void store_out(void *out, int64_t i, float x) {
  if constexpr (std::is_same<OutT, float>::value)
    static_cast<float *>(out)[i] = x;
  else
    static_cast<__nv_bfloat16 *>(out)[i] = __float2bfloat16_rn(x);
}

// Reduce-scatter of the G partial scores over the kLanesPerSlot lanes of a slot.  v[i]
// holds the lane's partial of head (i ^ hsel); afterwards the return value is the full
// score of head hsel.  (Partner lane c ^ m has hsel ^ (G/2...) so its upper half holds the
// heads of our lower half.)
template <int G, int LPS>
__device__ __forceinline__ float reduce_scores(float (&v)[G]) {
#pragma unroll
  for (int n = G, m = LPS / 2; n > 1; n >>= 1, m >>= 1) {
#pragma unroll
    for (int i = 0; i < n / 2; ++i) v[i] += __shfl_xor_sync(kFull, v[i + n / 2], m);
  }
  float s = v[0];
#pragma unroll
  for (int m = LPS / (2 * G); m >= 1; m >>= 1) s += __shfl_xor_sync(kFull, s, m);
  return s;
}

// Consumer-warp barrier on an mbarrier (bounded; returns false on timeout/abort).
__device__ __forceinline__ bool consumer_sync(uint64_t *bar, uint32_t &phase,
                                              volatile int *flags) {
  __syncwarp();
  if ((threadIdx.x & 31) == 0) mbar_arrive(bar);
  const bool ok = warp_wait(bar, phase, flags);
  phase ^= 1u;
  return ok;
}

// ------------------------------------------------------------------------------------
// The kernel
// ------------------------------------------------------------------------------------
template <int D, int G, int E, typename OutT>
__global__ void __launch_bounds__(Shape<D, G, E>::kThreads, Shape<D, G, E>::kMinBlocks)
    decode_attn_kernel(const AttnView v) {
  using S = Shape<D, G, E>;
  constexpr int LPS = S::kLanesPerSlot;
  extern __shared__ __align__(128) uint8_t smem[];
  uint8_t *stages = smem;
  uint8_t *qbufs = smem + S::kOffQ;
  uint64_t *full = reinterpret_cast<uint64_t *>(smem + S::kOffBar);
  uint64_t *empty = full + S::kStages;
  uint64_t *sync_bar = empty + S::kStages;
  int4 *info = reinterpret_cast<int4 *>(smem + S::kOffInfo);
  float *merge_acc = reinterpret_cast<float *>(smem + S::kOffMergeAcc);
  float2 *merge_ml = reinterpret_cast<float2 *>(smem + S::kOffMergeML);
  volatile int *flags = reinterpret_cast<volatile int *>(smem + S::kOffFlags);  // abort, last
  int32_t *cum = reinterpret_cast<int32_t *>(smem + S::kOffCum);  // [B+1] chunk prefix
  int32_t *lens = cum + v.batch + 1;                               // [B] slots

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int B = v.batch, Hkv = v.n_kv_heads;

  if (tid == 0) {
    for (int s = 0; s < S::kStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], S::kConsumerWarps);
    }
    mbar_init(sync_bar, S::kConsumerWarps);
    flags[0] = 0;
    flags[1] = 0;
    fence_mbar_init();
  }
  if (warp == 0) {  // chunks per sequence and their prefix sums
    int run = 0;
    for (int b0 = 0; b0 < B; b0 += 32) {
      const int b = b0 + lane;
      int n = 0;
      if (b < B) {
        int L = v.num_slots[b];
        if (L < 0 || L > v.max_slots) {
          record_error(v.err, HAM_DEVERR_SLOTS);
          L = L < 0 ? 0 : v.max_slots;
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
  __syncthreads();

  const int64_t W = (int64_t)Hkv * cum[B];
  // Sequences with no slots attend to nothing: their output is 0.  Segment s is zeroed by
  // CTA s % gridDim.x (before any CTA may leave for lack of chunks).
  for (int s = blockIdx.x; s < B * Hkv; s += gridDim.x) {
    const int b = s / Hkv;
    if (cum[b + 1] != cum[b]) continue;
    for (int idx = tid; idx < G * D; idx += blockDim.x)
      store_out<OutT>(v.out, (int64_t)s * G * D + idx, 0.f);
  }
  // Only min(gridDim.x, W) CTAs take part, so that every range holds at least one chunk:
  // the CTAs touching a segment are then exactly first..last (no idle CTA in between).
  const int C = plan_ctas(W, gridDim.x);
  if ((int)blockIdx.x >= C) return;
  const int64_t x0 = plan_cta_begin(W, C, blockIdx.x);
  const int64_t x1 = plan_cta_begin(W, C, (int64_t)blockIdx.x + 1);
  const int nchunks = (int)(x1 - x0);

  // ---------------------------------------------------------------- producer warp
  if (warp == S::kConsumerWarps) {
    const uint64_t pol = policy_evict_first();
    int it = 0, nseg = 0;
    for (int base = 0; base < nchunks; base += 32) {
      const int nb = min(32, nchunks - base);
      int seg = 0, valid = 0, fl = 0;
      long long off = 0;
      if (lane < nb) {  // decode chunk x0 + base + lane
        const int64_t x = x0 + base + lane;
        int lo = 0, hi = B - 1;
        while (lo < hi) {
          const int mid = (lo + hi + 1) >> 1;
          if ((int64_t)Hkv * cum[mid] <= x) lo = mid; else hi = mid - 1;
        }
        const int b = lo;
        const int nch = cum[b + 1] - cum[b];
        const int r = (int)(x - (int64_t)Hkv * cum[b]);
        const int g = r / nch, c = r - g * nch;
        seg = b * Hkv + g;
        valid = min(kChunkSlots, lens[b] - c * kChunkSlots);
        const int slot0 = c * kChunkSlots;
        const int page = v.page_table[(int64_t)b * v.max_pages + slot0 / v.page_slots];
        const bool page_ok = page >= 0 && page < v.pool_pages;
        off = (((long long)(page_ok ? page : 0) * Hkv + g) * v.page_slots +
               slot0 % v.page_slots) * D;
        fl = (page_ok ? kPageOk : 0) | ((c == 0 || x == x0) ? kFirst : 0) |
             ((c == nch - 1 || x == x1 - 1) ? kLast : 0);
      }
      bool stop = false;
      for (int j = 0; j < nb; ++j) {
        const int s_seg = __shfl_sync(kFull, seg, j);
        const int s_valid = __shfl_sync(kFull, valid, j);
        const int s_fl = __shfl_sync(kFull, fl, j);
        const long long s_off = __shfl_sync(kFull, off, j);
        int failed = 0;
        if (lane == 0) {
          const int stage = it % S::kStages;
          const uint32_t ph = (uint32_t)(it / S::kStages) & 1u;
          if (!thread_wait(&empty[stage], ph ^ 1u, flags, true)) {
            record_error(v.err, HAM_DEVERR_TIMEOUT);
            flags[0] = 1;
            failed = 1;
          } else {
            int qb = -1;
            if (s_fl & kFirst) qb = nseg++ % S::kQBufs;
            info[stage] = make_int4(s_seg, s_valid, s_fl, qb);
            uint32_t bytes = (s_fl & kPageOk) ? (uint32_t)S::kStageBytes : 0u;
            if (qb >= 0) bytes += S::kQBytes;
            if (bytes) mbar_arrive_tx(&full[stage], bytes);
            else mbar_arrive(&full[stage]);
            uint8_t *dst = stages + stage * S::kStageBytes;
            if (s_fl & kPageOk) {
              bulk_load(dst, v.k_pool + s_off, S::kChunkBytes, &full[stage], pol);
              bulk_load(dst + S::kChunkBytes, v.v_pool + s_off, S::kChunkBytes, &full[stage], pol);
            } else {
              record_error(v.err, HAM_DEVERR_PAGE);
            }
            if (qb >= 0)
              bulk_load(qbufs + qb * S::kQBytes, v.q + (int64_t)s_seg * G * D, S::kQBytes,
                        &full[stage]);
          }
        }
        if (__shfl_sync(kFull, failed, 0)) {
          stop = true;
          break;
        }
        ++it;
      }
      if (stop) break;
    }
    // Let every copy this CTA issued land before the CTA can exit.
    if (lane == 0) {
      for (int i = max(0, it - S::kStages); i < it; ++i)
        thread_wait(&full[i % S::kStages], (uint32_t)(i / S::kStages) & 1u, flags, false);
    }
    return;
  }

  // ---------------------------------------------------------------- consumer warps
  const int sg = lane / LPS, c = lane % LPS;
  const int hsel = c / S::kHeadLanes;           // the head this lane's score ends up in
  const int slot = warp * S::kSlotsPerWarp + sg;  // slot within the chunk
  const int ctid = warp * 32 + lane;
  const float qscale = rsqrtf((float)D) * 1.4426950408889634f;  // 1/sqrt(d) * log2(e)

  float2 q2[G][E / 2];   // [i]: head (i ^ hsel), this lane's elements, pre-scaled
  float2 acc[G][E / 2];  // same head order
  float m[G];            // running max per head (same order), uniform over the warp
  float l_own = 0.f;     // running sum of this lane's head over its slots
#pragma unroll
  for (int i = 0; i < G; ++i) {
    m[i] = -INFINITY;
#pragma unroll
    for (int e = 0; e < E / 2; ++e) acc[i][e] = make_float2(0.f, 0.f);
  }
  uint32_t sync_phase = 0;

  for (int it = 0; it < nchunks; ++it) {
    const int stage = it % S::kStages;
    if (!warp_wait(&full[stage], (uint32_t)(it / S::kStages) & 1u, flags)) {
      if (lane == 0) {
        record_error(v.err, HAM_DEVERR_TIMEOUT);
        flags[0] = 1;
      }
      return;
    }
    const int4 inf = info[stage];
    if (inf.z & kFirst) {  // query heads of a new segment
      const uint8_t *qb = qbufs + inf.w * S::kQBytes;
#pragma unroll
      for (int i = 0; i < G; ++i) {
        const uint8_t *qh = qb + (i ^ hsel) * D * 2;
#pragma unroll
        for (int t = 0; t < S::kPieces; ++t) {
          const uint4 w = *reinterpret_cast<const uint4 *>(qh + (t * LPS + c) * 16);
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            const float2 f = bf16x2_to_float2(word_of(w, j));
            q2[i][t * 4 + j] = make_float2(f.x * qscale, f.y * qscale);
          }
        }
      }
    }
    if (inf.z & kPageOk) {
      const uint8_t *kb = stages + stage * S::kStageBytes + slot * (D * 2);
      const uint8_t *vb = kb + S::kChunkBytes;
      const bool valid = slot < inf.y;
      uint4 kr[S::kPieces], vr[S::kPieces];
#pragma unroll
      for (int t = 0; t < S::kPieces; ++t)
        kr[t] = *reinterpret_cast<const uint4 *>(kb + (t * LPS + c) * 16);
#pragma unroll
      for (int t = 0; t < S::kPieces; ++t)
        vr[t] = *reinterpret_cast<const uint4 *>(vb + (t * LPS + c) * 16);
      // q.k partials, two elements per packed FMA
      float2 part[G];
#pragma unroll
      for (int i = 0; i < G; ++i) part[i] = make_float2(0.f, 0.f);
#pragma unroll
      for (int t = 0; t < S::kPieces; ++t) {
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const float2 kf = bf16x2_to_float2(word_of(kr[t], j));
#pragma unroll
          for (int i = 0; i < G; ++i) part[i] = __ffma2_rn(q2[i][t * 4 + j], kf, part[i]);
        }
      }
      float sc[G];
#pragma unroll
      for (int i = 0; i < G; ++i) sc[i] = part[i].x + part[i].y;
      float s = reduce_scores<G, LPS>(sc);
      s = valid ? s : -INFINITY;
      float tmax = s;
#pragma unroll
      for (int o = LPS; o < 32; o <<= 1) tmax = fmaxf(tmax, __shfl_xor_sync(kFull, tmax, o));
      if (__any_sync(kFull, tmax > m[0] + kRescaleSlack)) {
#pragma unroll
        for (int i = 0; i < G; ++i) {
          const float tm = __shfl_sync(kFull, tmax, (i ^ hsel) * S::kHeadLanes);
          const float mn = fmaxf(m[i], tm);
          const float alpha = (mn == -INFINITY) ? 1.f : ex2(m[i] - mn);
#pragma unroll
          for (int e = 0; e < E / 2; ++e) acc[i][e] = __fmul2_rn(acc[i][e], make_float2(alpha, alpha));
          if (i == 0) l_own *= alpha;
          m[i] = mn;
        }
      }
      const float p = valid ? ex2(s - m[0]) : 0.f;
      l_own += p;
      float ph[G];
#pragma unroll
      for (int i = 0; i < G; ++i)
        ph[i] = __shfl_sync(kFull, p, sg * LPS + (i ^ hsel) * S::kHeadLanes);
      if (!valid) {
#pragma unroll
        for (int t = 0; t < S::kPieces; ++t) vr[t] = make_uint4(0u, 0u, 0u, 0u);
      }
#pragma unroll
      for (int t = 0; t < S::kPieces; ++t) {
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const float2 vf = bf16x2_to_float2(word_of(vr[t], j));
#pragma unroll
          for (int i = 0; i < G; ++i)
            acc[i][t * 4 + j] = __ffma2_rn(make_float2(ph[i], ph[i]), vf, acc[i][t * 4 + j]);
        }
      }
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(&empty[stage]);

    if (!(inf.z & kLast)) continue;

    // ------------------------------------------------------------ end of a segment
    const int seg = inf.x;
#pragma unroll
    for (int o = LPS; o < 32; o <<= 1) {  // sum the warp's slot groups
#pragma unroll
      for (int i = 0; i < G; ++i) {
#pragma unroll
        for (int e = 0; e < E / 2; ++e) {
          acc[i][e].x += __shfl_xor_sync(kFull, acc[i][e].x, o);
          acc[i][e].y += __shfl_xor_sync(kFull, acc[i][e].y, o);
        }
      }
      l_own += __shfl_xor_sync(kFull, l_own, o);
    }
    if (sg == 0) {
#pragma unroll
      for (int i = 0; i < G; ++i) {
        float *dst = merge_acc + (warp * G + (i ^ hsel)) * D;
#pragma unroll
        for (int t = 0; t < S::kPieces; ++t) {
          float4 *d4 = reinterpret_cast<float4 *>(dst + (t * LPS + c) * 8);
          d4[0] = make_float4(acc[i][t * 4 + 0].x, acc[i][t * 4 + 0].y, acc[i][t * 4 + 1].x,
                              acc[i][t * 4 + 1].y);
          d4[1] = make_float4(acc[i][t * 4 + 2].x, acc[i][t * 4 + 2].y, acc[i][t * 4 + 3].x,
                              acc[i][t * 4 + 3].y);
        }
      }
      if (c % S::kHeadLanes == 0) merge_ml[warp * G + hsel] = make_float2(m[0], l_own);
    }
    bool ok = consumer_sync(sync_bar, sync_phase, flags);

    const int b = seg / Hkv, g = seg - b * Hkv;
    const int nch = cum[b + 1] - cum[b];
    const int64_t X0 = (int64_t)Hkv * cum[b] + (int64_t)g * nch;
    const int first = plan_owner(W, C, X0), last = plan_owner(W, C, X0 + nch - 1);
    const bool multi = first != last;
    const int64_t pidx = (int64_t)blockIdx.x + seg;
    if (ok) {
      for (int idx = ctid; idx < G * D; idx += S::kConsumerThreads) {
        const int h = idx / D, d = idx - h * D;
        float M = -INFINITY;
#pragma unroll
        for (int w = 0; w < S::kConsumerWarps; ++w) M = fmaxf(M, merge_ml[w * G + h].x);
        float num = 0.f, den = 0.f;
#pragma unroll
        for (int w = 0; w < S::kConsumerWarps; ++w) {
          const float2 ml = merge_ml[w * G + h];
          const float f = (ml.x == -INFINITY) ? 0.f : ex2(ml.x - M);
          num += f * merge_acc[(w * G + h) * D + d];
          den += f * ml.y;
        }
        if (!multi) {
          store_out<OutT>(v.out, ((int64_t)seg * G + h) * D + d, num / den);
        } else {
          v.part_acc[(pidx * G + h) * D + d] = num;
          if (d == 0) v.part_ml[pidx * G + h] = make_float2(M, den);
        }
      }
    }
    if (ok && multi) {
      __threadfence();
      ok = consumer_sync(sync_bar, sync_phase, flags);
      if (ok && ctid == 0) {
        const uint32_t ticket = atomicAdd(&v.tickets[seg], 1u);
        flags[1] = (ticket == (uint32_t)(last - first)) ? 1 : 0;
      }
      if (ok) ok = consumer_sync(sync_bar, sync_phase, flags);
      if (ok && flags[1]) {  // last CTA of the segment: merge the partials in CTA order
        __threadfence();
        for (int idx = ctid; idx < G * D; idx += S::kConsumerThreads) {
          const int h = idx / D, d = idx - h * D;
          float M = -INFINITY;
          for (int k = first; k <= last; ++k)
            M = fmaxf(M, __ldcg(&v.part_ml[((int64_t)k + seg) * G + h]).x);
          float num = 0.f, den = 0.f;
          for (int k = first; k <= last; ++k) {
            const int64_t pk = (int64_t)k + seg;
            const float2 ml = __ldcg(&v.part_ml[pk * G + h]);
            const float f = ex2(ml.x - M);
            num += f * __ldcg(&v.part_acc[(pk * G + h) * D + d]);
            den += f * ml.y;
          }
          store_out<OutT>(v.out, ((int64_t)seg * G + h) * D + d, num / den);
        }
        if (ctid == 0) v.tickets[seg] = 0u;
      }
    }
    if (ok) ok = consumer_sync(sync_bar, sync_phase, flags);  // merge buffers free again
    if (!ok) {
      if (lane == 0) {
        record_error(v.err, HAM_DEVERR_TIMEOUT);
        flags[0] = 1;
      }
      return;
    }
#pragma unroll
    for (int i = 0; i < G; ++i) {
      m[i] = -INFINITY;
#pragma unroll
      for (int e = 0; e < E / 2; ++e) acc[i][e] = make_float2(0.f, 0.f);
    }
    l_own = 0.f;
  }
}

// ------------------------------------------------------------------------------------
// Dispatch
// ------------------------------------------------------------------------------------
template <int D, int G, int E, typename OutT>
struct Instance {
  using S = Shape<D, G, E>;
  static const void *fn() { return reinterpret_cast<const void *>(&decode_attn_kernel<D, G, E, OutT>); }
  // Allow the largest dynamic shared memory any batch needs, once per device.
  static cudaError_t configure() {
    static std::mutex mu;
    static bool done[64] = {};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    std::lock_guard<std::mutex> lock(mu);
    if (dev >= 0 && dev < 64 && done[dev]) return cudaSuccess;
    e = cudaFuncSetAttribute(&decode_attn_kernel<D, G, E, OutT>,
                             cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)S::smem_bytes(kMaxBatch));
    if (e == cudaSuccess && dev >= 0 && dev < 64) done[dev] = true;
    return e;
  }
  static cudaError_t launch(const AttnView &v, cudaStream_t stream) {
    cudaError_t e = configure();
    if (e != cudaSuccess) return e;
    decode_attn_kernel<D, G, E, OutT>
        <<<v.ctas, S::kThreads, S::smem_bytes(v.batch), stream>>>(v);
    return cudaGetLastError();
  }
  static int ctas_per_sm(int batch) {
    if (configure() != cudaSuccess) return 0;
    int n = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, &decode_attn_kernel<D, G, E, OutT>,
                                                      S::kThreads, S::smem_bytes(batch)) !=
        cudaSuccess)
      return 0;
    return n;
  }
};

// head_dim 128 keeps 16 elements per lane (8 lanes per slot) unless the group is 8, where
// 8 elements per lane keep the register budget; head_dim 64 uses 8 elements per lane.
template <typename OutT, typename F>
cudaError_t dispatch(int head_dim, int group, F &&f) {
  switch (head_dim * 16 + group) {
    case 128 * 16 + 1: return f(Instance<128, 1, 16, OutT>());
    case 128 * 16 + 2: return f(Instance<128, 2, 16, OutT>());
    case 128 * 16 + 4: return f(Instance<128, 4, 16, OutT>());
    case 128 * 16 + 8: return f(Instance<128, 8, 8, OutT>());
    case 64 * 16 + 1: return f(Instance<64, 1, 8, OutT>());
    case 64 * 16 + 2: return f(Instance<64, 2, 8, OutT>());
    case 64 * 16 + 4: return f(Instance<64, 4, 8, OutT>());
    case 64 * 16 + 8: return f(Instance<64, 8, 8, OutT>());
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace

bool attention_supported(int head_dim, int group) {
  return (head_dim == 64 || head_dim == 128) &&
         (group == 1 || group == 2 || group == 4 || group == 8);
}

cudaError_t launch_attention(const AttnView &v, int head_dim, int group, int out_dtype,
                             cudaStream_t stream) {
  if (v.ctas < 1) return cudaErrorInvalidConfiguration;
  auto go = [&](auto inst) { return decltype(inst)::launch(v, stream); };
  return out_dtype == HAM_DTYPE_F32 ? dispatch<float>(head_dim, group, go)
                                    : dispatch<__nv_bfloat16>(head_dim, group, go);
}

int attention_ctas_per_sm(int head_dim, int group, int batch) {
  int n = 0;
  dispatch<__nv_bfloat16>(head_dim, group, [&](auto inst) {
    n = decltype(inst)::ctas_per_sm(batch);
    return cudaSuccess;
  });
  return n;
}

}  // namespace ham
