// Split-KV GQA decode attention over the paged smashed-KV cache (sm_103a).
//
// What it computes (HAMburger, arXiv 2505.20438): one KV set per macro-step (Sec. 3.1,
// Sec. 3.7 "Token Fusion"), so a decode step is plain softmax attention of each query head
// over the slot list of its sequence, scale 1/sqrt(d), query head h reading KV head h / G
// (Llama-3.2 base model, Sec. 4.1).  Decoding re-reads the whole cache every step and is
// bound by memory bandwidth (Sec. 2.3), so the kernel moves every K/V byte from HBM once
// per (sequence, KV head) and keeps everything else off the critical path:
//
//  * Split plan: the 16-slot chunks of all (sequence, KV head) segments are numbered
//    contiguously and cut into equal ranges, one per CTA (ham_internal.cuh).  Ragged
//    batches balance for free; the plan is computed on the device from the slot counters,
//    so the launch never waits on the host.
//  * Producer warp: one lane issues TMA tensor copies (cp.async.bulk.tensor, 128-byte
//    swizzle) of a chunk's K rows and V rows into a shared-memory ring, completing on
//    mbarriers, with an L2 evict-first hint.  The swizzle keeps the ldmatrix reads below
//    free of bank conflicts (head_dim 64) or 2-way (head_dim 128).  The query heads of a
//    segment ride on the first stage of that segment (1-D bulk copy).
//  * Consumer warp: the G query heads of the group are padded to 8 and a chunk is a
//    16 x head_dim x 8 contraction on the tensor cores (mma.sync m16n8k16, bf16 in, fp32
//    accumulate): S^T = K Q^T with slots as rows, then O^T += V^T P^T with P^T moved into
//    the B-operand layout by movmatrix.  The online softmax is fp32 in the exp2 domain with
//    a lazy running max (rescale only when a score exceeds it by more than 2^8).
//  * Combine: a segment covered by one CTA is written directly; otherwise each CTA writes a
//    partial (max, sum, acc) and a second, fully parallel kernel (one thread per output
//    element, launched with programmatic dependent launch so its launch overlaps this
//    kernel's tail) merges the partials in CTA order.  The result does not depend on
//    timing or page ids.  (A fused last-CTA merge was measured first: one warp merging
//    ~15 partials through L2 serialised 12-18 us at the end of every launch.)
//
// Caches of FP8 (e4m3) rows have their own pass (ham_attn_fp8.cu: tcgen05 products over
// 128-slot tiles) with the same plan and partials; the combine kernels below serve both.
//
// Every wait is bounded (about 2 s); a wait that runs out records HAM_DEVERR_TIMEOUT,
// lets the CTA's copies land and returns.  No trap, no unbounded spin.
#include <cuda.h>
#include <cuda_bf16.h>

#include <mutex>
#include <type_traits>

#include "ham_attn.cuh"
#include "ham_internal.cuh"
#include "ham_ptx.cuh"

namespace ham {
namespace {

constexpr float kRescaleSlack = 8.0f;  // log2 units

// ------------------------------------------------------------------------------------
// Shape of one kernel instance
// ------------------------------------------------------------------------------------
template <int D>
struct Shape {
  static constexpr int kChunkBytes = kChunkSlots * D * 2;   // K (or V) rows of one chunk
  static constexpr int kStageBytes = 2 * kChunkBytes;
  static constexpr int kStages = 32768 / kStageBytes;       // 32 KiB ring
  static constexpr int kQBufs = kStages + 1;
  static constexpr int kThreads = 64;                       // consumer warp, producer warp
  static constexpr int kSteps = D / 16;                     // k-steps of q.k, m-tiles of p.v
  static constexpr int kLinesPerRow = D / 64;               // 128-byte swizzle lines per row
  static constexpr int kOffQ = kStages * kStageBytes;       // from a 1024-byte aligned base
  static_assert(D == 64 || D == 128, "head_dim 64 or 128");
  static_assert(kStages >= 2, "ring depth");
};

// Per-segment buffer: the group's q heads, and for the fused step also the fp32 (cos, sin)
// row of the new slot's position.
template <int D>
struct SegBuf {
  int q_bytes, stride;
  __host__ __device__ SegBuf(int group, bool step)
      : q_bytes(group * D * 2), stride(align_up(group * D * 2 + (step ? (D / 2) * 8 : 0), 128)) {}
  __host__ __device__ int cs_off() const { return q_bytes; }
};

// Shared memory map after the per-segment buffers (runtime: depends on group and batch).
template <int D>
struct Layout {
  int off_bar, off_info, off_flags, off_cum, total;
  __host__ __device__ Layout(int group, bool step, int batch) {
    using S = Shape<D>;
    off_bar = S::kOffQ + S::kQBufs * SegBuf<D>(group, step).stride;
    off_info = align_up(off_bar + 2 * S::kStages * 8, 16);
    off_flags = off_info + S::kStages * 16;
    off_cum = off_flags + 16;
    // cum [B+1], lens [B], and for the fused step the new slot's position and the append
    // flag [B] each
    total = off_cum + 4 * (batch + 1) + 4 * batch * (step ? 3 : 1);
  }
};

// Byte offset of the 16-byte piece `c` (elements c*8 .. c*8+7) of slot row `slot` inside a
// chunk tile written by the swizzled TMA copy.
template <int D>
__device__ __forceinline__ uint32_t tile_offset(int slot, int c) {
  return swizzle128_offset(slot, c, Shape<D>::kLinesPerRow);
}

__device__ __forceinline__ float bf16_bits_to_float(uint16_t b) {
  return __uint_as_float((uint32_t)b << 16);
}
__device__ __forceinline__ double bf16_bits_to_double(uint16_t b) {
  return (double)__uint_as_float((uint32_t)b << 16);
}

// One element of the rotated pair (i, i + D/2), rounded once to bf16: y_i = x_i c - x_{i+D/2} s
// for the low half, y_{i+D/2} = x_{i+D/2} c + x_i s for the high half (explicit fp64
// operations, no FMA: the textbook formula as ham_kv_append evaluates it).
__device__ __forceinline__ uint16_t rotate_elem(double self, double other, double c, double s,
                                                bool high) {
  const double y = high ? __dadd_rn(__dmul_rn(self, c), __dmul_rn(other, s))
                        : __dsub_rn(__dmul_rn(self, c), __dmul_rn(other, s));
  return __bfloat16_as_ushort(__double2bfloat16(y));
}

// ------------------------------------------------------------------------------------
// The kernel
// ------------------------------------------------------------------------------------
template <int D, typename OutT, bool kStep>
__global__ void __launch_bounds__(Shape<D>::kThreads)
    decode_attn_kernel(const __grid_constant__ CUtensorMap tmap_k,
                       const __grid_constant__ CUtensorMap tmap_v, const AttnView v) {
  using S = Shape<D>;
  const int B = v.batch, Hkv = v.n_kv_heads, G = v.group;
  const SegBuf<D> sb(G, kStep);
  const Layout<D> lay(G, kStep, B);
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = reinterpret_cast<uint8_t *>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t *stages = smem;
  uint8_t *qbufs = smem + S::kOffQ;
  uint64_t *full = reinterpret_cast<uint64_t *>(smem + lay.off_bar);
  uint64_t *empty = full + S::kStages;
  int4 *info = reinterpret_cast<int4 *>(smem + lay.off_info);
  volatile int *flags = reinterpret_cast<volatile int *>(smem + lay.off_flags);  // abort
  int32_t *cum = reinterpret_cast<int32_t *>(smem + lay.off_cum);  // [B+1] chunk prefix
  int32_t *lens = cum + B + 1;                                      // [B] slots attended
  int32_t *posb = lens + B;                                         // [B] new slot position
  int32_t *appb = posb + B;                                         // [B] 1: append happens

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const bool early = v.early != 0;

  if (tid == 0) {
    for (int s = 0; s < S::kStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    flags[0] = 0;
    fence_mbar_init();
  }
  if (tid == 32) {
    prefetch_tensormap(&tmap_k);
    prefetch_tensormap(&tmap_v);
  }
  // Programmatic dependent launch.  Everything above overlaps the previous kernel's tail.  If
  // the host found that the previous launch on this stream wrote nothing of this layer
  // (`early`), the counters, the plan, the page table and the first K/V copies also run
  // before the dependency wait: they are this layer's library state, which no running kernel
  // writes.  Caller inputs (q, k_new, v_new, pos, ntok) and the shared scratch are touched only
  // after it.  The combine kernel that follows may be scheduled once the wait has returned.
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
        // fused step: the pass attends over the stored slots; the combine kernel adds the
        // appended one.  Its position, unless the caller gives it, is library state.
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
  __syncthreads();

  const int64_t W = (int64_t)Hkv * cum[B];
  // Only min(gridDim.x, W) CTAs take part, so that every range holds at least one chunk:
  // the CTAs touching a segment are then exactly first..last (no idle CTA in between).
  const int C = plan_ctas(W, gridDim.x);
  const bool active_cta = (int)blockIdx.x < C;
  const int64_t x0 = active_cta ? plan_cta_begin(W, C, blockIdx.x) : 0;
  const int64_t x1 = active_cta ? plan_cta_begin(W, C, (int64_t)blockIdx.x + 1) : 0;
  const int nchunks = (int)(x1 - x0);

  // Producer lanes decode 32 chunks at a time: lane j holds chunk base + j.
  auto decode = [&](int base, int &seg, int &valid, int &fl, int &row0) {
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
    row0 = ((page_ok ? page : 0) * Hkv + g) * v.page_slots + slot0 % v.page_slots;
    fl = (page_ok ? kPageOk : 0) | ((c == 0 || x == x0) ? kFirst : 0) |
         ((c == nch - 1 || x == x1 - 1) ? kLast : 0);
  };

  // The first ring's worth of K/V copies.  Their stages expect the K/V bytes now and arrive
  // (with the bytes of q and the step rows, if the stage opens a segment) after the wait.
  int seg0 = 0, valid0 = 0, fl0 = 0, row00 = 0, pre = 0;
  if (warp == 1 && active_cta) {
    const int nb = min(32, nchunks);
    if (lane < nb) decode(0, seg0, valid0, fl0, row00);
    pre = min(nb, S::kStages);
    const uint64_t pol = policy_evict_first();
    // The first segment's q into L2 while the previous kernel ends (a prefetch reads nothing
    // into the CTA: the copy below, after the dependency wait, takes q as that kernel left it)
    if (early && lane == 0 && nb > 0)
      bulk_prefetch_l2(v.q + (int64_t)seg0 * G * D, (uint32_t)sb.q_bytes);  // lane 0: chunk 0
    for (int j = 0; j < pre; ++j) {
      const int s_fl = __shfl_sync(kFull, fl0, j);
      const int s_row = __shfl_sync(kFull, row00, j);
      if (lane == 0 && (s_fl & kPageOk)) {
        uint8_t *dst = stages + j * S::kStageBytes;
        mbar_expect_tx(&full[j], (uint32_t)S::kStageBytes);
        tma_load_3d(dst, &tmap_k, 0, 0, s_row, &full[j], pol);
        tma_load_3d(dst + S::kChunkBytes, &tmap_v, 0, 0, s_row, &full[j], pol);
      }
    }
  }
  if (early) {
    grid_dependency_wait();
    grid_launch_dependents();
  }
  // The first segment's q (buffer 0, stage 0): its copy needs nothing of what warp 0 reads
  // next, so it is under way meanwhile.
  if (warp == 1 && active_cta && lane == 0) {
    mbar_expect_tx(&full[0], (uint32_t)sb.q_bytes);
    bulk_load(qbufs, v.q + (int64_t)seg0 * G * D, (uint32_t)sb.q_bytes, &full[0]);
  }
  if constexpr (kStep) {
    // Caller inputs of the append: explicit positions, and whether each append happens.
    // (Computing the flags after the block barrier instead, in the consumer warp alone while
    // the producer went on, made the pass 20-35% slower.)
    if (warp == 0) {
      if (v.step.pos)
        for (int b = lane; b < B; b += 32) posb[b] = v.step.pos[b];
      for (int b = lane; b < B; b += 32) {
        int L = v.num_slots[b];
        const bool bad = L < 0 || L > v.max_slots;
        L = L < 0 ? 0 : (bad ? v.max_slots : L);
        const int t = v.step.ntok[b];
        // 0: append; else the error that stops it (same order as ham_kv_append)
        const int why = t < 1 ? HAM_DEVERR_NTOK
                        : bad ? HAM_DEVERR_SLOTS
                        : L == v.max_slots ? HAM_DEVERR_CAPACITY : 0;
        appb[b] = why == 0;
        if (blockIdx.x == 0) v.step.stash[b] = make_int4(L, why, posb[b], t);
      }
    }
  }
  // Sequences with no slots attend to nothing: their output is 0.  Segment s is zeroed by
  // CTA s % gridDim.x (before any CTA may leave for lack of chunks).
  for (int s = blockIdx.x; s < B * Hkv; s += gridDim.x) {
    const int b = s / Hkv;
    if (cum[b + 1] != cum[b]) continue;
    for (int idx = tid; idx < G * D; idx += blockDim.x)
      store_out<OutT>(v.out, (int64_t)s * G * D + idx, 0.f);
    if (tid == 0) v.seg_range[s] = make_int2(-1, -1);
  }
  __syncthreads();
  if (!active_cta) return;

  // ring and data waits: the launch's limit; the final drain of in-flight copies keeps 2 s
  const uint64_t wait_lim = data_wait_limit(v.wait_ns);
  // ---------------------------------------------------------------- producer warp
  if (warp == 1) {
    const uint64_t pol = policy_evict_first();
    int it = 0, nseg = 0;
    for (int base = 0; base < nchunks; base += 32) {
      const int nb = min(32, nchunks - base);
      int seg = seg0, valid = valid0, fl = fl0, row0 = row00;
      if (base > 0 && lane < nb) decode(base, seg, valid, fl, row0);
      bool stop = false;
      for (int j = 0; j < nb; ++j) {
        const int s_seg = __shfl_sync(kFull, seg, j);
        const int s_valid = __shfl_sync(kFull, valid, j);
        const int s_fl = __shfl_sync(kFull, fl, j);
        const int s_row = __shfl_sync(kFull, row0, j);
        const bool issued = it < pre;  // K/V already on their way (first ring)
        int failed = 0;
        if (lane == 0) {
          const int stage = it % S::kStages;
          const uint32_t ph = (uint32_t)(it / S::kStages) & 1u;
          if (!issued && !thread_wait(&empty[stage], ph ^ 1u, flags, true, wait_lim)) {
            record_error(v.err, HAM_DEVERR_TIMEOUT);
            flags[0] = 1;
            failed = 1;
          } else {
            int qb = -1;
            bool tabled = false;
            const int b = s_seg / Hkv;
            if (s_fl & kFirst) qb = nseg++ % S::kQBufs;
            info[stage] = make_int4(s_seg, s_valid, s_fl, qb);
            uint32_t bytes = ((s_fl & kPageOk) && !issued) ? (uint32_t)S::kStageBytes : 0u;
            if (qb >= 0) {
              if (it > 0) bytes += (uint32_t)sb.q_bytes;  // (the first one is on its way)
              if constexpr (kStep) {
                const int64_t p = posb[b];
                tabled = p >= 0 && p < v.step.rope_positions;
                bytes += tabled ? (uint32_t)(D / 2) * 8 : 0u;
              }
            }
            if (bytes) mbar_arrive_tx(&full[stage], bytes);
            else mbar_arrive(&full[stage]);
            uint8_t *dst = stages + stage * S::kStageBytes;
            if (!(s_fl & kPageOk)) {
              record_error(v.err, HAM_DEVERR_PAGE);
            } else if (!issued) {
              tma_load_3d(dst, &tmap_k, 0, 0, s_row, &full[stage], pol);
              tma_load_3d(dst + S::kChunkBytes, &tmap_v, 0, 0, s_row, &full[stage], pol);
            }
            if (qb >= 0) {
              uint8_t *qdst = qbufs + qb * sb.stride;
              if (it > 0)
                bulk_load(qdst, v.q + (int64_t)s_seg * G * D, (uint32_t)sb.q_bytes, &full[stage]);
              if constexpr (kStep) {  // (cos, sin) of the new slot's position
                if (tabled)
                  bulk_load(qdst + sb.cs_off(),
                            v.step.rope_table_f + (int64_t)posb[b] * (D / 2), (D / 2) * 8,
                            &full[stage]);
              }
            }
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

  // ---------------------------------------------------------------- consumer warp
  // Fragment coordinates (mma.sync m16n8k16): row r0 / r0 + 8, column pair 2 * cq.
  const int r0 = lane >> 2, cq = lane & 3;
  const int h0 = 2 * cq, h1 = 2 * cq + 1;  // the two heads of this lane's S / O columns
  const bool hv0 = h0 < G, hv1 = h1 < G;
  const float qscale = rsqrtf((float)D) * 1.4426950408889634f;  // 1/sqrt(d) * log2(e)
  // ldmatrix row addresses (per lane) inside a chunk tile
  const int a_slot = 8 * ((lane >> 3) & 1) + (lane & 7);  // K as A: rows 0-15, k-halves
  const int a_half = lane >> 4;
  const int v_slot = 8 * (lane >> 4) + (lane & 7);        // V^T as A (transposed load)
  const int v_half = (lane >> 3) & 1;

  uint32_t qb[S::kSteps][2];  // B fragments of Q^T for the current segment
  float o[S::kSteps][4];      // O^T fragments: rows = head_dim, columns = heads
  float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;
  int cur_qb = 0;
#pragma unroll
  for (int t = 0; t < S::kSteps; ++t) {
    o[t][0] = o[t][1] = o[t][2] = o[t][3] = 0.f;
    qb[t][0] = qb[t][1] = 0u;
  }

  for (int it = 0; it < nchunks; ++it) {
    const int stage = it % S::kStages;
    if (!warp_wait(&full[stage], (uint32_t)(it / S::kStages) & 1u, flags, wait_lim)) {
      if (lane == 0) {
        record_error(v.err, HAM_DEVERR_TIMEOUT);
        flags[0] = 1;
      }
      return;
    }
    const int4 inf = info[stage];
    if (inf.z & kFirst) {  // Q^T fragments of a new segment (heads >= G are zero)
      cur_qb = inf.w;
      const uint16_t *q = reinterpret_cast<const uint16_t *>(qbufs + cur_qb * sb.stride);
#pragma unroll
      for (int t = 0; t < S::kSteps; ++t) {
        if (r0 < G) {
          qb[t][0] = *reinterpret_cast<const uint32_t *>(q + r0 * D + 16 * t + 2 * cq);
          qb[t][1] = *reinterpret_cast<const uint32_t *>(q + r0 * D + 16 * t + 8 + 2 * cq);
        } else {
          qb[t][0] = qb[t][1] = 0u;
        }
      }
      if constexpr (kStep) {
        const int b = inf.x / Hkv;
        float2 *cs = reinterpret_cast<float2 *>(qbufs + cur_qb * sb.stride + sb.cs_off());
        if (appb[b]) {
          const int64_t p = posb[b];
          if (!(p >= 0 && p < v.step.rope_positions))
            fill_cs_row(cs, p, v.step.inv_freq, D / 2, lane);
        }
        if (appb[b] && r0 < G) {
          // Turn this lane's q elements by the new slot's position, in registers (fp32; the
          // exact fp64 rotation goes to the cache and q_rot).  Fragment t holds columns
          // 16t + 2cq + {0, 1} and 16t + 8 + 2cq + {0, 1}; the partner of column j < D/2 is
          // j + D/2, the same place of fragment t + kSteps/2.
#pragma unroll
          for (int t = 0; t < S::kSteps / 2; ++t) {
#pragma unroll
            for (int e = 0; e < 2; ++e) {
              const int j = 16 * t + 8 * e + 2 * cq;
              const uint32_t lo = qb[t][e], hi = qb[t + S::kSteps / 2][e];
              const float a0 = __uint_as_float(lo << 16), a1 = __uint_as_float(lo & 0xFFFF0000u);
              const float b0 = __uint_as_float(hi << 16), b1 = __uint_as_float(hi & 0xFFFF0000u);
              const float2 c0 = cs[j], c1 = cs[j + 1];
              qb[t][e] = pack_bf16x2(a0 * c0.x - b0 * c0.y, a1 * c1.x - b1 * c1.y);
              qb[t + S::kSteps / 2][e] = pack_bf16x2(b0 * c0.x + a0 * c0.y, b1 * c1.x + a1 * c1.y);
            }
          }
        }
      }
    }
    if (inf.z & kPageOk) {
      uint8_t *kt = stages + stage * S::kStageBytes;
      uint8_t *vt = kt + S::kChunkBytes;
      const int nvalid = inf.y;
      const bool patch = nvalid < kChunkSlots;
      if (patch) {  // rows past the sequence end never reach the MMA
        for (int i = lane; i < (kChunkSlots - nvalid) * (D / 8); i += 32) {
          const int slot = nvalid + i / (D / 8), c = i % (D / 8);
          *reinterpret_cast<uint4 *>(vt + tile_offset<D>(slot, c)) = make_uint4(0, 0, 0, 0);
        }
      }
      if (patch) __syncwarp();
      const uint32_t kbase = smem_u32(kt), vbase = smem_u32(vt);
      // S^T (16 slots x 8 heads) = K (16 x D) . Q^T (D x 8), two accumulators for ILP
      float sa[4] = {0.f, 0.f, 0.f, 0.f}, sb4[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
      for (int t = 0; t < S::kSteps; ++t) {
        uint32_t a[4];
        ldmatrix_x4(a, kbase + tile_offset<D>(a_slot, 2 * t + a_half));
        if (t & 1) mma_16816(sb4, a, qb[t][0], qb[t][1]);
        else mma_16816(sa, a, qb[t][0], qb[t][1]);
      }
      const bool v0 = r0 < nvalid, v1 = r0 + 8 < nvalid;
      const float x0 = (v0 && hv0) ? (sa[0] + sb4[0]) * qscale : -INFINITY;
      const float x1 = (v0 && hv1) ? (sa[1] + sb4[1]) * qscale : -INFINITY;
      const float x2 = (v1 && hv0) ? (sa[2] + sb4[2]) * qscale : -INFINITY;
      const float x3 = (v1 && hv1) ? (sa[3] + sb4[3]) * qscale : -INFINITY;
      float t0 = fmaxf(x0, x2), t1 = fmaxf(x1, x3);
#pragma unroll
      for (int off = 4; off < 32; off <<= 1) {
        t0 = fmaxf(t0, __shfl_xor_sync(kFull, t0, off));
        t1 = fmaxf(t1, __shfl_xor_sync(kFull, t1, off));
      }
      if (__any_sync(kFull, t0 > m0 + kRescaleSlack || t1 > m1 + kRescaleSlack)) {
        const float n0 = fmaxf(m0, t0), n1 = fmaxf(m1, t1);
        const float a0 = (n0 == -INFINITY) ? 1.f : ex2(m0 - n0);
        const float a1 = (n1 == -INFINITY) ? 1.f : ex2(m1 - n1);
#pragma unroll
        for (int t = 0; t < S::kSteps; ++t) {
          o[t][0] *= a0;
          o[t][2] *= a0;
          o[t][1] *= a1;
          o[t][3] *= a1;
        }
        l0 *= a0;
        l1 *= a1;
        m0 = n0;
        m1 = n1;
      }
      const float p0 = (x0 == -INFINITY) ? 0.f : ex2(x0 - m0);
      const float p1 = (x1 == -INFINITY) ? 0.f : ex2(x1 - m1);
      const float p2 = (x2 == -INFINITY) ? 0.f : ex2(x2 - m0);
      const float p3 = (x3 == -INFINITY) ? 0.f : ex2(x3 - m1);
      const uint32_t pk0 = pack_bf16x2(p0, p1);  // slot r0:     heads h0, h1
      const uint32_t pk1 = pack_bf16x2(p2, p3);  // slot r0 + 8: heads h0, h1
      // the softmax sum uses the same rounded weights the MMA sees
      l0 += __uint_as_float(pk0 << 16) + __uint_as_float(pk1 << 16);
      l1 += __uint_as_float(pk0 & 0xFFFF0000u) + __uint_as_float(pk1 & 0xFFFF0000u);
      const uint32_t bp0 = movmatrix_trans(pk0);  // P^T B fragment, slots 0-7
      const uint32_t bp1 = movmatrix_trans(pk1);  // slots 8-15
      // O^T (D x 8 heads) += V^T (D x 16 slots) . P^T (16 slots x 8 heads)
#pragma unroll
      for (int t = 0; t < S::kSteps; ++t) {
        uint32_t a[4];
        ldmatrix_x4_trans(a, vbase + tile_offset<D>(v_slot, 2 * t + v_half));
        mma_16816(o[t], a, bp0, bp1);
      }
      if (patch) fence_proxy_async_smem();  // patched rows vs the next TMA into this stage
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(&empty[stage]);

    if (!(inf.z & kLast)) continue;

    // ------------------------------------------------------------ end of a segment
    const int seg = inf.x;
#pragma unroll
    for (int off = 4; off < 32; off <<= 1) {
      l0 += __shfl_xor_sync(kFull, l0, off);
      l1 += __shfl_xor_sync(kFull, l1, off);
    }
    const int b = seg / Hkv, g = seg - b * Hkv;
    const int nch = cum[b + 1] - cum[b];
    const int64_t X0 = (int64_t)Hkv * cum[b] + (int64_t)g * nch;
    const int first = plan_owner(W, C, X0), last = plan_owner(W, C, X0 + nch - 1);
    const int64_t obase = (int64_t)seg * G * D;
    // The whole segment is ours: normalise and store (fused step: the combine kernel still has
    // to add the appended slot, so the state always goes to the partials).
    if (!kStep && first == last) {
      // (a segment whose only slot was a refused append has l = 0: its output is 0)
      const float i0 = l0 > 0.f ? 1.f / l0 : 0.f, i1 = l1 > 0.f ? 1.f / l1 : 0.f;
#pragma unroll
      for (int t = 0; t < S::kSteps; ++t) {
        const int d0 = 16 * t + r0;
        if (hv0) {
          store_out<OutT>(v.out, obase + (int64_t)h0 * D + d0, o[t][0] * i0);
          store_out<OutT>(v.out, obase + (int64_t)h0 * D + d0 + 8, o[t][2] * i0);
        }
        if (hv1) {
          store_out<OutT>(v.out, obase + (int64_t)h1 * D + d0, o[t][1] * i1);
          store_out<OutT>(v.out, obase + (int64_t)h1 * D + d0 + 8, o[t][3] * i1);
        }
      }
    } else {  // partial state of this CTA; the combine kernel merges first..last
      const int64_t pidx = (int64_t)blockIdx.x + seg;
      float *pacc = v.part_acc + pidx * G * D;
#pragma unroll
      for (int t = 0; t < S::kSteps; ++t) {
        const int d0 = 16 * t + r0;
        if (hv0) {
          pacc[h0 * D + d0] = o[t][0];
          pacc[h0 * D + d0 + 8] = o[t][2];
        }
        if (hv1) {
          pacc[h1 * D + d0] = o[t][1];
          pacc[h1 * D + d0 + 8] = o[t][3];
        }
      }
      if (r0 == 0) {
        if (hv0) v.part_ml[pidx * G + h0] = make_float2(m0, l0);
        if (hv1) v.part_ml[pidx * G + h1] = make_float2(m1, l1);
      }
    }
    if (lane == 0 && (int)blockIdx.x == first) v.seg_range[seg] = make_int2(first, last);
#pragma unroll
    for (int t = 0; t < S::kSteps; ++t) o[t][0] = o[t][1] = o[t][2] = o[t][3] = 0.f;
    m0 = m1 = -INFINITY;
    l0 = l1 = 0.f;
  }
}

// ------------------------------------------------------------------------------------
// Combine: out[seg][h][d] = sum_k 2^(m_k - M) acc_k[h][d] / sum_k 2^(m_k - M) l_k over the
// CTAs k = first..last of the segment, M = max_k m_k (split-softmax merge, in CTA order, in
// batches of kBatch partials whose loads are in flight together).  One thread per pair of
// elements (h, i) and (h, i + D/2) of an output row: both share the head's (max, sum), and for
// the fused step they are the pair that RoPE turns together.  Blocks of kCombineThreads cover
// one segment's G*D/2 pairs (whole heads).
//
// Fused step: the pass covered the stored slots; the appended slot enters here as one more
// term of the merge: score q.k / sqrt(d) with q and the new key turned by the new position in
// fp32 and rounded to bf16 as in the pass, weight 2^(score - M'), value v_new.  The same
// threads commit the slot: the fp64 rotation of q (q_rot) and, for h = 0, of the new key,
// rounded once to bf16 as ham_kv_append computes them, and the new value row.  Slot metadata
// and counters are committed once no CTA can still read the counters.
//
// The kernel is scheduled (programmatic dependent launch) once every attention CTA has passed
// its own dependency wait, and then idles until the attention grid ends.  Two kernels use that:
//  * combine_kernel (batches up to kCombinePlanBatch, and for the fused step a grid of at most
//    one CTA per SM, so that it sits beside the attention grid): before the wait, the segment's
//    CTA range from the slot counters with the attention's split plan, and for the fused step
//    the append record as the pass forms it, the rotations, q_rot and the new slot's rows, none
//    of which the pass reads (it covers the stored slots, and the rows of slot n that its last
//    chunk copies are masked there).  Each CTA then reports that it has read the counters; the
//    last one to report commits the metadata and counters of every sequence after its wait (one
//    thread per sequence), so that no CTA of the grid reads a counter it has advanced.
//  * combine_late_kernel (otherwise): everything after the wait, from the range and the append
//    record the attention pass stored; each sequence's lead thread (KV head 0) commits.
// The decode attention alone (no step) writes no counter and plans early whenever the batch
// allows.  (Measured: with thousands of segments the grid is not resident beside the pass, and
// the CTAs that start after it would do the early work on the critical path.)
// ------------------------------------------------------------------------------------
constexpr int kCombineThreads = 128;
// Early mode: when the pass gives its CTAs 16 to 128 chunks each, combine_kernel lets the next
// kernel be scheduled at its start instead of after its wait.  The next attention grid's CTAs
// then take the SM slots that this pass's CTAs free (and the spare one) and plan and prefetch
// while this pass ends; their dependency wait still covers this grid, and what they read before
// it is as before (state the immediately preceding kernel does not write; this pass, two
// launches back, writes only its own handle's scratch and outputs, which a following kernel
// touches only after its wait).  Measured per step: -2.6% (bf16) and -7% (FP8) at batch 8 x 4096
// slots, -1.5% and -4% at 8192; unconditionally it cost 18% on the 32-layer stack at batch 1
// (4 chunks a CTA) and 1.5% at batch 4 x 65536 (215 chunks a CTA), hence the window.
constexpr int kTriggerChunksMin = 16, kTriggerChunksMax = 128;
constexpr int kCombinePlanBatch = kCombineThreads;  // batches whose plan the combine computes
static_assert(kCombineThreads % 64 == 0, "a block holds whole heads of head_dim 64 or 128");

// (cos, sin) of position p for pair i: the fp64 table, or fp64 sincos past it.
__device__ __forceinline__ double2 rope_cs(const StepArgs &st, int64_t p, int half, int i) {
  if (p >= 0 && p < st.rope_positions) return st.rope_table[p * half + i];
  double s, c;
  sincos((double)p * st.inv_freq[i], &s, &c);
  return make_double2(c, s);
}

// One rotation pair at (c, s): the fp64 rotations of q and of the new key, each rounded once
// to bf16 (the stored bits), and the pair's share of the new slot's score, q.k with both turned
// in fp32 and rounded to bf16 as in the attention pass.  Not inlined (fp64 code, two callers).
struct PairTurn {
  uint16_t qc0, qc1, kc0, kc1;
  float share;
  float qr0, qr1;  // q turned in fp32 and rounded to bf16 (the pass's q)
};
__device__ __noinline__ PairTurn turn_pair(double c, double sn, uint16_t q0, uint16_t q1,
                                           uint16_t k0, uint16_t k1) {
  PairTurn r;
  const double x0 = bf16_bits_to_double(q0), x1 = bf16_bits_to_double(q1);
  r.qc0 = rotate_elem(x0, x1, c, sn, false);
  r.qc1 = rotate_elem(x1, x0, c, sn, true);
  const double y0 = bf16_bits_to_double(k0), y1 = bf16_bits_to_double(k1);
  r.kc0 = rotate_elem(y0, y1, c, sn, false);
  r.kc1 = rotate_elem(y1, y0, c, sn, true);
  const float cf = (float)c, sf = (float)sn;
  const float a0 = bf16_bits_to_float(q0), a1 = bf16_bits_to_float(q1);
  const float b0 = bf16_bits_to_float(k0), b1 = bf16_bits_to_float(k1);
  const float qr0 = __bfloat162float(__float2bfloat16_rn(a0 * cf - a1 * sf));
  const float qr1 = __bfloat162float(__float2bfloat16_rn(a1 * cf + a0 * sf));
  const float kr0 = __bfloat162float(__float2bfloat16_rn(b0 * cf - b1 * sf));
  const float kr1 = __bfloat162float(__float2bfloat16_rn(b1 * cf + b0 * sf));
  r.share = qr0 * kr0 + qr1 * kr1;
  r.qr0 = qr0;
  r.qr1 = qr1;
  return r;
}

// FP8 pools, fused step: one of the new slot's rows (the rotated key, or the value) as the
// append encodes it (encode_e4m3_row's rule: e = E - 8 of the row's largest magnitude, clamped;
// each element times 2^-e rounded to e4m3 with saturation), from the pair (x0, x1) = elements
// (i, i + D/2) each thread of a head holds.  The row maximum runs over the head's D/2 threads:
// warp shuffles, and at D = 128 the head's two warps meet in `red` (one float a warp).  Every
// thread of the block calls it (zeros where a thread has no pair).  Returns the codes, e and the
// decoded values code 2^e (exact bf16 values: the rows the cache holds).
struct Fp8Pair {
  uint8_t c0, c1;
  int e;
  float d0, d1;
};
__device__ __forceinline__ Fp8Pair fp8_encode_pair(float x0, float x1, int half, float *red) {
  float a = fmaxf(fabsf(x0), fabsf(x1));
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) a = fmaxf(a, __shfl_xor_sync(kFull, a, off));
  if (half > 32) {
    const int warp = threadIdx.x >> 5;
    if ((threadIdx.x & 31) == 0) red[warp] = a;
    __syncthreads();
    a = fmaxf(red[warp & ~1], red[warp | 1]);
    __syncthreads();
  }
  Fp8Pair r;
  r.e = 0;
  if (a > 0.f) {
    int E = 0;
    frexpf(a, &E);
    r.e = min(max(E - 8, kFp8ExpMin), kFp8ExpMax);
  }
  r.c0 = (uint8_t)__nv_cvt_float_to_fp8(ldexpf(x0, -r.e), __NV_SATFINITE, __NV_E4M3);
  r.c1 = (uint8_t)__nv_cvt_float_to_fp8(ldexpf(x1, -r.e), __NV_SATFINITE, __NV_E4M3);
  const float s = pow2i(r.e);
  r.d0 = __half2float(__half(__nv_cvt_fp8_to_halfraw(r.c0, __NV_E4M3))) * s;
  r.d1 = __half2float(__half(__nv_cvt_fp8_to_halfraw(r.c1, __NV_E4M3))) * s;
  return r;
}

// FP8 pools, fused step: the new slot's codes of this thread's pair (elements i, i + D/2) of
// KV head g's key and value rows, and (i == 0) their exponents, at slot n of page `page`.
__device__ __forceinline__ void fp8_store_pair(const AttnView &v, int page, int g, int n, int i,
                                               int half, const Fp8Pair &k, const Fp8Pair &val) {
  const int P = v.page_slots, D = 2 * half, s = n % P;
  const int64_t ph = (int64_t)page * v.n_kv_heads + g;
  uint8_t *kc = reinterpret_cast<uint8_t *>(v.step.k_pool);
  uint8_t *vc = reinterpret_cast<uint8_t *>(v.step.v_pool);
  kc[(ph * P + s) * D + i] = k.c0;
  kc[(ph * P + s) * D + i + half] = k.c1;
  const int sv = s - s % kChunkSlots + fp8_v_slot_byte(s % kChunkSlots);
  vc[(ph * D + i) * P + sv] = val.c0;
  vc[(ph * D + i + half) * P + sv] = val.c1;
  if (i == 0) {
    int8_t *e = v.step.kv_exp + (ph * (P / kChunkSlots) + s / kChunkSlots) * 32 + s % kChunkSlots;
    e[0] = (int8_t)k.e;
    e[kChunkSlots] = (int8_t)val.e;
  }
}

// The append record (n, 0 or the error that stops it, position, ntok) of a sequence from its
// slot counter, token counter and the caller's ntok / pos, as the attention pass forms it.
__device__ __forceinline__ int4 append_record(const AttnView &v, int Lraw, int64_t tokens,
                                              int t, const int32_t *pos_b) {
  const bool bad = Lraw < 0 || Lraw > v.max_slots;
  const int n = Lraw < 0 ? 0 : (bad ? v.max_slots : Lraw);
  const int why = t < 1 ? HAM_DEVERR_NTOK
                  : bad ? HAM_DEVERR_SLOTS
                  : n == v.max_slots ? HAM_DEVERR_CAPACITY : 0;
  const int64_t p = pos_b ? (int64_t)*pos_b : (v.step.pos_mode == HAM_POS_SLOT ? (int64_t)n : tokens);
  return make_int4(n, why, (int)p, t);
}

// Online merge of the partials of CTAs lo..hi for the pair (h, i), (h, i + D/2) of segment
// seg, in CTA order, kBatch partials per round trip.
template <int kBatch>
__device__ __forceinline__ void merge_partials(const AttnView &v, int seg, int h, int i,
                                               int half, int D, int lo, int hi, float &M,
                                               float &num0, float &num1, float &den) {
  const int G = v.group;
  for (int k0b = lo; k0b <= hi; k0b += kBatch) {
    float2 ml[kBatch];
    float a0[kBatch], a1[kBatch];
#pragma unroll
    for (int j = 0; j < kBatch; ++j) {
      const int64_t pi = (int64_t)k0b + j + seg;
      const bool in = k0b + j <= hi;
      const float *acc = v.part_acc + pi * G * D + (int64_t)h * D;
      ml[j] = in ? __ldcg(&v.part_ml[pi * G + h]) : make_float2(-INFINITY, 0.f);
      a0[j] = in ? __ldcg(acc + i) : 0.f;
      a1[j] = in ? __ldcg(acc + i + half) : 0.f;
    }
    float bm = M;
#pragma unroll
    for (int j = 0; j < kBatch; ++j) bm = fmaxf(bm, ml[j].x);
    const float scale = (M == -INFINITY) ? 0.f : ex2(M - bm);
    num0 *= scale;
    num1 *= scale;
    den *= scale;
#pragma unroll
    for (int j = 0; j < kBatch; ++j) {
      const float w = (ml[j].x == -INFINITY) ? 0.f : ex2(ml[j].x - bm);
      num0 += w * a0[j];
      num1 += w * a1[j];
      den += w * ml[j].y;
    }
    M = bm;
  }
}

template <typename OutT, bool kStep, int kBatch>
__global__ void __launch_bounds__(kCombineThreads) combine_kernel(const AttnView v, int D,
                                                                  int blocks_per_seg) {
  const int G = v.group, Hkv = v.n_kv_heads, half = D / 2, B = v.batch;
  const int seg = blockIdx.x / blocks_per_seg;
  const int part = blockIdx.x % blocks_per_seg;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int idx = part * kCombineThreads + tid;  // pair index within the segment
  const bool active = idx < G * half;
  const int h = idx / half, i = idx - h * half;
  const int b = seg / Hkv, g = seg - b * Hkv;
  const int64_t orow = ((int64_t)seg * G + h) * D;  // row (b, g*G + h) of q / q_rot / out
  const StepArgs &st = v.step;
  __shared__ int red[3][kCombineThreads / 32];
  __shared__ float head_sum[kCombineThreads / 32];
  __shared__ float fp8_red[kCombineThreads / 32];
  __shared__ int commit_all;  // fused step: this CTA commits every sequence
  const bool fp8 = v.kv_exp != nullptr;  // FP8 pools

  // ---- the segment's CTA range (split plan, as the attention computes it)
  int first = -1, last = -1;
  bool heavy = false;  // the same in every CTA
  int Lt = 0;  // thread t < B: the slot counter of sequence t
  {
    int nch = 0;
    if (tid < B) {
      Lt = v.num_slots[tid];
      nch = chunks_of(Lt < 0 ? 0 : (Lt > v.max_slots ? v.max_slots : Lt));
    }
    int tot = nch, pre = tid < b ? nch : 0, own = tid == b ? nch : 0;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      tot += __shfl_xor_sync(kFull, tot, off);
      pre += __shfl_xor_sync(kFull, pre, off);
      own += __shfl_xor_sync(kFull, own, off);
    }
    if (lane == 0) {
      red[0][warp] = tot;
      red[1][warp] = pre;
      red[2][warp] = own;
    }
    __syncthreads();
    int T = 0, P = 0, N = 0;
#pragma unroll
    for (int w = 0; w < kCombineThreads / 32; ++w) {
      T += red[0][w];
      P += red[1][w];
      N += red[2][w];
    }
    // A pass that streams kTriggerChunksMin..Max chunks a CTA lets the next kernel be scheduled
    // now (see above); a shorter or a longer one keeps the trigger after the wait.
    const int64_t Wt = (int64_t)Hkv * T;
    const int64_t Ct = plan_ctas(Wt, v.ctas);
    heavy = Wt > 0 && Wt >= (int64_t)kTriggerChunksMin * Ct && Wt <= (int64_t)kTriggerChunksMax * Ct;
    if (N > 0) {
      const int64_t W = (int64_t)Hkv * T;
      const int C = plan_ctas(W, v.ctas);
      const int64_t X0 = (int64_t)Hkv * P + (int64_t)g * N;
      first = plan_owner(W, C, X0);
      last = plan_owner(W, C, X0 + N - 1);
    }
  }

  if (heavy) grid_launch_dependents();

  // ---- fused step: record, rotations, q_rot and the new slot's rows; then the report
  int4 rec = make_int4(0, 0, 0, 0);
  uint16_t v0 = 0, v1 = 0;
  float vd0 = 0.f, vd1 = 0.f;  // FP8 pools: the new value pair as the cache holds it
  float dot = 0.f;
  int4 crec = make_int4(0, 0, 0, 0);  // committing CTA, thread t < B: sequence t
  int64_t ctok = 0;
  int cpage = -1;
  if constexpr (kStep) {
    uint16_t q0 = 0, q1 = 0, k0 = 0, k1 = 0;
    if (active) {  // caller inputs: final once the attention grid started
      q0 = v.q[orow + i];
      q1 = v.q[orow + i + half];
      k0 = st.k_new[(int64_t)seg * D + i];
      k1 = st.k_new[(int64_t)seg * D + i + half];
      v0 = st.v_new[(int64_t)seg * D + i];
      v1 = st.v_new[(int64_t)seg * D + i + half];
    }
    const int64_t tb = (!st.pos && st.pos_mode == HAM_POS_TOKEN) ? st.num_tokens[b] : 0;
    rec = append_record(v, v.num_slots[b], tb, st.ntok[b], st.pos ? st.pos + b : nullptr);
    float share = 0.f;
    PairTurn pt{};
    int page = -1;
    if (rec.y == 0 && active) {
      const double2 cs = rope_cs(st, rec.z, half, i);
      pt = turn_pair(cs.x, cs.y, q0, q1, k0, k1);
      share = pt.share;
      if (st.q_rot) {
        st.q_rot[orow + i] = pt.qc0;
        st.q_rot[orow + i + half] = pt.qc1;
      }
      if (h == 0) page = v.page_table[(int64_t)b * v.max_pages + rec.x / v.page_slots];
      if (h == 0 && !fp8 && page >= 0 && page < v.pool_pages) {  // the new slot's rows of head g
        const int64_t row = (((int64_t)page * Hkv + g) * v.page_slots + rec.x % v.page_slots) * D;
        st.k_pool[row + i] = pt.kc0;
        st.k_pool[row + i + half] = pt.kc1;
        st.v_pool[row + i] = v0;
        st.v_pool[row + i + half] = v1;
      }
    }
    if (fp8) {  // encode the rows as the append does; the new slot's term takes the decoded ones
      const bool mine = rec.y == 0 && active;
      const Fp8Pair kp = fp8_encode_pair(mine ? bf16_bits_to_float(pt.kc0) : 0.f,
                                         mine ? bf16_bits_to_float(pt.kc1) : 0.f, half, fp8_red);
      const Fp8Pair vp = fp8_encode_pair(mine ? bf16_bits_to_float(v0) : 0.f,
                                         mine ? bf16_bits_to_float(v1) : 0.f, half, fp8_red);
      if (mine) {
        share = pt.qr0 * kp.d0 + pt.qr1 * kp.d1;
        vd0 = vp.d0;
        vd1 = vp.d1;
        if (h == 0 && page >= 0 && page < v.pool_pages)
          fp8_store_pair(v, page, g, rec.x, i, half, kp, vp);
      }
    }
    // the score of head h: one warp at d = 64, two at d = 128 (they meet in shared memory)
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) share += __shfl_xor_sync(kFull, share, off);
    if (lane == 0) head_sum[warp] = share;
    __syncthreads();  // (also: every counter read of this CTA is consumed)
    dot = half > 32 ? head_sum[warp & ~1] + head_sum[warp | 1] : head_sum[warp];
    if (tid == 0) {  // report; the last CTA to report commits every sequence
      __threadfence();
      const bool lastcta = atomicAdd(st.arrive, 1) == (int)gridDim.x - 1;
      if (lastcta) {
        *st.arrive = 0;
        __threadfence();
      }
      commit_all = lastcta;
    }
    __syncthreads();
    if (commit_all && tid < B) {  // its record, token count and page, while the pass runs
      ctok = st.num_tokens[tid];
      crec = append_record(v, Lt, ctok, st.ntok[tid], st.pos ? st.pos + tid : nullptr);
      if (crec.y == 0) cpage = v.page_table[(int64_t)tid * v.max_pages + crec.x / v.page_slots];
    }
  }

  grid_dependency_wait();  // the attention grid's partials
  // The next kernel may be scheduled now; its own dependency wait still covers this grid.
  if (!heavy) grid_launch_dependents();

  const bool merge = first >= 0 && (kStep || first != last);
  float M = -INFINITY, num0 = 0.f, num1 = 0.f, den = 0.f;
  if (active && merge)
    merge_partials<kBatch>(v, seg, h, i, half, D, first, last, M, num0, num1, den);

  if constexpr (kStep) {
    const bool appended = rec.y == 0;
    if (appended && active) {  // the appended slot: one more term of the merge
      const float x = dot * (rsqrtf((float)D) * 1.4426950408889634f);  // log2 domain
      const float bm = fmaxf(M, x);
      const float scale = (M == -INFINITY) ? 0.f : ex2(M - bm);
      const float w = ex2(x - bm);
      num0 = num0 * scale + w * (fp8 ? vd0 : bf16_bits_to_float(v0));
      num1 = num1 * scale + w * (fp8 ? vd1 : bf16_bits_to_float(v1));
      den = den * scale + w;
    }
    if (active && (merge || appended)) {
      const float inv = den > 0.f ? 1.f / den : 0.f;
      store_out<OutT>(v.out, orow + i, num0 * inv);
      store_out<OutT>(v.out, orow + i + half, num1 * inv);
    }
    // slot metadata and counters of sequence t (committing CTA, thread t), or the error that
    // stopped its append
    if (!commit_all || tid >= B) return;
    if (crec.y != 0) {
      record_error(v.err, crec.y);
      return;
    }
    if (cpage < 0 || cpage >= v.pool_pages) {  // the pass recorded HAM_DEVERR_PAGE too
      record_error(v.err, HAM_DEVERR_PAGE);
      return;
    }
    const int64_t meta = (int64_t)cpage * v.page_slots + crec.x % v.page_slots;
    st.slot_pos[meta] = crec.z;
    st.slot_ntok[meta] = crec.w;
    st.num_slots[tid] = crec.x + 1;
    st.num_tokens[tid] = ctok + crec.w;
  } else {
    if (active && merge) {
      const float inv = den > 0.f ? 1.f / den : 0.f;  // 0: every slot masked
      store_out<OutT>(v.out, orow + i, num0 * inv);
      store_out<OutT>(v.out, orow + i + half, num1 * inv);
    }
  }
}

template <typename OutT, bool kStep>
__global__ void __launch_bounds__(kCombineThreads) combine_late_kernel(const AttnView v, int D,
                                                                       int blocks_per_seg) {
  const int G = v.group, Hkv = v.n_kv_heads, half = D / 2;
  const int seg = blockIdx.x / blocks_per_seg;
  const int part = blockIdx.x % blocks_per_seg;
  const int idx = part * kCombineThreads + threadIdx.x;  // pair index within the segment
  const bool active = idx < G * half;
  const int h = idx / half, i = idx - h * half;
  const int64_t orow = ((int64_t)seg * G + h) * D;  // row (b, g*G + h) of q / q_rot / out
  const bool fp8 = v.kv_exp != nullptr;              // FP8 pools

  grid_dependency_wait();  // the attention grid's partials, ranges and append records
  // The next kernel may be scheduled now; its own dependency wait still covers this grid.
  grid_launch_dependents();

  const int2 r = v.seg_range[seg];
  // fused step: the append record and this thread's operands, then cos/sin and the page
  int4 rec = make_int4(0, 0, 0, 0);
  uint16_t q0 = 0, q1 = 0, k0 = 0, k1 = 0, v0 = 0, v1 = 0;
  double c = 1.0, sn = 0.0;
  int page = -1;
  bool app = false;
  int64_t tokens = 0;  // lead thread: the sequence's token count before the step
  if constexpr (kStep) {
    const StepArgs &st = v.step;
    const int b = seg / Hkv;
    rec = st.stash[b];  // (n, 0 or the error that stops the append, position, ntok)
    if (idx == 0 && seg - b * Hkv == 0) tokens = st.num_tokens[b];
    app = rec.y == 0;
    if (active) {
      q0 = v.q[orow + i];
      q1 = v.q[orow + i + half];
      k0 = st.k_new[(int64_t)seg * D + i];
      k1 = st.k_new[(int64_t)seg * D + i + half];
      v0 = st.v_new[(int64_t)seg * D + i];
      v1 = st.v_new[(int64_t)seg * D + i + half];
    }
    if (app && active) {
      const int64_t p = rec.z;
      if (p >= 0 && p < st.rope_positions) {
        const double2 e = st.rope_table[p * half + i];
        c = e.x;
        sn = e.y;
      } else {
        sincos((double)p * st.inv_freq[i], &sn, &c);
      }
      if (h == 0) page = v.page_table[(int64_t)b * v.max_pages + rec.x / v.page_slots];
    }
  }
  const bool merge = r.x >= 0 && (kStep || r.x != r.y);
  float M = -INFINITY, num0 = 0.f, num1 = 0.f, den = 0.f;
  if (active && merge) merge_partials<8>(v, seg, h, i, half, D, r.x, r.y, M, num0, num1, den);

  // fused step: the exact (fp64) rotations it commits (cos/sin were loaded before the merge,
  // whose loads are therefore not held up by them)
  uint16_t qc0 = 0, qc1 = 0, kc0 = 0, kc1 = 0;
  if constexpr (kStep) {
    if (app && active) {
      if (v.step.q_rot) {
        const double x0 = bf16_bits_to_double(q0), x1 = bf16_bits_to_double(q1);
        qc0 = rotate_elem(x0, x1, c, sn, false);
        qc1 = rotate_elem(x1, x0, c, sn, true);
      }
      if (h == 0 || fp8) {  // (FP8: every head scores the new slot with the stored key)
        const double x0 = bf16_bits_to_double(k0), x1 = bf16_bits_to_double(k1);
        kc0 = rotate_elem(x0, x1, c, sn, false);
        kc1 = rotate_elem(x1, x0, c, sn, true);
      }
    }
  }

  if constexpr (kStep) {
    // Score of the appended slot for head h: the pair's share of q.k, summed over the D/2
    // threads of the head (one warp at d = 64, two at d = 128, whose sums meet in shared
    // memory).  Every thread of the block takes part, so no thread has left yet.
    __shared__ float head_sum[kCombineThreads / 32];
    __shared__ float fp8_red[kCombineThreads / 32];
    float share = 0.f, qr0 = 0.f, qr1 = 0.f;
    if (app && active) {
      const float cf = (float)c, sf = (float)sn;
      const float x0 = bf16_bits_to_float(q0), x1 = bf16_bits_to_float(q1);
      const float y0 = bf16_bits_to_float(k0), y1 = bf16_bits_to_float(k1);
      qr0 = __bfloat162float(__float2bfloat16_rn(x0 * cf - x1 * sf));
      qr1 = __bfloat162float(__float2bfloat16_rn(x1 * cf + x0 * sf));
      const float kr0 = __bfloat162float(__float2bfloat16_rn(y0 * cf - y1 * sf));
      const float kr1 = __bfloat162float(__float2bfloat16_rn(y1 * cf + y0 * sf));
      share = qr0 * kr0 + qr1 * kr1;
    }
    // FP8 pools: the rows encoded as the append encodes them; the new slot's term takes the
    // decoded ones (every thread of the block takes part in the row maxima)
    Fp8Pair kp{}, vp{};
    if (fp8) {
      const bool mine = app && active;
      kp = fp8_encode_pair(mine ? bf16_bits_to_float(kc0) : 0.f,
                           mine ? bf16_bits_to_float(kc1) : 0.f, half, fp8_red);
      vp = fp8_encode_pair(mine ? bf16_bits_to_float(v0) : 0.f,
                           mine ? bf16_bits_to_float(v1) : 0.f, half, fp8_red);
      if (mine) share = qr0 * kp.d0 + qr1 * kp.d1;
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) share += __shfl_xor_sync(kFull, share, off);
    const int warp = threadIdx.x >> 5;
    if ((threadIdx.x & 31) == 0) head_sum[warp] = share;
    __syncthreads();
    const float dot = half > 32 ? head_sum[warp & ~1] + head_sum[warp | 1] : head_sum[warp];
    if (app && active) {
      const float x = dot * (rsqrtf((float)D) * 1.4426950408889634f);  // log2 domain
      const float bm = fmaxf(M, x);
      const float scale = (M == -INFINITY) ? 0.f : ex2(M - bm);
      const float w = ex2(x - bm);
      num0 = num0 * scale + w * (fp8 ? vp.d0 : bf16_bits_to_float(v0));
      num1 = num1 * scale + w * (fp8 ? vp.d1 : bf16_bits_to_float(v1));
      den = den * scale + w;
    }
    if (active && (merge || app)) {
      const float inv = den > 0.f ? 1.f / den : 0.f;
      store_out<OutT>(v.out, orow + i, num0 * inv);
      store_out<OutT>(v.out, orow + i + half, num1 * inv);
    }

    const StepArgs &st = v.step;
    const int b = seg / Hkv, g = seg - b * Hkv;
    const bool lead = g == 0 && idx == 0;  // one thread per sequence
    if (!app) {                            // no append for this sequence
      if (lead) record_error(v.err, rec.y);
      return;
    }
    if (!active) return;
    if (st.q_rot) {
      st.q_rot[orow + i] = qc0;
      st.q_rot[orow + i + half] = qc1;
    }
    if (h != 0) return;
    if (page < 0 || page >= v.pool_pages) {  // the pass recorded HAM_DEVERR_PAGE
      if (lead) record_error(v.err, HAM_DEVERR_PAGE);
      return;
    }
    const int n = rec.x;
    if (fp8) {
      fp8_store_pair(v, page, g, n, i, half, kp, vp);
    } else {
      const int64_t row = (((int64_t)page * Hkv + g) * v.page_slots + n % v.page_slots) * D;
      st.k_pool[row + i] = kc0;
      st.k_pool[row + i + half] = kc1;
      st.v_pool[row + i] = v0;
      st.v_pool[row + i + half] = v1;
    }
    if (lead) {
      const int64_t meta = (int64_t)page * v.page_slots + n % v.page_slots;
      st.slot_pos[meta] = rec.z;
      st.slot_ntok[meta] = rec.w;
      st.num_slots[b] = n + 1;
      st.num_tokens[b] = tokens + rec.w;
    }
  } else {
    if (active && merge) {
      const float inv = den > 0.f ? 1.f / den : 0.f;  // 0: every slot masked
      store_out<OutT>(v.out, orow + i, num0 * inv);
      store_out<OutT>(v.out, orow + i + half, num1 * inv);
    }
  }
}

// Early mode: the plan fits one block (batch <= kCombinePlanBatch), and for the fused step the
// grid sits beside the attention grid (at most one CTA per SM).
inline bool combine_early(const AttnView &v, int64_t combine_ctas, bool step) {
  return v.batch <= kCombinePlanBatch && (!step || combine_ctas <= (int64_t)v.sms);
}

// Early mode's merge batch: a segment spans about ctas / segments + 1 CTAs when the lengths
// are equal, and 32 or 16 partials in flight save round trips when there are that many.
template <typename OutT, bool kStep>
cudaError_t launch_combine(const AttnView &v, int head_dim, cudaStream_t stream) {
  const int per_seg = (v.group * head_dim / 2 + kCombineThreads - 1) / kCombineThreads;
  const int64_t segs = (int64_t)v.batch * v.n_kv_heads;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)(segs * per_seg));
  cfg.blockDim = dim3(kCombineThreads);
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  if (!combine_early(v, segs * per_seg, kStep))
    return cudaLaunchKernelEx(&cfg, combine_late_kernel<OutT, kStep>, v, head_dim, per_seg);
  if ((int64_t)v.ctas >= 24 * segs)
    return cudaLaunchKernelEx(&cfg, combine_kernel<OutT, kStep, 32>, v, head_dim, per_seg);
  if ((int64_t)v.ctas >= 7 * segs)
    return cudaLaunchKernelEx(&cfg, combine_kernel<OutT, kStep, 16>, v, head_dim, per_seg);
  return cudaLaunchKernelEx(&cfg, combine_kernel<OutT, kStep, 8>, v, head_dim, per_seg);
}

// ------------------------------------------------------------------------------------
// Dispatch
// ------------------------------------------------------------------------------------
template <int D, typename OutT, bool kStep>
struct Instance {
  using S = Shape<D>;
  static auto fn() { return &decode_attn_kernel<D, OutT, kStep>; }
  static size_t smem_bytes(int group, int batch) {
    return 1024 + (size_t)Layout<D>(group, kStep, batch).total;
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
                             (int)smem_bytes(kMaxGroup, kMaxBatch));
    if (e == cudaSuccess && dev >= 0 && dev < 64) done[dev] = true;
    return e;
  }
  static cudaError_t launch(const CUtensorMap &tk, const CUtensorMap &tv, const AttnView &v,
                            cudaStream_t stream) {
    cudaError_t e = configure();
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)v.ctas);
    cfg.blockDim = dim3(S::kThreads);
    cfg.dynamicSmemBytes = smem_bytes(v.group, v.batch);
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    e = cudaLaunchKernelEx(&cfg, decode_attn_kernel<D, OutT, kStep>, tk, tv, v);
    if (e != cudaSuccess) return e;
    return launch_combine<OutT, kStep>(v, D, stream);
  }
  static int ctas_per_sm(int group, int batch) {
    if (configure() != cudaSuccess) return 0;
    int n = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, fn(), S::kThreads,
                                                      smem_bytes(group, batch)) != cudaSuccess)
      return 0;
    return n;
  }
};

template <typename OutT, bool kStep, typename F>
cudaError_t dispatch(int head_dim, F &&f) {
  if (head_dim == 128) return f(Instance<128, OutT, kStep>());
  if (head_dim == 64) return f(Instance<64, OutT, kStep>());
  return cudaErrorInvalidValue;
}

}  // namespace

bool attention_supported(int head_dim, int group) {
  return (head_dim == 64 || head_dim == 128) && group >= 1 && group <= kMaxGroup;
}

cudaError_t launch_attention(const CUtensorMap &tk, const CUtensorMap &tv, const AttnView &v,
                             int head_dim, int out_dtype, cudaStream_t stream) {
  if (v.ctas < 1 || v.group < 1 || v.group > kMaxGroup) return cudaErrorInvalidConfiguration;
  auto go = [&](auto inst) { return decltype(inst)::launch(tk, tv, v, stream); };
  if (v.kv_exp) {  // FP8 pools: the tcgen05 pass, then the same combine kernel
    if (head_dim != kFp8HeadDim) return cudaErrorInvalidValue;
    cudaError_t e = launch_fp8_attention_pass(tk, tv, v, out_dtype, false, stream);
    if (e != cudaSuccess) return e;
    return out_dtype == HAM_DTYPE_F32 ? launch_combine<float, false>(v, kFp8HeadDim, stream)
                                      : launch_combine<__nv_bfloat16, false>(v, kFp8HeadDim, stream);
  }
  return out_dtype == HAM_DTYPE_F32 ? dispatch<float, false>(head_dim, go)
                                    : dispatch<__nv_bfloat16, false>(head_dim, go);
}

cudaError_t launch_decode_step(const CUtensorMap &tk, const CUtensorMap &tv, const AttnView &v,
                               int head_dim, int out_dtype, cudaStream_t stream) {
  if (v.ctas < 1 || v.group < 1 || v.group > kMaxGroup) return cudaErrorInvalidConfiguration;
  auto go = [&](auto inst) { return decltype(inst)::launch(tk, tv, v, stream); };
  if (v.kv_exp) {  // FP8 pools: the tcgen05 pass, then the same combine kernel
    if (head_dim != kFp8HeadDim) return cudaErrorInvalidValue;
    cudaError_t e = launch_fp8_attention_pass(tk, tv, v, out_dtype, true, stream);
    if (e != cudaSuccess) return e;
    return out_dtype == HAM_DTYPE_F32 ? launch_combine<float, true>(v, kFp8HeadDim, stream)
                                      : launch_combine<__nv_bfloat16, true>(v, kFp8HeadDim, stream);
  }
  return out_dtype == HAM_DTYPE_F32 ? dispatch<float, true>(head_dim, go)
                                    : dispatch<__nv_bfloat16, true>(head_dim, go);
}

int attention_ctas_per_sm(int head_dim, int group, int batch, bool step, int out_dtype,
                          bool fp8) {
  if (fp8)
    return head_dim == kFp8HeadDim ? fp8_attention_ctas_per_sm(group, batch, step, out_dtype) : 0;
  int n = 0;
  auto q = [&](auto inst) {
    n = decltype(inst)::ctas_per_sm(group, batch);
    return cudaSuccess;
  };
  const bool f32 = out_dtype == HAM_DTYPE_F32;
  if (step) f32 ? dispatch<float, true>(head_dim, q) : dispatch<__nv_bfloat16, true>(head_dim, q);
  else f32 ? dispatch<float, false>(head_dim, q) : dispatch<__nv_bfloat16, false>(head_dim, q);
  return n;
}

cudaError_t configure_attention_instances() {
  cudaError_t e = Instance<128, __nv_bfloat16, false>::configure();
  if (e == cudaSuccess) e = Instance<64, __nv_bfloat16, false>::configure();
  if (e == cudaSuccess) e = Instance<128, float, false>::configure();
  if (e == cudaSuccess) e = Instance<64, float, false>::configure();
  return e;
}

}  // namespace ham
