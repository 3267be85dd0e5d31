// Micro-step attention: one step of a decoder whose per-sequence cache is a handful of slots.
//
// HAMburger's micro-step decoder (Sec. 3.3; Sec. 4.1: four layers with the base model's
// configuration) generates the tokens of a macro-step one by one, conditioned on hidden states
// of several middle layers of the base model as context.  Its attention reads only that local
// context and the micro-tokens produced so far, never the base model's cache, so its cost does
// not grow with the sequence (Sec. 3.7, the constant c of the speed-up model).  Per layer and
// micro-step the work is: rotate q and k at the new entry's position, append k and v, attend
// over at most 16 entries.  The general decode step (plan, split, combine: two launches) is
// built for caches of thousands of slots; here one kernel does everything:
//  - one CTA per (sequence, KV head); the CTAs of a sequence form a thread-block cluster, whose
//    barrier orders every CTA's read of the slot counter before rank 0 advances it;
//  - two dependent round trips to memory: the counters and the page entry together with the
//    query heads and the new key and value, then the cos/sin at the position together with the
//    old entries; the new key (rotated in fp64 from the handle's cos/sin table and rounded once
//    to bf16, the bits ham_kv_append stores) and the rotated query heads of the group are kept
//    in shared memory;
//  - a warp per query head: each lane holds head_dim / 32 elements, a dot product is a
//    5-step shuffle reduction, the softmax (fp32, exact exp) and the weighted sum of values
//    stay in registers.
#include <cuda_bf16.h>

#include "ham_micro.cuh"
#include "ham_ptx.cuh"

namespace ham {
namespace {

constexpr int kMicroThreads = 128;
constexpr int kMicroWarps = kMicroThreads / 32;

__device__ __forceinline__ float bf16_value(uint16_t b) { return __uint_as_float((uint32_t)b << 16); }
__device__ __forceinline__ double bf16_value_d(uint16_t b) { return (double)bf16_value(b); }
__device__ __forceinline__ uint16_t to_bf16_bits(double x) {
  return __bfloat16_as_ushort(__double2bfloat16(x));
}

// (x[i], x[i + half]) turned by the angle with cosine c and sine s: x0 c - x1 s, x1 c + x0 s in
// fp64 with explicit _rn operations (no contraction), rounded once to bf16.
__device__ __forceinline__ void turn_pair(const uint16_t *src, uint16_t *dst, int i, int half,
                                          double c, double s) {
  const double x0 = bf16_value_d(src[i]), x1 = bf16_value_d(src[i + half]);
  dst[i] = to_bf16_bits(__dsub_rn(__dmul_rn(x0, c), __dmul_rn(x1, s)));
  dst[i + half] = to_bf16_bits(__dadd_rn(__dmul_rn(x1, c), __dmul_rn(x0, s)));
}

template <int D>
__global__ void __launch_bounds__(kMicroThreads) micro_step_kernel(MicroView v) {
  constexpr int HALF = D / 2;
  constexpr int PER = D / 32;        // elements of a row per lane
  constexpr int VEC = D / 8;         // 16-byte pieces of a row
  const int b = blockIdx.x, g = blockIdx.y;
  const int G = v.n_q_heads / v.n_kv_heads;
  const int Hkv = v.n_kv_heads;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  __shared__ __align__(16) uint16_t ks[kMicroMaxSlots][D];
  __shared__ __align__(16) uint16_t vs[kMicroMaxSlots][D];
  __shared__ __align__(16) uint16_t qs[8][D];     // the group's query heads (turned in place)
  __shared__ __align__(16) uint16_t kn[D], vn[D]; // the new key (unrotated) and value
  __shared__ double cos_t[HALF], sin_t[HALF];
  __shared__ int32_t s_ok, s_n, s_old, s_ntok;
  __shared__ int64_t s_pos, s_page;

  grid_dependency_wait();
  grid_launch_dependents();
  // First round trip: the counters and the page entry, and (not depending on them) the query
  // heads and the new key and value.
  const uint16_t *q_src = v.q + ((int64_t)b * v.n_q_heads + (int64_t)g * G) * D;
  const int64_t kv_off = ((int64_t)b * Hkv + g) * D;
  if (threadIdx.x == 0) {
    const int32_t n = v.num_slots[b];
    const int32_t t = v.ntok[b];
    int32_t err = 0;
    if (t < 1) err = HAM_DEVERR_NTOK;
    else if (n < 0 || n >= v.max_slots) err = n < 0 ? HAM_DEVERR_SLOTS : HAM_DEVERR_CAPACITY;
    int64_t page = v.page_table[(int64_t)b * v.max_pages];   // the sequence's only page
    int32_t old = n < 0 ? 0 : (n > v.max_slots ? v.max_slots : n);
    if (page < 0 || page >= v.pool_pages) {
      if (!err) err = HAM_DEVERR_PAGE;
      page = 0;
      old = 0;   // nothing readable: the sequence attends over no slot
    }
    if (err && g == 0) record_error(v.err, err);
    s_ok = err ? 0 : 1;
    s_n = n;
    s_old = old;
    s_ntok = t;
    s_page = page;
    s_pos = v.pos ? (int64_t)v.pos[b] : (v.pos_mode == HAM_POS_SLOT ? (int64_t)n : v.num_tokens[b]);
  }
  for (int idx = threadIdx.x; idx < (G + 2) * VEC; idx += kMicroThreads) {
    const int r = idx / VEC, e = idx % VEC;
    if (r < G)
      reinterpret_cast<uint4 *>(qs[r])[e] = reinterpret_cast<const uint4 *>(q_src + r * D)[e];
    else if (r == G)
      reinterpret_cast<uint4 *>(kn)[e] = reinterpret_cast<const uint4 *>(v.k_new + kv_off)[e];
    else
      reinterpret_cast<uint4 *>(vn)[e] = reinterpret_cast<const uint4 *>(v.v_new + kv_off)[e];
  }
  __syncthreads();
  // Second round trip: cos/sin at the position, the old entries of the page.
  const bool ok = s_ok != 0;
  const int old = s_old;
  const int64_t p = s_pos;
  if (ok && threadIdx.x < HALF) {
    double c, s;
    if (p >= 0 && p < v.rope_positions) {
      const double2 t = v.rope_table[p * HALF + threadIdx.x];
      c = t.x;
      s = t.y;
    } else {
      sincos((double)p * v.inv_freq[threadIdx.x], &s, &c);
    }
    cos_t[threadIdx.x] = c;
    sin_t[threadIdx.x] = s;
  }
  const int64_t row0 = (s_page * Hkv + g) * v.page_slots;    // row of slot 0, this KV head
  for (int idx = threadIdx.x; idx < old * VEC; idx += kMicroThreads) {
    const int j = idx / VEC, e = idx % VEC;
    reinterpret_cast<uint4 *>(ks[j])[e] = reinterpret_cast<const uint4 *>(v.k_pool + (row0 + j) * D)[e];
    reinterpret_cast<uint4 *>(vs[j])[e] = reinterpret_cast<const uint4 *>(v.v_pool + (row0 + j) * D)[e];
  }
  __syncthreads();   // cos/sin ready
  if (ok) {   // turn the queries in place and the new key into its slot; copy the new value
    const int n = s_n;
    for (int idx = threadIdx.x; idx < (G + 1) * HALF; idx += kMicroThreads) {
      const int r = idx / HALF, i = idx % HALF;
      if (r < G) turn_pair(qs[r], qs[r], i, HALF, cos_t[i], sin_t[i]);
      else turn_pair(kn, ks[n], i, HALF, cos_t[i], sin_t[i]);
    }
    for (int e = threadIdx.x; e < VEC; e += kMicroThreads)
      reinterpret_cast<uint4 *>(vs[n])[e] = reinterpret_cast<const uint4 *>(vn)[e];
  }
  __syncthreads();
  if (ok) {   // the new slot's rows and the rotated queries
    const int n = s_n;
    for (int e = threadIdx.x; e < 2 * VEC; e += kMicroThreads) {
      uint16_t *pool = e < VEC ? v.k_pool : v.v_pool;
      const uint16_t *src = e < VEC ? ks[n] : vs[n];
      reinterpret_cast<uint4 *>(pool + (row0 + n) * D)[e % VEC] =
          reinterpret_cast<const uint4 *>(src)[e % VEC];
    }
    if (v.q_rot) {
      uint16_t *dst = v.q_rot + ((int64_t)b * v.n_q_heads + (int64_t)g * G) * D;
      for (int idx = threadIdx.x; idx < G * VEC; idx += kMicroThreads)
        reinterpret_cast<uint4 *>(dst)[idx] = reinterpret_cast<const uint4 *>(qs[idx / VEC])[idx % VEC];
    }
  }
  // every CTA of the sequence has read the counter: rank 0 advances it
  asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory");
  asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory");
  if (ok && g == 0 && threadIdx.x == 0) {
    const int64_t meta = s_page * v.page_slots + s_n;
    v.slot_pos[meta] = (int32_t)p;
    v.slot_ntok[meta] = s_ntok;
    v.num_slots[b] = s_n + 1;
    v.num_tokens[b] += s_ntok;
  }

  // attention of the group's query heads over the L entries, one warp per head
  const int L = ok ? s_n + 1 : old;
  const float scale = rsqrtf((float)D);
  for (int hl = warp; hl < G; hl += kMicroWarps) {
    float qv[PER];
#pragma unroll
    for (int e = 0; e < PER; ++e) qv[e] = bf16_value(qs[hl][lane * PER + e]);
    float sc[kMicroMaxSlots];
    float m = -INFINITY;
#pragma unroll
    for (int j = 0; j < kMicroMaxSlots; ++j) {
      if (j < L) {
        float part = 0.f;
#pragma unroll
        for (int e = 0; e < PER; ++e) part = fmaf(qv[e], bf16_value(ks[j][lane * PER + e]), part);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) part += __shfl_xor_sync(kFull, part, o);
        sc[j] = part * scale;
        m = fmaxf(m, sc[j]);
      }
    }
    float acc[PER];
#pragma unroll
    for (int e = 0; e < PER; ++e) acc[e] = 0.f;
    float l = 0.f;
#pragma unroll
    for (int j = 0; j < kMicroMaxSlots; ++j) {
      if (j < L) {
        const float w = expf(sc[j] - m);
        l += w;
#pragma unroll
        for (int e = 0; e < PER; ++e) acc[e] = fmaf(w, bf16_value(vs[j][lane * PER + e]), acc[e]);
      }
    }
    const float inv = L > 0 ? 1.f / l : 0.f;
    const int64_t o = ((int64_t)b * v.n_q_heads + (int64_t)g * G + hl) * D + lane * PER;
    if (v.out_f32) {
      float *dst = static_cast<float *>(v.out) + o;
#pragma unroll
      for (int e = 0; e < PER; ++e) dst[e] = acc[e] * inv;
    } else {
      uint16_t *dst = static_cast<uint16_t *>(v.out) + o;
#pragma unroll
      for (int e = 0; e < PER; ++e) dst[e] = __bfloat16_as_ushort(__float2bfloat16_rn(acc[e] * inv));
    }
  }
}

template <int D>
cudaError_t launch_d(const MicroView &v, cudaStream_t stream) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)v.batch, (unsigned)v.n_kv_heads);
  cfg.blockDim = dim3(kMicroThreads);
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = 1;
  attr[1].val.clusterDim.y = (unsigned)v.n_kv_heads;
  attr[1].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, micro_step_kernel<D>, v);
}

}  // namespace

cudaError_t launch_micro(const MicroView &v, cudaStream_t stream) {
  return v.head_dim == 64 ? launch_d<64>(v, stream) : launch_d<128>(v, stream);
}

}  // namespace ham
