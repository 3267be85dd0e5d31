// Fused RoPE + append of the slot a macro-step produces (HAMburger Sec. 3.1: one KV set
// per macro-step; Sec. 3.2: the merged embedding enters at an offset position).  An FP8
// cache stores the rotated bf16 key and the value encoded as e4m3 rows with a power-of-two
// scale (encode_e4m3_row).
//
// One thread-block cluster per sequence, one CTA per KV head (or a few).  The rotation is
// computed in fp64 and rounded once to bf16 (nearest, ties to even).  cos and sin of
// p * base^(-2i/d) come from a table the host fills at allocation with libm (positions the
// cache can reach); past the table the kernel falls back to fp64 sincos.  With fp64
// operands the stored bits are the correctly rounded exact rotation except within ~1e-16
// relative of a bf16 rounding boundary, so an independent fp64 implementation reproduces
// them (and with tabled cos/sin the operands are the ones such an implementation gets).
#include <cuda_bf16.h>

#include "ham_internal.cuh"

namespace ham {
namespace {

constexpr int kAppendThreads = 64;
constexpr int kMaxHalfDim = 64;    // head_dim <= 128
constexpr int kMaxCluster = 8;     // portable thread-block cluster size
constexpr int kMaxRows = 2 * 2 + 2 * 8;  // staged rows of 128 elements: k, v, up to 8 q heads
                                          // per KV head, for up to 2 KV heads of d=64

__device__ __forceinline__ double bf16_bits_to_double(uint16_t b) {
  return (double)__uint_as_float((uint32_t)b << 16);
}

__device__ __forceinline__ uint16_t double_to_bf16_bits(double x) {
  return __bfloat16_as_ushort(__double2bfloat16(x));
}

// Rotate the pair (x[i], x[i + half]) of one row by the angle whose cos/sin are (c, s).
// Explicit _rn operations: no FMA contraction, the same operation sequence as the
// textbook formula x0 c - x1 s, x1 c + x0 s.
__device__ __forceinline__ void rotate_pair(const uint16_t *src, uint16_t *dst, int i, int half,
                                            double c, double s) {
  const double x0 = bf16_bits_to_double(src[i]);
  const double x1 = bf16_bits_to_double(src[i + half]);
  const double y0 = __dsub_rn(__dmul_rn(x0, c), __dmul_rn(x1, s));
  const double y1 = __dadd_rn(__dmul_rn(x1, c), __dmul_rn(x0, s));
  dst[i] = double_to_bf16_bits(y0);
  dst[i + half] = double_to_bf16_bits(y1);
}

// Block (b, y) handles KV heads [y * kv_per_block, ...) of sequence b and their query heads;
// the blocks of one sequence form a thread-block cluster.  Every block reads the slot
// counter, the cluster barrier orders those reads before cluster rank 0 advances it.
// Everything that does not depend on the counter (frequencies, the new k/v/q rows) is
// fetched in the same round trip as the counter, so the chain is counter -> page -> store.
__global__ void __launch_bounds__(kAppendThreads) append_kernel(AppendView v) {
  const int32_t b = blockIdx.x;
  const int d = v.head_dim, half = d / 2;
  const int G = v.n_q_heads / v.n_kv_heads;
  const int g0 = blockIdx.y * v.kv_per_block;
  const int ng = min(v.kv_per_block, v.n_kv_heads - g0);  // KV heads of this block
  __shared__ double cos_t[kMaxHalfDim], sin_t[kMaxHalfDim];
  __shared__ __align__(16) uint16_t rows[kMaxRows * 128];  // k rows, v rows, q rows
  __shared__ int32_t s_ok;
  __shared__ int64_t s_pos, s_row_meta;
  __shared__ int32_t s_n, s_ntok;

  // Library-owned constant: safe to read before the previous kernel has finished.
  const double inv_freq = threadIdx.x < half ? v.inv_freq[threadIdx.x] : 0.0;
  // Programmatic dependent launch: wait for the previous kernel (which may still read q or
  // write the counters), then let the next one start its prologue.
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

  // stage the new rows: ng k rows, ng v rows, ng*G q rows (16-byte vectors)
  const int vec = d / 8;
  uint16_t *k_s = rows, *v_s = rows + ng * d, *q_s = rows + 2 * ng * d;
  for (int i = threadIdx.x; i < ng * vec; i += blockDim.x) {
    const int64_t src = ((int64_t)b * v.n_kv_heads + g0) * d;
    reinterpret_cast<uint4 *>(k_s)[i] = reinterpret_cast<const uint4 *>(v.k_new + src)[i];
    reinterpret_cast<uint4 *>(v_s)[i] = reinterpret_cast<const uint4 *>(v.v_new + src)[i];
  }
  if (v.q) {
    const int64_t src = ((int64_t)b * v.n_q_heads + (int64_t)g0 * G) * d;
    for (int i = threadIdx.x; i < ng * G * vec; i += blockDim.x)
      reinterpret_cast<uint4 *>(q_s)[i] = reinterpret_cast<const uint4 *>(v.q + src)[i];
  }
  // every thread learns the position, so the cos/sin fetch overlaps the page lookup
  const int32_t n = v.num_slots[b];
  const int64_t p = v.pos ? (int64_t)v.pos[b] : (v.pos_mode == HAM_POS_SLOT ? (int64_t)n : v.num_tokens[b]);
  const bool tabled = p >= 0 && p < v.rope_positions;
  double2 cs_sn = make_double2(1.0, 0.0);
  if (tabled && threadIdx.x < half) cs_sn = v.rope_table[p * half + threadIdx.x];
  if (threadIdx.x == 0) {
    const int32_t t = v.ntok[b];
    int32_t err = 0;
    if (t < 1) {
      err = HAM_DEVERR_NTOK;
    } else if (n < 0 || n >= v.max_slots) {
      err = n < 0 ? HAM_DEVERR_SLOTS : HAM_DEVERR_CAPACITY;
    }
    int64_t page = -1;
    if (!err) {
      page = v.page_table[(int64_t)b * v.max_pages + n / v.page_slots];
      if (page < 0 || page >= v.pool_pages) err = HAM_DEVERR_PAGE;
    }
    if (err && blockIdx.y == 0) record_error(v.err, err);
    s_ok = err ? 0 : 1;
    s_n = n;
    s_ntok = t;
    s_pos = p;
    s_row_meta = err ? 0 : page * v.page_slots + n % v.page_slots;
  }
  // every block of the sequence has read the counters (cluster barrier, also a block barrier)
  asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory");
  asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory");
  if (!s_ok) return;
  if (blockIdx.y == 0 && threadIdx.x == 0) {
    v.slot_pos[s_row_meta] = (int32_t)s_pos;
    v.slot_ntok[s_row_meta] = s_ntok;
    v.num_slots[b] = s_n + 1;
    v.num_tokens[b] += s_ntok;
  }
  if (threadIdx.x < half) {
    if (!tabled) sincos((double)p * inv_freq, &cs_sn.y, &cs_sn.x);
    cos_t[threadIdx.x] = cs_sn.x;
    sin_t[threadIdx.x] = cs_sn.y;
  }
  __syncthreads();
  const int64_t page = s_row_meta / v.page_slots;
  const int32_t row = (int32_t)(s_row_meta % v.page_slots);
  if (v.kv_exp) {
    // FP8 pools (head_dim 128): the key is rotated and rounded to bf16 exactly as below, then
    // each row is encoded by one warp (codes, V transposed within its page, and exponents)
    // ng * (2 + G) <= kMaxRows at head_dim 128 (append_kv_per_block), G >= 1: ng <= 6
    __shared__ __align__(16) uint16_t k_rot[(kMaxRows / 3) * kFp8HeadDim];
    for (int idx = threadIdx.x; idx < ng * half; idx += blockDim.x) {
      const int j = idx / half, i = idx % half;
      rotate_pair(k_s + j * d, k_rot + j * d, i, half, cos_t[i], sin_t[i]);
    }
    __syncthreads();
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, P = v.page_slots;
    uint8_t *kc = reinterpret_cast<uint8_t *>(v.k_pool), *vc = reinterpret_cast<uint8_t *>(v.v_pool);
    for (int r = warp; r < 2 * ng; r += kAppendThreads / 32) {
      const int j = r >> 1;
      const bool is_v = (r & 1) != 0;
      const uint16_t *src = (is_v ? v_s : k_rot) + j * d + 4 * lane;
      float x[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) x[i] = __uint_as_float((uint32_t)src[i] << 16);
      uint32_t codes;
      const int e = encode_e4m3_row(x, codes);
      const int64_t ph = page * v.n_kv_heads + g0 + j;  // (page, head) block
      if (!is_v) {
        *reinterpret_cast<uint32_t *>(kc + (ph * P + row) * kFp8HeadDim + 4 * lane) = codes;
      } else {
        const int sv = row - row % kChunkSlots + fp8_v_slot_byte(row % kChunkSlots);
#pragma unroll
        for (int i = 0; i < 4; ++i)
          vc[(ph * kFp8HeadDim + 4 * lane + i) * P + sv] = (uint8_t)(codes >> (8 * i));
      }
      if (lane == 0)
        v.kv_exp[(ph * (P / kChunkSlots) + row / kChunkSlots) * 32 + (is_v ? kChunkSlots : 0) +
                 row % kChunkSlots] = (int8_t)e;
    }
  } else {
    for (int idx = threadIdx.x; idx < ng * half; idx += blockDim.x) {  // keys
      const int j = idx / half, i = idx % half;
      const int64_t dst = ((page * v.n_kv_heads + g0 + j) * v.page_slots + row) * d;
      rotate_pair(k_s + j * d, v.k_pool + dst, i, half, cos_t[i], sin_t[i]);
    }
    for (int idx = threadIdx.x; idx < ng * vec; idx += blockDim.x) {  // values, bit copy
      const int j = idx / vec, e = idx % vec;
      const int64_t dst = ((page * v.n_kv_heads + g0 + j) * v.page_slots + row) * d;
      reinterpret_cast<uint4 *>(v.v_pool + dst)[e] = reinterpret_cast<const uint4 *>(v_s + j * d)[e];
    }
  }
  if (v.q) {  // the query heads, turned at the same position, written back in place
    for (int idx = threadIdx.x; idx < ng * G * half; idx += blockDim.x) {
      const int h = idx / half, i = idx % half;
      uint16_t *dst = v.q + ((int64_t)b * v.n_q_heads + (int64_t)g0 * G + h) * d;
      rotate_pair(q_s + h * d, dst, i, half, cos_t[i], sin_t[i]);
    }
  }
}

}  // namespace

// KV heads per append block, so that one sequence's blocks fit a portable cluster and a
// block's staged rows fit its shared buffer.
int append_kv_per_block(int n_q_heads, int n_kv_heads, int head_dim) {
  const int group = n_q_heads / n_kv_heads;
  int per = (n_kv_heads + kMaxCluster - 1) / kMaxCluster;
  if (per * (2 + group) * head_dim > kMaxRows * 128) return 0;
  return per;
}

cudaError_t launch_append(const AppendView &v, cudaStream_t stream) {
  const int blocks = (v.n_kv_heads + v.kv_per_block - 1) / v.kv_per_block;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)v.batch, (unsigned)blocks);
  cfg.blockDim = dim3(kAppendThreads);
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = 1;
  attr[1].val.clusterDim.y = (unsigned)blocks;
  attr[1].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, append_kernel, v);
}

}  // namespace ham
