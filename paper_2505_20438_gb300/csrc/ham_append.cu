// Fused RoPE + append of the slot a macro-step produces (HAMburger Sec. 3.1: one KV set
// per macro-step; Sec. 3.2: the merged embedding enters at an offset position).
//
// One CTA per sequence.  The rotation is computed in fp64 from an fp64 frequency table
// (base^(-2i/d), made on the host) and fp64 sin/cos, then rounded once to bf16
// (nearest, ties to even).  Doing the whole rotation in fp64 makes the stored bits the
// correctly rounded value of the exact rotation except within ~1e-16 relative of a bf16
// rounding boundary, so an independent fp64 implementation reproduces them.
#include <cuda_bf16.h>

#include "ham_internal.cuh"

namespace ham {
namespace {

constexpr int kAppendThreads = 256;
constexpr int kMaxHalfDim = 64;  // head_dim <= 128

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

__global__ void __launch_bounds__(kAppendThreads) append_kernel(AppendView v) {
  const int32_t b = blockIdx.x;
  const int d = v.head_dim, half = d / 2;
  __shared__ double cos_t[kMaxHalfDim], sin_t[kMaxHalfDim];
  __shared__ int32_t s_ok;
  __shared__ int64_t s_pos, s_row_meta;
  __shared__ int32_t s_n, s_ntok;

  if (threadIdx.x == 0) {
    const int32_t n = v.num_slots[b];
    const int32_t t = v.ntok[b];
    int32_t ok = 1;
    if (t < 1) {
      record_error(v.err, HAM_DEVERR_NTOK);
      ok = 0;
    } else if (n < 0 || n >= v.max_slots) {
      record_error(v.err, n < 0 ? HAM_DEVERR_SLOTS : HAM_DEVERR_CAPACITY);
      ok = 0;
    }
    int64_t page = -1;
    if (ok) {
      page = v.page_table[(int64_t)b * v.max_pages + n / v.page_slots];
      if (page < 0 || page >= v.pool_pages) {
        record_error(v.err, HAM_DEVERR_PAGE);
        ok = 0;
      }
    }
    s_ok = ok;
    s_n = n;
    s_ntok = t;
    s_pos = v.pos ? (int64_t)v.pos[b] : (v.pos_mode == HAM_POS_SLOT ? (int64_t)n : v.num_tokens[b]);
    s_row_meta = page * v.page_slots + (ok ? n % v.page_slots : 0);
  }
  __syncthreads();
  if (!s_ok) return;
  const int64_t p = s_pos;
  for (int i = threadIdx.x; i < half; i += blockDim.x) {
    double s, c;
    sincos((double)p * v.inv_freq[i], &s, &c);
    cos_t[i] = c;
    sin_t[i] = s;
  }
  __syncthreads();

  const int64_t page = s_row_meta / v.page_slots;
  const int32_t row = (int32_t)(s_row_meta % v.page_slots);
  // keys: rotate and store into the slot's rows of every KV head
  for (int idx = threadIdx.x; idx < v.n_kv_heads * half; idx += blockDim.x) {
    const int g = idx / half, i = idx % half;
    const uint16_t *src = v.k_new + ((int64_t)b * v.n_kv_heads + g) * d;
    uint16_t *dst = v.k_pool + ((page * v.n_kv_heads + g) * v.page_slots + row) * d;
    rotate_pair(src, dst, i, half, cos_t[i], sin_t[i]);
  }
  // values: bit copy in 16-byte vectors
  const int vec_per_row = d / 8;
  for (int idx = threadIdx.x; idx < v.n_kv_heads * vec_per_row; idx += blockDim.x) {
    const int g = idx / vec_per_row, e = idx % vec_per_row;
    const uint4 *src = reinterpret_cast<const uint4 *>(v.v_new + ((int64_t)b * v.n_kv_heads + g) * d);
    uint4 *dst = reinterpret_cast<uint4 *>(v.v_pool + ((page * v.n_kv_heads + g) * v.page_slots + row) * d);
    dst[e] = src[e];
  }
  // query heads of this sequence, rotated in place at the same position
  if (v.q) {
    for (int idx = threadIdx.x; idx < v.n_q_heads * half; idx += blockDim.x) {
      const int h = idx / half, i = idx % half;
      uint16_t *qh = v.q + ((int64_t)b * v.n_q_heads + h) * d;
      rotate_pair(qh, qh, i, half, cos_t[i], sin_t[i]);
    }
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    v.slot_pos[s_row_meta] = (int32_t)p;
    v.slot_ntok[s_row_meta] = s_ntok;
    v.num_slots[b] = s_n + 1;
    v.num_tokens[b] += s_ntok;
  }
}

}  // namespace

cudaError_t launch_append(const AppendView &v, cudaStream_t stream) {
  append_kernel<<<v.batch, kAppendThreads, 0, stream>>>(v);
  return cudaGetLastError();
}

}  // namespace ham
