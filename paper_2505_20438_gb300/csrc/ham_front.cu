// Macro-step layer front: q/k/v projection of the layer input, RoPE at the new slot's position
// and the append, in one kernel (HAMburger Sec. 3.1: a macro-step is one forward of the base
// model and stores one key/value set; Sec. 3.2: it enters at an offset position; Sec. 4.1: the
// Llama base model, whose attention layers project the normalised input with bias-free
// linear maps).
//
// Decoding batches are small (a handful of sequences), so the projection is a weight stream:
// every byte of the fused weight [W_q; W_k; W_v] is read once per call and each is used for
// `batch` multiply-adds.  The kernel is bound by HBM bandwidth.  Layout of the work:
//  - a CTA owns 16 output rows of one head, chosen as the 8 rotation pairs (i, i + d/2) for
//    i = p0 .. p0+7, so that the rotation is local to the CTA (and to a thread, below);
//  - eight warps split the hidden dimension; each streams its 16 rows straight from HBM into
//    registers with 16-byte loads, U steps of 32 columns per batch of loads, and multiplies them
//    on the tensor cores (mma.m16n8k16, weights as the 16-row A operand, 8 sequences as the B
//    columns);
//  - the inner dimension is permuted consistently on both operands: a thread's 16-byte load
//    covers 8 consecutive columns, which the mma reads as columns {2t, 2t+1, 2t+8, 2t+9} of
//    two k-steps.  A dot product does not depend on the order of its terms, so no shuffle,
//    transposition or shared-memory staging is needed;
//  - a ninth warp reads the sequences' counters, token counts and pages and fetches the cos/sin
//    of the CTA's 8 frequencies at each sequence's position while the others stream, so neither
//    dependent lookup sits on a streaming warp's path;
//  - after a cross-warp sum in shared memory, the accumulator of a thread holds both elements
//    of a rotation pair for two sequences; the rotation is evaluated in fp64 from the handle's
//    fp64 cos/sin table and rounded once to bf16;
//  - every CTA reads the slot counters of its sequences; the last CTA of a grid row to finish
//    (an arrival counter) advances them, so no CTA sees a counter another has already moved.
//
// Tried and dropped (Llama-3-8B layer, batch 8): a shared-memory ring filled by per-thread
// 16-byte cp.async copies kept more bytes in flight but ran at half the speed (the copies
// throttled the load/store pipe); staging each warp's slice of x in shared memory by bulk copies
// so that the batches could be 6 steps deep was 50% slower (every CTA pulls all of x from L2 at
// once, 25 MB per call, before its first weights arrive).

#include <cuda_bf16.h>

#include "ham_front.cuh"
#include "ham_ptx.cuh"

namespace ham {
namespace {

constexpr int kFrontWarps = 8;                        // warps streaming the weights
constexpr int kFrontThreads = (kFrontWarps + 1) * 32;  // + the warp that reads the state

__device__ __forceinline__ uint4 ld_weights(const uint16_t *p) {
  return __ldcs(reinterpret_cast<const uint4 *>(p));   // streamed once: evict first
}
__device__ __forceinline__ uint4 ld_input(const uint16_t *p) {
  return __ldg(reinterpret_cast<const uint4 *>(p));
}
__device__ __forceinline__ void prefetch_l2(const void *p) {
  asm volatile("prefetch.global.L2 [%0];" ::"l"(p));
}
__device__ __forceinline__ uint16_t bf16_bits(double x) {
  return __bfloat16_as_ushort(__double2bfloat16(x));
}
__device__ __forceinline__ uint16_t bf16_bits_f(float x) {
  return __bfloat16_as_ushort(__float2bfloat16_rn(x));
}

// Rotate (a0, a1) = elements (i, i + d/2) by the angle whose cos/sin are (c, s), in fp64 with
// explicit _rn operations (no contraction): a0 c - a1 s, a1 c + a0 s.
__device__ __forceinline__ void rotate_store(float a0, float a1, double c, double s,
                                             uint16_t *dst0, uint16_t *dst1) {
  const double x0 = (double)a0, x1 = (double)a1;
  *dst0 = bf16_bits(__dsub_rn(__dmul_rn(x0, c), __dmul_rn(x1, s)));
  *dst1 = bf16_bits(__dadd_rn(__dmul_rn(x1, c), __dmul_rn(x0, s)));
}

// NT: n-tiles of 8 sequences per CTA row (1..4); U: 32-column steps whose loads are issued
// together.
template <int NT, int U>
__global__ void __launch_bounds__(kFrontThreads, NT == 1 ? 3 : 2) front_kernel(FrontView v) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int gid = lane >> 2, tig = lane & 3;
  const int d = v.head_dim, half = d >> 1;
  const int tiles_per_head = d >> 4;
  const int hh = blockIdx.x / tiles_per_head;            // fused head index
  const int p0 = (blockIdx.x % tiles_per_head) * 8;      // pairs p0 .. p0 + 7
  const int b_base = blockIdx.y * kFrontBatchTile;
  const int H = v.hidden;
  const int cols = H / kFrontWarps;                       // hidden columns of one warp
  const int steps = cols >> 5;
  const bool rotated = hh < v.n_q_heads + v.n_kv_heads;  // a q or k head

  __shared__ float red[kFrontWarps][NT * 4][32];  // cross-warp partial sums
  __shared__ double2 s_cs[NT * 8][8];            // (cos, sin) of pair p0 + j at s_pos[bl]
  __shared__ int64_t s_row[kFrontBatchTile];     // page * page_slots + slot % page_slots, -1: none
  __shared__ int64_t s_pos[kFrontBatchTile];
  __shared__ int32_t s_n[kFrontBatchTile], s_ntok[kFrontBatchTile];
  __shared__ int32_t s_last;

  if (warp == kFrontWarps) {
    // The state warp: lane t covers sequence b_base + t of this CTA row.  Every CTA of the row
    // derives the same values from the counters.
    grid_dependency_wait();
    grid_launch_dependents();
    const int b = b_base + lane;
    int64_t row = -1, p = 0;
    int32_t n = 0, t = 0;
    if (b < v.batch) {
      n = v.num_slots[b];
      t = v.ntok[b];
      int32_t err = 0;
      if (t < 1) {
        err = HAM_DEVERR_NTOK;
      } else if (n < 0) {
        err = HAM_DEVERR_SLOTS;
      } else if (n >= v.max_slots) {
        err = HAM_DEVERR_CAPACITY;
      } else {
        const int64_t page = v.page_table[(int64_t)b * v.max_pages + n / v.page_slots];
        if (page < 0 || page >= v.pool_pages) err = HAM_DEVERR_PAGE;
        else row = page * v.page_slots + n % v.page_slots;
      }
      p = v.pos ? (int64_t)v.pos[b] : (v.pos_mode == HAM_POS_SLOT ? (int64_t)n : v.num_tokens[b]);
      if (err && blockIdx.x == 0) record_error(v.err, err);
    }
    s_row[lane] = row;
    s_pos[lane] = p;
    s_n[lane] = n;
    s_ntok[lane] = t;
    if (rotated && row >= 0 && lane < NT * 8) {
      if (p >= 0 && p < v.rope_positions) {
        double2 cs[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) cs[j] = v.rope_table[p * half + p0 + j];
#pragma unroll
        for (int j = 0; j < 8; ++j) s_cs[lane][j] = cs[j];
      } else {
        for (int j = 0; j < 8; ++j) {
          double sn, cs;
          sincos((double)p * v.inv_freq[p0 + j], &sn, &cs);
          s_cs[lane][j] = make_double2(cs, sn);
        }
      }
    }
  } else {
    const int64_t col0 = (int64_t)warp * cols + tig * 8;
    const uint16_t *w_lo = v.w + ((int64_t)hh * d + p0 + gid) * H + col0;
    const uint16_t *w_hi = w_lo + (int64_t)half * H;
    // The weights are not written by kernels (a prefetch into L2 is safe in any case): pull
    // the first columns while the previous kernel on the stream finishes.
    for (int u = 0; u < U && u < steps; ++u) {
      prefetch_l2(w_lo + u * 32);
      prefetch_l2(w_hi + u * 32);
    }
    grid_dependency_wait();
    grid_launch_dependents();

    const uint16_t *x_row[NT];
    bool x_ok[NT];
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
      const int b = b_base + nt * 8 + gid;
      x_ok[nt] = b < v.batch;
      x_row[nt] = v.x + (int64_t)(x_ok[nt] ? b : 0) * H + col0;
    }
    float acc[NT][4];
#pragma unroll
    for (int nt = 0; nt < NT; ++nt)
#pragma unroll
      for (int e = 0; e < 4; ++e) acc[nt][e] = 0.f;

    const uint4 zero = make_uint4(0u, 0u, 0u, 0u);
    int s = 0;
#pragma unroll 1
    for (; s + U <= steps; s += U) {
      uint4 wa[U], wb[U], xa[U][NT];
#pragma unroll
      for (int u = 0; u < U; ++u) {
        wa[u] = ld_weights(w_lo + (s + u) * 32);
        wb[u] = ld_weights(w_hi + (s + u) * 32);
      }
#pragma unroll
      for (int u = 0; u < U; ++u)
#pragma unroll
        for (int nt = 0; nt < NT; ++nt)
          xa[u][nt] = x_ok[nt] ? ld_input(x_row[nt] + (s + u) * 32) : zero;
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const uint32_t a0[4] = {wa[u].x, wb[u].x, wa[u].y, wb[u].y};
        const uint32_t a1[4] = {wa[u].z, wb[u].z, wa[u].w, wb[u].w};
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) {
          mma_16816(acc[nt], a0, xa[u][nt].x, xa[u][nt].y);
          mma_16816(acc[nt], a1, xa[u][nt].z, xa[u][nt].w);
        }
      }
    }
#pragma unroll 1
    for (; s < steps; ++s) {   // steps not a multiple of U
      const uint4 wa = ld_weights(w_lo + s * 32), wb = ld_weights(w_hi + s * 32);
      const uint32_t a0[4] = {wa.x, wb.x, wa.y, wb.y};
      const uint32_t a1[4] = {wa.z, wb.z, wa.w, wb.w};
#pragma unroll
      for (int nt = 0; nt < NT; ++nt) {
        const uint4 xv = x_ok[nt] ? ld_input(x_row[nt] + s * 32) : zero;
        mma_16816(acc[nt], a0, xv.x, xv.y);
        mma_16816(acc[nt], a1, xv.z, xv.w);
      }
    }
#pragma unroll
    for (int nt = 0; nt < NT; ++nt)
#pragma unroll
      for (int e = 0; e < 4; ++e) red[warp][nt * 4 + e][lane] = acc[nt][e];
  }
  __syncthreads();
  // Every CTA of this row has read the counters once it gets here (the reads precede the
  // barrier above); the last one to arrive commits them after its stores.
  const bool fp8 = v.kv_exp != nullptr;
  if (threadIdx.x == 0) {
    __threadfence();
    s_last = atomicAdd(&v.arrive[blockIdx.y], 1) == (int)gridDim.x - 1;
  }

  if (warp < NT) {
    const int nt = warp;
    float c[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      float t = 0.f;
#pragma unroll
      for (int w = 0; w < kFrontWarps; ++w) t += red[w][nt * 4 + e][lane];
      c[e] = t;
    }
    // c[0], c[1]: element i of sequences bl, bl + 1; c[2], c[3]: element i + d/2 of the same
    const int i = p0 + gid;
    const int Hq = v.n_q_heads, Hkv = v.n_kv_heads;
#pragma unroll
    for (int e2 = 0; e2 < 2; ++e2) {
      const int bl = nt * 8 + tig * 2 + e2;
      const int b = b_base + bl;
      if (b >= v.batch) continue;
      const float a0 = c[e2], a1 = c[2 + e2];
      const int64_t row = s_row[bl];
      if (hh < Hq) {
        uint16_t *dst = v.q_rot + ((int64_t)b * Hq + hh) * d;
        if (row >= 0) {
          const double2 cs = s_cs[bl][gid];
          rotate_store(a0, a1, cs.x, cs.y, dst + i, dst + i + half);
        } else {  // no append for this sequence: the query stays unrotated
          dst[i] = bf16_bits_f(a0);
          dst[i + half] = bf16_bits_f(a1);
        }
      } else if (row >= 0 && fp8) {  // staged as bf16; the row's last CTA encodes it
        const int g = rotated ? hh - Hq : hh - Hq - Hkv;
        uint16_t *dst = v.stage + (((int64_t)b * Hkv + g) * 2 + (rotated ? 0 : 1)) * d;
        if (rotated) {
          const double2 cs = s_cs[bl][gid];
          rotate_store(a0, a1, cs.x, cs.y, dst + i, dst + i + half);
        } else {
          dst[i] = bf16_bits_f(a0);
          dst[i + half] = bf16_bits_f(a1);
        }
      } else if (row >= 0) {
        const int g = rotated ? hh - Hq : hh - Hq - Hkv;
        const int64_t page = row / v.page_slots, r = row % v.page_slots;
        const int64_t off = ((page * Hkv + g) * v.page_slots + r) * d;
        if (rotated) {
          const double2 cs = s_cs[bl][gid];
          rotate_store(a0, a1, cs.x, cs.y, v.k_pool + off + i, v.k_pool + off + i + half);
        } else {
          v.v_pool[off + i] = bf16_bits_f(a0);
          v.v_pool[off + i + half] = bf16_bits_f(a1);
        }
      }
    }
  }
  if (fp8) __threadfence();  // each thread's staged elements: visible to the encoding CTA
  __syncthreads();
  if (fp8 && hh >= v.n_q_heads) {
    // FP8 pools: the 8 CTAs of one key (or value) head each staged 16 elements of its rows; the
    // last of them to finish encodes the head's rows of this CTA row as ham_kv_append does
    // (encode_e4m3_row: one warp a row of 128 elements, 4 a lane; codes, V transposed within
    // its page, exponents).  Sixteen heads encode in parallel, a round trip each.
    __shared__ int32_t s_enc;
    const int Hkv = v.n_kv_heads, kv_head = hh - v.n_q_heads;  // keys 0 .. Hkv-1, then values
    int32_t *cnt = v.enc_arrive + (int64_t)blockIdx.y * 2 * Hkv + kv_head;
    if (threadIdx.x == 0) {
      __threadfence();
      s_enc = atomicAdd(cnt, 1) == tiles_per_head - 1;
    }
    __syncthreads();
    if (s_enc) {
      __threadfence();
      const bool is_v = !rotated;
      const int g = is_v ? kv_head - Hkv : kv_head, P = v.page_slots;
      const int nb = min(kFrontBatchTile, v.batch - b_base);
      uint8_t *kc = reinterpret_cast<uint8_t *>(v.k_pool);
      uint8_t *vc = reinterpret_cast<uint8_t *>(v.v_pool);
      for (int bl = warp; bl < nb; bl += kFrontWarps + 1) {
        const int64_t row = s_row[bl];
        if (row < 0) continue;  // (uniform over the warp)
        const uint16_t *src = v.stage + (((int64_t)(b_base + bl) * Hkv + g) * 2 + (is_v ? 1 : 0)) *
                                            kFp8HeadDim + 4 * lane;
        float x[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) x[e] = __uint_as_float((uint32_t)__ldcg(src + e) << 16);
        uint32_t codes;
        const int ex = encode_e4m3_row(x, codes);
        const int64_t page = row / P, sl = row % P;
        const int64_t ph = page * Hkv + g;  // (page, head) block
        if (!is_v) {
          *reinterpret_cast<uint32_t *>(kc + (ph * P + sl) * kFp8HeadDim + 4 * lane) = codes;
        } else {
          const int64_t sv = sl - sl % kChunkSlots + fp8_v_slot_byte((int)(sl % kChunkSlots));
#pragma unroll
          for (int e = 0; e < 4; ++e)
            vc[(ph * kFp8HeadDim + 4 * lane + e) * P + sv] = (uint8_t)(codes >> (8 * e));
        }
        if (lane == 0)
          v.kv_exp[(ph * (P / kChunkSlots) + sl / kChunkSlots) * 32 + (is_v ? kChunkSlots : 0) +
                   sl % kChunkSlots] = (int8_t)ex;
      }
      if (threadIdx.x == 0) *cnt = 0;  // for the next call
    }
  }
  if (s_last && threadIdx.x < kFrontBatchTile) {
    __threadfence();
    const int b = b_base + threadIdx.x;
    const int64_t row = s_row[threadIdx.x];
    if (b < v.batch && row >= 0) {
      v.slot_pos[row] = (int32_t)s_pos[threadIdx.x];
      v.slot_ntok[row] = s_ntok[threadIdx.x];
      v.num_slots[b] = s_n[threadIdx.x] + 1;
      v.num_tokens[b] += s_ntok[threadIdx.x];
    }
    if (threadIdx.x == 0) v.arrive[blockIdx.y] = 0;
  }
}

template <int NT, int U>
cudaError_t launch_nt(const FrontView &v, cudaStream_t stream) {
  cudaLaunchConfig_t cfg = {};
  const int tiles = (v.n_q_heads + 2 * v.n_kv_heads) * v.head_dim / 16;
  cfg.gridDim = dim3((unsigned)tiles, (unsigned)((v.batch + kFrontBatchTile - 1) / kFrontBatchTile));
  cfg.blockDim = dim3(kFrontThreads);
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, front_kernel<NT, U>, v);
}

}  // namespace

cudaError_t launch_front(const FrontView &v, cudaStream_t stream) {
  const int rows = v.batch < kFrontBatchTile ? v.batch : kFrontBatchTile;
  switch ((rows + 7) / 8) {
    case 1: return launch_nt<1, 4>(v, stream);
    case 2: return launch_nt<2, 4>(v, stream);
    case 3: return launch_nt<3, 2>(v, stream);
    default: return launch_nt<4, 2>(v, stream);
  }
}

}  // namespace ham
