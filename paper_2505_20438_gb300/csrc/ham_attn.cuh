// Pieces shared by the two decode-attention passes of libham.so: the bf16 pass (ham_attn.cu,
// mma.sync over 16-slot chunks) and the FP8 pass (ham_attn_fp8.cu, tcgen05 over 128-slot
// tiles).  Both follow the same split plan (ham_internal.cuh) and hand the same partials to the
// combine kernel in ham_attn.cu.
#pragma once

#include <cuda_bf16.h>
#include <stdint.h>

#include <type_traits>

#include "ham_internal.cuh"
#include "ham_ptx.cuh"

namespace ham {
namespace {

constexpr int kFirst = 1, kLast = 2, kPageOk = 4;  // chunk (and stage) flags
constexpr int kMaxGroup = 8;                       // query heads of a KV head

__host__ __device__ constexpr int align_up(int x, int a) { return (x + a - 1) / a * a; }

template <typename OutT>
__device__ __forceinline__ void store_out(void *out, int64_t i, float x) {
  if constexpr (std::is_same<OutT, float>::value)
    static_cast<float *>(out)[i] = x;
  else
    static_cast<__nv_bfloat16 *>(out)[i] = __float2bfloat16_rn(x);
}

// Position of the slot a fused step appends to sequence b (slot index n or tokens so far,
// unless given).
__device__ __forceinline__ int64_t step_position(const StepArgs &st, int b, int n) {
  if (st.pos) return st.pos[b];
  return st.pos_mode == HAM_POS_SLOT ? (int64_t)n : st.num_tokens[b];
}

// Positions past the fp32 (cos, sin) table: one warp fills the segment's row in shared memory
// itself (fp64 sincos rounded to fp32), so that the rotations always read the row.  A bulk copy
// may later reuse the buffer (hence the proxy fence).
__device__ __forceinline__ void fill_cs_row(float2 *cs_row, int64_t p, const double *inv_freq,
                                            int half, int lane) {
  for (int i = lane; i < half; i += 32) {
    double sd, cd;
    sincos((double)p * inv_freq[i], &sd, &cd);
    cs_row[i] = make_float2((float)cd, (float)sd);
  }
  fence_proxy_async_smem();
  __syncwarp();
}

}  // namespace
}  // namespace ham
