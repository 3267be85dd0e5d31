// Weight-streaming projections on the 5th-generation tensor cores (sm_103a), used by the
// compositional embedder (Sec. 3.2, Sec. 4.1: a multi-head cross-attention and a linear layer
// whose dense products, at decoding batches, read far more weight bytes than token bytes).
//
//   Y[s][rows][ldy] (fp32, columns 0..F-1) = X[rows][K_s] . W[F][K_s]^T,
//   K_s the s-th of `splits` column ranges of whole 64-column tiles, as even as the tile count
//   allows (the consumer sums the parts in a fixed order)
//
// One CTA per (128 output features, column range s, one or two row tiles of 128 rows: two when
// the call has more than 128 rows; a last partial tile of features or rows reads zeros past the
// matrix and stores nothing there), one CTA an SM: X is
// the A operand (its rows in the TMEM lanes), W the B operand (N = 128 features), both K-major
// 64-column tiles in the layout of the 128-byte swizzle, in two shared-memory rings.  W comes
// either pre-tiled (tile_weights: each 128 x 64 tile one contiguous, already swizzled 16 KiB
// block, moved by a 1-D bulk copy: whole DRAM pages instead of 128-byte pieces of 128 rows) or
// through a TMA tensor map; X always through a tensor map (it is small and stays in L2); an X
// stage always spans the 128 rows of the A layout, rows past the call's tile are never loaded
// and only reach accumulator rows that are never stored.  Two MMA warps take alternate k-tiles
// into two fp32 accumulators in tensor memory (one thread issues a tcgen05.mma only about
// every 125 cycles, measured on GB300).  Eight epilogue warps (two a TMEM lane quarter, one
// half of the features each) add them: a thread holds 32 consecutive features of one row,
// writes them into the (free) W ring in the 128-byte swizzle layout (no bank conflicts), and
// each warp stores its 32 x 32 boxes with TMA (whole lines; the rows past the call clip at the
// tensor's edge).  One scalar store an element (one warp a scheduler) was instruction-latency
// bound at about 4 us a CTA; 16-byte stores from a thread a row touched 32 lines an instruction
// and took about 2 us.  With programmatic dependent launch the first
// W tiles are requested before the dependency wait (they never depend on an earlier kernel); X
// only after it.  Every wait is bounded (about 2 s); a wait that runs out records
// HAM_DEVERR_TIMEOUT, lets the CTA's copies and products complete and returns.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cstring>

#include "ham_internal.cuh"
#include "ham_ptx.cuh"

namespace ham {
namespace {

constexpr int kGemmM = 128;                 // output features per CTA (the MMA's N)
constexpr int kGemmKTile = 64;              // K columns per stage: 128 bytes of a row
constexpr int kGemmWBytes = kGemmM * 128;   // a W tile
constexpr int kGemmRows = 128;              // rows per CTA (the MMA's M, TMEM lanes)
constexpr int kGemmXBytes = kGemmRows * 128;
constexpr int kGemmEpiWarp0 = 3;            // producer 0, MMA 1 and 2, epilogue 3..10
constexpr int kGemmThreads = 11 * 32;
constexpr int kGemmSmemBudget = 200 * 1024; // one CTA an SM: deep rings
constexpr uint32_t kGemmTmemCols = 256;     // two accumulators of 128 columns
constexpr int kGemmStages = 6;              // each ring: W tiles from HBM, X tiles from L2
constexpr int kGemmStages2 = 4;             // the same with two row tiles a CTA

// Row tiles a CTA: one up to 128 rows; above, two (both MMA warps then share each weight tile,
// one accumulator each), so that a call's grid stays one wave and reads the weights half as often.
inline int gemm_row_tiles(int rows) { return rows > kGemmRows ? 2 : 1; }
constexpr int gemm_smem(int stages, int rt) {
  return 1024 + stages * (kGemmWBytes + rt * kGemmXBytes) + (4 * stages + 1) * 8 + 16;
}
static_assert(gemm_smem(kGemmStages, 1) <= kGemmSmemBudget && gemm_smem(kGemmStages2, 2) <= kGemmSmemBudget,
              "rings exceed the shared-memory budget");
static_assert(kGemmStages2 * kGemmWBytes >= (kGemmM / 32) * 16384,
              "the epilogue stages a row tile's 128 x 128 fp32 boxes in the weight ring");

struct GemmPlan {
  int nt, rt, stages, smem;
};

GemmPlan gemm_plan(int rows) {
  GemmPlan p;
  p.nt = gemm_row_tile(rows);
  p.rt = gemm_row_tiles(rows);
  p.stages = p.rt == 2 ? kGemmStages2 : kGemmStages;
  p.smem = gemm_smem(p.stages, p.rt);
  return p;
}

// Byte offset of element (r, k) of a 128-row x 64-column bf16 tile in the 128-byte swizzle (the
// layout a TMA copy with that swizzle writes into 1024-byte aligned shared memory).
__device__ __forceinline__ uint32_t sw128_tile_offset(int r, int k) {
  return (uint32_t)(r * 128 + ((((k >> 3) ^ (r & 7)) & 7) << 4) + (k & 7) * 2);
}

// One thread per 16-byte piece of the tiled layout: W [F][K] row-major -> Wt
// [ceil(F/128)][ceil(K/64)][tile], zeros past the matrix.
__global__ void tile_weights_kernel(const __nv_bfloat16 *__restrict__ W, int F, int K,
                                    uint8_t *__restrict__ Wt) {
  const int kt_total = (K + kGemmKTile - 1) / kGemmKTile;
  const int64_t pieces = (int64_t)((F + kGemmM - 1) / kGemmM) * kt_total * (kGemmWBytes / 16);
  const int64_t p = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (p >= pieces) return;
  const int64_t tile = p / (kGemmWBytes / 16);
  const int in = (int)(p % (kGemmWBytes / 16));  // piece (row r, 8-column group c) of the tile
  const int r = in / 8, c = in % 8;
  const int mt = (int)(tile / kt_total), kt = (int)(tile % kt_total);
  const int row = mt * kGemmM + r, col0 = kt * kGemmKTile + 8 * c;
  uint16_t v[8];
#pragma unroll
  for (int e = 0; e < 8; ++e)
    v[e] = row < F && col0 + e < K
               ? __bfloat16_as_ushort(W[(int64_t)row * K + col0 + e])
               : (uint16_t)0;
  *reinterpret_cast<uint4 *>(Wt + tile * kGemmWBytes + sw128_tile_offset(r, 8 * c)) =
      make_uint4(v[0] | (uint32_t)v[1] << 16, v[2] | (uint32_t)v[3] << 16,
                 v[4] | (uint32_t)v[5] << 16, v[6] | (uint32_t)v[7] << 16);
}

__global__ void __launch_bounds__(kGemmThreads, 1)
    gemm_xwt_kernel(const __grid_constant__ CUtensorMap tw, const uint8_t *__restrict__ wt,
                    int kt_total, const __grid_constant__ CUtensorMap tx,
                    const __grid_constant__ CUtensorMap ty, int tma_y, float *__restrict__ Y,
                    int64_t ldy, int32_t *err, int rows, int F, int nt, int rt, int stages,
                    int pdl) {
  const int m0 = blockIdx.x * kGemmM, split = blockIdx.y, n0 = blockIdx.z * kGemmRows * rt;
  // k-tiles [kt0, kt1) of this split; columns past K read as zeros
  const int kt0 = (int)((int64_t)split * kt_total / gridDim.y);
  const int kt1 = (int)((int64_t)(split + 1) * kt_total / gridDim.y);
  const int k0 = kt0 * kGemmKTile, nk = kt1 - kt0;
  // one row tile: two accumulators for alternate k-tiles (two issuing warps) and their sum;
  // two row tiles: one accumulator a row tile, every k-tile
  const bool two = rt == 1 && nk > 1;
  const int xs = rt * kGemmXBytes;  // an X stage
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = reinterpret_cast<uint8_t *>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t *wring = smem, *xring = smem + stages * kGemmWBytes;
  uint64_t *w_full = reinterpret_cast<uint64_t *>(xring + stages * xs);
  uint64_t *w_empty = w_full + stages, *x_full = w_empty + stages;
  uint64_t *x_empty = x_full + stages, *acc_full = x_empty + stages;
  uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(acc_full + 1);
  volatile int *abort_flag = reinterpret_cast<volatile int *>(tmem_slot + 1);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  // the next kernel may be scheduled now: it waits for this grid before reading its output
  grid_launch_dependents();
  if (tid == 0) {
    for (int s = 0; s < stages; ++s) {
      mbar_init(&w_full[s], 1);
      mbar_init(&w_empty[s], rt);  // every MMA warp that reads the stage commits
      mbar_init(&x_full[s], 1);
      mbar_init(&x_empty[s], rt);
    }
    mbar_init(acc_full, 2);  // one commit per MMA warp
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    if (!wt) prefetch_tensormap(&tw);
    prefetch_tensormap(&tx);
  }
  if (warp == 1) tmem_alloc<kGemmTmemCols>(tmem_slot);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  int wi = 0, xi = 0;  // W and X tiles the producer requested

  if (warp == 0) {
    // ------------------------------------------------------------ producer (lane 0)
    if (lane == 0) {
      const uint64_t pol_w = policy_evict_first();  // each weight byte is read once a call
      const uint64_t pol_x = policy_evict_last();   // every feature tile reads the rows
      const uint8_t *wsrc =
          wt ? wt + ((int64_t)blockIdx.x * kt_total + kt0) * (int64_t)kGemmWBytes : nullptr;
      auto load_w = [&](int t, int s) {
        mbar_arrive_tx(&w_full[s], (uint32_t)kGemmWBytes);
        if (wt)
          bulk_load(wring + s * kGemmWBytes, wsrc + (int64_t)t * kGemmWBytes,
                    (uint32_t)kGemmWBytes, &w_full[s]);
        else
          tma_load_2d(wring + s * kGemmWBytes, &tw, k0 + t * kGemmKTile, m0, &w_full[s], pol_w);
      };
      // W tiles of the first stages (the whole column range when it fits) before the dependency
      // wait: they never depend on an earlier kernel
      const int wpre = min(stages, nk);
      for (int t = 0; t < wpre; ++t) load_w(t, t);
      wi = wpre;
      if (pdl) grid_dependency_wait();
      // then in k order: tile t's W (past the first stages) and X, each once its stage is free
      for (int t = 0; t < nk; ++t) {
        const int s = t % stages;
        const uint32_t par = (uint32_t)((t / stages) - 1) & 1u;
        if (t >= wpre) {
          if (!thread_wait(&w_empty[s], par, abort_flag, true)) break;
          load_w(t, s);
          wi = t + 1;
        }
        if (t >= stages && !thread_wait(&x_empty[s], par, abort_flag, true)) break;
        mbar_arrive_tx(&x_full[s], (uint32_t)(rt * nt * 128));
        for (int r = 0; r < rt; ++r)  // (a row tile past the rows reads zeros)
          tma_load_2d(xring + s * xs + r * kGemmXBytes, &tx, k0 + t * kGemmKTile,
                      n0 + r * kGemmRows, &x_full[s], pol_x);
        xi = t + 1;
      }
      if (xi < nk && !*abort_flag) {  // a wait ran out
        record_error(err, HAM_DEVERR_TIMEOUT);
        *abort_flag = 1;
      }
    }
  } else if (warp == 1 || warp == 2) {
    // ------------------------------------------------------------ MMA issue (lane 0)
    // One row tile: warp 1 the even k-tiles into columns 0..127, warp 2 the odd ones into
    // columns 128..255 (a single k-tile: warp 1 alone).  Two row tiles: warp 1 + r row tile r
    // into columns 128 r.., every k-tile.
    const int par = warp - 1;
    const int step = two ? 2 : 1;
    const uint32_t acc = tmem + (uint32_t)(par * kGemmM);
    const uint32_t idesc = idesc_bf16(kGemmRows, kGemmM, false);  // K-major X and W
    bool ok = true, first = true;
    const int t0 = rt == 2 ? 0 : two ? par : (par == 0 ? 0 : nk);
    const int xoff = rt == 2 ? par * kGemmXBytes : 0;
    for (int t = t0; t < nk; t += step) {
      const int s = t % stages;
      const uint32_t ph = (uint32_t)(t / stages) & 1u;
      if (!warp_wait(&w_full[s], ph, abort_flag) || !warp_wait(&x_full[s], ph, abort_flag)) {
        ok = false;
        break;
      }
      if (lane == 0) {
        tc_fence_after();
        const uint32_t xa = smem_u32(xring + s * xs + xoff);
        const uint32_t wa = smem_u32(wring + s * kGemmWBytes);
#pragma unroll
        for (int kk = 0; kk < kGemmKTile / 16; ++kk)
          tc_mma(acc, smem_desc_sw128(xa + kk * 32, 16, 1024),
                 smem_desc_sw128(wa + kk * 32, 16, 1024), idesc, !first || kk > 0);
        tc_commit(&w_empty[s]);
        tc_commit(&x_empty[s]);
      }
      first = false;
      __syncwarp();
    }
    if (!ok && lane == 0 && !*abort_flag) {
      record_error(err, HAM_DEVERR_TIMEOUT);
      *abort_flag = 1;
    }
    if (lane == 0) tc_commit(acc_full);  // also when nothing was issued
    __syncwarp();
  } else {
    // ------------------------------------------------------------ epilogue (warps 3-10)
    // Thread = TMEM lane = row of the row tile; the warp's half of the 128 features, 32 at a
    // time (one row tile: both accumulators added; two: each row tile's own, one after the other
    // through the same staging boxes).  tcgen05.ld is warp-collective: every lane loads, lanes
    // past the rows store nothing.
    const int quarter = warp & 3, half = (warp - kGemmEpiWarp0) >> 2;
    const uint32_t t_row = tmem + ((uint32_t)(quarter * 32) << 16);
    const bool ok = warp_wait(acc_full, 0u, abort_flag) && !__any_sync(kFull, *abort_flag != 0);
    if (ok) tc_fence_after();
    if (ok && tma_y && lane == 0) prefetch_tensormap(&ty);
    for (int rtile = 0; ok && rtile < rt; ++rtile) {
      if (rtile > 0 && tma_y) {  // the previous row tile's boxes have left the staging area
        if (lane == 0) bulk_wait_all();
        __syncwarp();
      }
      const int nb = n0 + rtile * kGemmRows;  // the row tile's first row
      const int n = nb + quarter * 32 + lane;
      const uint32_t t_acc = t_row + (uint32_t)(rtile * kGemmM);
      float *yrow = Y + ((int64_t)split * rows + n) * ldy;
      const bool vec = (ldy & 3) == 0 && (reinterpret_cast<uintptr_t>(Y) & 15u) == 0;
      for (int c0 = half * (kGemmM / 2); c0 < (half + 1) * (kGemmM / 2); c0 += 32) {
        uint32_t a[32], b[32];
        tmem_ld32(t_acc + c0, a);
        if (two) tmem_ld32(t_row + kGemmM + c0, b);
        tmem_wait_ld();
        float v[32];
#pragma unroll
        for (int j = 0; j < 32; ++j) v[j] = __uint_as_float(a[j]) + (two ? __uint_as_float(b[j]) : 0.f);
        const int f = m0 + c0;
        if (tma_y) {
          // 32 rows x 128 bytes of chunk c0 / 32, quarter `quarter`: 1024-byte aligned
          uint8_t *box = wring + (c0 / 32) * 16384 + quarter * 4096;
#pragma unroll
          for (int q = 0; q < 8; ++q)
            *reinterpret_cast<float4 *>(box + lane * 128 + ((q ^ (lane & 7)) << 4)) =
                make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0 && f < F && nb + quarter * 32 < rows) {
            tma_store_3d(&ty, box, f, nb + quarter * 32, split);
            bulk_commit_group();
          }
        } else if (n < rows && f < F) {
          if (vec && f + 32 <= F) {
            float4 *dst = reinterpret_cast<float4 *>(yrow + f);
#pragma unroll
            for (int q = 0; q < 8; ++q)
              dst[q] = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
          } else {
#pragma unroll
            for (int j = 0; j < 32; ++j)
              if (f + j < F) yrow[f + j] = v[j];
          }
        }
      }
    }
    if (ok && tma_y && lane == 0) bulk_wait_all();  // the boxes are written (and the ring read)
  }
  // the products are complete (acc_full) and the epilogue has read them: free the columns
  tc_fence_before();
  __syncthreads();
  if (warp == 0 && lane == 0 && *abort_flag) {
    // after an abort, every copy this CTA issued lands before the CTA can exit (without one,
    // the MMA warps waited for every copy)
    for (int t = max(0, wi - stages); t < wi; ++t)
      thread_wait(&w_full[t % stages], (uint32_t)(t / stages) & 1u, abort_flag, false);
    for (int t = max(0, xi - stages); t < xi; ++t)
      thread_wait(&x_full[t % stages], (uint32_t)(t / stages) & 1u, abort_flag, false);
  }
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc<kGemmTmemCols>(tmem);
  }
}

}  // namespace

int gemm_row_tile(int rows) {
  const int r = rows < kGemmRows ? rows : kGemmRows;
  const int t = ((r + 15) / 16) * 16;
  return t < 16 ? 16 : t;
}

// SMs of the current device (cached per device).
int device_sms() {
  static int sms[64] = {};
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 0 || dev >= 64) return 148;
  if (!sms[dev] && cudaDeviceGetAttribute(&sms[dev], cudaDevAttrMultiProcessorCount, dev) !=
                       cudaSuccess)
    sms[dev] = 148;
  return sms[dev];
}

// Column splits: as many CTAs as fit in one wave (one resident an SM) stream the weights, at most
// max_splits (each split is one more part to sum) and at most one split a 64-column tile.
int gemm_splits(int F, int K, int rows, int max_splits) {
  const int rpc = kGemmRows * gemm_row_tiles(rows);  // rows a CTA
  const int tiles = ((F + kGemmM - 1) / kGemmM) * ((rows + rpc - 1) / rpc);
  const int kt = (K + kGemmKTile - 1) / kGemmKTile;
  const int s = std::min(std::min(max_splits, kt), device_sms() / std::max(tiles, 1));
  return std::max(s, 1);
}

size_t tiled_weight_bytes(int F, int K) {
  return (size_t)((F + kGemmM - 1) / kGemmM) * ((K + kGemmKTile - 1) / kGemmKTile) * kGemmWBytes;
}

cudaError_t tile_weights(const void *W, int F, int K, void *Wt, cudaStream_t stream) {
  const int64_t pieces = (int64_t)tiled_weight_bytes(F, K) / 16;
  tile_weights_kernel<<<(unsigned)((pieces + 255) / 256), 256, 0, stream>>>(
      static_cast<const __nv_bfloat16 *>(W), F, K, static_cast<uint8_t *>(Wt));
  return cudaGetLastError();
}

cudaError_t launch_gemm_xwt(const CUtensorMap *tw, const void *wt, const CUtensorMap &tx,
                            float *Y, int64_t ldy, int32_t *err, int rows, int F, int K,
                            int splits, bool pdl, cudaStream_t stream) {
  if (rows < 1 || F < 1 || K < 1 || splits < 1 || ldy < F || (!tw && !wt) ||
      splits > (K + kGemmKTile - 1) / kGemmKTile || ((uintptr_t)wt & 15u))
    return cudaErrorInvalidValue;
  const GemmPlan p = gemm_plan(rows);
  static bool configured[64] = {};
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 0 || dev >= 64 || !configured[dev]) {
    cudaError_t e = cudaFuncSetAttribute(gemm_xwt_kernel,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         kGemmSmemBudget);
    if (e != cudaSuccess) return e;
    if (dev >= 0 && dev < 64) configured[dev] = true;
  }
  CUtensorMap no_map;
  memset(&no_map, 0, sizeof no_map);
  // the parts through TMA stores when their layout allows it, else plain stores
  CUtensorMap ty;
  const bool tma_y = (ldy & 3) == 0 && ((uintptr_t)Y & 15u) == 0 &&
                     make_parts_tensor_map(&ty, Y, splits, rows, F, ldy) == 0;
  if (!tma_y) ty = no_map;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)((F + kGemmM - 1) / kGemmM), (unsigned)splits,
                     (unsigned)((rows + kGemmRows * p.rt - 1) / (kGemmRows * p.rt)));
  cfg.blockDim = dim3(kGemmThreads);
  cfg.dynamicSmemBytes = (size_t)p.smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, gemm_xwt_kernel, tw ? *tw : no_map,
                            static_cast<const uint8_t *>(wt), (K + kGemmKTile - 1) / kGemmKTile,
                            tx, ty, tma_y ? 1 : 0, Y, ldy, err, rows, F, p.nt, p.rt, p.stages,
                            pdl ? 1 : 0);
}

}  // namespace ham
