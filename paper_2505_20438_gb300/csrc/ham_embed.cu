// Compositional embedder (HAMburger, arXiv 2505.20438, Sec. 3.2, Sec. 3.4, Sec. 4.1).
//
// The tokens a macro-step produced for a sequence (1..max_patch) become one hidden state of
// the model width H before the base model's next forward: a multi-head cross-attention with
// the mean of the token embeddings as its query, keys and values from the embeddings plus a
// learned embedding of each token's place in the patch, then a linear layer; one token skips
// the module.  On the GPU, four launches:
//
//  1. QKV = X [T][H] . [W_q; W_k; W_v]^T in fp32 (gemm_xwt_kernel, the tcgen05 weight-streaming
//     projection of ham_gemm.cu, in split parts that the next kernel sums).  Because the projections
//     are linear, W_q mean(x) = mean(W_q x), and W_{k,v} (x_i + P[i]) = W_{k,v} x_i + W_{k,v} P[i]:
//     the position terms KVP = [W_k; W_v] P^T are computed once when the handle is made.
//  2. fuse_kernel, one warp per (sequence, head): the mean query, k_i and v_i with their
//     position terms, the scaled scores, softmax over the patch (fp32) and o, the loads of the
//     patch a round trip a part.  o goes out as two bf16 parts, hi = bf16(o) and lo = bf16(o - hi),
//     stacked as 2B rows, so that the output projection sees about 16 bits of it.
//  3. [o_hi; o_lo] . W_o^T in fp32 (the same projection kernel over the 2B rows: the weights are
//     read once; launched with programmatic dependent launch, it requests its first W_o tiles
//     while the fusion kernel still runs).
//  4. finish_kernel: the state is the two products' sum rounded to bf16, or for a sequence of
//     one token its embedding bit for bit; a token count outside 1..max_patch (or rows outside
//     the call's tokens) gives zeros and sets the error word.
// Every launch is a programmatic dependent launch of the one before (the next call's
// projection included): it is scheduled while its predecessor runs, reads only inputs and
// weights until its dependency wait, and waits before the first read of what the predecessor
// wrote; the four are a chain of short latency-bound steps, so the overlap is most of the gain.
// The weights (4 H^2 bf16) dominate the bytes of a call: memory-bound at decoding batches,
// where the token rows are far fewer than the weight rows.
// With token ids (ham_embed_tokens) step 1 is a lookup: the projections of every vocabulary
// entry, [W_q; W_k; W_v] E[v], are tabulated once in fp32, and the fusion kernel reads the rows
// of the ids.  A call then reads W_o (H^2 bf16) and 12 H bytes per token instead of 4 H^2.
#include <cuda.h>
#include <cuda_bf16.h>

#include <cstdarg>
#include <cstdint>
#include <cstdio>
#include <algorithm>
#include <cstring>

#include "ham_internal.cuh"
#include "ham_ptx.cuh"

struct ham_embedder {
  ham_embed_config cfg{};
  int device = 0;
  CUtensorMap tmap_wkv{};        // [W_k; W_v] rows of wqkv, 128-row boxes (position terms)
  uint8_t *wqkv_t = nullptr;     // [W_q; W_k; W_v] and W_o pre-tiled for the projection kernel
  uint8_t *wo_t = nullptr;
  __nv_bfloat16 *wqkv = nullptr; // [3H][H]
  __nv_bfloat16 *wo = nullptr;   // [H][H]
  float *kvp = nullptr;          // [max_patch][2H]: W_k P[i], W_v P[i]
  int32_t vocab = 0;             // entries of the vocabulary tables (0: none set)
  __nv_bfloat16 *table_e = nullptr; // [vocab][H]: the token embeddings
  float *table_qkv = nullptr;    // [vocab][3H] fp32: [W_q; W_k; W_v] E[v]
  float *qkv = nullptr;          // [parts][rows][3H] fp32: split parts of the Q/K/V projection
  float *part2 = nullptr;        // [parts][2 batch][H] fp32: the output projection of o_hi, o_lo
  __nv_bfloat16 *o = nullptr;    // [2][batch][H]: o's hi and lo bf16 parts
  int32_t *err = nullptr;        // device error word
  int32_t *host_err = nullptr;   // pinned read-back
};

namespace ham {
namespace {

constexpr int kMaxPatch = 8;  // tokens per sequence, at most (ham_embed_config.max_patch)

int efail(int status, const char *fmt, ...) {
  char msg[256];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(msg, sizeof msg, fmt, ap);
  va_end(ap);
  return set_last_error(status, msg);
}

bool aligned16(const void *p) { return ((uintptr_t)p & 15u) == 0; }

// One warp per (sequence b, head h); lane j owns head elements j, j + 32, ... (kPer of them).
// qkv: nparts parts of [T][3H] fp32, summed here; or, with token ids, the tabulated rows
// [vocab][3H] of the ids (one part).
template <int kPer>
__global__ void __launch_bounds__(256) fuse_kernel(const float *__restrict__ qkv, int nparts,
                                                   const float *__restrict__ kvp,
                                                   const int32_t *__restrict__ offsets,
                                                   __nv_bfloat16 *__restrict__ o,
                                                   __nv_bfloat16 *__restrict__ o_lo, int32_t *err,
                                                   const int32_t *__restrict__ ids, int vocab,
                                                   int batch, int total, int H, int n_heads,
                                                   int max_patch, float scale) {
  // the output projection may be scheduled now: it reads only its weights until its dependency
  // wait, which waits for this whole grid
  grid_launch_dependents();
  // launched dependent on the Q/K/V projection: everything before the wait reads only the call's
  // inputs and the handle's tables; the wait precedes the first read of its parts
  const int warp = (int)((blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5);
  const int lane = threadIdx.x & 31;
  if (warp >= batch * n_heads) return;
  const int b = warp / n_heads, h = warp - b * n_heads;
  const int hd = kPer * 32;
  const int t0 = offsets[b], n = offsets[b + 1] - t0;
  // a sequence's rows must lie in the call's token rows, and its ids in the vocabulary
  bool bad = n < 1 || n > max_patch || t0 < 0 || t0 + n > total;
  int row[kMaxPatch];
#pragma unroll
  for (int i = 0; i < kMaxPatch; ++i) {
    row[i] = t0 + i;
    if (ids && !bad && i < n) {
      row[i] = ids[t0 + i];
      bad = bad || row[i] < 0 || row[i] >= vocab;
    }
  }
  __nv_bfloat16 *orow = o + (int64_t)b * H + (int64_t)h * hd;
  __nv_bfloat16 *lorow = o_lo + (int64_t)b * H + (int64_t)h * hd;
  if (bad || n == 1) {  // the finish kernel handles these rows; O is not used for them
    if (bad && h == 0 && lane == 0) record_error(err, HAM_DEVERR_NTOK);
#pragma unroll
    for (int e = 0; e < kPer; ++e) orow[lane + 32 * e] = lorow[lane + 32 * e] = __float2bfloat16_rn(0.f);
    return;
  }
  const int64_t ld = 3 * (int64_t)H, part = (int64_t)total * ld;
  const int64_t col = (int64_t)h * hd + lane;
  const bool tabulated = ids != nullptr;  // the tables were written when the handle was made
  // the patch's loads a round trip at a time: the position terms, then each part's q, k and v
  // rows of every token at once (the parts are added in their order)
  float qv[kMaxPatch][kPer], kv[kMaxPatch][kPer], vv[kMaxPatch][kPer];
#pragma unroll
  for (int i = 0; i < kMaxPatch; ++i) {
    const bool in = i < n;
    const float *pp = kvp + (int64_t)(in ? i : 0) * 2 * H + col;
#pragma unroll
    for (int e = 0; e < kPer; ++e) {
      qv[i][e] = 0.f;
      kv[i][e] = in ? pp[32 * e] : 0.f;
      vv[i][e] = in ? pp[H + 32 * e] : 0.f;
    }
  }
  if (!tabulated) grid_dependency_wait();
  for (int sp = 0; sp < nparts; ++sp) {
    const float *base = qkv + sp * part + col;
#pragma unroll
    for (int i = 0; i < kMaxPatch; ++i) {
      const bool in = i < n;
      const float *r = base + (int64_t)(in ? row[i] : row[0]) * ld;
#pragma unroll
      for (int e = 0; e < kPer; ++e) {
        qv[i][e] += in ? r[32 * e] : 0.f;
        kv[i][e] += in ? r[H + 32 * e] : 0.f;
        vv[i][e] += in ? r[2 * H + 32 * e] : 0.f;
      }
    }
  }
  float q[kPer];
  const float inv_n = 1.f / (float)n;
#pragma unroll
  for (int e = 0; e < kPer; ++e) {
    float sum = 0.f;
#pragma unroll
    for (int i = 0; i < kMaxPatch; ++i) sum += qv[i][e];
    q[e] = sum * inv_n;
  }
  // scores (the reductions of the patch's tokens interleave), softmax over the patch
  float s[kMaxPatch];
#pragma unroll
  for (int i = 0; i < kMaxPatch; ++i) {
    float part_s = 0.f;
#pragma unroll
    for (int e = 0; e < kPer; ++e) part_s += q[e] * kv[i][e];
    s[i] = part_s;
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1)
#pragma unroll
    for (int i = 0; i < kMaxPatch; ++i) s[i] += __shfl_xor_sync(0xffffffffu, s[i], off);
  float smax = -INFINITY;
#pragma unroll
  for (int i = 0; i < kMaxPatch; ++i)
    if (i < n) smax = fmaxf(smax, s[i] * scale);
  float den = 0.f;
#pragma unroll
  for (int i = 0; i < kMaxPatch; ++i) {
    s[i] = i < n ? expf(s[i] * scale - smax) : 0.f;
    den += s[i];
  }
  const float inv = 1.f / den;
#pragma unroll
  for (int e = 0; e < kPer; ++e) {
    float acc = 0.f;
#pragma unroll
    for (int i = 0; i < kMaxPatch; ++i) acc += s[i] * vv[i][e];
    // o as two bf16 parts, o = hi + lo to about 16 bits, for the output projection
    const float ov = acc * inv;
    const __nv_bfloat16 hi = __float2bfloat16_rn(ov);
    orow[lane + 32 * e] = hi;
    lorow[lane + 32 * e] = __float2bfloat16_rn(ov - __bfloat162float(hi));
  }
}

// out[b] = the sum of the output parts rounded to bf16; a sequence of one token gets its
// embedding bit for bit; a bad count gets zeros.  Eight elements per thread.
// With token ids, x is the vocabulary's embedding table and a token's row is its id; an id
// outside the vocabulary makes its sequence bad.
__global__ void finish_kernel(const float *__restrict__ part, int nparts,
                              const __nv_bfloat16 *__restrict__ x,
                              const int32_t *__restrict__ offsets, __nv_bfloat16 *__restrict__ out,
                              const int32_t *__restrict__ ids, int vocab, int batch, int total,
                              int H, int max_patch) {
  // the next call's projection may be scheduled now (it waits for this grid before its first
  // read of anything a call writes); launched dependent on the output projection, this kernel
  // reads the call's inputs first and waits before the first read of the parts
  grid_launch_dependents();
  const int b = blockIdx.y;
  const int j = 8 * (blockIdx.x * blockDim.x + threadIdx.x);
  if (b >= batch || j >= H) return;
  const int t0 = offsets[b], n = offsets[b + 1] - t0;
  bool bad = n < 1 || n > max_patch || t0 < 0 || t0 + n > total;
  int xrow = t0;
  if (ids && !bad) {
    xrow = ids[t0];
    for (int i = 0; i < n; ++i) {
      const int id = ids[t0 + i];
      bad = bad || id < 0 || id >= vocab;
    }
  }
  uint4 v = make_uint4(0, 0, 0, 0);
  if (!bad && n == 1) {
    v = *reinterpret_cast<const uint4 *>(x + (int64_t)xrow * H + j);
  } else if (!bad) {
    grid_dependency_wait();
    // the parts added in their order, loaded kBatch at a time (one round trip each batch)
    constexpr int kBatch = 10;
    float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
    for (int sp0 = 0; sp0 < nparts; sp0 += kBatch) {
      float4 lo[kBatch], hi[kBatch];
#pragma unroll
      for (int u = 0; u < kBatch; ++u) {
        if (sp0 + u < nparts) {
          const float4 *p = reinterpret_cast<const float4 *>(
              part + ((int64_t)(sp0 + u) * batch + b) * H + j);
          lo[u] = p[0];
          hi[u] = p[1];
        }
      }
#pragma unroll
      for (int u = 0; u < kBatch; ++u) {
        if (sp0 + u < nparts) {
          acc[0] += lo[u].x; acc[1] += lo[u].y; acc[2] += lo[u].z; acc[3] += lo[u].w;
          acc[4] += hi[u].x; acc[5] += hi[u].y; acc[6] += hi[u].z; acc[7] += hi[u].w;
        }
      }
    }
    uint32_t w[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const uint32_t lo = __bfloat16_as_ushort(__float2bfloat16_rn(acc[2 * e]));
      const uint32_t hi = __bfloat16_as_ushort(__float2bfloat16_rn(acc[2 * e + 1]));
      w[e] = lo | (hi << 16);
    }
    v = make_uint4(w[0], w[1], w[2], w[3]);
  }
  *reinterpret_cast<uint4 *>(out + (int64_t)b * H + j) = v;
}

}  // namespace
}  // namespace ham

namespace ham {
namespace {

// parts[s][rows][ldy] = X[rows][K_s] . W[n_out][K_s]^T in fp32 on the tensor cores, W pre-tiled
// (wt) or through a tensor map (tw); returns the number of parts (the K splits: `splits`, or 0
// for the kernel's choice of at most kMaxSplits), or -1 on failure.
// Split caps: each split is one more part for the fusion (Q/K/V) or finish (output) kernel to
// read; the output projection, whose weights are fewer, needs more CTAs to stream them.
constexpr int kMaxSplitsQKV = 3, kMaxSplitsOut = 4;
int project(ham_embedder *e, cudaStream_t s, const CUtensorMap *tw, const void *wt,
            const __nv_bfloat16 *X, float *parts, int rows, int n_out, int K, int64_t ldy,
            int splits, bool pdl, int max_splits = kMaxSplitsQKV) {
  CUtensorMap tx;
  if (make_matrix_tensor_map(&tx, X, rows, K, gemm_row_tile(rows)) != 0) return -1;
  const int S = splits > 0 ? splits : gemm_splits(n_out, K, rows, max_splits);
  if (launch_gemm_xwt(tw, wt, tx, parts, ldy, e->err, rows, n_out, K, S, pdl, s) != cudaSuccess)
    return -1;
  return S;
}

// Largest parts x rows of a projection of up to max_rows rows (the part buffer's size).
size_t max_part_rows(int n_out, int K, int min_rows, int max_rows, int step, int max_splits) {
  size_t best = 0;
  for (int r = min_rows; r <= max_rows; r += step)
    best = std::max(best, (size_t)gemm_splits(n_out, K, r, max_splits) * (size_t)r);
  return best;
}

// A launch with programmatic dependent launch: the kernel may start before the previous one on
// the stream ends, and waits for it (griddepcontrol.wait) before reading what it wrote.
template <typename... KArgs, typename... Args>
cudaError_t launch_dependent(void (*kernel)(KArgs...), dim3 grid, dim3 block, cudaStream_t s,
                             Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = 0;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
}

// The four launches of a call.  Without ids, xb is the call's token rows and step 1 is the
// projection GEMM; with ids, xb is the vocabulary's embedding table and the fusion kernel
// reads the tabulated projections of the ids.
int run_embed(ham_embedder *e, const __nv_bfloat16 *xb, const int32_t *ids,
              const int32_t *offsets, int32_t batch, int32_t total_tokens, void *out,
              void *stream) {
  const ham_embed_config &c = e->cfg;
  if (batch < 1 || batch > c.max_batch)
    return efail(HAM_EINVAL, "batch %d outside 1..%d", batch, c.max_batch);
  if (total_tokens < batch || total_tokens > batch * c.max_patch)
    return efail(HAM_EINVAL, "total_tokens %d outside %d..%d", total_tokens, batch,
                 batch * c.max_patch);
  if (!aligned16(out) || ((uintptr_t)offsets & 3u))
    return efail(HAM_EINVAL, "out must be 16-byte aligned, offsets 4-byte aligned");
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev != e->device) cudaSetDevice(e->device);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const int H = c.hidden, hd = H / c.n_heads;
  int rc = HAM_OK;
  __nv_bfloat16 *o_lo = e->o + (size_t)batch * H;  // rows batch..2 batch-1 of one [2B][H] block
  const float *qkv = ids ? e->table_qkv : e->qkv;
  int qkv_parts = 1;
  if (!ids) {
    qkv_parts = project(e, s, nullptr, e->wqkv_t, xb, e->qkv, total_tokens, 3 * H, H, 3 * H,
                        0, true);
    if (qkv_parts < 1) rc = efail(HAM_ECUDA, "Q/K/V projection launch failed");
  }
  if (rc == HAM_OK) {
    const int warps = batch * c.n_heads;
    const dim3 grid((unsigned)((warps + 7) / 8)), block(256);
    const float scale = 1.f / sqrtf((float)hd);
    auto fuse = hd == 32 ? fuse_kernel<1> : hd == 64 ? fuse_kernel<2> : fuse_kernel<4>;
    cudaError_t ce = launch_dependent(fuse, grid, block, s, qkv, qkv_parts, (const float *)e->kvp,
                                      offsets, e->o, o_lo, e->err, ids, (int)e->vocab, (int)batch,
                                      (int)total_tokens, H, c.n_heads, c.max_patch, scale);
    if (ce != cudaSuccess) rc = efail(HAM_ECUDA, "fuse launch: %s", cudaGetErrorString(ce));
  }
  int out_parts = 0;
  if (rc == HAM_OK) {  // o_hi and o_lo stacked as 2B rows: the weights are read once
    out_parts = project(e, s, nullptr, e->wo_t, e->o, e->part2, 2 * batch, H, H, H, 0, true,
                        kMaxSplitsOut);
    if (out_parts < 1) rc = efail(HAM_ECUDA, "output projection launch failed");
  }
  if (rc == HAM_OK) {
    const dim3 grid((unsigned)((H / 8 + 127) / 128), (unsigned)batch), block(128);
    cudaError_t ce = launch_dependent(finish_kernel, grid, block, s, (const float *)e->part2,
                                      2 * out_parts, xb, offsets,
                                      static_cast<__nv_bfloat16 *>(out), ids, (int)e->vocab,
                                      (int)batch, (int)total_tokens, H, c.max_patch);
    if (ce != cudaSuccess) rc = efail(HAM_ECUDA, "finish launch: %s", cudaGetErrorString(ce));
  }
  if (dev != e->device) cudaSetDevice(dev);
  return rc;
}

}  // namespace
}  // namespace ham

using ham::efail;

extern "C" {

int ham_embedder_free(ham_embedder *e) {
  if (!e) return HAM_OK;
  int dev = 0;
  cudaGetDevice(&dev);
  cudaSetDevice(e->device);
  cudaFree(e->wqkv);
  cudaFree(e->wo);
  cudaFree(e->wqkv_t);
  cudaFree(e->wo_t);
  cudaFree(e->kvp);
  cudaFree(e->table_e);
  cudaFree(e->table_qkv);
  cudaFree(e->qkv);
  cudaFree(e->part2);
  cudaFree(e->o);
  cudaFree(e->err);
  cudaFreeHost(e->host_err);
  cudaSetDevice(dev);
  delete e;
  return HAM_OK;
}

int ham_embedder_alloc(const ham_embed_config *cfg, const void *wq, const void *wk,
                       const void *wv, const void *wo, const void *pos, ham_embedder **out) {
  if (!cfg || !out) return efail(HAM_EINVAL, "cfg and out are required");
  *out = nullptr;
  const int H = cfg->hidden, nh = cfg->n_heads;
  if (nh < 1 || H < 1 || H % nh != 0 || H % 8 != 0)
    return efail(HAM_EINVAL, "hidden %d must be a multiple of n_heads %d and of 8", H, nh);
  const int hd = H / nh;
  if (hd != 32 && hd != 64 && hd != 128)
    return efail(HAM_EUNSUPPORTED, "head_dim %d: 32, 64 or 128", hd);
  if (cfg->max_batch < 1 || cfg->max_patch < 1 || cfg->max_patch > ham::kMaxPatch)
    return efail(HAM_EINVAL, "max_batch >= 1 and max_patch in 1..%d", ham::kMaxPatch);
  if (!wq || !wk || !wv || !wo || !pos) return efail(HAM_EINVAL, "weights are required");
  if (!ham::aligned16(wq) || !ham::aligned16(wk) || !ham::aligned16(wv) || !ham::aligned16(wo) ||
      !ham::aligned16(pos))
    return efail(HAM_EINVAL, "weights must be 16-byte aligned");
  ham_embedder *e = new ham_embedder();
  e->cfg = *cfg;
  cudaGetDevice(&e->device);
  const size_t hh = (size_t)H * H;
  const size_t rows = (size_t)cfg->max_batch * cfg->max_patch;
  cudaError_t ce = cudaSuccess;
  auto alloc = [&](void **p, size_t bytes) {
    if (ce == cudaSuccess) ce = cudaMalloc(p, bytes);
  };
  alloc(reinterpret_cast<void **>(&e->wqkv), 3 * hh * 2);
  alloc(reinterpret_cast<void **>(&e->wo), hh * 2);
  alloc(reinterpret_cast<void **>(&e->wqkv_t), ham::tiled_weight_bytes(3 * H, H));
  alloc(reinterpret_cast<void **>(&e->wo_t), ham::tiled_weight_bytes(H, H));
  alloc(reinterpret_cast<void **>(&e->kvp), (size_t)cfg->max_patch * 2 * H * 4);
  // split parts of the projections, for the largest parts x rows any call can produce
  alloc(reinterpret_cast<void **>(&e->qkv),
        ham::max_part_rows(3 * H, H, 1, (int)rows, 1, ham::kMaxSplitsQKV) * 3 * H * 4);
  alloc(reinterpret_cast<void **>(&e->part2),
        ham::max_part_rows(H, H, 2, 2 * cfg->max_batch, 2, ham::kMaxSplitsOut) * H * 4);
  alloc(reinterpret_cast<void **>(&e->o), 2 * (size_t)cfg->max_batch * H * 2);
  alloc(reinterpret_cast<void **>(&e->err), 4);
  if (ce == cudaSuccess) ce = cudaMallocHost(reinterpret_cast<void **>(&e->host_err), 4);
  if (ce != cudaSuccess) {
    cudaGetLastError();
    ham_embedder_free(e);
    return efail(HAM_ENOMEM, "embedder allocation failed");
  }
  ce = cudaMemcpy(e->wqkv, wq, hh * 2, cudaMemcpyDeviceToDevice);
  if (ce == cudaSuccess) ce = cudaMemcpy(e->wqkv + hh, wk, hh * 2, cudaMemcpyDeviceToDevice);
  if (ce == cudaSuccess) ce = cudaMemcpy(e->wqkv + 2 * hh, wv, hh * 2, cudaMemcpyDeviceToDevice);
  if (ce == cudaSuccess) ce = cudaMemcpy(e->wo, wo, hh * 2, cudaMemcpyDeviceToDevice);
  if (ce == cudaSuccess) ce = cudaMemset(e->err, 0, 4);
  if (ce != cudaSuccess) {
    cudaGetLastError();
    ham_embedder_free(e);
    return efail(HAM_ECUDA, "embedder set-up: %s", cudaGetErrorString(ce));
  }
  // the projection kernel's tiled weights, and a tensor map of [W_k; W_v] for the position terms
  int tr = ham::tile_weights(e->wqkv, 3 * H, H, e->wqkv_t, nullptr) == cudaSuccess &&
                   ham::tile_weights(e->wo, H, H, e->wo_t, nullptr) == cudaSuccess
               ? 0
               : -1;
  if (tr == 0) tr = ham::make_matrix_tensor_map(&e->tmap_wkv, e->wqkv + hh, 2 * (int64_t)H, H, 128);
  // position terms: KVP [max_patch][2H] = P [max_patch][H] . [W_k; W_v]^T (one part)
  if (tr == 0 && ham::project(e, nullptr, &e->tmap_wkv, nullptr,
                              static_cast<const __nv_bfloat16 *>(pos), e->kvp, cfg->max_patch,
                              2 * H, H, 2 * H, 1, false) != 1)
    tr = -1;
  if (tr == 0 && cudaDeviceSynchronize() != cudaSuccess) tr = -1;
  if (tr != 0) {
    cudaGetLastError();
    ham_embedder_free(e);
    return efail(HAM_ECUDA, "embedder set-up (tensor maps or position terms) failed");
  }
  *out = e;
  return HAM_OK;
}

int ham_embed(ham_embedder *e, const void *x, const int32_t *offsets, int32_t batch,
              int32_t total_tokens, void *out, void *stream) {
  ham::ApiRange nvtx_range("ham_embed");
  if (!e || !x || !offsets || !out) return efail(HAM_EINVAL, "null argument");
  if (!ham::aligned16(x)) return efail(HAM_EINVAL, "x must be 16-byte aligned");
  return ham::run_embed(e, static_cast<const __nv_bfloat16 *>(x), nullptr, offsets, batch,
                        total_tokens, out, stream);
}

int ham_embed_tokens(ham_embedder *e, const int32_t *ids, const int32_t *offsets,
                     int32_t batch, int32_t total_tokens, void *out, void *stream) {
  ham::ApiRange nvtx_range("ham_embed_tokens");
  if (!e || !ids || !offsets || !out) return efail(HAM_EINVAL, "null argument");
  if (e->vocab < 1) return efail(HAM_EINVAL, "no vocabulary set (ham_embedder_set_vocab)");
  if ((uintptr_t)ids & 3u) return efail(HAM_EINVAL, "ids must be 4-byte aligned");
  return ham::run_embed(e, e->table_e, ids, offsets, batch, total_tokens, out, stream);
}

int ham_embedder_set_vocab(ham_embedder *e, const void *table, int32_t vocab) {
  if (!e || !table) return efail(HAM_EINVAL, "null argument");
  const int H = e->cfg.hidden;
  if (vocab < 1 || (int64_t)vocab * 3 * H > INT32_MAX)
    return efail(HAM_EINVAL, "vocab %d outside 1..%lld", vocab,
                 (long long)(INT32_MAX / (3 * (int64_t)H)));
  if (!ham::aligned16(table)) return efail(HAM_EINVAL, "table must be 16-byte aligned");
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev != e->device) cudaSetDevice(e->device);
  cudaFree(e->table_e);
  cudaFree(e->table_qkv);
  e->table_e = nullptr;
  e->table_qkv = nullptr;
  e->vocab = 0;
  int rc = HAM_OK;
  cudaError_t ce = cudaMalloc(reinterpret_cast<void **>(&e->table_e), (size_t)vocab * H * 2);
  if (ce == cudaSuccess)
    ce = cudaMalloc(reinterpret_cast<void **>(&e->table_qkv), (size_t)vocab * 3 * H * 4);
  if (ce != cudaSuccess) {
    cudaGetLastError();
    rc = efail(HAM_ENOMEM, "vocabulary tables (%d entries) do not fit", vocab);
  }
  if (rc == HAM_OK) {
    ce = cudaMemcpy(e->table_e, table, (size_t)vocab * H * 2, cudaMemcpyDeviceToDevice);
    // the tabulated projections: [vocab][3H] = E [vocab][H] . [W_q; W_k; W_v]^T, fp32 (one part)
    if (ce == cudaSuccess &&
        ham::project(e, nullptr, nullptr, e->wqkv_t, e->table_e, e->table_qkv, vocab, 3 * H, H,
                     3 * H, 1, false) != 1)
      ce = cudaErrorLaunchFailure;
    if (ce == cudaSuccess) ce = cudaDeviceSynchronize();
    if (ce != cudaSuccess) {
      cudaGetLastError();
      rc = efail(HAM_ECUDA, "vocabulary tabulation: %s", cudaGetErrorString(ce));
    }
  }
  if (rc == HAM_OK) {
    e->vocab = vocab;
  } else {
    cudaFree(e->table_e);
    cudaFree(e->table_qkv);
    e->table_e = nullptr;
    e->table_qkv = nullptr;
  }
  if (dev != e->device) cudaSetDevice(dev);
  return rc;
}

int ham_embedder_status(ham_embedder *e, void *stream, int32_t *device_code) {
  if (!e) return efail(HAM_EINVAL, "null handle");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  cudaError_t ce = cudaMemcpyAsync(e->host_err, e->err, 4, cudaMemcpyDeviceToHost, s);
  if (ce == cudaSuccess) ce = cudaMemsetAsync(e->err, 0, 4, s);
  if (ce == cudaSuccess) ce = cudaStreamSynchronize(s);
  if (ce != cudaSuccess) return efail(HAM_ECUDA, "status read: %s", cudaGetErrorString(ce));
  if (device_code) *device_code = *e->host_err;
  if (*e->host_err != 0) return efail(HAM_EDEVICE, "device error word = %d", *e->host_err);
  return HAM_OK;
}

}  // extern "C"
