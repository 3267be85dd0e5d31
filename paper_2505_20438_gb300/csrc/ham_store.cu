// Paged smashed-KV store: allocation, page tables, counters, fill/export and the C ABI
// entry points that are not kernels of the decode path.
//
// A macro-step of HAMburger stores one KV set for all tokens it fused (Sec. 3.1, Sec. 3.7
// "Token Fusion"), so the store is a per-sequence list of slots, each with the position it
// was rotated at (Sec. 3.2) and its token count.
#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <map>
#include <mutex>
#include <utility>
#include <vector>

#include "ham_internal.cuh"
#include "ham_front.cuh"
#include "ham_micro.cuh"
#include "ham_prefill.cuh"

namespace {

thread_local char g_last_error[512] = "";

int fail(int status, const char *fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_last_error, sizeof g_last_error, fmt, ap);
  va_end(ap);
  return status;
}

int cuda_fail(cudaError_t e, const char *what) {
  return fail(HAM_ECUDA, "%s: %s", what, cudaGetErrorString(e));
}

#define HAM_CUDA(call)                                   \
  do {                                                   \
    cudaError_t e_ = (call);                             \
    if (e_ != cudaSuccess) return cuda_fail(e_, #call);  \
  } while (0)

bool aligned16(const void *p) { return ((uintptr_t)p & 15u) == 0; }

size_t round_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

uint64_t splitmix64(uint64_t &s) {
  uint64_t z = (s += 0x9E3779B97F4A7C15ull);
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

// Page ids of every sequence: sequential for seed 0, else the first batch*max_pages ids of
// a seeded Fisher-Yates shuffle of the pool.
std::vector<int32_t> reserve_pages(int32_t batch, int32_t max_pages, int64_t pool_pages,
                                   uint64_t seed) {
  std::vector<int32_t> ids((size_t)pool_pages);
  for (int64_t i = 0; i < pool_pages; ++i) ids[(size_t)i] = (int32_t)i;
  if (seed != 0) {
    uint64_t s = seed;
    for (int64_t i = pool_pages - 1; i > 0; --i) {
      int64_t j = (int64_t)(splitmix64(s) % (uint64_t)(i + 1));
      std::swap(ids[(size_t)i], ids[(size_t)j]);
    }
  }
  ids.resize((size_t)batch * (size_t)max_pages);
  return ids;
}

int check_layer(const ham_kv *kv, int32_t layer) {
  if (!kv) return fail(HAM_EINVAL, "null handle");
  if (layer < 0 || layer >= kv->cfg.layers)
    return fail(HAM_EINVAL, "layer %d outside [0, %d)", layer, kv->cfg.layers);
  return HAM_OK;
}

// Run host code on the handle's device, restoring the caller's device afterwards.
struct DeviceGuard {
  int prev = -1;
  explicit DeviceGuard(int dev) {
    if (cudaGetDevice(&prev) == cudaSuccess && prev != dev) cudaSetDevice(dev);
    else prev = -1;
  }
  ~DeviceGuard() {
    if (prev >= 0) cudaSetDevice(prev);
  }
};

int64_t pool_rows(const ham_kv *kv) {
  return kv->cfg.pool_pages * kv->cfg.n_kv_heads * (int64_t)kv->cfg.page_slots;
}

// The K (which 0) or V (1) pool of a layer: bf16 elements, or for FP8 pools the code block
// (uint8, behind a uint16_t pointer that nothing dereferences as bf16).
uint16_t *layer_pool(const ham_kv *kv, int32_t layer, int which) {
  if (kv->fp8) {
    const ham::Fp8Layer f = ham::fp8_layer(kv->pool, pool_rows(kv), layer);
    return reinterpret_cast<uint16_t *>(which ? f.v : f.k);
  }
  return kv->pool + ((size_t)layer * 2 + (size_t)which) * (size_t)kv->pool_elems;
}
int8_t *layer_exp(const ham_kv *kv, int32_t layer) {
  return kv->fp8 ? ham::fp8_layer(kv->pool, pool_rows(kv), layer).e : nullptr;
}
// Bytes of one layer's pools.
size_t layer_pool_bytes(const ham_kv *kv) {
  return kv->fp8 ? ham::fp8_layer_bytes(pool_rows(kv))
                 : 2 * (size_t)kv->pool_elems * sizeof(uint16_t);
}
int fp8_unsupported(const ham_kv *kv, const char *call) {
  return kv->fp8 ? fail(HAM_EUNSUPPORTED, "%s: not available for an FP8 (e4m3) cache", call) : 0;
}

// ---------------------------------------------------------------------------------------
// Early start.  The attention kernels are launched with programmatic dependent launch and can
// read their layer's counters, page table and pools before their dependency wait, which lets
// the plan and the first K/V copies overlap the previous kernel, provided that kernel does not
// write them.  Every kernel of this library waits for its own predecessor before letting its
// successor start, so when an attention grid starts, everything before the immediately
// preceding kernel has completed; only that kernel may still run.  The library remembers, per
// stream (and per stream capture), the last launch it made and which (handle, layer) state it
// writes, and allows the early start only when that launch is known and leaves this layer
// alone.  Kernels of other code in between are harmless: they cannot write a handle's state
// (only these calls do), and an unknown predecessor means no early start.
// ---------------------------------------------------------------------------------------
struct LastLaunch {
  const ham_kv *kv;
  int32_t layer;  // -1: every layer
  bool writes;    // wrote the layer's counters, pools or slot metadata
};
std::mutex g_launch_mu;
std::map<std::pair<uintptr_t, unsigned long long>, LastLaunch> g_last_launch;

std::pair<uintptr_t, unsigned long long> launch_key(void *stream) {
  cudaStreamCaptureStatus st = cudaStreamCaptureStatusNone;
  unsigned long long id = 0;
  if (cudaStreamGetCaptureInfo(static_cast<cudaStream_t>(stream), &st, &id) != cudaSuccess) {
    cudaGetLastError();
    id = ~0ull;  // unknown: gets its own (always conservative) entry
  } else if (st != cudaStreamCaptureStatusActive) {
    id = 0;
  }
  return {(uintptr_t)stream, id};
}

bool may_start_early(const ham_kv *kv, int32_t layer, void *stream) {
  const auto key = launch_key(stream);
  std::lock_guard<std::mutex> lock(g_launch_mu);
  const auto it = g_last_launch.find(key);
  if (it == g_last_launch.end()) return false;
  const LastLaunch &l = it->second;
  return !(l.kv == kv && l.writes && (l.layer == layer || l.layer < 0));
}

void note_launch(const ham_kv *kv, int32_t layer, void *stream, bool writes) {
  const auto key = launch_key(stream);
  std::lock_guard<std::mutex> lock(g_launch_mu);
  if (g_last_launch.size() > 4096) g_last_launch.clear();  // forgetting is always safe
  g_last_launch[key] = LastLaunch{kv, layer, writes};
}

// Byte offsets of everything ham_kv_alloc carves out of the handle's metadata allocation (each
// piece 256-byte aligned).  Recomputed from the configuration where a call needs a piece the
// handle keeps no pointer to.
struct MetaLayout {
  size_t pos, ntok, pt, ns, nt, inv_freq, err, acc, ml, sr, stash, arrive, pf_seq, pf_pos;
  size_t pf_part, pf_ml;  // ham_prefill's split partials (bf16 caches; empty for FP8)
  size_t front_stage;     // ham_qkv_append on FP8 caches: the new rows as bf16 (else empty)
  size_t front_enc;       // ... and the per-head arrival counters of its encoding
  size_t front;   // ham_qkv_append: one arrival counter per grid row
  size_t total;
};

MetaLayout meta_layout(const ham_config &cfg, int32_t max_ctas, int64_t max_pages) {
  const int group = cfg.n_q_heads / cfg.n_kv_heads;
  const size_t slots_meta = (size_t)cfg.pool_pages * cfg.page_slots * sizeof(int32_t);
  const size_t n_seg = (size_t)cfg.batch * cfg.n_kv_heads;
  const size_t n_part = (size_t)max_ctas + n_seg;
  size_t off = 0;
  auto carve = [&](size_t bytes) {
    size_t at = off;
    off = round_up(off + bytes, 256);
    return at;
  };
  MetaLayout m{};
  m.pos = carve(slots_meta);
  m.ntok = carve(slots_meta);
  m.pt = carve((size_t)cfg.batch * (size_t)max_pages * sizeof(int32_t));
  m.ns = carve((size_t)cfg.layers * cfg.batch * sizeof(int32_t));
  m.nt = carve((size_t)cfg.layers * cfg.batch * sizeof(int64_t));
  m.inv_freq = carve((size_t)(cfg.head_dim / 2) * sizeof(double));
  m.err = carve(sizeof(int32_t));
  m.acc = carve(n_part * group * cfg.head_dim * sizeof(float));
  m.ml = carve(n_part * group * sizeof(float2));
  m.sr = carve(n_seg * sizeof(int2));
  m.stash = carve((size_t)cfg.batch * sizeof(int4));
  m.arrive = carve(sizeof(int32_t));
  m.pf_seq = carve((size_t)cfg.batch * sizeof(int4));
  m.pf_pos = carve((size_t)cfg.batch * cfg.max_slots_per_seq * sizeof(int2));
  {  // (max_ctas is 8 x the SMs)
    const bool fp8 = cfg.kv_dtype == HAM_KV_E4M3;
    const size_t floats = fp8 ? 0 : ham::prefill_part_floats(max_ctas / 8, cfg.head_dim);
    m.pf_part = carve(floats * sizeof(float));
    m.pf_ml = carve(floats / (size_t)cfg.head_dim * sizeof(float2));
  }
  m.front = carve((size_t)ham::kFrontMaxRows * sizeof(int32_t));
  m.front_stage = carve(cfg.kv_dtype == HAM_KV_E4M3
                            ? (size_t)cfg.batch * cfg.n_kv_heads * 2 * cfg.head_dim * sizeof(uint16_t)
                            : 0);
  m.front_enc = carve(cfg.kv_dtype == HAM_KV_E4M3
                          ? (size_t)ham::kFrontMaxRows * 2 * cfg.n_kv_heads * sizeof(int32_t)
                          : 0);
  m.total = off;
  return m;
}

}  // namespace

// ------------------------------------------------------------------------------------
// fill kernel (test and bench set-up: logical cache -> pages)
// ------------------------------------------------------------------------------------
namespace ham {

int set_last_error(int status, const char *msg) { return fail(status, "%s", msg); }

__global__ void fill_rows_kernel(FillView v) {
  const int32_t b = blockIdx.y;
  const int32_t count = v.counts[b];
  if (count < 0 || count > v.lmax || count > v.max_slots) return;  // reported by fill_meta
  const int vec_per_row = v.head_dim / 8;  // 16-byte vectors per (slot, KV head) row
  const int64_t vec_per_slot = (int64_t)v.n_kv_heads * vec_per_row;
  const int64_t first = (int64_t)blockIdx.x * 16;  // 16 slots per block
  for (int64_t idx = threadIdx.x; idx < 16 * vec_per_slot; idx += blockDim.x) {
    const int64_t j = first + idx / vec_per_slot;
    if (j >= count) continue;
    const int32_t g = (int32_t)((idx % vec_per_slot) / vec_per_row);
    const int32_t e = (int32_t)(idx % vec_per_row);
    const int32_t page = v.page_table[(int64_t)b * v.max_pages + j / v.page_slots];
    if (page < 0 || page >= v.pool_pages) {
      record_error(v.err, HAM_DEVERR_PAGE);
      continue;
    }
    const int64_t dst = (((int64_t)page * v.n_kv_heads + g) * v.page_slots + j % v.page_slots) *
                        v.head_dim / 8 + e;
    const int64_t src = (((int64_t)b * v.lmax + j) * v.n_kv_heads + g) * vec_per_row + e;
    reinterpret_cast<uint4 *>(v.k_pool)[dst] = reinterpret_cast<const uint4 *>(v.k_log)[src];
    reinterpret_cast<uint4 *>(v.v_pool)[dst] = reinterpret_cast<const uint4 *>(v.v_log)[src];
  }
}

// FP8 pools: one warp per (sequence b, slot j, KV head g) row pair; the K and the V row are
// each encoded (encode_e4m3_row) and stored as codes (V transposed within its page) and
// exponents.  Blocks of 8 warps; grid (ceil(lmax * Hkv / 8), batch).
__global__ void fill_rows_fp8_kernel(FillView v) {
  const int32_t b = blockIdx.y;
  const int32_t count = v.counts[b];
  if (count < 0 || count > v.lmax || count > v.max_slots) return;  // reported by fill_meta
  const int lane = threadIdx.x & 31;
  const int64_t r = (int64_t)blockIdx.x * (blockDim.x / 32) + threadIdx.x / 32;
  const int32_t j = (int32_t)(r / v.n_kv_heads), g = (int32_t)(r % v.n_kv_heads);
  if (j >= count) return;
  const int32_t page = v.page_table[(int64_t)b * v.max_pages + j / v.page_slots];
  if (page < 0 || page >= v.pool_pages) {
    if (lane == 0) record_error(v.err, HAM_DEVERR_PAGE);
    return;
  }
  const int P = v.page_slots, s = j % P;
  const int64_t src = (((int64_t)b * v.lmax + j) * v.n_kv_heads + g) * kFp8HeadDim + 4 * lane;
  const int64_t ph = (int64_t)page * v.n_kv_heads + g;  // (page, head) block
  float xk[4], xv[4];
  const uint2 kb = *reinterpret_cast<const uint2 *>(v.k_log + src);
  const uint2 vb = *reinterpret_cast<const uint2 *>(v.v_log + src);
  xk[0] = __uint_as_float(kb.x << 16); xk[1] = __uint_as_float(kb.x & 0xFFFF0000u);
  xk[2] = __uint_as_float(kb.y << 16); xk[3] = __uint_as_float(kb.y & 0xFFFF0000u);
  xv[0] = __uint_as_float(vb.x << 16); xv[1] = __uint_as_float(vb.x & 0xFFFF0000u);
  xv[2] = __uint_as_float(vb.y << 16); xv[3] = __uint_as_float(vb.y & 0xFFFF0000u);
  uint32_t ck, cv;
  const int ek = encode_e4m3_row(xk, ck), ev = encode_e4m3_row(xv, cv);
  uint8_t *kc = reinterpret_cast<uint8_t *>(v.k_pool), *vc = reinterpret_cast<uint8_t *>(v.v_pool);
  *reinterpret_cast<uint32_t *>(kc + (ph * P + s) * kFp8HeadDim + 4 * lane) = ck;
  const int sv = s - s % kChunkSlots + fp8_v_slot_byte(s % kChunkSlots);
#pragma unroll
  for (int i = 0; i < 4; ++i)
    vc[(ph * kFp8HeadDim + 4 * lane + i) * P + sv] = (uint8_t)(cv >> (8 * i));
  if (lane == 0) {
    int8_t *e = v.kv_exp + (ph * (P / kChunkSlots) + s / kChunkSlots) * 32 + s % kChunkSlots;
    e[0] = (int8_t)ek;
    e[kChunkSlots] = (int8_t)ev;
  }
}

__global__ void fill_meta_kernel(FillView v) {
  const int32_t b = blockIdx.x;
  const int32_t count = v.counts[b];
  __shared__ long long partial[32];
  if (count < 0 || count > v.lmax || count > v.max_slots) {
    if (threadIdx.x == 0) record_error(v.err, HAM_DEVERR_SLOTS);
    return;
  }
  long long tokens = 0;
  for (int32_t j = threadIdx.x; j < count; j += blockDim.x) {
    const int32_t page = v.page_table[(int64_t)b * v.max_pages + j / v.page_slots];
    const int32_t t = v.ntok ? v.ntok[(int64_t)b * v.lmax + j] : 1;
    tokens += t;
    if (page < 0 || page >= v.pool_pages) continue;  // reported by fill_rows
    const int64_t m = (int64_t)page * v.page_slots + j % v.page_slots;
    v.slot_pos[m] = v.pos ? v.pos[(int64_t)b * v.lmax + j] : j;
    v.slot_ntok[m] = t;
  }
  for (int o = 16; o > 0; o >>= 1) tokens += __shfl_xor_sync(0xffffffffu, tokens, o);
  if ((threadIdx.x & 31) == 0) partial[threadIdx.x / 32] = tokens;
  __syncthreads();
  if (threadIdx.x == 0) {
    long long total = 0;
    for (int w = 0; w < (int)(blockDim.x / 32); ++w) total += partial[w];
    v.num_slots[b] = count;
    v.num_tokens[b] = total;
  }
}

__global__ void set_lengths_kernel(int32_t *num_slots, int64_t *num_tokens,
                                   const int32_t *new_slots, const int64_t *new_tokens,
                                   int32_t batch, int32_t max_slots, int32_t *err) {
  const int32_t b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= batch) return;
  const int32_t n = new_slots[b];
  if (n < 0 || n > max_slots) {
    record_error(err, HAM_DEVERR_SLOTS);
    return;
  }
  num_slots[b] = n;
  if (new_tokens) num_tokens[b] = new_tokens[b];
}

namespace {
using EncodeTiled = CUresult (*)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *,
                                 const cuuint64_t *, const cuuint64_t *, const cuuint32_t *,
                                 const cuuint32_t *, CUtensorMapInterleave, CUtensorMapSwizzle,
                                 CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
EncodeTiled tensor_map_encoder() {
  static EncodeTiled encode = nullptr;
  if (!encode) {
    void *fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault,
                                         &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess || !fn)
      return nullptr;
    encode = reinterpret_cast<EncodeTiled>(fn);
  }
  return encode;
}
}  // namespace

int make_rows_tensor_map(CUtensorMap *map, const void *base, int64_t rows, int heads,
                         int head_dim, int box_heads, int box_rows) {
  EncodeTiled encode = tensor_map_encoder();
  if (!encode) return -1;
  const cuuint64_t dims[4] = {64, (cuuint64_t)(head_dim / 64), (cuuint64_t)heads,
                              (cuuint64_t)rows};
  const cuuint64_t strides[3] = {128, (cuuint64_t)head_dim * 2,
                                 (cuuint64_t)heads * head_dim * 2};  // bytes, dims 1..3
  const cuuint32_t box[4] = {64, 1, (cuuint32_t)box_heads, (cuuint32_t)box_rows};
  const cuuint32_t estride[4] = {1, 1, 1, 1};
  return (int)encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void *>(base), dims,
                     strides, box, estride, CU_TENSOR_MAP_INTERLEAVE_NONE,
                     CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                     CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
}

int make_matrix_tensor_map(CUtensorMap *map, const void *base, int64_t rows, int64_t cols,
                           int box_rows) {
  EncodeTiled encode = tensor_map_encoder();
  if (!encode) return -1;
  const cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
  const cuuint64_t strides[1] = {(cuuint64_t)cols * 2};  // bytes of a row
  const cuuint32_t box[2] = {64, (cuuint32_t)box_rows};
  const cuuint32_t estride[2] = {1, 1};
  return (int)encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(base), dims,
                     strides, box, estride, CU_TENSOR_MAP_INTERLEAVE_NONE,
                     CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                     CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
}

int make_parts_tensor_map(CUtensorMap *map, void *base, int splits, int64_t rows, int64_t cols,
                          int64_t ld) {
  EncodeTiled encode = tensor_map_encoder();
  if (!encode) return -1;
  const cuuint64_t dims[3] = {(cuuint64_t)cols, (cuuint64_t)rows, (cuuint64_t)splits};
  const cuuint64_t strides[2] = {(cuuint64_t)ld * 4, (cuuint64_t)(rows * ld) * 4};  // bytes
  const cuuint32_t box[3] = {32, 32, 1};
  const cuuint32_t estride[3] = {1, 1, 1};
  return (int)encode(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 3, base, dims, strides, box, estride,
                     CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
}

int make_fp8_k_tensor_map(CUtensorMap *map, const void *k_codes, int64_t rows) {
  EncodeTiled encode = tensor_map_encoder();
  if (!encode) return -1;
  const cuuint64_t dims[2] = {(cuuint64_t)kFp8HeadDim, (cuuint64_t)rows};
  const cuuint64_t strides[1] = {(cuuint64_t)kFp8HeadDim};  // bytes of a row
  const cuuint32_t box[2] = {(cuuint32_t)kFp8HeadDim, (cuuint32_t)kChunkSlots};
  const cuuint32_t estride[2] = {1, 1};
  return (int)encode(map, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<void *>(k_codes), dims,
                     strides, box, estride, CU_TENSOR_MAP_INTERLEAVE_NONE,
                     CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                     CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
}

int make_fp8_v_tensor_map(CUtensorMap *map, const void *v_codes, int64_t rows_d, int page_slots) {
  EncodeTiled encode = tensor_map_encoder();
  if (!encode) return -1;
  const cuuint64_t dims[2] = {(cuuint64_t)page_slots, (cuuint64_t)rows_d};
  const cuuint64_t strides[1] = {(cuuint64_t)page_slots};  // bytes of a (page, head, d) row
  const cuuint32_t box[2] = {(cuuint32_t)kChunkSlots, (cuuint32_t)kFp8HeadDim};
  const cuuint32_t estride[2] = {1, 1};
  return (int)encode(map, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<void *>(v_codes), dims,
                     strides, box, estride, CU_TENSOR_MAP_INTERLEAVE_NONE,
                     CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                     CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
}

int make_pool_tensor_map(CUtensorMap *map, const void *pool, int64_t rows, int head_dim,
                         bool half_box) {
  EncodeTiled encode = tensor_map_encoder();
  if (!encode) return -1;
  const cuuint64_t dims[3] = {64, (cuuint64_t)(head_dim / 64), (cuuint64_t)rows};
  const cuuint64_t strides[2] = {128, (cuuint64_t)head_dim * 2};  // bytes, dims 1 and 2
  const cuuint32_t box[3] = {64, half_box ? 1u : (cuuint32_t)(head_dim / 64),
                             (cuuint32_t)kChunkSlots};
  const cuuint32_t estride[3] = {1, 1, 1};
  return (int)encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(pool), dims,
                     strides, box, estride, CU_TENSOR_MAP_INTERLEAVE_NONE,
                     CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                     CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
}

cudaError_t launch_fill(const FillView &v, cudaStream_t stream) {
  if (v.lmax > 0 && v.kv_exp) {
    dim3 grid((unsigned)(((int64_t)v.lmax * v.n_kv_heads + 7) / 8), (unsigned)v.batch);
    fill_rows_fp8_kernel<<<grid, 256, 0, stream>>>(v);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  } else if (v.lmax > 0) {
    dim3 grid((unsigned)((v.lmax + 15) / 16), (unsigned)v.batch);
    fill_rows_kernel<<<grid, 256, 0, stream>>>(v);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  fill_meta_kernel<<<v.batch, 256, 0, stream>>>(v);
  return cudaGetLastError();
}

}  // namespace ham

// ------------------------------------------------------------------------------------
// C ABI
// ------------------------------------------------------------------------------------
extern "C" {

const char *ham_last_error(void) { return g_last_error; }

int ham_kv_alloc(const ham_config *cfg_in, ham_kv **out) {
  if (!out) return fail(HAM_EINVAL, "out is NULL");
  *out = nullptr;
  if (!cfg_in) return fail(HAM_EINVAL, "config is NULL");
  ham_config cfg = *cfg_in;
  if (cfg.layers < 1 || cfg.batch < 1 || cfg.batch > ham::kMaxBatch || cfg.n_q_heads < 1 ||
      cfg.n_kv_heads < 1 || cfg.n_q_heads % cfg.n_kv_heads != 0)
    return fail(HAM_EINVAL, "bad shape: layers %d batch %d (max %d) heads %d/%d", cfg.layers,
                cfg.batch, ham::kMaxBatch, cfg.n_q_heads, cfg.n_kv_heads);
  if (cfg.page_slots < ham::kChunkSlots || cfg.page_slots % ham::kChunkSlots != 0)
    return fail(HAM_EINVAL, "page_slots %d must be a positive multiple of %d", cfg.page_slots,
                ham::kChunkSlots);
  if (cfg.max_slots_per_seq < 1)
    return fail(HAM_EINVAL, "max_slots_per_seq %d must be >= 1", cfg.max_slots_per_seq);
  if (cfg.pos_mode != HAM_POS_SLOT && cfg.pos_mode != HAM_POS_TOKEN)
    return fail(HAM_EINVAL, "pos_mode %d", cfg.pos_mode);
  if (!(cfg.rope_base > 1.0) || !std::isfinite(cfg.rope_base))
    return fail(HAM_EINVAL, "rope_base must be finite and > 1");
  if (cfg.kv_dtype != HAM_KV_BF16 && cfg.kv_dtype != HAM_KV_E4M3)
    return fail(HAM_EINVAL, "kv_dtype %d", cfg.kv_dtype);
  if (cfg.kv_dtype == HAM_KV_E4M3 && cfg.head_dim != ham::kFp8HeadDim)
    return fail(HAM_EUNSUPPORTED, "FP8 pools: head_dim %d (only %d is compiled)", cfg.head_dim,
                ham::kFp8HeadDim);
  const int group = cfg.n_q_heads / cfg.n_kv_heads;
  if (!ham::attention_supported(cfg.head_dim, group) ||
      ham::append_kv_per_block(cfg.n_q_heads, cfg.n_kv_heads, cfg.head_dim) == 0)
    return fail(HAM_EUNSUPPORTED, "head_dim %d / group %d not compiled (head_dim 64 or 128, "
                "group 1, 2, 4 or 8)", cfg.head_dim, group);
  const int64_t max_pages =
      ((int64_t)cfg.max_slots_per_seq + cfg.page_slots - 1) / cfg.page_slots;
  const int64_t need_pages = (int64_t)cfg.batch * max_pages;
  if (need_pages > INT32_MAX) return fail(HAM_EINVAL, "page table too large");
  // The attention kernel counts 16-slot chunks of the whole batch in int32.
  if ((int64_t)cfg.batch * ham::chunks_of(cfg.max_slots_per_seq) * cfg.n_kv_heads > INT32_MAX)
    return fail(HAM_EINVAL, "batch * max_slots_per_seq too large");
  if (cfg.pool_pages == 0) cfg.pool_pages = need_pages;
  if (cfg.pool_pages < need_pages)
    return fail(HAM_ECAPACITY, "pool of %lld pages < %lld pages reserved by the page tables",
                (long long)cfg.pool_pages, (long long)need_pages);
  if (cfg.pool_pages > INT32_MAX) return fail(HAM_EINVAL, "pool_pages above int32 range");
  // TMA row coordinates of the pools are int32
  if (cfg.pool_pages * cfg.n_kv_heads * (int64_t)cfg.page_slots > INT32_MAX)
    return fail(HAM_EINVAL, "pool_pages * n_kv_heads * page_slots above int32 range");
  // FP8: the transposed value blocks are addressed by (page, head, element) rows
  if (cfg.kv_dtype == HAM_KV_E4M3 &&
      cfg.pool_pages * cfg.n_kv_heads * (int64_t)ham::kFp8HeadDim > INT32_MAX)
    return fail(HAM_EINVAL, "pool_pages * n_kv_heads * 128 above int32 range");

  int dev = 0;
  HAM_CUDA(cudaGetDevice(&dev));
  int sms = 0;
  HAM_CUDA(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));

  ham_kv *kv = new ham_kv();
  kv->cfg = cfg;
  kv->device = dev;
  kv->num_sms = sms;
  kv->max_pages = (int32_t)max_pages;
  kv->max_ctas = 8 * sms;
  kv->pool_elems = cfg.pool_pages * cfg.n_kv_heads * (int64_t)cfg.page_slots * cfg.head_dim;
  kv->fp8 = cfg.kv_dtype == HAM_KV_E4M3 ? 1 : 0;

  const size_t pool_bytes = (size_t)cfg.layers * layer_pool_bytes(kv);
  const MetaLayout lay = meta_layout(cfg, kv->max_ctas, max_pages);
  const size_t off = lay.total;
  kv->scratch_bytes = (int64_t)(off - lay.acc);

  {
    const int per_sm = ham::attention_ctas_per_sm(cfg.head_dim, group, cfg.batch, false,
                                                  HAM_DTYPE_BF16, kv->fp8 != 0);
    const int per_sm_step = ham::attention_ctas_per_sm(cfg.head_dim, group, cfg.batch, true,
                                                       HAM_DTYPE_BF16, kv->fp8 != 0);
    if (per_sm <= 0 || per_sm_step <= 0) {
      delete kv;
      return fail(HAM_ECUDA, "attention kernel cannot be resident on an SM");
    }
    kv->default_ctas =
        std::min(ham::default_attention_ctas(sms, per_sm, kv->fp8 != 0), kv->max_ctas);
    kv->default_step_ctas =
        std::min(ham::default_attention_ctas(sms, per_sm_step, kv->fp8 != 0), kv->max_ctas);
  }
  cudaError_t e = cudaMalloc(&kv->pool, pool_bytes);
  if (e != cudaSuccess) {
    delete kv;
    cudaGetLastError();
    return fail(HAM_ENOMEM, "cudaMalloc of %zu pool bytes: %s", pool_bytes, cudaGetErrorString(e));
  }
  e = cudaMalloc(&kv->meta, off);
  if (e == cudaSuccess) e = cudaMallocHost(&kv->host_stage, 256 + (size_t)cfg.batch * 16);
  if (e != cudaSuccess) {
    cudaGetLastError();
    ham_kv_free(kv);
    return fail(HAM_ENOMEM, "allocation of the cache metadata failed");
  }
  kv->slot_pos = reinterpret_cast<int32_t *>(kv->meta + lay.pos);
  kv->slot_ntok = reinterpret_cast<int32_t *>(kv->meta + lay.ntok);
  kv->page_table = reinterpret_cast<int32_t *>(kv->meta + lay.pt);
  kv->num_slots = reinterpret_cast<int32_t *>(kv->meta + lay.ns);
  kv->num_tokens = reinterpret_cast<int64_t *>(kv->meta + lay.nt);
  kv->inv_freq = reinterpret_cast<double *>(kv->meta + lay.inv_freq);
  kv->err = reinterpret_cast<int32_t *>(kv->meta + lay.err);
  kv->part_acc = reinterpret_cast<float *>(kv->meta + lay.acc);
  kv->part_ml = reinterpret_cast<float2 *>(kv->meta + lay.ml);
  kv->seg_range = reinterpret_cast<int2 *>(kv->meta + lay.sr);
  kv->stash = reinterpret_cast<int4 *>(kv->meta + lay.stash);
  kv->arrive = reinterpret_cast<int32_t *>(kv->meta + lay.arrive);
  kv->prefill_seq = reinterpret_cast<int4 *>(kv->meta + lay.pf_seq);
  kv->prefill_rows = reinterpret_cast<int2 *>(kv->meta + lay.pf_pos);
  if (!kv->fp8) {
    kv->prefill_part = reinterpret_cast<float *>(kv->meta + lay.pf_part);
    kv->prefill_part_ml = reinterpret_cast<float2 *>(kv->meta + lay.pf_ml);
  }

  // Zeroed pool: slots past a sequence's length hold zeros, never uninitialised bits (FP8:
  // zero codes and exponents, the encoding of a zero row).
  e = cudaMemset(kv->pool, 0, pool_bytes);
  if (e == cudaSuccess) e = cudaMemset(kv->meta, 0, off);
  std::vector<int32_t> pt = reserve_pages(cfg.batch, kv->max_pages, cfg.pool_pages, cfg.page_seed);
  if (e == cudaSuccess)
    e = cudaMemcpy(kv->page_table, pt.data(), pt.size() * sizeof(int32_t), cudaMemcpyHostToDevice);
  // RoPE frequencies theta_i / pos = base^(-2i/d), fp64 (rotate-half pairs (i, i + d/2)).
  std::vector<double> inv_freq((size_t)cfg.head_dim / 2);
  for (int i = 0; i < cfg.head_dim / 2; ++i)
    inv_freq[(size_t)i] = pow(cfg.rope_base, -(2.0 * (double)i) / (double)cfg.head_dim);
  if (e == cudaSuccess)
    e = cudaMemcpy(kv->inv_freq, inv_freq.data(), inv_freq.size() * sizeof(double),
                   cudaMemcpyHostToDevice);
  // (cos, sin) of p * inv_freq[i] for every position a sequence can reach by slot index (or
  // 4 tokens per slot), in fp64 (stored bits) and fp32 (the attention pass), both tables
  // capped at 512 MiB together (~350k positions at head_dim 128); the kernels fall back to
  // sincos beyond, which on this GPU's narrow fp64 pipe costs microseconds per launch.
  if (e == cudaSuccess) {
    const int64_t half = cfg.head_dim / 2;
    const int64_t reach = (int64_t)cfg.max_slots_per_seq * (cfg.pos_mode == HAM_POS_TOKEN ? 4 : 1);
    const int64_t cap = (int64_t)(512u << 20) /
                        (half * (int64_t)(sizeof(double2) + sizeof(float2) + sizeof(float4)));
    kv->rope_positions = std::min(reach, cap);
    std::vector<double2> table((size_t)(kv->rope_positions * half));
    std::vector<float2> table_f(table.size());
    std::vector<float4> table_ff(table.size());  // (c_hi, c_lo, s_hi, s_lo): c = c_hi + c_lo
    for (int64_t p = 0; p < kv->rope_positions; ++p)
      for (int64_t i = 0; i < half; ++i) {
        const double theta = (double)p * inv_freq[(size_t)i];
        const double c = cos(theta), s = sin(theta);
        table[(size_t)(p * half + i)] = make_double2(c, s);
        table_f[(size_t)(p * half + i)] = make_float2((float)c, (float)s);
        const float ch = (float)c, sh = (float)s;
        table_ff[(size_t)(p * half + i)] =
            make_float4(ch, (float)(c - (double)ch), sh, (float)(s - (double)sh));
      }
    e = cudaMalloc(&kv->rope_table, table.size() * sizeof(double2));
    if (e == cudaSuccess)
      e = cudaMemcpy(kv->rope_table, table.data(), table.size() * sizeof(double2),
                     cudaMemcpyHostToDevice);
    if (e == cudaSuccess) e = cudaMalloc(&kv->rope_table_f, table_f.size() * sizeof(float2));
    if (e == cudaSuccess)
      e = cudaMemcpy(kv->rope_table_f, table_f.data(), table_f.size() * sizeof(float2),
                     cudaMemcpyHostToDevice);
    if (e == cudaSuccess) e = cudaMalloc(&kv->rope_table_ff, table_ff.size() * sizeof(float4));
    if (e == cudaSuccess)
      e = cudaMemcpy(kv->rope_table_ff, table_ff.data(), table_ff.size() * sizeof(float4),
                     cudaMemcpyHostToDevice);
  }
  if (e != cudaSuccess) {
    int rc = cuda_fail(e, "initialising the cache");
    ham_kv_free(kv);
    return rc;
  }
  kv->tmaps.resize((size_t)cfg.layers * 2);
  kv->tmaps_half.resize((size_t)cfg.layers * 2);
  const int64_t rows = cfg.pool_pages * cfg.n_kv_heads * (int64_t)cfg.page_slots;
  for (int layer = 0; layer < cfg.layers; ++layer) {
    if (kv->fp8) {  // the code blocks; the half-box maps (prefill) stay unused
      const ham::Fp8Layer f = ham::fp8_layer(kv->pool, rows, layer);
      int r = ham::make_fp8_k_tensor_map(&kv->tmaps[(size_t)layer * 2], f.k, rows);
      if (r == 0)
        r = ham::make_fp8_v_tensor_map(&kv->tmaps[(size_t)layer * 2 + 1], f.v,
                                       rows / cfg.page_slots * ham::kFp8HeadDim, cfg.page_slots);
      memset(&kv->tmaps_half[(size_t)layer * 2], 0, 2 * sizeof(CUtensorMap));
      if (r != 0) {
        ham_kv_free(kv);
        return fail(HAM_ECUDA, "cuTensorMapEncodeTiled failed (CUresult %d)", r);
      }
      continue;
    }
    for (int which = 0; which < 2; ++which) {
      int r = ham::make_pool_tensor_map(&kv->tmaps[(size_t)layer * 2 + which],
                                        layer_pool(kv, layer, which), rows, cfg.head_dim, false);
      if (r == 0)
        r = ham::make_pool_tensor_map(&kv->tmaps_half[(size_t)layer * 2 + which],
                                      layer_pool(kv, layer, which), rows, cfg.head_dim, true);
      if (r != 0) {
        ham_kv_free(kv);
        return fail(HAM_ECUDA, "cuTensorMapEncodeTiled failed (CUresult %d)", r);
      }
    }
  }
  *out = kv;
  return HAM_OK;
}

int ham_kv_free(ham_kv *kv) {
  if (!kv) return HAM_OK;
  DeviceGuard guard(kv->device);
  cudaDeviceSynchronize();
  if (kv->pool) cudaFree(kv->pool);
  if (kv->meta) cudaFree(kv->meta);
  if (kv->rope_table) cudaFree(kv->rope_table);
  if (kv->rope_table_f) cudaFree(kv->rope_table_f);
  if (kv->rope_table_ff) cudaFree(kv->rope_table_ff);
  if (kv->host_stage) cudaFreeHost(kv->host_stage);
  delete kv;
  return HAM_OK;
}

int ham_kv_get_info(const ham_kv *kv, ham_kv_info *info) {
  if (!kv || !info) return fail(HAM_EINVAL, "null argument");
  memset(info, 0, sizeof *info);
  info->cfg = kv->cfg;
  info->max_pages_per_seq = kv->max_pages;
  info->attn_ctas = kv->attn_ctas > 0 ? kv->attn_ctas : kv->default_ctas;
  info->num_sms = kv->num_sms;
  info->device = kv->device;
  info->pool_bytes = (int64_t)layer_pool_bytes(kv);
  info->scratch_bytes = kv->scratch_bytes;
  return HAM_OK;
}

int ham_kv_set_attn_ctas(ham_kv *kv, int32_t ctas) {
  if (!kv) return fail(HAM_EINVAL, "null handle");
  if (ctas < 0 || ctas > kv->max_ctas)
    return fail(HAM_EINVAL, "ctas %d outside [0, %d]", ctas, kv->max_ctas);
  kv->attn_ctas = ctas;
  return HAM_OK;
}

int ham_kv_set_wait_limit_ns(ham_kv *kv, uint64_t ns) {
  if (!kv) return fail(HAM_EINVAL, "null handle");
  constexpr uint64_t kDefaultNs = 2000000000ull;  // the kernels' default bound, 2 s
  if (ns > kDefaultNs)
    return fail(HAM_EINVAL, "limit %llu ns above the default %llu", (unsigned long long)ns,
                (unsigned long long)kDefaultNs);
  kv->wait_ns = ns;
  return HAM_OK;
}

int ham_kv_append(ham_kv *kv, int32_t layer, void *q_inout, const void *k_new,
                  const void *v_new, const int32_t *pos, const int32_t *ntok, void *stream) {
  ham::ApiRange nvtx_range("ham_kv_append");
  int rc = check_layer(kv, layer);
  if (rc) return rc;
  if (!k_new || !v_new || !ntok) return fail(HAM_EINVAL, "k_new, v_new and ntok are required");
  if (!aligned16(k_new) || !aligned16(v_new) || (q_inout && !aligned16(q_inout)))
    return fail(HAM_EINVAL, "q/k/v must be 16-byte aligned");
  if (((uintptr_t)ntok & 3u) || ((uintptr_t)pos & 3u))
    return fail(HAM_EINVAL, "pos/ntok must be 4-byte aligned");
  DeviceGuard guard(kv->device);
  ham::AppendView v{};
  v.k_pool = layer_pool(kv, layer, 0);
  v.v_pool = layer_pool(kv, layer, 1);
  v.kv_exp = layer_exp(kv, layer);
  v.slot_pos = kv->slot_pos;
  v.slot_ntok = kv->slot_ntok;
  v.page_table = kv->page_table;
  v.num_slots = kv->num_slots + (size_t)layer * kv->cfg.batch;
  v.num_tokens = kv->num_tokens + (size_t)layer * kv->cfg.batch;
  v.inv_freq = kv->inv_freq;
  v.rope_table = kv->rope_table;
  v.rope_positions = kv->rope_positions;
  v.q = static_cast<uint16_t *>(q_inout);
  v.k_new = static_cast<const uint16_t *>(k_new);
  v.v_new = static_cast<const uint16_t *>(v_new);
  v.pos = pos;
  v.ntok = ntok;
  v.err = kv->err;
  v.pool_pages = kv->cfg.pool_pages;
  v.batch = kv->cfg.batch;
  v.n_q_heads = kv->cfg.n_q_heads;
  v.n_kv_heads = kv->cfg.n_kv_heads;
  v.head_dim = kv->cfg.head_dim;
  v.page_slots = kv->cfg.page_slots;
  v.max_pages = kv->max_pages;
  v.max_slots = kv->cfg.max_slots_per_seq;
  v.pos_mode = kv->cfg.pos_mode;
  v.kv_per_block = ham::append_kv_per_block(v.n_q_heads, v.n_kv_heads, v.head_dim);
  cudaError_t e = ham::launch_append(v, static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "append launch");
  note_launch(kv, layer, stream, true);
  return HAM_OK;
}

int ham_decode_attn_ex(ham_kv *kv, int32_t layer, const void *q, void *out, int32_t out_dtype,
                       void *stream) {
  ham::ApiRange nvtx_range("ham_decode_attn_ex");
  int rc = check_layer(kv, layer);
  if (rc) return rc;
  if (!q || !out) return fail(HAM_EINVAL, "q and out are required");
  if (!aligned16(q) || !aligned16(out)) return fail(HAM_EINVAL, "q/out must be 16-byte aligned");
  if (out_dtype != HAM_DTYPE_BF16 && out_dtype != HAM_DTYPE_F32)
    return fail(HAM_EINVAL, "out_dtype %d", out_dtype);
  DeviceGuard guard(kv->device);
  const int group = kv->cfg.n_q_heads / kv->cfg.n_kv_heads;
  const int ctas = kv->attn_ctas > 0 ? kv->attn_ctas : kv->default_ctas;
  ham::AttnView v{};
  v.k_pool = layer_pool(kv, layer, 0);
  v.v_pool = layer_pool(kv, layer, 1);
  v.kv_exp = layer_exp(kv, layer);
  v.page_table = kv->page_table;
  v.num_slots = kv->num_slots + (size_t)layer * kv->cfg.batch;
  v.q = static_cast<const uint16_t *>(q);
  v.out = out;
  v.part_acc = kv->part_acc;
  v.part_ml = kv->part_ml;
  v.seg_range = kv->seg_range;
  v.err = kv->err;
  v.pool_pages = kv->cfg.pool_pages;
  v.batch = kv->cfg.batch;
  v.n_kv_heads = kv->cfg.n_kv_heads;
  v.group = group;
  v.page_slots = kv->cfg.page_slots;
  v.max_pages = kv->max_pages;
  v.max_slots = kv->cfg.max_slots_per_seq;
  v.ctas = ctas;
  v.sms = kv->num_sms;
  v.wait_ns = kv->wait_ns;
  v.early = may_start_early(kv, layer, stream) ? 1 : 0;
  cudaError_t e = ham::launch_attention(kv->tmaps[(size_t)layer * 2], kv->tmaps[(size_t)layer * 2 + 1],
                                        v, kv->cfg.head_dim, out_dtype,
                                        static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "attention launch");
  note_launch(kv, layer, stream, false);
  return HAM_OK;
}

namespace {
bool overlaps(const void *a, size_t a_bytes, const void *b, size_t b_bytes) {
  const uintptr_t a0 = (uintptr_t)a, b0 = (uintptr_t)b;
  return a && b && a0 < b0 + b_bytes && b0 < a0 + a_bytes;
}
}  // namespace

int ham_qkv_append(ham_kv *kv, int32_t layer, const void *x, const void *w_qkv, int32_t hidden,
                   const int32_t *pos, const int32_t *ntok, void *q_rot, void *stream) {
  ham::ApiRange nvtx_range("ham_qkv_append");
  int rc = check_layer(kv, layer);
  if (rc) return rc;
  if (!x || !w_qkv || !ntok || !q_rot) return fail(HAM_EINVAL, "x, w_qkv, ntok and q_rot are required");
  if (!aligned16(x) || !aligned16(w_qkv) || !aligned16(q_rot))
    return fail(HAM_EINVAL, "x, w_qkv and q_rot must be 16-byte aligned");
  if (((uintptr_t)ntok & 3u) || ((uintptr_t)pos & 3u))
    return fail(HAM_EINVAL, "pos/ntok must be 4-byte aligned");
  if (hidden < ham::kFrontHiddenQuantum || hidden % ham::kFrontHiddenQuantum != 0 || hidden > (1 << 20))
    return fail(HAM_EINVAL, "hidden %d must be a positive multiple of %d (at most 2^20)", hidden,
                ham::kFrontHiddenQuantum);
  const ham_config &c = kv->cfg;
  if (c.head_dim != 64 && c.head_dim != 128)
    return fail(HAM_EUNSUPPORTED, "layer front: head_dim %d not compiled", c.head_dim);
  const size_t d = (size_t)c.head_dim, B = (size_t)c.batch;
  const size_t x_bytes = B * (size_t)hidden * 2;
  const size_t w_bytes = (size_t)(c.n_q_heads + 2 * c.n_kv_heads) * d * (size_t)hidden * 2;
  const size_t q_bytes = B * (size_t)c.n_q_heads * d * 2;
  const size_t pool_bytes = (size_t)c.layers * layer_pool_bytes(kv);
  if (overlaps(q_rot, q_bytes, x, x_bytes) || overlaps(q_rot, q_bytes, w_qkv, w_bytes) ||
      overlaps(q_rot, q_bytes, kv->pool, pool_bytes) || overlaps(x, x_bytes, kv->pool, pool_bytes) ||
      overlaps(w_qkv, w_bytes, kv->pool, pool_bytes))
    return fail(HAM_EINVAL, "q_rot, x, w_qkv and the cache must not overlap");
  DeviceGuard guard(kv->device);
  const MetaLayout lay = meta_layout(c, kv->max_ctas, kv->max_pages);
  ham::FrontView v{};
  v.x = static_cast<const uint16_t *>(x);
  v.w = static_cast<const uint16_t *>(w_qkv);
  v.q_rot = static_cast<uint16_t *>(q_rot);
  v.k_pool = layer_pool(kv, layer, 0);
  v.v_pool = layer_pool(kv, layer, 1);
  v.slot_pos = kv->slot_pos;
  v.slot_ntok = kv->slot_ntok;
  v.page_table = kv->page_table;
  v.num_slots = kv->num_slots + (size_t)layer * c.batch;
  v.num_tokens = kv->num_tokens + (size_t)layer * c.batch;
  v.inv_freq = kv->inv_freq;
  v.rope_table = kv->rope_table;
  v.rope_positions = kv->rope_positions;
  v.pos = pos;
  v.ntok = ntok;
  v.arrive = reinterpret_cast<int32_t *>(kv->meta + lay.front);
  v.kv_exp = layer_exp(kv, layer);  // FP8 pools: encoded by the front's last CTAs
  v.stage = kv->fp8 ? reinterpret_cast<uint16_t *>(kv->meta + lay.front_stage) : nullptr;
  v.enc_arrive = kv->fp8 ? reinterpret_cast<int32_t *>(kv->meta + lay.front_enc) : nullptr;
  v.err = kv->err;
  v.pool_pages = c.pool_pages;
  v.batch = c.batch;
  v.hidden = hidden;
  v.n_q_heads = c.n_q_heads;
  v.n_kv_heads = c.n_kv_heads;
  v.head_dim = c.head_dim;
  v.page_slots = c.page_slots;
  v.max_pages = kv->max_pages;
  v.max_slots = c.max_slots_per_seq;
  v.pos_mode = c.pos_mode;
  cudaError_t e = ham::launch_front(v, static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "layer front launch");
  note_launch(kv, layer, stream, true);
  return HAM_OK;
}

int ham_decode_step(ham_kv *kv, int32_t layer, const void *q, void *q_rot, const void *k_new,
                    const void *v_new, const int32_t *pos, const int32_t *ntok, void *out,
                    int32_t out_dtype, void *stream) {
  ham::ApiRange nvtx_range("ham_decode_step");
  int rc = check_layer(kv, layer);
  if (rc) return rc;
  if (!q || !k_new || !v_new || !ntok || !out)
    return fail(HAM_EINVAL, "q, k_new, v_new, ntok and out are required");
  if (!aligned16(q) || !aligned16(k_new) || !aligned16(v_new) || !aligned16(out) ||
      (q_rot && !aligned16(q_rot)))
    return fail(HAM_EINVAL, "q/q_rot/k/v/out must be 16-byte aligned");
  if (((uintptr_t)ntok & 3u) || ((uintptr_t)pos & 3u))
    return fail(HAM_EINVAL, "pos/ntok must be 4-byte aligned");
  if (out_dtype != HAM_DTYPE_BF16 && out_dtype != HAM_DTYPE_F32)
    return fail(HAM_EINVAL, "out_dtype %d", out_dtype);
  const ham_config &c = kv->cfg;
  const int group = c.n_q_heads / c.n_kv_heads;
  {  // outputs are written while q is still being read
    const size_t n = (size_t)c.batch * c.n_q_heads * c.head_dim;
    const size_t out_bytes = n * (out_dtype == HAM_DTYPE_F32 ? 4 : 2);
    if (overlaps(q, n * 2, out, out_bytes) || overlaps(q_rot, n * 2, q, n * 2) ||
        overlaps(q_rot, n * 2, out, out_bytes))
      return fail(HAM_EINVAL, "q, q_rot and out must not overlap");
  }
  DeviceGuard guard(kv->device);
  ham::AttnView v{};
  v.k_pool = layer_pool(kv, layer, 0);
  v.v_pool = layer_pool(kv, layer, 1);
  v.kv_exp = layer_exp(kv, layer);
  v.page_table = kv->page_table;
  v.num_slots = kv->num_slots + (size_t)layer * c.batch;
  v.q = static_cast<const uint16_t *>(q);
  v.out = out;
  v.part_acc = kv->part_acc;
  v.part_ml = kv->part_ml;
  v.seg_range = kv->seg_range;
  v.err = kv->err;
  v.pool_pages = c.pool_pages;
  v.batch = c.batch;
  v.n_kv_heads = c.n_kv_heads;
  v.group = group;
  v.page_slots = c.page_slots;
  v.max_pages = kv->max_pages;
  v.max_slots = c.max_slots_per_seq;
  v.ctas = kv->attn_ctas > 0 ? kv->attn_ctas : kv->default_step_ctas;
  v.sms = kv->num_sms;
  v.wait_ns = kv->wait_ns;
  ham::StepArgs &st = v.step;
  st.k_new = static_cast<const uint16_t *>(k_new);
  st.v_new = static_cast<const uint16_t *>(v_new);
  st.q_rot = static_cast<uint16_t *>(q_rot);
  st.pos = pos;
  st.ntok = ntok;
  st.num_slots = kv->num_slots + (size_t)layer * c.batch;
  st.num_tokens = kv->num_tokens + (size_t)layer * c.batch;
  st.slot_pos = kv->slot_pos;
  st.slot_ntok = kv->slot_ntok;
  st.k_pool = layer_pool(kv, layer, 0);
  st.v_pool = layer_pool(kv, layer, 1);
  st.kv_exp = layer_exp(kv, layer);
  st.inv_freq = kv->inv_freq;
  st.rope_table = kv->rope_table;
  st.rope_table_f = kv->rope_table_f;
  st.rope_positions = kv->rope_positions;
  st.stash = kv->stash;
  st.arrive = kv->arrive;
  st.pos_mode = c.pos_mode;
  v.early = may_start_early(kv, layer, stream) ? 1 : 0;
  cudaError_t e = ham::launch_decode_step(kv->tmaps[(size_t)layer * 2],
                                          kv->tmaps[(size_t)layer * 2 + 1], v, c.head_dim,
                                          out_dtype, static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "decode step launch");
  note_launch(kv, layer, stream, true);
  return HAM_OK;
}

int ham_micro_step(ham_kv *kv, int32_t layer, const void *q, void *q_rot, const void *k_new,
                   const void *v_new, const int32_t *pos, const int32_t *ntok, void *out,
                   int32_t out_dtype, void *stream) {
  ham::ApiRange nvtx_range("ham_micro_step");
  int rc = check_layer(kv, layer);
  if (rc) return rc;
  if ((rc = fp8_unsupported(kv, "ham_micro_step")) != 0) return rc;
  if (!q || !k_new || !v_new || !ntok || !out)
    return fail(HAM_EINVAL, "q, k_new, v_new, ntok and out are required");
  if (!aligned16(q) || !aligned16(k_new) || !aligned16(v_new) || !aligned16(out) ||
      (q_rot && !aligned16(q_rot)))
    return fail(HAM_EINVAL, "q/q_rot/k/v/out must be 16-byte aligned");
  if (((uintptr_t)ntok & 3u) || ((uintptr_t)pos & 3u))
    return fail(HAM_EINVAL, "pos/ntok must be 4-byte aligned");
  if (out_dtype != HAM_DTYPE_BF16 && out_dtype != HAM_DTYPE_F32)
    return fail(HAM_EINVAL, "out_dtype %d", out_dtype);
  const ham_config &c = kv->cfg;
  if (c.max_slots_per_seq > ham::kMicroMaxSlots || c.n_kv_heads > ham::kMicroMaxKvHeads ||
      (c.head_dim != 64 && c.head_dim != 128))
    return fail(HAM_EUNSUPPORTED, "micro step: needs max_slots_per_seq <= %d, n_kv_heads <= %d, "
                "head_dim 64 or 128 (have %d, %d, %d)", ham::kMicroMaxSlots,
                ham::kMicroMaxKvHeads, c.max_slots_per_seq, c.n_kv_heads, c.head_dim);
  {  // outputs are written while q is still being read
    const size_t n = (size_t)c.batch * c.n_q_heads * c.head_dim;
    const size_t out_bytes = n * (out_dtype == HAM_DTYPE_F32 ? 4 : 2);
    const size_t kv_bytes = (size_t)c.batch * c.n_kv_heads * c.head_dim * 2;
    const size_t pool_bytes = (size_t)c.layers * 2 * (size_t)kv->pool_elems * 2;
    if (overlaps(q, n * 2, out, out_bytes) || overlaps(q_rot, n * 2, q, n * 2) ||
        overlaps(q_rot, n * 2, out, out_bytes) || overlaps(out, out_bytes, kv->pool, pool_bytes) ||
        overlaps(q_rot, n * 2, kv->pool, pool_bytes) || overlaps(k_new, kv_bytes, kv->pool, pool_bytes) ||
        overlaps(v_new, kv_bytes, kv->pool, pool_bytes))
      return fail(HAM_EINVAL, "q, q_rot, out and the cache must not overlap");
  }
  DeviceGuard guard(kv->device);
  ham::MicroView v{};
  v.q = static_cast<const uint16_t *>(q);
  v.q_rot = static_cast<uint16_t *>(q_rot);
  v.k_new = static_cast<const uint16_t *>(k_new);
  v.v_new = static_cast<const uint16_t *>(v_new);
  v.pos = pos;
  v.ntok = ntok;
  v.out = out;
  v.k_pool = layer_pool(kv, layer, 0);
  v.v_pool = layer_pool(kv, layer, 1);
  v.slot_pos = kv->slot_pos;
  v.slot_ntok = kv->slot_ntok;
  v.page_table = kv->page_table;
  v.num_slots = kv->num_slots + (size_t)layer * c.batch;
  v.num_tokens = kv->num_tokens + (size_t)layer * c.batch;
  v.inv_freq = kv->inv_freq;
  v.rope_table = kv->rope_table;
  v.rope_positions = kv->rope_positions;
  v.err = kv->err;
  v.pool_pages = c.pool_pages;
  v.batch = c.batch;
  v.n_q_heads = c.n_q_heads;
  v.n_kv_heads = c.n_kv_heads;
  v.head_dim = c.head_dim;
  v.page_slots = c.page_slots;
  v.max_pages = kv->max_pages;
  v.max_slots = c.max_slots_per_seq;
  v.pos_mode = c.pos_mode;
  v.out_f32 = out_dtype == HAM_DTYPE_F32 ? 1 : 0;
  cudaError_t e = ham::launch_micro(v, static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "micro step launch");
  note_launch(kv, layer, stream, true);
  return HAM_OK;
}

int ham_prefill(ham_kv *kv, int32_t layer, void *q_inout, const void *k_new, const void *v_new,
                const int32_t *offsets, const int32_t *pos, const int32_t *ntok,
                int32_t total_rows, void *out, int32_t out_dtype, void *stream) {
  ham::ApiRange nvtx_range("ham_prefill");
  int rc = check_layer(kv, layer);
  if (rc) return rc;
  if ((rc = fp8_unsupported(kv, "ham_prefill")) != 0) return rc;
  if (out_dtype != HAM_DTYPE_BF16 && out_dtype != HAM_DTYPE_F32)
    return fail(HAM_EINVAL, "out_dtype %d", out_dtype);
  const ham_config &c = kv->cfg;
  if (total_rows < 0 || (int64_t)total_rows > (int64_t)c.batch * c.max_slots_per_seq)
    return fail(HAM_EINVAL, "total_rows %d outside 0..batch * max_slots_per_seq", total_rows);
  if (total_rows == 0) return HAM_OK;  // nothing to store or attend (the buffers may be NULL)
  if (!q_inout || !k_new || !v_new || !offsets || !out)
    return fail(HAM_EINVAL, "q_inout, k_new, v_new, offsets and out are required");
  if (!aligned16(q_inout) || !aligned16(k_new) || !aligned16(v_new) || !aligned16(out))
    return fail(HAM_EINVAL, "q/k/v/out must be 16-byte aligned");
  if (((uintptr_t)offsets & 3u) || ((uintptr_t)pos & 3u) || ((uintptr_t)ntok & 3u))
    return fail(HAM_EINVAL, "offsets/pos/ntok must be 4-byte aligned");
  const int group = c.n_q_heads / c.n_kv_heads;
  if (!ham::prefill_supported(c.head_dim, group))
    return fail(HAM_EUNSUPPORTED, "prefill: head_dim %d / group %d not compiled", c.head_dim,
                group);
  const size_t T = (size_t)total_rows, d = (size_t)c.head_dim;
  const size_t q_bytes = T * c.n_q_heads * d * 2, kv_bytes = T * c.n_kv_heads * d * 2;
  const size_t out_bytes = T * c.n_q_heads * d * (out_dtype == HAM_DTYPE_F32 ? 4 : 2);
  const size_t pool_bytes = (size_t)c.layers * 2 * (size_t)kv->pool_elems * 2;
  if (overlaps(q_inout, q_bytes, out, out_bytes) || overlaps(q_inout, q_bytes, k_new, kv_bytes) ||
      overlaps(q_inout, q_bytes, v_new, kv_bytes) || overlaps(out, out_bytes, k_new, kv_bytes) ||
      overlaps(out, out_bytes, v_new, kv_bytes) || overlaps(q_inout, q_bytes, kv->pool, pool_bytes) ||
      overlaps(out, out_bytes, kv->pool, pool_bytes) || overlaps(k_new, kv_bytes, kv->pool, pool_bytes) ||
      overlaps(v_new, kv_bytes, kv->pool, pool_bytes))
    return fail(HAM_EINVAL, "q_inout, out, k_new, v_new and the cache must not overlap");
  const int64_t blocks = (int64_t)total_rows / ham::prefill_query_rows(group) + c.batch;
  if (blocks > 65535)
    return fail(HAM_EINVAL, "total_rows %d: split the chunk (at most %lld query blocks a call)",
                total_rows, 65535LL);
  DeviceGuard guard(kv->device);
  ham::PrefillView v{};
  v.k_pool = layer_pool(kv, layer, 0);
  v.v_pool = layer_pool(kv, layer, 1);
  v.slot_pos = kv->slot_pos;
  v.slot_ntok = kv->slot_ntok;
  v.page_table = kv->page_table;
  v.num_slots = kv->num_slots + (size_t)layer * c.batch;
  v.num_tokens = kv->num_tokens + (size_t)layer * c.batch;
  v.rope_table_ff = kv->rope_table_ff;
  v.inv_freq = kv->inv_freq;
  v.rope_positions = kv->rope_positions;
  v.q = static_cast<uint16_t *>(q_inout);
  v.k_new = static_cast<const uint16_t *>(k_new);
  v.v_new = static_cast<const uint16_t *>(v_new);
  v.offsets = offsets;
  v.pos = pos;
  v.ntok = ntok;
  v.out = out;
  v.wait_ns = kv->wait_ns;
  v.seq_info = kv->prefill_seq;
  v.row_info = kv->prefill_rows;
  // Split over slots when the grid would leave SMs idle (a short chunk, whatever the cache
  // holds: the kernel keeps one split for sequences with few cached slots).
  {
    const int64_t base = (int64_t)c.n_kv_heads * blocks;
    int Z = 1;
    if (kv->prefill_part && 2 * base <= kv->num_sms) {
      Z = (int)std::min<int64_t>(ham::kPrefillMaxSplits, kv->num_sms / base);
      while (Z > 1 && (size_t)Z * T * c.n_q_heads * d >
                          ham::prefill_part_floats(kv->num_sms, c.head_dim))
        --Z;
    }
    v.splits = Z;
    v.part_o = kv->prefill_part;
    v.part_ml = kv->prefill_part_ml;
  }
  v.err = kv->err;
  v.pool_pages = c.pool_pages;
  v.batch = c.batch;
  v.rows = total_rows;
  v.n_q_heads = c.n_q_heads;
  v.n_kv_heads = c.n_kv_heads;
  v.head_dim = c.head_dim;
  v.page_slots = c.page_slots;
  v.max_pages = kv->max_pages;
  v.max_slots = c.max_slots_per_seq;
  v.pos_mode = c.pos_mode;
  cudaError_t e = ham::launch_prefill(kv->tmaps_half[(size_t)layer * 2],
                                      kv->tmaps_half[(size_t)layer * 2 + 1], v, out_dtype,
                                      static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "prefill launch");
  note_launch(kv, layer, stream, true);
  return HAM_OK;
}

int ham_decode_attn(ham_kv *kv, int32_t layer, const void *q, void *out, void *stream) {
  return ham_decode_attn_ex(kv, layer, q, out, HAM_DTYPE_BF16, stream);
}

int ham_kv_layer_lengths(ham_kv *kv, int32_t layer, int32_t *num_slots_host,
                         int64_t *num_tokens_host, void *stream) {
  int rc = check_layer(kv, layer);
  if (rc) return rc;
  DeviceGuard guard(kv->device);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const int B = kv->cfg.batch;
  uint8_t *h = static_cast<uint8_t *>(kv->host_stage);
  int32_t *h_err = reinterpret_cast<int32_t *>(h);
  int64_t *h_tok = reinterpret_cast<int64_t *>(h + 64);
  int32_t *h_slots = reinterpret_cast<int32_t *>(h + 64 + (size_t)B * 8);
  HAM_CUDA(cudaMemcpyAsync(h_slots, kv->num_slots + (size_t)layer * B, B * sizeof(int32_t),
                           cudaMemcpyDeviceToHost, s));
  HAM_CUDA(cudaMemcpyAsync(h_tok, kv->num_tokens + (size_t)layer * B, B * sizeof(int64_t),
                           cudaMemcpyDeviceToHost, s));
  HAM_CUDA(cudaMemcpyAsync(h_err, kv->err, sizeof(int32_t), cudaMemcpyDeviceToHost, s));
  HAM_CUDA(cudaStreamSynchronize(s));
  if (num_slots_host) memcpy(num_slots_host, h_slots, B * sizeof(int32_t));
  if (num_tokens_host) memcpy(num_tokens_host, h_tok, B * sizeof(int64_t));
  if (*h_err != 0) return fail(HAM_EDEVICE, "device error word = %d", *h_err);
  return HAM_OK;
}

int ham_slot_lengths(ham_kv *kv, int32_t *num_slots_host, int64_t *num_tokens_host,
                     void *stream) {
  if (!kv) return fail(HAM_EINVAL, "null handle");
  return ham_kv_layer_lengths(kv, kv->cfg.layers - 1, num_slots_host, num_tokens_host, stream);
}

int ham_kv_status(ham_kv *kv, void *stream, int32_t *device_code) {
  if (!kv) return fail(HAM_EINVAL, "null handle");
  DeviceGuard guard(kv->device);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  int32_t *h_err = static_cast<int32_t *>(kv->host_stage);
  HAM_CUDA(cudaMemcpyAsync(h_err, kv->err, sizeof(int32_t), cudaMemcpyDeviceToHost, s));
  HAM_CUDA(cudaMemsetAsync(kv->err, 0, sizeof(int32_t), s));
  HAM_CUDA(cudaStreamSynchronize(s));
  if (device_code) *device_code = *h_err;
  if (*h_err != 0) return fail(HAM_EDEVICE, "device error word = %d", *h_err);
  return HAM_OK;
}

int ham_kv_set_page_table(ham_kv *kv, const int32_t *host_pt) {
  if (!kv || !host_pt) return fail(HAM_EINVAL, "null argument");
  const size_t n = (size_t)kv->cfg.batch * kv->max_pages;
  std::vector<uint8_t> used((size_t)kv->cfg.pool_pages, 0);
  for (size_t i = 0; i < n; ++i) {
    int32_t p = host_pt[i];
    if (p < 0 || p >= kv->cfg.pool_pages)
      return fail(HAM_EINVAL, "page table entry %zu = %d outside [0, %lld)", i, p,
                  (long long)kv->cfg.pool_pages);
    if (used[(size_t)p]++) return fail(HAM_EINVAL, "page %d appears twice", p);
  }
  DeviceGuard guard(kv->device);
  HAM_CUDA(cudaDeviceSynchronize());
  HAM_CUDA(cudaMemcpy(kv->page_table, host_pt, n * sizeof(int32_t), cudaMemcpyHostToDevice));
  return HAM_OK;
}

int ham_kv_get_page_table(const ham_kv *kv, int32_t *host_pt) {
  if (!kv || !host_pt) return fail(HAM_EINVAL, "null argument");
  DeviceGuard guard(kv->device);
  HAM_CUDA(cudaMemcpy(host_pt, kv->page_table,
                      (size_t)kv->cfg.batch * kv->max_pages * sizeof(int32_t),
                      cudaMemcpyDeviceToHost));
  return HAM_OK;
}

int ham_kv_fill(ham_kv *kv, int32_t layer, const void *k_log, const void *v_log,
                const int32_t *pos, const int32_t *ntok, const int32_t *counts, int32_t lmax,
                void *stream) {
  ham::ApiRange nvtx_range("ham_kv_fill");
  int rc = check_layer(kv, layer);
  if (rc) return rc;
  if (!counts || lmax < 0 || (lmax > 0 && (!k_log || !v_log)))
    return fail(HAM_EINVAL, "counts, lmax >= 0 and (for lmax > 0) k_log, v_log are required");
  if ((k_log && !aligned16(k_log)) || (v_log && !aligned16(v_log)))
    return fail(HAM_EINVAL, "k_log/v_log must be 16-byte aligned");
  DeviceGuard guard(kv->device);
  ham::FillView v{};
  v.k_pool = layer_pool(kv, layer, 0);
  v.v_pool = layer_pool(kv, layer, 1);
  v.kv_exp = layer_exp(kv, layer);
  v.slot_pos = kv->slot_pos;
  v.slot_ntok = kv->slot_ntok;
  v.page_table = kv->page_table;
  v.num_slots = kv->num_slots + (size_t)layer * kv->cfg.batch;
  v.num_tokens = kv->num_tokens + (size_t)layer * kv->cfg.batch;
  v.k_log = static_cast<const uint16_t *>(k_log);
  v.v_log = static_cast<const uint16_t *>(v_log);
  v.pos = pos;
  v.ntok = ntok;
  v.counts = counts;
  v.err = kv->err;
  v.pool_pages = kv->cfg.pool_pages;
  v.batch = kv->cfg.batch;
  v.n_kv_heads = kv->cfg.n_kv_heads;
  v.head_dim = kv->cfg.head_dim;
  v.page_slots = kv->cfg.page_slots;
  v.max_pages = kv->max_pages;
  v.max_slots = kv->cfg.max_slots_per_seq;
  v.lmax = lmax;
  cudaError_t e = ham::launch_fill(v, static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "fill launch");
  note_launch(kv, layer, stream, true);
  return HAM_OK;
}

int ham_kv_export(ham_kv *kv, int32_t layer, void *k_dst, void *v_dst, int32_t *pos_dst,
                  int32_t *ntok_dst, void *stream) {
  ham::ApiRange nvtx_range("ham_kv_export");
  int rc = check_layer(kv, layer);
  if (rc) return rc;
  DeviceGuard guard(kv->device);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const size_t pool_bytes = (size_t)kv->pool_elems * (kv->fp8 ? 1 : sizeof(uint16_t));
  const size_t meta_bytes = (size_t)kv->cfg.pool_pages * kv->cfg.page_slots * sizeof(int32_t);
  if (k_dst) HAM_CUDA(cudaMemcpyAsync(k_dst, layer_pool(kv, layer, 0), pool_bytes, cudaMemcpyDefault, s));
  if (v_dst) HAM_CUDA(cudaMemcpyAsync(v_dst, layer_pool(kv, layer, 1), pool_bytes, cudaMemcpyDefault, s));
  if (pos_dst) HAM_CUDA(cudaMemcpyAsync(pos_dst, kv->slot_pos, meta_bytes, cudaMemcpyDefault, s));
  if (ntok_dst) HAM_CUDA(cudaMemcpyAsync(ntok_dst, kv->slot_ntok, meta_bytes, cudaMemcpyDefault, s));
  return HAM_OK;
}

int ham_kv_export_scales(ham_kv *kv, int32_t layer, void *e_dst, void *stream) {
  int rc = check_layer(kv, layer);
  if (rc) return rc;
  if (!kv->fp8) return fail(HAM_EINVAL, "not an FP8 cache");
  if (!e_dst) return fail(HAM_EINVAL, "e_dst is required");
  DeviceGuard guard(kv->device);
  HAM_CUDA(cudaMemcpyAsync(e_dst, layer_exp(kv, layer), (size_t)pool_rows(kv) * 2,
                           cudaMemcpyDefault, static_cast<cudaStream_t>(stream)));
  return HAM_OK;
}

int ham_kv_set_lengths(ham_kv *kv, int32_t layer, const int32_t *num_slots,
                       const int64_t *num_tokens, void *stream) {
  ham::ApiRange nvtx_range("ham_kv_set_lengths");
  int rc = check_layer(kv, layer);
  if (rc) return rc;
  if (!num_slots) return fail(HAM_EINVAL, "num_slots is required");
  DeviceGuard guard(kv->device);
  const int B = kv->cfg.batch;
  ham::set_lengths_kernel<<<(B + 127) / 128, 128, 0, static_cast<cudaStream_t>(stream)>>>(
      kv->num_slots + (size_t)layer * B, kv->num_tokens + (size_t)layer * B, num_slots,
      num_tokens, B, kv->cfg.max_slots_per_seq, kv->err);
  HAM_CUDA(cudaGetLastError());
  note_launch(kv, layer, stream, true);
  return HAM_OK;
}

int ham_kv_reset(ham_kv *kv, void *stream) {
  if (!kv) return fail(HAM_EINVAL, "null handle");
  DeviceGuard guard(kv->device);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const size_t n = (size_t)kv->cfg.layers * kv->cfg.batch;
  HAM_CUDA(cudaMemsetAsync(kv->num_slots, 0, n * sizeof(int32_t), s));
  HAM_CUDA(cudaMemsetAsync(kv->num_tokens, 0, n * sizeof(int64_t), s));
  note_launch(kv, -1, stream, true);
  return HAM_OK;
}

int ham_split_plan(int32_t batch, int32_t n_kv_heads, const int32_t *num_slots_host,
                   int32_t ctas, int64_t *cta_begin, int32_t *seg_first_cta,
                   int32_t *seg_last_cta) {
  if (batch < 1 || n_kv_heads < 1 || ctas < 1 || !num_slots_host)
    return fail(HAM_EINVAL, "bad plan arguments");
  std::vector<int64_t> cum((size_t)batch + 1, 0);
  for (int32_t b = 0; b < batch; ++b) {
    if (num_slots_host[b] < 0) return fail(HAM_EINVAL, "negative slot count");
    cum[(size_t)b + 1] = cum[(size_t)b] + ham::chunks_of(num_slots_host[b]);
  }
  const int64_t W = (int64_t)n_kv_heads * cum[(size_t)batch];
  const int32_t C = ham::plan_ctas(W, ctas);  // CTAs that get chunks; the rest stay idle
  if (cta_begin)
    for (int32_t c = 0; c <= ctas; ++c)
      cta_begin[c] = C ? ham::plan_cta_begin(W, C, c < C ? c : C) : 0;
  for (int32_t b = 0; b < batch; ++b) {
    const int64_t nch = cum[(size_t)b + 1] - cum[(size_t)b];
    for (int32_t g = 0; g < n_kv_heads; ++g) {
      const int64_t s = (int64_t)b * n_kv_heads + g;
      const int64_t x0 = (int64_t)n_kv_heads * cum[(size_t)b] + g * nch;
      const int32_t first = nch ? ham::plan_owner(W, C, x0) : -1;
      const int32_t last = nch ? ham::plan_owner(W, C, x0 + nch - 1) : -1;
      if (seg_first_cta) seg_first_cta[s] = first;
      if (seg_last_cta) seg_last_cta[s] = last;
    }
  }
  return HAM_OK;
}

}  // extern "C"
