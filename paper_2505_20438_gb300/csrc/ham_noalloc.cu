// Decode attention that allocates nothing: the split-attention scratch (partial softmax
// states and per-segment CTA ranges) lives in a file-scope device array instead of memory
// owned by a ham_kv handle, and the caller passes every input and output.
//
// The array's name in host code is only a host-side stand-in: kernels must be given the
// device address, which cudaGetSymbolAddress returns per device.  That lookup, and the
// shared-memory attribute of all four attention instances (bf16 / fp32 output, head_dim 64 /
// 128), happen on the first call on each device, whatever that call's dtype and head_dim.
#include <cstdio>
#include <cstring>
#include <mutex>

#include "ham_internal.cuh"

namespace {

constexpr size_t kScratchBytes = 8u << 20;  // 8 MiB per device, held until the process exits

static __device__ __align__(256) unsigned char g_attn_scratch[kScratchBytes];

int noalloc_fail(int status, const char *msg) { return ham::set_last_error(status, msg); }

struct DeviceSetup {
  void *scratch = nullptr;
  int num_sms = 0;
  bool done = false;
};

std::mutex g_setup_mu;
DeviceSetup g_setup[64];

size_t align256(size_t x) { return (x + 255) / 256 * 256; }

}  // namespace

extern "C" {

int ham_decode_attn_noalloc(const ham_attn_args *a, void *stream) {
  ham::ApiRange nvtx_range("ham_decode_attn_noalloc");
  if (!a) return noalloc_fail(HAM_EINVAL, "args is NULL");
  if (!a->k_pool || !a->v_pool || !a->page_table || !a->num_slots || !a->q || !a->out)
    return noalloc_fail(HAM_EINVAL, "k_pool, v_pool, page_table, num_slots, q and out are required");
  if (a->batch < 1 || a->batch > ham::kMaxBatch || a->n_kv_heads < 1 || a->n_q_heads < 1 ||
      a->n_q_heads % a->n_kv_heads != 0 || a->page_slots < ham::kChunkSlots ||
      a->page_slots % ham::kChunkSlots != 0 || a->max_pages < 1 || a->max_slots < 0 ||
      (int64_t)a->max_slots > (int64_t)a->max_pages * a->page_slots || a->pool_pages < 1 ||
      a->ctas < 0 || (a->out_dtype != HAM_DTYPE_BF16 && a->out_dtype != HAM_DTYPE_F32))
    return noalloc_fail(HAM_EINVAL, "bad shape or settings in ham_attn_args");
  const int group = a->n_q_heads / a->n_kv_heads;
  if (!ham::attention_supported(a->head_dim, group))
    return noalloc_fail(HAM_EUNSUPPORTED, "head_dim must be 64 or 128 and the group 1..8");
  const int64_t rows = a->pool_pages * a->n_kv_heads * (int64_t)a->page_slots;
  if (rows > INT32_MAX) return noalloc_fail(HAM_EINVAL, "pool too large for int32 TMA rows");
  const uintptr_t align_or = (uintptr_t)a->k_pool | (uintptr_t)a->v_pool | (uintptr_t)a->q |
                             (uintptr_t)a->out;
  if (align_or & 15u) return noalloc_fail(HAM_EINVAL, "pools, q and out must be 16-byte aligned");

  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64)
    return noalloc_fail(HAM_ECUDA, "no usable current CUDA device");
  DeviceSetup setup;
  {
    std::lock_guard<std::mutex> lock(g_setup_mu);
    DeviceSetup &s = g_setup[dev];
    if (!s.done) {  // once per device, with that device current
      void *p = nullptr;
      cudaError_t e = cudaGetSymbolAddress(&p, g_attn_scratch);
      if (e != cudaSuccess || !p) {
        cudaGetLastError();
        return noalloc_fail(HAM_ECUDA, "cudaGetSymbolAddress of the static scratch failed");
      }
      int sms = 0;
      if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
        return noalloc_fail(HAM_ECUDA, "cannot read the SM count");
      // every attention instance this entry point can launch (bf16 / fp32 output, head_dim 64
      // / 128) gets its attribute now, so that no later call makes one, inside a capture or not
      if (ham::configure_attention_instances() != cudaSuccess) {
        cudaGetLastError();
        return noalloc_fail(HAM_ECUDA, "cannot set the attention kernels' shared-memory size");
      }
      s.scratch = p;
      s.num_sms = sms;
      s.done = true;
    }
    setup = s;
  }

  int ctas = a->ctas;
  if (ctas == 0) {
    const int per_sm =
        ham::attention_ctas_per_sm(a->head_dim, group, a->batch, false, a->out_dtype);
    if (per_sm <= 0) return noalloc_fail(HAM_ECUDA, "attention kernel cannot be resident");
    ctas = ham::default_attention_ctas(setup.num_sms, per_sm);
  }
  // scratch: partial (acc, max/sum) for each (CTA, segment) incidence, then segment ranges
  const size_t n_seg = (size_t)a->batch * a->n_kv_heads;
  const size_t n_part = (size_t)ctas + n_seg;
  const size_t acc_bytes = align256(n_part * group * a->head_dim * sizeof(float));
  const size_t ml_bytes = align256(n_part * group * sizeof(float2));
  const size_t seg_bytes = align256(n_seg * sizeof(int2));
  if (acc_bytes + ml_bytes + seg_bytes > kScratchBytes) {
    char msg[200];
    snprintf(msg, sizeof msg,
             "needs %zu scratch bytes for %d CTAs and %zu segments; the static scratch holds "
             "%zu (use fewer CTAs, a smaller batch, or ham_decode_attn)",
             acc_bytes + ml_bytes + seg_bytes, ctas, n_seg, kScratchBytes);
    return noalloc_fail(HAM_EINVAL, msg);
  }

  CUtensorMap tk, tv;
  if (ham::make_pool_tensor_map(&tk, a->k_pool, rows, a->head_dim, false) != 0 ||
      ham::make_pool_tensor_map(&tv, a->v_pool, rows, a->head_dim, false) != 0)
    return noalloc_fail(HAM_ECUDA, "cuTensorMapEncodeTiled failed for the pools");

  unsigned char *base = static_cast<unsigned char *>(setup.scratch);
  ham::AttnView v{};
  v.k_pool = static_cast<const uint16_t *>(a->k_pool);
  v.v_pool = static_cast<const uint16_t *>(a->v_pool);
  v.page_table = a->page_table;
  v.num_slots = a->num_slots;
  v.q = static_cast<const uint16_t *>(a->q);
  v.out = a->out;
  v.part_acc = reinterpret_cast<float *>(base);
  v.part_ml = reinterpret_cast<float2 *>(base + acc_bytes);
  v.seg_range = reinterpret_cast<int2 *>(base + acc_bytes + ml_bytes);
  v.err = a->err;
  v.pool_pages = a->pool_pages;
  v.batch = a->batch;
  v.n_kv_heads = a->n_kv_heads;
  v.group = group;
  v.page_slots = a->page_slots;
  v.max_pages = a->max_pages;
  v.max_slots = a->max_slots;
  v.ctas = ctas;
  v.sms = setup.num_sms;
  cudaError_t e = ham::launch_attention(tk, tv, v, a->head_dim, a->out_dtype,
                                        static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) {
    char msg[200];
    snprintf(msg, sizeof msg, "attention launch: %s", cudaGetErrorString(e));
    return noalloc_fail(HAM_ECUDA, msg);
  }
  return HAM_OK;
}

}  // extern "C"
