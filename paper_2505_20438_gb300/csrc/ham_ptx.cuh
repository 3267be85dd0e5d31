// Inline-PTX wrappers shared by the attention kernels of libham.so (sm_103a): shared-memory
// addresses, mbarriers, TMA copies, ldmatrix / movmatrix, the bf16 mma.sync tile, programmatic
// dependent launch, and the bounded mbarrier waits every kernel uses (no unbounded spin).
#pragma once

#include <cuda.h>
#include <stdint.h>

namespace ham {
namespace {

constexpr uint32_t kFull = 0xffffffffu;
constexpr uint64_t kWaitLimitNs = 2000000000ull;   // bounded waits: 2 s

// ------------------------------------------------------------------------------------
// PTX wrappers
// ------------------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_u32(const void *p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ uint64_t global_timer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
__device__ __forceinline__ void mbar_init(uint64_t *bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count)
               : "memory");
}
__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
__device__ __forceinline__ void mbar_arrive(uint64_t *bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}
__device__ __forceinline__ void mbar_arrive_tx(uint64_t *bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(bytes)
               : "memory");
}
// Add `bytes` to the transaction count of the current phase without arriving.
__device__ __forceinline__ void mbar_expect_tx(uint64_t *bar, uint32_t bytes) {
  asm volatile("mbarrier.expect_tx.relaxed.cta.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(bytes)
               : "memory");
}
__device__ __forceinline__ bool mbar_test(uint64_t *bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
      " selp.u32 %0, 1, 0, p;\n}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}
// Non-blocking test of an mbarrier phase (never suspends the thread, unlike try_wait).
__device__ __forceinline__ bool mbar_poll(uint64_t *bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n"
      " selp.u32 %0, 1, 0, p;\n}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}
__device__ __forceinline__ uint64_t policy_evict_last() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
  return p;
}
__device__ __forceinline__ uint64_t policy_evict_first() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}
// 1-D bulk copy global -> shared (TMA engine); 16-byte aligned, size % 16 == 0.
__device__ __forceinline__ void bulk_load(void *dst, const void *src, uint32_t bytes,
                                          uint64_t *bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1], %2, [%3];" ::"r"(smem_u32(dst)),
      "l"(src), "r"(bytes), "r"(smem_u32(bar))
      : "memory");
}
// Rank-3 tiled TMA copy of the box at (x, y, z) of `map` into shared memory.
__device__ __forceinline__ void tma_load_3d(void *dst, const CUtensorMap *map, int x, int y,
                                            int z, uint64_t *bar, uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      ".L2::cache_hint [%0], [%1, {%2, %3, %4}], [%5], %6;" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(z), "r"(smem_u32(bar)),
      "l"(policy)
      : "memory");
}
__device__ __forceinline__ void prefetch_tensormap(const CUtensorMap *map) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(map)) : "memory");
}
__device__ __forceinline__ void ldmatrix_x4(uint32_t (&r)[4], uint32_t addr) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(addr));
}
__device__ __forceinline__ void ldmatrix_x4_trans(uint32_t (&r)[4], uint32_t addr) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(addr));
}
__device__ __forceinline__ uint32_t movmatrix_trans(uint32_t a) {
  uint32_t d;
  asm volatile("movmatrix.sync.aligned.m8n8.trans.b16 %0, %1;" : "=r"(d) : "r"(a));
  return d;
}
// D += A * B for one 16x8x16 tile: A 16x16 bf16 (row), B 16x8 bf16 (col), D fp32.
__device__ __forceinline__ void mma_16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0,
                                          uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 "
      "{%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, {%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
// Two fp32 -> packed bf16 (round to nearest even): lo in bits 0..15, hi in 16..31.
__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  uint32_t d;
  asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(d) : "f"(hi), "f"(lo));
  return d;
}
__device__ __forceinline__ void grid_dependency_wait() {
  asm volatile("griddepcontrol.wait;" ::: "memory");
}
__device__ __forceinline__ void grid_launch_dependents() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}
__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// One thread waits on an mbarrier phase, bounded.  honor_abort: give up early once another
// warp has aborted (not used while draining in-flight copies).
// limit_ns: how long to wait (the default, 2 s, unless a caller shortened its data waits).  A
// shortened limit polls without suspending (try_wait may sleep for longer than the limit), so
// that it is honoured to within a poll.
__device__ bool thread_wait(uint64_t *bar, uint32_t parity, volatile int *abort_flag,
                            bool honor_abort, uint64_t limit_ns = kWaitLimitNs) {
  if (limit_ns < kWaitLimitNs) {
    const uint64_t t0 = global_timer_ns();
    while (!mbar_poll(bar, parity)) {
      if (honor_abort && *abort_flag) return false;
      if (global_timer_ns() - t0 > limit_ns) return false;
    }
    return true;
  }
  if (mbar_test(bar, parity)) return true;
  const uint64_t t0 = global_timer_ns();
  for (uint32_t n = 1;; ++n) {
    if (mbar_test(bar, parity)) return true;
    if ((n & 15u) == 0) {
      if (honor_abort && *abort_flag) return false;
      if (global_timer_ns() - t0 > limit_ns) return false;
    }
  }
}

// The whole warp waits on an mbarrier phase, bounded; the result is warp-uniform.
__device__ bool warp_wait(uint64_t *bar, uint32_t parity, volatile int *abort_flag,
                          uint64_t limit_ns = kWaitLimitNs) {
  if (limit_ns < kWaitLimitNs) {  // shortened: poll without suspending, lane 0 keeps the time
    const uint64_t t0 = global_timer_ns();
    for (;;) {
      if (__all_sync(kFull, mbar_poll(bar, parity))) return true;
      int stop = 0;
      if ((threadIdx.x & 31) == 0)
        stop = (*abort_flag != 0) || (global_timer_ns() - t0 > limit_ns);
      if (__shfl_sync(kFull, stop, 0)) return false;
    }
  }
  if (__all_sync(kFull, mbar_test(bar, parity))) return true;
  const uint64_t t0 = global_timer_ns();
  for (uint32_t n = 1;; ++n) {
    if (__all_sync(kFull, mbar_test(bar, parity))) return true;
    if ((n & 15u) == 0) {
      int stop = 0;
      if ((threadIdx.x & 31) == 0)
        stop = (*abort_flag != 0) || (global_timer_ns() - t0 > limit_ns);
      if (__shfl_sync(kFull, stop, 0)) return false;
    }
  }
}

// Byte offset of the 16-byte piece `c` (elements 8c .. 8c+7) of row `row` in a tile written by a
// TMA copy with the 128-byte swizzle: rows are split into 128-byte lines (line = row *
// lines_per_row + c / 8) and the piece index inside a line is XORed with line % 8.  The tile
// must start on a 1024-byte boundary.
// Data-wait limit of a launch: the caller's (nonzero) value, else the default.
__device__ __forceinline__ uint64_t data_wait_limit(uint64_t wait_ns) {
  return wait_ns ? wait_ns : kWaitLimitNs;
}

__device__ __forceinline__ uint32_t swizzle128_offset(int row, int c, int lines_per_row) {
  const int line = row * lines_per_row + (c >> 3);
  return (uint32_t)(line * 128 + (((c & 7) ^ (line & 7)) << 4));
}

}  // namespace
}  // namespace ham
