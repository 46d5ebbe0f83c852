// sf_device.cuh - device-side building blocks shared by the libstagefrontier
// kernels: mbarrier / bulk-tensor-copy PTX wrappers, a bounded barrier wait,
// warp reductions on 64-bit keys, and the status word.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "stagefrontier.h"

namespace sf {

constexpr unsigned kFull = 0xffffffffu;
// A device wait gives up after this many nanoseconds of %globaltimer; one
// tile normally lands in microseconds.
constexpr uint64_t kWaitLimitNs = 2000000000ull;

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ uint64_t global_timer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}

// Make mbarrier initialisation visible to the async (TMA) proxy.
__device__ __forceinline__ void fence_barrier_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(bytes)
               : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// Wait for the phase of `bar` with the given parity to complete.  Returns
// false, without waiting further, once *abort is set or after `limit_ns` of
// %globaltimer; the caller then records SF_ST_TIMEOUT and runs to completion
// without data.
__device__ __forceinline__ bool mbar_wait_bounded(uint64_t* bar, uint32_t parity, volatile int* abort,
                                                  uint64_t limit_ns = kWaitLimitNs) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = global_timer_ns();
  for (uint32_t i = 1;; ++i) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((i & 63u) == 0u) {
      if (*abort) return false;
      if (global_timer_ns() - t0 > limit_ns) {
        *abort = 1;
        return false;
      }
    }
  }
}

// Wait (bounded by kWaitLimitNs, no abort flag) for a phase; used to let
// copies still in flight land before a CTA exits.  Returns false on timeout.
__device__ __forceinline__ bool mbar_wait_timeout(uint64_t* bar, uint32_t parity) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = global_timer_ns();
  while (!mbar_try_wait(bar, parity))
    if (global_timer_ns() - t0 > kWaitLimitNs) return false;
  return true;
}

__device__ __forceinline__ unsigned char* align_1024(unsigned char* p) {
  return p + ((1024u - (smem_u32(p) & 1023u)) & 1023u);
}

// 2-D tiled bulk tensor copy global -> shared, completion counted in bytes on `bar`.
__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, int32_t x, int32_t y,
                                            uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3}], [%4];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(smem_u32(bar))
      : "memory");
}

__device__ __forceinline__ void prefetch_tensormap(const CUtensorMap* map) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(map)) : "memory");
}

// Named barrier among `count` threads (a multiple of 32), id 1..15.
__device__ __forceinline__ void named_barrier(uint32_t id, uint32_t count) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(count) : "memory");
}

// Unsigned 64-bit max over the full warp with two 32-bit redux steps:
// the high words decide, the low words break ties among the winners.
__device__ __forceinline__ uint64_t warp_max_u64(uint64_t v) {
  const unsigned hi = static_cast<unsigned>(v >> 32);
  const unsigned lo = static_cast<unsigned>(v);
  const unsigned mhi = __reduce_max_sync(kFull, hi);
  const unsigned mlo = __reduce_max_sync(kFull, hi == mhi ? lo : 0u);
  return (static_cast<uint64_t>(mhi) << 32) | mlo;
}

__device__ __forceinline__ uint64_t warp_min_u64(uint64_t v) {
  const unsigned hi = static_cast<unsigned>(v >> 32);
  const unsigned lo = static_cast<unsigned>(v);
  const unsigned mhi = __reduce_min_sync(kFull, hi);
  const unsigned mlo = __reduce_min_sync(kFull, hi == mhi ? lo : 0xffffffffu);
  return (static_cast<uint64_t>(mhi) << 32) | mlo;
}

// Histogram scan of one radix pass: the digit d whose bin holds rank `rem`
// among the counted values, and the count of values in lower bins.  Each lane
// owns 8 consecutive bins (h[0..7] = bins 8*lane .. 8*lane+7); the lane whose
// range holds `rem` is found with one warp scan and one ballot, and the bin
// within it by counting the inclusive prefixes not above `rem` (every lane
// does the arithmetic; the owner's result is broadcast).
__device__ __forceinline__ void bins_find(const uint32_t (&h)[8], uint32_t rem, int lane, uint32_t& digit,
                                          uint32_t& below) {
  uint32_t c[8];  // inclusive prefix within the lane's 8 bins
  c[0] = h[0];
#pragma unroll
  for (int q = 1; q < 8; ++q) c[q] = c[q - 1] + h[q];
  uint32_t incl = c[7];
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t up = __shfl_up_sync(kFull, incl, o);
    if (lane >= o) incl += up;
  }
  const uint32_t excl = incl - c[7];
  const int owner = __ffs(__ballot_sync(kFull, excl <= rem && rem < incl)) - 1;
  const uint32_t r = rem - excl;  // rank within the owner's bins
  uint32_t j = 0, bl = 0;
#pragma unroll
  for (int q = 0; q < 7; ++q) {
    const bool past = c[q] <= r;  // bin q lies wholly below rank r
    j += past ? 1u : 0u;
    bl = past ? c[q] : bl;
  }
  digit = __shfl_sync(kFull, 8u * lane + j, owner);
  below = __shfl_sync(kFull, excl + bl, owner);
}

// bins_find over a 256-bin shared-memory histogram (16-byte aligned).
__device__ __forceinline__ void hist_find(const uint32_t* hist, uint32_t rem, int lane, uint32_t& digit,
                                          uint32_t& below) {
  const uint4 h0 = reinterpret_cast<const uint4*>(hist)[2 * lane];
  const uint4 h1 = reinterpret_cast<const uint4*>(hist)[2 * lane + 1];
  const uint32_t h[8] = {h0.x, h0.y, h0.z, h0.w, h1.x, h1.y, h1.z, h1.w};
  bins_find(h, rem, lane, digit, below);
}

// Programmatic dependent launch.  A kernel launched with programmatic stream
// serialization may start while the previous kernel on its stream still runs,
// once every CTA of that kernel has called griddep_launch_dependents() (or
// has exited); griddep_wait() returns when the previous kernel has completed
// and its memory operations are visible, and at once for a kernel launched
// without that attribute.
__device__ __forceinline__ void griddep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void griddep_launch_dependents() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

__device__ __forceinline__ void report(uint32_t* status, uint32_t bits) {
  if (status != nullptr && bits != 0u) atomicOr(status, bits);
}

// Status bits from the OR of the high words of every duration (sign bit:
// negative; bits 47..62: >= 2^47) and of every rank total.
__device__ __forceinline__ uint32_t range_bits(uint32_t d_hi_or, uint32_t total_hi_or) {
  uint32_t b = 0;
  if (d_hi_or & 0x80000000u) b |= SF_ST_NEGATIVE;
  if ((d_hi_or & 0x7fff8000u) || (total_hi_or & 0xffff8000u)) b |= SF_ST_RANGE;
  return b;
}

// 128-bit accumulation into two uint64 words with order-independent carries.
__device__ __forceinline__ void atomic_add_u128(uint64_t* p, unsigned __int128 v) {
  const unsigned long long lo = static_cast<unsigned long long>(v);
  const unsigned long long hi = static_cast<unsigned long long>(v >> 64);
  const unsigned long long old = atomicAdd(reinterpret_cast<unsigned long long*>(p), lo);
  const unsigned long long carry = (old + lo < old) ? 1ull : 0ull;
  if (hi + carry) atomicAdd(reinterpret_cast<unsigned long long*>(p + 1), hi + carry);
}

}  // namespace sf
