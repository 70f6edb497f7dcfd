// Bounded mbarrier waits shared by the kernels that use mbarrier pipelines.
// A wait never spins forever: after `budget` SM cycles it raises the CTA's
// abort flag, records TQ_ETIMEOUT * 1000 + where in the search status word
// (read back by tq_search_check) and returns false, so the kernel can stop,
// drain what it has in flight and return with the context still usable.
#pragma once

#include <cstdint>

#include "tq_internal.h"

namespace tq {

constexpr long long kWaitCycles = kWaitCyclesMax;

__device__ __forceinline__ uint32_t wait_smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ bool mbar_try_wait_parity(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}"
      : "=r"(ok)
      : "r"(wait_smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// Waits for the phase of `bar` with the given parity; false on timeout or
// when another thread of the CTA has already raised `abort_flag`.
__device__ __forceinline__ bool bounded_wait(uint64_t* bar, uint32_t parity, volatile int* abort_flag, int* err,
                                             int where, long long budget) {
  const long long t0 = clock64();
  for (uint32_t i = 0;; ++i) {
    if (mbar_try_wait_parity(bar, parity)) return true;
    if ((i & 63) == 63) {
      if (*abort_flag) return false;
      if (clock64() - t0 > budget) {
        *abort_flag = 1;
        atomicExch(err, TQ_ETIMEOUT * 1000 + where);
        return false;
      }
    }
  }
}

}  // namespace tq
