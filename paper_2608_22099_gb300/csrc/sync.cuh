// sync.cuh -- bounded mbarrier handshakes inside one CTA.
//
// Every wait polls with a clock64 budget; when the budget runs out the waiter
// raises a shared abort flag and returns false, and every other waiter of the
// CTA sees the flag and returns false too, so a protocol slip ends the kernel
// with an error status instead of a hang.
#pragma once

#include <cstdint>

namespace bandlu {

// About one second at the GB300's clocks: far above any legitimate wait here.
constexpr long long kWaitLimitCycles = 2000000000ll;

__device__ __forceinline__ unsigned smem_addr(const void *p) {
  return (unsigned)__cvta_generic_to_shared(p);
}

__device__ __forceinline__ void mbar_init(unsigned long long *bar, unsigned count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(count) : "memory");
}

// Arrive once (release semantics at CTA scope).
__device__ __forceinline__ void mbar_arrive(unsigned long long *bar) {
  asm volatile(
      "{\n\t.reg .b64 st;\n\t"
      "mbarrier.arrive.shared::cta.b64 st, [%0];\n\t}" ::"r"(smem_addr(bar))
      : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(unsigned long long *bar, unsigned parity) {
  unsigned ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_addr(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// Wait for the completion of the phase with the given parity.  Called by all
// 32 lanes of a warp; the result is warp-uniform.
__device__ __forceinline__ bool mbar_wait_warp(unsigned long long *bar, unsigned parity, volatile int *abort_flag) {
  bool ok = true;
  if (!mbar_try_wait(bar, parity)) {
    const long long t0 = clock64();
    for (unsigned it = 1;; ++it) {
      if (mbar_try_wait(bar, parity)) break;
      if ((it & 31u) == 0) {
        if (*abort_flag) {
          ok = false;
          break;
        }
        if (clock64() - t0 > kWaitLimitCycles) {
          *abort_flag = 1;
          ok = false;
          break;
        }
      }
    }
  }
  return __all_sync(0xffffffffu, ok);  // one call site: lanes reconverge here
}

}  // namespace bandlu
