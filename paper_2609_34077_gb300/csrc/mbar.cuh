// Shared-memory mbarriers (sm_90+ PTX) with bounded waits, used by the tensor-core expert GEMMs
// (gemm_tc.cu). Not part of the C ABI.
#pragma once

#include "common.cuh"

namespace mcft {

// Limit of every bounded mbarrier wait: after it the waiter records MCFT_ERR_TIMEOUT and returns.
constexpr uint64_t kTimeoutNs = 2000000000ull;

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
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
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
      " selp.u32 %0, 1, 0, p;\n}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// Wait for the phase of `parity` to complete; false if the kernel is aborting or 2 s passed.
__device__ inline bool mbar_wait(uint64_t* bar, uint32_t parity, volatile int* abort,
                                 unsigned* err) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  for (uint32_t i = 1;; ++i) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((i & 31) == 0) {
      if (*abort) return false;
      if (globaltimer_ns() - t0 > kTimeoutNs) {
        *abort = 1;
        set_error(err, kErrTimeout);
        return false;
      }
    }
  }
}

// Bounded wait used while draining (ignores the abort flag).
__device__ inline void mbar_wait_drain(uint64_t* bar, uint32_t parity, unsigned* err) {
  const uint64_t t0 = globaltimer_ns();
  while (!mbar_try_wait(bar, parity)) {
    if (globaltimer_ns() - t0 > kTimeoutNs) {
      set_error(err, kErrTimeout);
      return;
    }
  }
}

}  // namespace mcft
