// Device-side timing and the bounded grid barrier shared by the cooperative decode kernels.
// An Args type provides bar_count (unsigned*), bar_base (unsigned), err (int*) and
// barrier_timeout_ns; FERR_BARRIER_TIMEOUT is the sticky error bit set on a timeout.
#pragma once
#include <stdint.h>

#include "fused.cuh"

namespace moe {
namespace dev {

__device__ __forceinline__ uint64_t gtimer() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ unsigned ld_acquire_u32(const unsigned* p) {
  unsigned v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

// Grid-wide barrier over co-resident CTAs with a bounded wait. Each CTA's arrival is one
// release-add on a counter that only grows; barrier number n of a launch completes when the
// counter reaches bar_base + n * gridDim.x, which every CTA polls with acquire loads. Bounded: after
// a.barrier_timeout_ns the waiting CTA sets FERR_BARRIER_TIMEOUT and gives up. Returns false (in
// every thread of the CTA alike) once a fatal error flag is set, so that all CTAs leave the
// kernel together.
template <typename Args>
__device__ bool grid_sync(const Args& a, unsigned& nbar) {
  __shared__ int s_abort;
  __syncthreads();
  nbar++;
  if (threadIdx.x == 0) {
    const unsigned target = a.bar_base + nbar * gridDim.x;
    __threadfence();
    asm volatile("red.release.gpu.global.add.u32 [%0], %1;" ::"l"(a.bar_count), "r"(1u) : "memory");
    if ((int)(ld_acquire_u32(a.bar_count) - target) < 0) {
      const uint64_t t0 = gtimer();
      while ((int)(ld_acquire_u32(a.bar_count) - target) < 0) {
        if (*(volatile int*)a.err & FERR_FATAL) break;
        if (gtimer() - t0 > a.barrier_timeout_ns) {
          atomicOr(a.err, FERR_BARRIER_TIMEOUT);
          break;
        }
        __nanosleep(20);
      }
    }
    s_abort = *(volatile int*)a.err & FERR_FATAL;
  }
  __syncthreads();
  return s_abort == 0;
}

}  // namespace dev
}  // namespace moe
