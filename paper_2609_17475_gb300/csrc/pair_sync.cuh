// Named-barrier helpers for kernels whose warps work in pairs on one chunk
// (the packed verifiers): barrier id 1 + pair index, 64 threads.
#pragma once
#include "common.cuh"

namespace jfkv {

// both warps of pair `id - 1` meet; every thread learns whether both passed `ok`
__device__ __forceinline__ bool pair_sync_and(int id, bool ok) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred p, q;\n\t"
      "setp.ne.u32 q, %1, 0;\n\t"
      "bar.red.and.pred p, %2, 64, q;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}\n"
      : "=r"(r) : "r"((uint32_t)ok), "r"(id) : "memory");
  return r != 0;
}

__device__ __forceinline__ void pair_sync(int id) {
  asm volatile("bar.sync %0, 64;\n" ::"r"(id) : "memory");
}

}  // namespace jfkv
