// Self-test of the bounded-wait give-up path that every kernel of the
// library takes when a copy it waits for does not land: the wait polls its
// mbarrier a fixed number of times, then the kernel ORs JF_DEV_ERR_TIMEOUT
// into its status word and returns instead of hanging.  Here the barrier's
// phase completes only if the kernel itself arrives (arrive != 0), so with
// arrive == 0 nothing ever completes it and the wait must give up.  No copy,
// no MMA and no other CTA is involved.
#include "common.cuh"

namespace jfkv {

__global__ void bounded_wait_selftest_kernel(int32_t* status, int arrive, uint32_t limit) {
  __shared__ __align__(8) uint64_t bar;
  if (threadIdx.x != 0) return;
  mbar_init(&bar, 1);
  fence_barrier_init();
  if (arrive) mbar_arrive(&bar);
  if (!mbar_wait_bounded(&bar, 0, limit)) flag_error(status, JF_DEV_ERR_TIMEOUT);
}

}  // namespace jfkv

extern "C" int jf_selftest_bounded_wait(int32_t* status, int32_t arrive, void* stream) {
  if (!status) return JF_ERR_INVALID_ARG;
  jfkv::bounded_wait_selftest_kernel<<<1, 32, 0, static_cast<cudaStream_t>(stream)>>>(
      status, arrive ? 1 : 0, 1u << 12);
  return cudaGetLastError() == cudaSuccess ? JF_OK : JF_ERR_CUDA;
}
