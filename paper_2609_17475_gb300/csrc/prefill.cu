// Prefill-chunk attention (placeholder until the tcgen05 kernel lands).
#include "common.cuh"

namespace jfkv {

int launch_prefill(const Geom&, const jf_kv_pool&, const CUtensorMap&, const int32_t*,
                   const void*, int32_t, int32_t, int32_t, float, int32_t, void*, void*,
                   cudaStream_t) {
  return JF_ERR_UNSUPPORTED;
}

}  // namespace jfkv
