// Page-gather checkpoint and restore scatter (Sec. 3.4: the checkpoint reads
// the request's page runs in place and emits one packed stream; restoration
// writes packed runs back into the existing pool).
//
// A pure copy: each CTA moves a 16 KiB slice of one page record with 16-byte
// vector loads, four in flight per thread, so the kernel runs at copy
// bandwidth.  page_bytes is always a multiple of 16.
#include "common.cuh"

namespace jfkv {

constexpr int CK_THREADS = 256;
constexpr int CK_UNROLL = 4;
constexpr int CK_SLICE = CK_THREADS * CK_UNROLL * 16;   // bytes per CTA

__global__ void __launch_bounds__(CK_THREADS)
page_copy_kernel(uint8_t* pool, int64_t num_pages, int64_t page_bytes,
                 const int32_t* page_table_row, uint8_t* blob, int32_t* err, int to_blob) {
  const int k = blockIdx.y;
  const int32_t page = page_table_row[k];
  if (page < 0 || page >= num_pages) {
    if (blockIdx.x == 0 && threadIdx.x == 0) flag_error(err, JF_DEV_ERR_PAGE_ID);
    return;
  }
  const int64_t nvec = page_bytes / 16;
  const int64_t v0 = (int64_t)blockIdx.x * (CK_SLICE / 16) + threadIdx.x;
  uint4* pg = reinterpret_cast<uint4*>(pool + (int64_t)page * page_bytes);
  uint4* bl = reinterpret_cast<uint4*>(blob + (int64_t)k * page_bytes);
  const uint4* src = to_blob ? pg : bl;
  uint4* dst = to_blob ? bl : pg;
  uint4 r[CK_UNROLL];
#pragma unroll
  for (int u = 0; u < CK_UNROLL; ++u) {
    const int64_t i = v0 + (int64_t)u * CK_THREADS;
    if (i < nvec) r[u] = __ldcs(src + i);
  }
#pragma unroll
  for (int u = 0; u < CK_UNROLL; ++u) {
    const int64_t i = v0 + (int64_t)u * CK_THREADS;
    if (i < nvec) __stcs(dst + i, r[u]);
  }
}

int launch_page_copy(const Geom& g, const jf_kv_pool& pool, const int32_t* page_table_row,
                     int32_t num_pages, void* blob, int32_t* err, bool to_blob,
                     cudaStream_t stream) {
  if (num_pages == 0) return JF_OK;
  const int64_t slices = (g.page_bytes + CK_SLICE - 1) / CK_SLICE;
  if (num_pages > 65535) return JF_ERR_UNSUPPORTED;
  dim3 grid((unsigned)slices, (unsigned)num_pages);
  page_copy_kernel<<<grid, CK_THREADS, 0, stream>>>(static_cast<uint8_t*>(pool.base),
                                                    g.num_pages, g.page_bytes, page_table_row,
                                                    static_cast<uint8_t*>(blob), err,
                                                    to_blob ? 1 : 0);
  return cudaGetLastError() == cudaSuccess ? JF_OK : JF_ERR_CUDA;
}

}  // namespace jfkv
