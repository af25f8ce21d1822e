// Quantize-on-append: bf16 K/V rows -> affine 4-bit group-64 codes in their
// page slots (Sec. 3.3 "pending cache writes"; Sec. 2 paged pool; App. A.1
// Table 3 midpoint thresholds with strict >).
//
// One vector (row, KV head, K|V) of D bf16 elements is handled by D/8 lanes,
// each loading 16 bytes (8 elements), so a warp reads 512 contiguous bytes at
// D = 256 and writes one 128-byte code row plus four 4-byte scale/bias words.
// The quantizer itself (quant.cuh) is shared with the fused decode.
#include "quant.cuh"

namespace jfkv {

struct AppendArgs {
  uint8_t* pool;
  int64_t num_pages;
  int64_t page_bytes;
  int64_t codes_region;
  int64_t sb_region;
  int32_t P;
  int32_t Hkv;
  const int32_t* page_table;
  int32_t pt_stride;
  int32_t num_requests;
  const int32_t* row_req;
  const int32_t* row_pos;
  const uint16_t* k;
  const uint16_t* v;
  int32_t n_rows;
  int32_t* err;
};

template <int D>
__global__ void __launch_bounds__(256) append_kernel(const AppendArgs a) {
  constexpr int LPV = D / 8;        // lanes per vector
  constexpr int VPW = 32 / LPV;     // vectors per warp
  const int lane = threadIdx.x & 31;
  const int64_t warp_id = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int li = lane % LPV;
  const int64_t vec = warp_id * VPW + lane / LPV;
  const int64_t total = (int64_t)a.n_rows * a.Hkv * 2;
  const bool active = vec < total;
  // programmatic dependent launch: the next kernel may be scheduled now (it
  // waits for this grid before reading the pool); this grid waits for the
  // previous kernel before it reads the rows, the table or the pool
  asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory");
  asm volatile("griddepcontrol.wait;\n" ::: "memory");

  int64_t row = 0;
  int kind = 0, head = 0;
  float x[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
  if (active) {
    row = vec / (2 * a.Hkv);
    const int rem = (int)(vec % (2 * a.Hkv));
    kind = rem / a.Hkv;
    head = rem % a.Hkv;
    load8_bf16((kind ? a.v : a.k) + (row * a.Hkv + head) * D + li * 8, x);
  }
  __nv_bfloat16 scale_h, bias_h;
  const uint32_t word = quantize8(x, scale_h, bias_h);
  if (!active) return;

  // destination slot
  const int32_t req = a.row_req[row];
  const int32_t pos = a.row_pos[row];
  if (req < 0 || req >= a.num_requests || pos < 0 || pos / a.P >= a.pt_stride) {
    if (li == 0) flag_error(a.err, JF_DEV_ERR_POSITION);
    return;
  }
  const int32_t page = a.page_table[(int64_t)req * a.pt_stride + pos / a.P];
  if (page < 0 || page >= a.num_pages) {
    if (li == 0) flag_error(a.err, JF_DEV_ERR_PAGE_ID);
    return;
  }
  store_quantized<D>(a.pool + (int64_t)page * a.page_bytes, a.codes_region, a.sb_region, a.P,
                     head, pos % a.P, kind, li, word, scale_h, bias_h);
}

int launch_append(const Geom& g, const jf_kv_pool& pool, const int32_t* page_table,
                  int32_t pt_stride, int32_t num_requests, const int32_t* row_req,
                  const int32_t* row_pos, const void* k, const void* v, int32_t n_rows,
                  int32_t* err, cudaStream_t stream) {
  AppendArgs a;
  a.pool = static_cast<uint8_t*>(pool.base);
  a.num_pages = g.num_pages;
  a.page_bytes = g.page_bytes;
  a.codes_region = g.codes_region;
  a.sb_region = g.sb_region;
  a.P = g.P;
  a.Hkv = g.Hkv;
  a.page_table = page_table;
  a.pt_stride = pt_stride;
  a.num_requests = num_requests;
  a.row_req = row_req;
  a.row_pos = row_pos;
  a.k = static_cast<const uint16_t*>(k);
  a.v = static_cast<const uint16_t*>(v);
  a.n_rows = n_rows;
  a.err = err;
  const int64_t vectors = (int64_t)n_rows * g.Hkv * 2;
  const int vpw = 32 / (g.D / 8);
  const int64_t warps = (vectors + vpw - 1) / vpw;
  const int64_t blocks = (warps + 7) / 8;
  if (blocks > 0x7FFFFFFF) return JF_ERR_INVALID_ARG;
  cudaLaunchAttribute pdl[1];
  pdl[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  pdl[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)blocks);
  cfg.blockDim = dim3(256);
  cfg.stream = stream;
  cfg.attrs = pdl;
  cfg.numAttrs = 1;
  const cudaError_t e = (g.D == 256) ? cudaLaunchKernelEx(&cfg, append_kernel<256>, a)
                                     : cudaLaunchKernelEx(&cfg, append_kernel<128>, a);
  return e == cudaSuccess ? JF_OK : JF_ERR_CUDA;
}

}  // namespace jfkv
