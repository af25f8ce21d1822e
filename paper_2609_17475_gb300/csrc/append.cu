// Quantize-on-append: bf16 K/V rows -> affine 4-bit group-64 codes in their
// page slots (Sec. 3.3 "pending cache writes"; Sec. 2 paged pool; App. A.1
// Table 3 midpoint thresholds with strict >).
//
// The K and V vectors of one (row, KV head) of D bf16 elements are handled by
// D/8 lanes, each loading 16 bytes (8 elements) of each, so a warp reads two
// 512-byte rows at D = 256 and writes two 128-byte code rows plus their
// 4-byte scale/bias words.
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
  constexpr int VPW = 32 / LPV;     // (row, KV head) pairs per warp: K and V vectors each
  const int lane = threadIdx.x & 31;
  const int64_t warp_id = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int li = lane % LPV;
  const int64_t vec = warp_id * VPW + lane / LPV;   // (row, head)
  const int64_t total = (int64_t)a.n_rows * a.Hkv;
  const bool active = vec < total;
  // programmatic dependent launch: the next kernel may be scheduled now (it
  // waits for this grid before reading the pool); this grid waits for the
  // previous kernel before it reads the rows, the table or the pool
  asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory");
  asm volatile("griddepcontrol.wait;\n" ::: "memory");

  int64_t row = 0;
  int head = 0;
  float xk[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
  float xv[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
  int32_t req = 0, pos = 0;
  if (active) {
    row = vec / a.Hkv;
    head = (int)(vec % a.Hkv);
    // the row's slot and its K and V elements are independent loads, issued
    // together; the page-table entry (which needs the slot) overlaps the
    // quantizer
    req = a.row_req[row];
    pos = a.row_pos[row];
    load8_bf16(a.k + (row * a.Hkv + head) * D + li * 8, xk);
    load8_bf16(a.v + (row * a.Hkv + head) * D + li * 8, xv);
  }
  const bool slot_ok = req >= 0 && req < a.num_requests && pos >= 0 && pos / a.P < a.pt_stride;
  const int32_t page =
      (active && slot_ok) ? a.page_table[(int64_t)req * a.pt_stride + pos / a.P] : -1;
  __nv_bfloat16 sk, bk, sv, bv;
  const uint32_t wk = quantize8(xk, sk, bk);
  const uint32_t wv = quantize8(xv, sv, bv);
  if (!active) return;

  // destination slot
  if (!slot_ok) {
    if (li == 0) flag_error(a.err, JF_DEV_ERR_POSITION);
    return;
  }
  if (page < 0 || page >= a.num_pages) {
    if (li == 0) flag_error(a.err, JF_DEV_ERR_PAGE_ID);
    return;
  }
  uint8_t* const base = a.pool + (int64_t)page * a.page_bytes;
  store_quantized<D>(base, a.codes_region, a.sb_region, a.P, head, pos % a.P, 0, li, wk, sk, bk);
  store_quantized<D>(base, a.codes_region, a.sb_region, a.P, head, pos % a.P, 1, li, wv, sv, bv);
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
  const int64_t pairs = (int64_t)n_rows * g.Hkv;   // (row, KV head): a K and a V vector
  const int vpw = 32 / (g.D / 8);
  const int64_t warps = (pairs + vpw - 1) / vpw;
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
