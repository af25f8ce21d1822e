// extern "C" entry points of libjfkv.so: host-side validation, TMA tensor-map
// construction and kernel dispatch.  See include/jfkv.h for the contract.
#include <cstdio>
#include <cstring>
#include <mutex>

#include "common.cuh"
#include "tq4.cuh"

namespace jfkv {
int launch_append(const Geom&, const jf_kv_pool&, const int32_t*, int32_t, int32_t,
                  const int32_t*, const int32_t*, const void*, const void*, int32_t, int32_t*,
                  cudaStream_t);
int launch_page_copy(const Geom&, const jf_kv_pool&, const int32_t*, int32_t, void*, int32_t*,
                     bool, cudaStream_t);
int launch_decode(const Geom&, const jf_kv_pool&, const CUtensorMap&, const int32_t*, int32_t,
                  const int32_t*, int32_t, const void*, int32_t, float, void*, void*, int32_t,
                  cudaStream_t, const void* k_new = nullptr, const void* v_new = nullptr,
                  int32_t q_len = 1);
size_t decode_workspace_bytes(int64_t B, int64_t Hq, int64_t D, int64_t S);
int tq4_codebook_host(int d, float* out);
int tq4_make_params(const jf_tq4_codec* codec, int d, Tq4Params* p);
int launch_tq4_append(const Geom&, const jf_kv_pool&, const Tq4Params&, const int32_t*, int32_t,
                      int32_t, const int32_t*, const int32_t*, const void*, const void*, int32_t,
                      int32_t*, cudaStream_t);
int launch_tq4_decode(const Geom&, const jf_kv_pool&, const CUtensorMap&, const Tq4Params&,
                      const int32_t*, int32_t, const int32_t*, int32_t, const void*, int32_t,
                      float, void*, void*, int32_t, cudaStream_t, const void*, const void*,
                      int32_t);
int decode_box_rows();
int launch_prefill(const Geom&, const jf_kv_pool&, const CUtensorMap&, const int32_t*,
                   const void*, int32_t, int32_t, int32_t, float, int32_t, void*, void*,
                   cudaStream_t);
int launch_prefill_batch(const Geom&, const jf_kv_pool&, const int32_t* const*, const int32_t*,
                         const int32_t*, const void*, const int64_t*, int32_t, int32_t, float,
                         int32_t, void*, void*, cudaStream_t, int32_t, int64_t,
                         const Tq4Params*);
size_t prefill_workspace_bytes(int64_t rows, int64_t Hq, int64_t D, int64_t S, int fmt);
int sm_count();
}  // namespace jfkv

using namespace jfkv;

namespace {

bool aligned(const void* p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

int check_pool(const jf_kv_pool* pool) {
  if (!pool || !pool->base) return JF_ERR_INVALID_ARG;
  if (!aligned(pool->base, 16)) return JF_ERR_INVALID_ARG;
  if (pool->num_pages < 1 || pool->num_kv_heads < 1) return JF_ERR_INVALID_ARG;
  if (pool->format != JF_FMT_AFFINE4_G64) return JF_ERR_UNSUPPORTED;
  if (pool->group_size != 64) return JF_ERR_UNSUPPORTED;
  if (pool->head_dim != 128 && pool->head_dim != 256) return JF_ERR_UNSUPPORTED;
  if (pool->page_size != 64 && pool->page_size != 128 && pool->page_size != 256)
    return JF_ERR_UNSUPPORTED;
  if (pool->num_kv_heads > 65535) return JF_ERR_UNSUPPORTED;
  if (pool->num_pages > 0x7FFFFFFFLL) return JF_ERR_UNSUPPORTED;
  return JF_OK;
}

// Pools of either format, for the entry points that take both (append,
// single-query decode, checkpoint, restore).  TQ4 pools need their codec.
int check_pool_any(const jf_kv_pool* pool) {
  if (!pool || pool->format != JF_FMT_TQ4) return check_pool(pool);
  if (!pool->base || !aligned(pool->base, 16)) return JF_ERR_INVALID_ARG;
  if (pool->num_pages < 1 || pool->num_kv_heads < 1) return JF_ERR_INVALID_ARG;
  if (!pool->tq4) return JF_ERR_INVALID_ARG;
  if (pool->head_dim != 128 && pool->head_dim != 256) return JF_ERR_UNSUPPORTED;
  if (pool->page_size != 64 && pool->page_size != 128 && pool->page_size != 256)
    return JF_ERR_UNSUPPORTED;
  if (pool->num_kv_heads > 65535) return JF_ERR_UNSUPPORTED;
  if (pool->num_pages > 0x7FFFFFFFLL) return JF_ERR_UNSUPPORTED;
  return JF_OK;
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess)
      p = nullptr;
    return reinterpret_cast<EncodeTiledFn>(p);
  }();
  return fn;
}

// 5-D map over the code rows of a pool: (byte in row, slot, KV head, K|V, page),
// box = (row bytes, rows_per_box, 1, 1, 1), 128B (or 64B) swizzle.
int make_codes_map(const Geom& g, void* base, int rows_per_box, CUtensorMap* map) {
  EncodeTiledFn enc = encode_fn();
  if (!enc) return JF_ERR_CUDA;
  cuuint64_t dims[5] = {(cuuint64_t)g.CB, (cuuint64_t)g.P, (cuuint64_t)g.Hkv, 2,
                        (cuuint64_t)g.num_pages};
  cuuint64_t strides[4] = {(cuuint64_t)g.CB, (cuuint64_t)g.P * g.CB,
                           (cuuint64_t)g.codes_region, (cuuint64_t)g.page_bytes};
  cuuint32_t box[5] = {(cuuint32_t)g.CB, (cuuint32_t)rows_per_box, 1, 1, 1};
  cuuint32_t estr[5] = {1, 1, 1, 1, 1};
  CUtensorMapSwizzle sw = g.CB == 128 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_64B;
  CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_UINT8, 5, base, dims, strides, box, estr,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, sw, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? JF_OK : JF_ERR_CUDA;
}

}  // namespace

extern "C" {

size_t jf_kv_page_bytes(int32_t num_kv_heads, int32_t page_size, int32_t head_dim) {
  if (num_kv_heads < 1 || page_size < 1 || (head_dim != 128 && head_dim != 256)) return 0;
  jf_kv_pool p{};
  p.num_pages = 1;
  p.page_size = page_size;
  p.num_kv_heads = num_kv_heads;
  p.head_dim = head_dim;
  return (size_t)make_geom(p).page_bytes;
}

size_t jf_kv_page_bytes_fmt(int32_t format, int32_t num_kv_heads, int32_t page_size,
                            int32_t head_dim) {
  if (format != JF_FMT_AFFINE4_G64 && format != JF_FMT_TQ4) return 0;
  if (num_kv_heads < 1 || page_size < 1 || (head_dim != 128 && head_dim != 256)) return 0;
  jf_kv_pool p{};
  p.num_pages = 1;
  p.page_size = page_size;
  p.num_kv_heads = num_kv_heads;
  p.head_dim = head_dim;
  p.format = format;
  return (size_t)make_geom(p).page_bytes;
}

int jf_tq4_codebook(int32_t head_dim, float* centroids) {
  if (!centroids || head_dim < 3 || head_dim > 65536) return JF_ERR_INVALID_ARG;
  return tq4_codebook_host(head_dim, centroids);
}

size_t jf_attn_workspace_bytes(int32_t batch, int32_t num_q_heads, int32_t num_kv_heads,
                               int32_t head_dim, int32_t num_splits) {
  if (batch < 1 || num_q_heads < 1 || num_kv_heads < 1 || num_splits < 1) return 0;
  if (num_q_heads % num_kv_heads) return 0;
  if (head_dim != 128 && head_dim != 256) return 0;
  return decode_workspace_bytes(batch, num_q_heads, head_dim, num_splits);
}

size_t jf_prefill_workspace_bytes(void) { return 256; }

int jf_kv_quantize_append(const jf_kv_pool* pool, const int32_t* page_table, int32_t pt_stride,
                          int32_t num_requests, const int32_t* row_req, const int32_t* row_pos,
                          const void* k, const void* v, int32_t n_rows, int32_t* err_flag,
                          void* stream) {
  int st = check_pool_any(pool);
  if (st) return st;
  if (n_rows < 0 || pt_stride < 1 || num_requests < 1) return JF_ERR_INVALID_ARG;
  if (n_rows == 0) return JF_OK;
  if (!page_table || !row_req || !row_pos || !k || !v) return JF_ERR_INVALID_ARG;
  if (!aligned(k, 16) || !aligned(v, 16)) return JF_ERR_INVALID_ARG;
  const Geom g = make_geom(*pool);
  if (pool->format == JF_FMT_TQ4) {
    Tq4Params prm;
    st = tq4_make_params(pool->tq4, g.D, &prm);
    if (st) return st;
    return launch_tq4_append(g, *pool, prm, page_table, pt_stride, num_requests, row_req,
                             row_pos, k, v, n_rows, err_flag, static_cast<cudaStream_t>(stream));
  }
  return launch_append(g, *pool, page_table, pt_stride, num_requests, row_req, row_pos, k, v,
                       n_rows, err_flag, static_cast<cudaStream_t>(stream));
}

static int decode_common(const jf_kv_pool* pool, const int32_t* page_table, int32_t pt_stride,
                         const int32_t* context_lens, int32_t batch, const void* k_new,
                         const void* v_new, const void* q, int32_t num_q_heads,
                         float softmax_scale, void* out, void* workspace, size_t workspace_bytes,
                         int32_t num_splits, void* stream, int32_t q_len = 1) {
  int st = check_pool_any(pool);
  if (st) return st;
  if (!page_table || !context_lens || !q || !out || !workspace) return JF_ERR_INVALID_ARG;
  if (batch < 1 || batch > 65535 || pt_stride < 1 || num_q_heads < 1) return JF_ERR_INVALID_ARG;
  if (num_q_heads % pool->num_kv_heads) return JF_ERR_INVALID_ARG;
  if (num_q_heads / pool->num_kv_heads > 8) return JF_ERR_UNSUPPORTED;
  if (num_splits < 1 || num_splits > 65535) return JF_ERR_INVALID_ARG;
  if (q_len < 1 || q_len > 4) return JF_ERR_INVALID_ARG;
  if (!(softmax_scale == softmax_scale)) return JF_ERR_INVALID_ARG;
  if (!aligned(q, 16) || !aligned(out, 16) || !aligned(workspace, 256)) return JF_ERR_INVALID_ARG;
  if (k_new && (!aligned(k_new, 16) || !aligned(v_new, 16))) return JF_ERR_INVALID_ARG;
  const size_t need = jf_attn_workspace_bytes(batch, q_len * num_q_heads, pool->num_kv_heads,
                                              pool->head_dim, num_splits);
  if (workspace_bytes < need) return JF_ERR_WORKSPACE_TOO_SMALL;
  const Geom g = make_geom(*pool);
  Tq4Params prm;
  if (pool->format == JF_FMT_TQ4) {
    st = tq4_make_params(pool->tq4, g.D, &prm);
    if (st) return st;
  }
  CUtensorMap tmap;
  st = make_codes_map(g, pool->base, decode_box_rows(), &tmap);
  if (st) return st;
  if (pool->format == JF_FMT_TQ4) {
    return launch_tq4_decode(g, *pool, tmap, prm, page_table, pt_stride, context_lens, batch, q,
                             num_q_heads, softmax_scale, out, workspace, num_splits,
                             static_cast<cudaStream_t>(stream), k_new, v_new, q_len);
  }
  return launch_decode(g, *pool, tmap, page_table, pt_stride, context_lens, batch, q,
                       num_q_heads, softmax_scale, out, workspace, num_splits,
                       static_cast<cudaStream_t>(stream), k_new, v_new, q_len);
}

int jf_paged_decode_attn(const jf_kv_pool* pool, const int32_t* page_table, int32_t pt_stride,
                         const int32_t* context_lens, int32_t batch, const void* q,
                         int32_t num_q_heads, float softmax_scale, void* out, void* workspace,
                         size_t workspace_bytes, int32_t num_splits, void* stream) {
  return decode_common(pool, page_table, pt_stride, context_lens, batch, nullptr, nullptr, q,
                       num_q_heads, softmax_scale, out, workspace, workspace_bytes, num_splits,
                       stream);
}

int jf_paged_verify_attn(const jf_kv_pool* pool, const int32_t* page_table, int32_t pt_stride,
                         const int32_t* context_lens, int32_t batch, const void* q,
                         int32_t q_len, int32_t num_q_heads, float softmax_scale, void* out,
                         void* workspace, size_t workspace_bytes, int32_t num_splits,
                         void* stream) {
  if (q_len < 1 || q_len > 4) return JF_ERR_INVALID_ARG;
  return decode_common(pool, page_table, pt_stride, context_lens, batch, nullptr, nullptr, q,
                       num_q_heads, softmax_scale, out, workspace, workspace_bytes, num_splits,
                       stream, q_len);
}

int jf_paged_decode_append_attn(const jf_kv_pool* pool, const int32_t* page_table,
                                int32_t pt_stride, const int32_t* context_lens, int32_t batch,
                                const void* k_new, const void* v_new, const void* q,
                                int32_t num_q_heads, float softmax_scale, void* out,
                                void* workspace, size_t workspace_bytes, int32_t num_splits,
                                void* stream) {
  if (!k_new || !v_new) return JF_ERR_INVALID_ARG;
  return decode_common(pool, page_table, pt_stride, context_lens, batch, k_new, v_new, q,
                       num_q_heads, softmax_scale, out, workspace, workspace_bytes, num_splits,
                       stream);
}

}  // extern "C"

namespace {

// The prefill kernel's geometry: 128 MMA rows per CTA (128 / G queries), two
// CTAs per pair, one CTA per SM, 64-position history tiles.
constexpr int64_t kPfRows = 128;
constexpr int64_t kPfTile = 64;

// Wave balance of one chunk over a long prefix (q_start >= 4 chunk_len, so
// its CTA pairs carry nearly equal work W, the prefix's history tiles).
// Pairs run num_sms / 2 at a time.  When the last wave would be partly
// empty, the query tiles that fill it become a tail: the head's pairs run as
// whole waves, and the tail's history is split k ways, so the tail costs
// ceil(pieces / slots) rounds of W / k instead of one more W.  The estimate
// adds a fixed cost for the split launch and its merge and a cost per round
// (0.07 W + 0.03 W per round, fitted on a 2,048-query chunk after 30,720
// positions at 24 / 4 heads, D = 256); the smallest k within 0.05 W of the
// best is taken, only if it beats the unsplit tail by 0.05 W and leaves
// every piece 8 history tiles or more.  head = chunk_len, k = 1: one launch.
struct PfTailPlan {
  int32_t head, k;
};

PfTailPlan prefill_tail_plan(int64_t G, int64_t Hkv, int64_t q_start, int64_t chunk_len,
                             int64_t num_sms) {
  PfTailPlan p{(int32_t)chunk_len, 1};
  if (G < 1 || G > kPfRows || Hkv < 1 || num_sms < 2 || chunk_len < 1 || q_start < 4 * chunk_len)
    return p;
  const int64_t slots = num_sms / 2;
  const int64_t qpp = 2 * (kPfRows / G);                // queries per CTA pair
  const int64_t pph = (chunk_len + qpp - 1) / qpp;      // pairs per KV head
  const int64_t rem = (pph * Hkv) % slots;
  if (pph * Hkv <= slots || rem == 0) return p;
  const int64_t t_tail = (rem + Hkv - 1) / Hkv;         // tail pairs per KV head
  if (t_tail >= pph) return p;
  const int64_t c_head = (pph - t_tail) * qpp;
  const int64_t min_tiles = (q_start + c_head + kPfTile) / kPfTile;   // first tail query's
  double est[9] = {0};
  double best = 1e30;
  for (int s = 2; s <= 8 && min_tiles / s >= 8; ++s) {
    const int64_t rounds = (t_tail * Hkv * s + slots - 1) / slots;
    est[s] = (double)rounds / s + 0.07 + 0.03 * (double)rounds;
    if (est[s] < best) best = est[s];
  }
  if (best > 0.95) return p;
  for (int s = 2; s <= 8; ++s)
    if (est[s] > 0 && est[s] <= best + 0.05) return PfTailPlan{(int32_t)c_head, s};
  return p;
}

// Workspace of the balanced form: the head launch (unsplit) and the tail
// launch (k splits) run one after the other on the same workspace.
size_t prefill_tail_workspace(const PfTailPlan& p, int64_t chunk_len, int64_t Hq, int64_t D,
                              int fmt) {
  const size_t h = prefill_workspace_bytes(p.head, Hq, D, 1, fmt);
  const size_t t = prefill_workspace_bytes(chunk_len - p.head, Hq, D, p.k, fmt);
  return h > t ? h : t;
}

}  // namespace

extern "C" {

size_t jf_prefill_chunk_workspace_bytes(const jf_kv_pool* pool, int32_t q_start,
                                        int32_t chunk_len, int32_t num_q_heads, int32_t num_sms) {
  if (check_pool_any(pool)) return 0;
  if (q_start < 0 || chunk_len < 0 || num_q_heads < 1 || num_sms < 0) return 0;
  if (num_q_heads % pool->num_kv_heads) return 0;
  const bool tq = pool->format == JF_FMT_TQ4;
  const size_t one = tq ? prefill_workspace_bytes(chunk_len, num_q_heads, pool->head_dim, 1,
                                                  JF_FMT_TQ4)
                        : jf_prefill_workspace_bytes();
  const PfTailPlan p = prefill_tail_plan(num_q_heads / pool->num_kv_heads, pool->num_kv_heads,
                                         q_start, chunk_len, num_sms ? num_sms : sm_count());
  if (p.k == 1) return one;
  const size_t bal = prefill_tail_workspace(p, chunk_len, num_q_heads, pool->head_dim,
                                            pool->format);
  return bal > one ? bal : one;
}

int jf_prefill_chunk_attn(const jf_kv_pool* pool, const int32_t* page_table_row, const void* q,
                          int32_t q_start, int32_t chunk_len, int32_t num_q_heads,
                          float softmax_scale, int32_t causal, void* out, void* workspace,
                          size_t workspace_bytes, void* stream) {
  int st = check_pool_any(pool);
  if (st) return st;
  if (!page_table_row || !q || !out || !workspace) return JF_ERR_INVALID_ARG;
  if (q_start < 0 || chunk_len < 0 || num_q_heads < 1) return JF_ERR_INVALID_ARG;
  if (num_q_heads % pool->num_kv_heads) return JF_ERR_INVALID_ARG;
  if (!(softmax_scale == softmax_scale)) return JF_ERR_INVALID_ARG;
  const bool tq = pool->format == JF_FMT_TQ4;
  const size_t need = tq ? prefill_workspace_bytes(chunk_len, num_q_heads, pool->head_dim, 1,
                                                   JF_FMT_TQ4)
                         : jf_prefill_workspace_bytes();
  if (workspace_bytes < need) return JF_ERR_WORKSPACE_TOO_SMALL;
  if (!aligned(q, 16) || !aligned(out, 16) || !aligned(workspace, tq ? 256 : 16))
    return JF_ERR_INVALID_ARG;
  if ((int64_t)q_start + chunk_len > 0x7FFFFFFF) return JF_ERR_INVALID_ARG;
  if (chunk_len == 0) return JF_OK;
  const Geom g = make_geom(*pool);
  if (num_q_heads / pool->num_kv_heads > 128) return JF_ERR_UNSUPPORTED;
  Tq4Params prm;
  if (tq) {
    st = tq4_make_params(pool->tq4, g.D, &prm);
    if (st) return st;
  }
  const cudaStream_t s = static_cast<cudaStream_t>(stream);
  const int64_t row0 = 0;
  const PfTailPlan p = prefill_tail_plan(num_q_heads / pool->num_kv_heads, pool->num_kv_heads,
                                         q_start, chunk_len, sm_count());
  if (p.k > 1 && aligned(workspace, 256) &&
      workspace_bytes >= prefill_tail_workspace(p, chunk_len, num_q_heads, g.D, pool->format)) {
    // the head's query tiles as whole waves, then the tail's with split histories
    const size_t row_bytes = (size_t)num_q_heads * g.D * 2;
    const int32_t t_start = q_start + p.head, t_len = chunk_len - p.head;
    const void* q_t = static_cast<const uint8_t*>(q) + (size_t)p.head * row_bytes;
    void* out_t = static_cast<uint8_t*>(out) + (size_t)p.head * row_bytes;
    st = launch_prefill_batch(g, *pool, &page_table_row, &q_start, &p.head, q, &row0, 1,
                              num_q_heads, softmax_scale, causal, out, workspace, s, 1, p.head,
                              tq ? &prm : nullptr);
    if (st) return st;
    return launch_prefill_batch(g, *pool, &page_table_row, &t_start, &t_len, q_t, &row0, 1,
                                num_q_heads, softmax_scale, causal, out_t, workspace, s, p.k,
                                t_len, tq ? &prm : nullptr);
  }
  if (tq)
    return launch_prefill_batch(g, *pool, &page_table_row, &q_start, &chunk_len, q, &row0, 1,
                                num_q_heads, softmax_scale, causal, out, workspace, s, 1,
                                chunk_len, &prm);
  CUtensorMap tmap{};
  return launch_prefill(g, *pool, tmap, page_table_row, q, q_start, chunk_len, num_q_heads,
                        softmax_scale, causal, out, workspace, s);
}

size_t jf_prefill_batch_workspace_bytes(int32_t format, int64_t total_rows, int32_t num_q_heads,
                                        int32_t head_dim, int32_t num_splits) {
  if (format != JF_FMT_AFFINE4_G64 && format != JF_FMT_TQ4) return 0;
  if (total_rows < 0 || num_q_heads < 1 || num_splits < 1 || num_splits > 65535) return 0;
  if (head_dim != 128 && head_dim != 256) return 0;
  return prefill_workspace_bytes(total_rows, num_q_heads, head_dim, num_splits, format);
}

int jf_prefill_batch_attn(const jf_kv_pool* pool, const int32_t* page_table, int32_t pt_stride,
                          int32_t batch, const int32_t* q_start, const int32_t* chunk_len,
                          const void* q, int32_t num_q_heads, float softmax_scale, int32_t causal,
                          int32_t num_splits, void* out, void* workspace, size_t workspace_bytes,
                          void* stream) {
  int st = check_pool_any(pool);
  if (st) return st;
  if (batch < 1 || pt_stride < 1 || num_q_heads < 1) return JF_ERR_INVALID_ARG;
  if (batch > JF_PREFILL_MAX_BATCH) return JF_ERR_UNSUPPORTED;
  if (!page_table || !q_start || !chunk_len || !q || !out || !workspace) return JF_ERR_INVALID_ARG;
  if (num_q_heads % pool->num_kv_heads) return JF_ERR_INVALID_ARG;
  if (num_q_heads / pool->num_kv_heads > 128) return JF_ERR_UNSUPPORTED;
  if (!(softmax_scale == softmax_scale)) return JF_ERR_INVALID_ARG;
  if (num_splits < 1 || num_splits > 65535) return JF_ERR_INVALID_ARG;
  if (!aligned(q, 16) || !aligned(out, 16) || !aligned(workspace, 256)) return JF_ERR_INVALID_ARG;
  const int32_t* rows[JF_PREFILL_MAX_BATCH];
  int64_t row0[JF_PREFILL_MAX_BATCH];
  int64_t acc = 0;
  for (int b = 0; b < batch; ++b) {
    if (q_start[b] < 0 || chunk_len[b] < 0) return JF_ERR_INVALID_ARG;
    if ((int64_t)q_start[b] + chunk_len[b] > (int64_t)pt_stride * pool->page_size)
      return JF_ERR_INVALID_ARG;   // the chunk must fit the request's page-table row
    rows[b] = page_table + (int64_t)b * pt_stride;
    row0[b] = acc;
    acc += chunk_len[b];
  }
  if (acc > 0x7FFFFFFF) return JF_ERR_INVALID_ARG;
  if (workspace_bytes <
      prefill_workspace_bytes(acc, num_q_heads, pool->head_dim, num_splits, pool->format))
    return JF_ERR_WORKSPACE_TOO_SMALL;
  if (acc == 0) return JF_OK;
  const Geom g = make_geom(*pool);
  Tq4Params prm;
  if (pool->format == JF_FMT_TQ4) {
    st = tq4_make_params(pool->tq4, g.D, &prm);
    if (st) return st;
  }
  return launch_prefill_batch(g, *pool, rows, q_start, chunk_len, q, row0, batch, num_q_heads,
                              softmax_scale, causal, out, workspace,
                              static_cast<cudaStream_t>(stream), num_splits, acc,
                              pool->format == JF_FMT_TQ4 ? &prm : nullptr);
}

int64_t jf_reservation_pages(int64_t prompt_len, int64_t output_len, int64_t g_out,
                             int32_t page_size) {
  if (prompt_len < 0 || output_len < 0 || g_out < 0 || page_size < 1) return -1;
  const int64_t out = output_len < g_out ? output_len : g_out;
  if (prompt_len > INT64_MAX - out - page_size) return -1;
  return (prompt_len + out + page_size - 1) / page_size;
}

int jf_kv_checkpoint(const jf_kv_pool* pool, const int32_t* page_table_row, int32_t num_pages,
                     void* dst, size_t dst_bytes, int32_t* err_flag, void* stream) {
  int st = check_pool_any(pool);
  if (st) return st;
  if (num_pages < 0) return JF_ERR_INVALID_ARG;
  if (num_pages == 0) return JF_OK;
  if (!page_table_row || !dst || !aligned(dst, 16)) return JF_ERR_INVALID_ARG;
  const Geom g = make_geom(*pool);
  if (dst_bytes < (size_t)num_pages * (size_t)g.page_bytes) return JF_ERR_INVALID_ARG;
  return launch_page_copy(g, *pool, page_table_row, num_pages, dst, err_flag, true,
                          static_cast<cudaStream_t>(stream));
}

int jf_kv_restore(const jf_kv_pool* pool, const int32_t* page_table_row, int32_t num_pages,
                  const void* src, size_t src_bytes, int32_t* err_flag, void* stream) {
  int st = check_pool_any(pool);
  if (st) return st;
  if (num_pages < 0) return JF_ERR_INVALID_ARG;
  if (num_pages == 0) return JF_OK;
  if (!page_table_row || !src || !aligned(src, 16)) return JF_ERR_INVALID_ARG;
  const Geom g = make_geom(*pool);
  if (src_bytes < (size_t)num_pages * (size_t)g.page_bytes) return JF_ERR_INVALID_ARG;
  return launch_page_copy(g, *pool, page_table_row, num_pages, const_cast<void*>(src), err_flag,
                          false, static_cast<cudaStream_t>(stream));
}

// ---------------------------------------------------------------------------
// Decode without a caller-supplied workspace: scratch in a file-scope device
// array.  In host code `jf_static_decode_ws` only names the symbol; its device
// address comes from cudaGetSymbolAddress, looked up once per device.
// ---------------------------------------------------------------------------
}  // extern "C"

static __device__ __align__(256) unsigned char jf_static_decode_ws[JF_STATIC_WORKSPACE_BYTES];

namespace {
constexpr int kMaxDevices = 256;
std::mutex g_static_ws_mu;
void* g_static_ws_ptr[kMaxDevices] = {};

// Device address of the static workspace on the current device (set-up on the
// first call per device, with that device current).
int static_workspace(void** out) {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess) return JF_ERR_CUDA;
  if (dev < 0 || dev >= kMaxDevices) return JF_ERR_UNSUPPORTED;
  std::lock_guard<std::mutex> lock(g_static_ws_mu);
  if (!g_static_ws_ptr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, jf_static_decode_ws) != cudaSuccess || !p) return JF_ERR_CUDA;
    g_static_ws_ptr[dev] = p;
  }
  *out = g_static_ws_ptr[dev];
  return JF_OK;
}
}  // namespace

extern "C" {

int jf_paged_decode_attn_noalloc(const jf_kv_pool* pool, const int32_t* page_table,
                                 int32_t pt_stride, const int32_t* context_lens, int32_t batch,
                                 const void* q, int32_t num_q_heads, float softmax_scale,
                                 void* out, int32_t num_splits, int32_t* err_flag, void* stream) {
  int st = check_pool(pool);
  if (st) return st;
  if (!page_table || !context_lens || !q || !out) return JF_ERR_INVALID_ARG;
  if (batch < 1 || batch > 65535 || pt_stride < 1 || num_q_heads < 1) return JF_ERR_INVALID_ARG;
  if (num_q_heads % pool->num_kv_heads) return JF_ERR_INVALID_ARG;
  if (num_q_heads / pool->num_kv_heads > 8) return JF_ERR_UNSUPPORTED;
  if (num_splits < 1 || num_splits > 65535) return JF_ERR_INVALID_ARG;
  if (!(softmax_scale == softmax_scale)) return JF_ERR_INVALID_ARG;
  if (!aligned(q, 16) || !aligned(out, 16)) return JF_ERR_INVALID_ARG;
  const size_t need = jf_attn_workspace_bytes(batch, num_q_heads, pool->num_kv_heads,
                                              pool->head_dim, num_splits);
  if (need == 0) return JF_ERR_INVALID_ARG;
  if (need > JF_STATIC_WORKSPACE_BYTES) return JF_ERR_WORKSPACE_TOO_SMALL;
  void* ws = nullptr;
  st = static_workspace(&ws);
  if (st) return st;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  // the status word is the only scratch that must start at zero
  if (cudaMemsetAsync(ws, 0, sizeof(int32_t), s) != cudaSuccess) return JF_ERR_CUDA;
  const Geom g = make_geom(*pool);
  CUtensorMap tmap;
  st = make_codes_map(g, pool->base, decode_box_rows(), &tmap);
  if (st) return st;
  st = launch_decode(g, *pool, tmap, page_table, pt_stride, context_lens, batch, q, num_q_heads,
                     softmax_scale, out, ws, num_splits, s);
  if (st) return st;
  if (err_flag &&
      cudaMemcpyAsync(err_flag, ws, sizeof(int32_t), cudaMemcpyDeviceToDevice, s) != cudaSuccess)
    return JF_ERR_CUDA;
  return JF_OK;
}

const char* jf_status_string(int status) {
  switch (status) {
    case JF_OK: return "JF_OK";
    case JF_ERR_INVALID_ARG: return "JF_ERR_INVALID_ARG";
    case JF_ERR_UNSUPPORTED: return "JF_ERR_UNSUPPORTED";
    case JF_ERR_WORKSPACE_TOO_SMALL: return "JF_ERR_WORKSPACE_TOO_SMALL";
    case JF_ERR_CUDA: return "JF_ERR_CUDA";
    default: return "JF_ERR_UNKNOWN";
  }
}

const char* jf_version(void) { return "jfkv 0.1 (sm_103a)"; }

}  // extern "C"
