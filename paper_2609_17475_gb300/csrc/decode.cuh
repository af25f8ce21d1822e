// Split-K decode pieces shared by the affine and TQ4 decode kernels: the
// per-call argument block, the split plans (per request and batch-wide) and
// the swizzled stage addressing.  Sec. 2, Eq. 3 motivates the fixed-size
// workspace these plans index; Sec. 3.1 the page-native decode.
#pragma once
#include "common.cuh"

namespace jfkv {

constexpr int DTOK = 32;      // positions per pipeline stage (one chunk)
constexpr int MIN_CPS = 16;   // minimum chunks per split (512 positions)
constexpr float DTAU = 4.f;   // log2 headroom before the reference maximum moves

struct DecodeArgs {
  const uint8_t* pool;
  int64_t num_pages;
  int64_t page_bytes;
  int64_t codes_region;   // bytes of one code region (K or V) in a page record
  int64_t sb_base;     // offset of the K scale/bias region in a page record
  int64_t sb_region;   // bytes of one scale/bias region (K or V)
  int32_t P, Hkv, Hq, G;
  int32_t log2P;        // P is a power of two
  const int32_t* page_table;
  int32_t pt_stride;
  const int32_t* ctx;
  const uint16_t* q;
  const uint16_t* knew;   // fused append: new K/V rows [B, Hkv, D], or null
  const uint16_t* vnew;
  uint16_t* out;
  float* part_ml;      // [B, Hq, S, 2]
  float* part_o;       // [B, Hq, S, D]
  int32_t* status;
  int32_t num_splits;   // workspace rows per (request, query row): the row stride
  int32_t plan_splits;  // per-request plans cut a request into at most this many splits
  float scale_log2;    // softmax_scale * log2(e)
  int32_t B;           // requests
  int32_t L;           // query tokens per request (1: decode; 2-4: packed verifier)
  int32_t NT;          // n-tiles per KV head: ceil(G * L / 8) groups of 8 (token, head) rows
  int32_t HqL;         // L * Hq: rows of q, out and the partials per request
  int32_t balanced;    // 1: batch split plan (balanced_plan), partial rows by global split
  int32_t span;        // 1: batch span plan (span_find), partial rows (piece + request)
  int32_t budget;      // balanced: target splits per KV head over the whole batch
};

__host__ __device__ inline void split_plan(int ctx, int num_splits, int& nch, int& cps,
                                           int& nsplit) {
  nch = (ctx + DTOK - 1) / DTOK;
  if (nch <= 0) { nch = 0; cps = MIN_CPS; nsplit = 0; return; }
  cps = (nch + num_splits - 1) / num_splits;
  if (cps < MIN_CPS) cps = MIN_CPS;
  nsplit = (nch + cps - 1) / cps;
}

// Batch split plan (B > 1).  Splits are sized for the whole batch, not per
// request: with T the chunks of all requests, every request is cut into
// pieces of cps = max(MIN_CPS, ceil(T / budget)) chunks, so each split CTA
// streams about the same bytes however unequal the contexts are.  Request b
// gets n_b = ceil(nch_b / cps) splits, numbered g0_b .. g0_b + n_b - 1 after
// those of requests 0 .. b-1; the global number g names the split's partial
// rows (g * Hq + hq).  Called by one whole warp; for a split CTA (x >= 0) it
// finds the request and split of global split x (b = -1 when x is past the
// last), for a merge CTA (want_b >= 0) the first global split and count of
// request want_b.
struct BalPlan {
  int b, split, nsplit, g0, cps;
};

static __device__ BalPlan balanced_plan(const DecodeArgs& a, int x, int want_b, int lane) {
  const int64_t cap = (int64_t)a.pt_stride * a.P;
  auto nch_of = [&](int bb) -> int {
    int64_t c = a.ctx[bb];
    c = c < 0 ? 0 : (c > cap ? cap : c);
    return (int)((c + DTOK - 1) / DTOK);
  };
  long long T = 0;
  for (int bb = lane; bb < a.B; bb += 32) T += nch_of(bb);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) T += __shfl_xor_sync(0xffffffffu, T, o);
  int cps = (int)((T + a.budget - 1) / a.budget);
  if (cps < MIN_CPS) cps = MIN_CPS;
  BalPlan p{-1, 0, 0, 0, cps};
  int base = 0;
  for (int b0 = 0; b0 < a.B; b0 += 32) {
    const int bb = b0 + lane;
    const int n = (bb < a.B) ? (nch_of(bb) + cps - 1) / cps : 0;
    int incl = n;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += y;
    }
    const int excl = base + incl - n;
    const bool hit = (x >= 0) ? (bb < a.B && x >= excl && x < excl + n) : (bb == want_b);
    const unsigned m = __ballot_sync(0xffffffffu, hit);
    if (m) {
      const int src = __ffs(m) - 1;
      p.b = __shfl_sync(0xffffffffu, bb, src);
      p.g0 = __shfl_sync(0xffffffffu, excl, src);
      p.nsplit = __shfl_sync(0xffffffffu, n, src);
      p.split = (x >= 0) ? x - p.g0 : 0;
      return p;
    }
    base += __shfl_sync(0xffffffffu, incl, 31);
  }
  return p;
}

// Span plan (batches of the affine decode).  The chunks of all requests are
// laid end to end (request 0 first), each request's run preceded by
// SPAN_HDR places that stand for the cost of starting a segment (query
// fragments, pipeline fill, the combine and its partial row), and cut into
// pieces of W places, W = max(MIN_CPS, ceil(T / budget)), T the total: every
// piece carries the same work however unequal the requests are, and a piece
// that starts a request streams that many fewer chunks (32 measured best:
// two requests 67.9 -> 64.6 us, 32 mixed requests 196-197 -> 191-193 us).  Piece x meets requests in
// segments; the segment of request b is one split whose partial rows are
// (x + b) * HqL + hq (along the sequence every piece or request boundary
// advances x + b, so the numbers never repeat, and a request's rows are
// contiguous: x0_b + b .. x1_b + b).  The workspace holds B * num_splits
// rows per query row, so budget <= B * (num_splits - 1) + 1.
constexpr int SPAN_HDR = 32;   // places standing for a segment's start (see above)

__device__ __forceinline__ int span_nch(const DecodeArgs& a, int b) {
  const int64_t cap = (int64_t)a.pt_stride * a.P;
  int64_t c = a.ctx[b];
  c = c < 0 ? 0 : (c > cap ? cap : c);
  const int n = (int)((c + DTOK - 1) / DTOK);
  return n > 0 ? n + SPAN_HDR : 0;   // a request's length in the sequence
}

// total chunks of the batch (every lane of the calling warp gets it)
static __device__ long long span_total(const DecodeArgs& a, int lane) {
  long long T = 0;
  for (int bb = lane; bb < a.B; bb += 32) T += span_nch(a, bb);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) T += __shfl_xor_sync(0xffffffffu, T, o);
  return T;
}

__host__ __device__ inline int span_width(long long T, int budget) {
  long long w = (T + budget - 1) / (budget > 0 ? budget : 1);
  return (int)(w < MIN_CPS ? MIN_CPS : w);
}

struct SpanHit {
  int b;            // request (-1: none)
  long long start;  // its first chunk in the batch sequence
  int nch;          // its chunks
};

// The request holding batch chunk `pos` (pos >= 0), or, with pos < 0, request
// want_b itself.  Called by a whole warp.
static __device__ SpanHit span_find(const DecodeArgs& a, long long pos, int lane,
                                    int want_b = -1) {
  long long base = 0;
  for (int b0 = 0; b0 < a.B; b0 += 32) {
    const int bb = b0 + lane;
    const int n = (bb < a.B) ? span_nch(a, bb) : 0;
    long long incl = n;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const long long y = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += y;
    }
    const long long excl = base + incl - n;
    const bool hit = (pos >= 0) ? (bb < a.B && n > 0 && pos >= excl && pos < excl + n)
                                : (bb == want_b);
    const unsigned m = __ballot_sync(0xffffffffu, hit);
    if (m) {
      const int src = __ffs(m) - 1;
      return SpanHit{__shfl_sync(0xffffffffu, bb, src), __shfl_sync(0xffffffffu, excl, src),
                     __shfl_sync(0xffffffffu, n, src)};
    }
    base += __shfl_sync(0xffffffffu, incl, 31);
  }
  return SpanHit{-1, 0, 0};
}

// Partial rows of request b under the span plan: rows row .. row + n - 1
// (n = 0 for an empty request).  Called by a whole warp.
struct SpanRows {
  int row, n;
};
static __device__ SpanRows span_rows(const DecodeArgs& a, int b, int lane) {
  const long long T = span_total(a, lane);
  const SpanHit h = span_find(a, -1, lane, b);
  if (h.nch <= 0) return SpanRows{0, 0};
  const int W = span_width(T, a.budget);
  const int x0 = (int)(h.start / W), x1 = (int)((h.start + h.nch - 1) / W);
  return SpanRows{x0 + b, x1 - x0 + 1};
}

// Context length of request b clamped to [0, pt_stride * P].  An out-of-range
// value is reported by the CTAs that own split 0 of request b (every request
// with at least one chunk has one; the merge kernel reports the others).
__device__ __forceinline__ int checked_ctx(const DecodeArgs& a, int b, int split) {
  int ctx = a.ctx[b];
  const int64_t cap = (int64_t)a.pt_stride * a.P;
  if (ctx < 0 || ctx > cap) {
    if (threadIdx.x == 0 && split == 0) flag_error(a.status, JF_DEV_ERR_POSITION);
    ctx = ctx < 0 ? 0 : (int)cap;
  }
  return ctx;
}

// Byte offset of 16-byte chunk `ch` of code row `t` inside a TMA-swizzled
// stage buffer (128B swizzle for 128-byte rows, 64B swizzle for 64-byte rows).
template <int CB>
__device__ __forceinline__ uint32_t swz(int t, int ch) {
  if constexpr (CB == 128)
    return t * 128 + ((ch ^ (t & 7)) << 4);
  else
    return t * 64 + ((ch ^ ((t >> 1) & 3)) << 4);
}

int sm_count();
// Merge phase for D = 128 or 256 (launched after a split kernel on `stream`).
int launch_decode_merge(const DecodeArgs& a, int D, int B, cudaStream_t stream);
// Packed verifier for NT >= 2 n-tiles per KV head (verify.cu): CTAs per KV
// head and split, and the split launch (+ merge).
int verify_pair_ctas(int NT);
int launch_verify_pairs(const CUtensorMap& tmap, const DecodeArgs& a, int D, int B,
                        cudaStream_t stream);

}  // namespace jfkv
