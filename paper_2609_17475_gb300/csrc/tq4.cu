// TQ4 KV format (Sec. 3.1 Eq. 4; App. A.1 Table 3): codebook construction,
// encode-on-append and page-native decode attention.
//
//   y = H_d S x / (sqrt(d) rho),   x_hat = rho_hat S H_d c[z] / sqrt(d)
//
// Codebook (host).  16 Lloyd-Max centroids for the density (1 - x^2)^((d-3)/2)
// on a 32,768-point grid over [-1 + 1e-6, 1 - 1e-6], quantile start, at most
// 100 updates, stop once the largest change is below 1e-6; fp64, rounded to
// fp32 at the end.
//
// Append.  One warp per vector (d/32 elements per lane).  The index decision
// z_j = #{k : u_j > T_k}, u = H_d S x, T_k = fp64(fp64(sqrt(d) rho) t_k), is
// made exactly: a fp32 Hadamard butterfly decides every element whose value
// lies farther than 2^-15 rho from every threshold (the fp32 butterfly is
// within 2^-17 rho of the exact value: 8 levels of rounding, each at most
// 2^-24 of a partial sum bounded by sum|x| <= sqrt(d) rho), and a warp with
// any closer element redoes its vector with the fp64 butterfly, which is
// exact for bf16 inputs whose magnitudes span less than 2^37, and compares
// those elements with the thresholds their fast-path bracket leaves open.
// rho is the fp32 rounding of the square root of the fp64 sum of squares,
// obtained from a certified double-float sum (fp64 only near a tie).
//
// Decode.  The query is rotated once per CTA, q' = H_d S_K q / sqrt(d), so
//   <q, K_t> = rho_hat_t <q', c[z_t]>,  sum_t p_t V_t = S_V H_d (sum_t p_t
//   rho_hat_t c[z_t]) / sqrt(d):
// the K and V indices only ever meet the 16 centroids, and the inverse
// rotation of V is one Hadamard transform per head at the end of the split.
// Centroids come from a shared-memory table indexed by a whole code byte (two
// indices -> f16x2), replicated per lane (word b * 32 + lane) so a warp's 32
// lookups never share a bank.  QK^T: A = looked-up K pairs [16 positions x
// 16 d] (ldmatrix gives a lane 4 code bytes of one position), B = q' [16 d x
// 8 heads].  PV: A = V pairs regrouped by position (ldmatrix.trans gives two
// positions' bytes; one byte permute per register), B = p_t rho_hat_t 2^-8 as
// f16 [16 positions x 8 heads].  Pipeline, split plans and the merge kernel
// are those of the affine decode.
#include <cmath>
#include <cfloat>
#include <vector>

#include "decode.cuh"
#include "tq4.cuh"

namespace jfkv {

// ---------------------------------------------------------------------------
// Host: codebook (App. A.1 Table 3)
// ---------------------------------------------------------------------------
int tq4_codebook_host(int d, float* out) {
  if (d < 3 || d > 65536 || !out) return JF_ERR_INVALID_ARG;
  constexpr int N = 32768, K = 16, MAX_UPDATES = 100;
  constexpr double TOL = 1e-6;
  std::vector<double> x(N), w(N);
  const double start = -1.0 + 1e-6, stop = 1.0 - 1e-6;
  const double step = (stop - start) / (double)(N - 1);
  for (int i = 0; i < N; ++i) x[i] = (double)i * step + start;
  x[N - 1] = stop;
  double wsum = 0.0;
  for (int i = 0; i < N; ++i) {
    const double u = 1.0 - x[i] * x[i];
    w[i] = std::pow(u, (double)(d - 3) / 2.0);
    wsum += w[i];
  }
  for (int i = 0; i < N; ++i) w[i] /= wsum;
  // quantile start: first grid point whose cumulative weight reaches (k + 1/2)/16
  double c[K];
  {
    double cdf = 0.0;
    int k = 0;
    for (int i = 0; i < N && k < K; ++i) {
      cdf += w[i];
      while (k < K && cdf >= (k + 0.5) / K) c[k++] = x[i];
    }
    while (k < K) { c[k] = x[N - 1]; ++k; }
  }
  for (int it = 0; it < MAX_UPDATES; ++it) {
    double t[K - 1];
    for (int k = 0; k < K - 1; ++k) t[k] = (c[k] + c[k + 1]) / 2.0;
    double mass[K] = {0}, mom[K] = {0};
    int k = 0;
    for (int i = 0; i < N; ++i) {   // the grid ascends: cell #{k : x > t_k}
      while (k < K - 1 && x[i] > t[k]) ++k;
      mass[k] += w[i];
      mom[k] += w[i] * x[i];
    }
    double change = 0.0;
    for (int j = 0; j < K; ++j) {
      if (mass[j] > 0.0) {
        const double nc = mom[j] / mass[j];
        change = std::fmax(change, std::fabs(nc - c[j]));
        c[j] = nc;
      }
    }
    if (change < TOL) break;
  }
  for (int j = 0; j < K; ++j) out[j] = (float)c[j];
  return JF_OK;
}

int tq4_make_params(const jf_tq4_codec* codec, int d, Tq4Params* p) {
  if (!codec || !p) return JF_ERR_INVALID_ARG;
  for (int k = 0; k < 16; ++k) {
    const float v = codec->centroids[k];
    if (!(std::fabs(v) < 1.0f)) return JF_ERR_INVALID_ARG;
    if (k > 0 && !(v > codec->centroids[k - 1])) return JF_ERR_INVALID_ARG;
    p->c[k] = v;
  }
  const float sd = (float)std::sqrt((double)d);
  for (int k = 0; k < 15; ++k) {
    volatile float s = p->c[k] + p->c[k + 1];   // fp32 rounding of the sum
    p->t[k] = s * 0.5f;
    p->tq[k] = sd * p->t[k];
  }
  // the append's fast path needs neighbouring thresholds more than 4 margins
  // (2^-15 rho each) apart; a codebook with closer ones decides every index
  // in fp64
  p->exact_all = 0;
  for (int k = 0; k < 14; ++k)
    if (!((double)p->tq[k + 1] - (double)p->tq[k] > 0x1p-12)) p->exact_all = 1;
  for (int j = 0; j < 8; ++j) p->sk[j] = p->sv[j] = 0u;
  for (int j = 0; j < d; ++j) {
    const int a = codec->signs_k[j], b = codec->signs_v[j];
    if ((a != 1 && a != -1) || (b != 1 && b != -1)) return JF_ERR_INVALID_ARG;
    if (a < 0) p->sk[j >> 5] |= 1u << (j & 31);
    if (b < 0) p->sv[j >> 5] |= 1u << (j & 31);
  }
  return JF_OK;
}

// ---------------------------------------------------------------------------
// Append (encode on write)
// ---------------------------------------------------------------------------
struct Tq4AppendArgs {
  uint8_t* pool;
  int64_t num_pages;
  int64_t page_bytes;
  int64_t codes_region;
  int64_t norm_region;
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

template <int E>
__device__ __forceinline__ void load_bf16(const uint16_t* src, float (&x)[E]) {
  if constexpr (E == 8) {
    const uint4 w = *reinterpret_cast<const uint4*>(src);
    const uint32_t ws[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) { x[2 * i] = bf16lo_to_f32(ws[i]); x[2 * i + 1] = bf16hi_to_f32(ws[i]); }
  } else {
    const uint2 w = *reinterpret_cast<const uint2*>(src);
    x[0] = bf16lo_to_f32(w.x); x[1] = bf16hi_to_f32(w.x);
    x[2] = bf16lo_to_f32(w.y); x[3] = bf16hi_to_f32(w.y);
  }
}

// Count of the 15 ascending thresholds T_k with u > T_k, by a branch-free
// 4-level search, and the thresholds bracketing u (lo < u <= hi; -inf / +inf
// past the ends).
__device__ __forceinline__ int bracket15(float u, const float (&T)[15], float& lo, float& hi) {
  const bool b3 = u > T[7];
  lo = b3 ? T[7] : -INFINITY;
  hi = b3 ? INFINITY : T[7];
  const float t2 = b3 ? T[11] : T[3];
  const bool b2 = u > t2;
  lo = b2 ? t2 : lo;
  hi = b2 ? hi : t2;
  const float t1 = b3 ? (b2 ? T[13] : T[9]) : (b2 ? T[5] : T[1]);
  const bool b1 = u > t1;
  lo = b1 ? t1 : lo;
  hi = b1 ? hi : t1;
  const float t0 = b3 ? (b2 ? (b1 ? T[14] : T[12]) : (b1 ? T[10] : T[8]))
                      : (b2 ? (b1 ? T[6] : T[4]) : (b1 ? T[2] : T[0]));
  const bool b0 = u > t0;
  lo = b0 ? t0 : lo;
  hi = b0 ? hi : t0;
  return (b3 ? 8 : 0) + (b2 ? 4 : 0) + (b1 ? 2 : 0) + (b0 ? 1 : 0);
}

// (s_hi, s_lo) += b for a double-float accumulator (Knuth's TwoSum; the
// error term of s_hi + b is exact)
__device__ __forceinline__ void two_sum_acc(float& sh, float& sl, float b) {
  const float s = __fadd_rn(sh, b);
  const float bb = __fsub_rn(s, sh);
  const float err = __fadd_rn(__fsub_rn(sh, __fsub_rn(s, bb)), __fsub_rn(b, bb));
  sh = s;
  sl = __fadd_rn(sl, err);
}

// Encode one vector of D bf16 elements (src) with a whole warp: returns this
// lane's E = D/32 indices (element E lane + e in bits 4e .. 4e+3) and sets
// rho (the fp32 norm; every lane gets the same value).  kind 0: K, 1: V.
template <int D>
__device__ __forceinline__ uint32_t tq4_encode(const uint16_t* src, int kind, const Tq4Params& prm,
                                               int lane, float& rho_out) {
  constexpr int E = D / 32;
  float x[E];
  load_bf16<E>(src + lane * E, x);
  const uint32_t sbits = ((kind ? prm.sv : prm.sk)[(lane * E) >> 5]) >> ((lane * E) & 31);

  // rho = RN32(sqrt(s)), s the fp64 sum of squares.  Squares of bf16 values
  // are exact in fp32; their sum is carried as a double-float (TwoSum, error
  // about 2^-40 s) and its square root rounded from r = RN32(sqrt(s_hi)) and
  // the exact residual s_hi - r^2 (one fma).  When the result lies within
  // 2^-10 half-ulp of a rounding boundary, or s is out of the safe range, the
  // warp recomputes s in fp64 (GB300's fp64 rate is low, so this stays rare).
  float sh = 0.f, sl = 0.f;
#pragma unroll
  for (int e = 0; e < E; ++e) two_sum_acc(sh, sl, __fmul_rn(x[e], x[e]));
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float bh = __shfl_xor_sync(0xffffffffu, sh, o);
    const float bl = __shfl_xor_sync(0xffffffffu, sl, o);
    two_sum_acc(sh, sl, bh);
    sl = __fadd_rn(sl, bl);
  }
  float rho;
  {
    const float r = __fsqrt_rn(sh);
    const float res = __fmaf_rn(-r, r, sh);                // exact: s_hi - r^2
    // sqrt(s) = r + dl up to ~2^-41 r; rounding boundaries at half an ulp on
    // either side (the spacing below a power of two is half the one above)
    const float dl = __fmul_rn(__fadd_rn(res, sl), __fdiv_rn(0.5f, r));
    const float up = __int_as_float(__float_as_int(r) + 1);
    const float dn = __int_as_float(__float_as_int(r) - 1);
    const float half = (dl > 0.f) ? 0.5f * (up - r) : 0.5f * (r - dn);
    const float ad = fabsf(dl);
    const bool sure = (sh >= 0x1p-100f) && (sh <= 0x1p+120f) &&
                      (fabsf(ad - half) > half * 0x1p-10f) && !(ad > 2.f * half);
    rho = (ad < half) ? r : (dl > 0.f ? up : dn);
    if (!sure) {   // uniform: every lane holds the same (sh, sl)
      double s = 0.0;
#pragma unroll
      for (int e = 0; e < E; ++e) s += (double)x[e] * (double)x[e];
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
      rho = __double2float_rn(sqrt(s));
    }
  }

  // fast path: fp32 butterfly, decided where no threshold is within 2^-15 rho
  float u[E];
#pragma unroll
  for (int e = 0; e < E; ++e) u[e] = ((sbits >> e) & 1u) ? -x[e] : x[e];
  warp_fwht<float, E>(u, lane);
  float T[15];
#pragma unroll
  for (int k = 0; k < 15; ++k) T[k] = rho * prm.tq[k];
  const float M = rho * 0x1p-15f;
  bool near = !(rho >= 1e-30f && rho <= 1e36f) || prm.exact_all;
  // thresholds are farther apart than 2M, so only the two bracketing ones can
  // lie within M of u
  uint32_t word = 0, nearmask = 0;
#pragma unroll
  for (int e = 0; e < E; ++e) {
    float lo, hi;
    const int z = bracket15(u[e], T, lo, hi);
    if (u[e] - lo <= M || hi - u[e] <= M) nearmask |= 1u << e;
    word |= (uint32_t)z << (4 * e);
  }
  near = near || (nearmask != 0);
  if (__any_sync(0xffffffffu, near)) {
    // exact path: fp64 butterfly; an element within M of a threshold compares
    // against the contract's threshold products T_k = fp64(fp64(sqrt(D) rho)
    // t_k) for its two bracketing thresholds (all 15 when the norm is outside
    // the fast path's range)
    double ud[E];
#pragma unroll
    for (int e = 0; e < E; ++e) ud[e] = ((sbits >> e) & 1u) ? -(double)x[e] : (double)x[e];
    warp_fwht<double, E>(ud, lane);
    const double r = (double)rho * sqrt((double)D);
    const bool all = !(rho >= 1e-30f && rho <= 1e36f) || prm.exact_all;
#pragma unroll
    for (int e = 0; e < E; ++e) {
      if (all || ((nearmask >> e) & 1u)) {
        const int zf = (word >> (4 * e)) & 0xF;
        const int k0 = all ? 0 : max(zf - 1, 0), k1 = all ? 15 : min(zf + 1, 15);
        int z = k0;
        for (int k = k0; k < k1; ++k) z += (ud[e] > r * (double)prm.t[k]) ? 1 : 0;
        word = (word & ~(0xFu << (4 * e))) | ((uint32_t)z << (4 * e));
      }
    }
  }

  rho_out = rho;
  return word;
}

// Store a lane's indices and (lane 0) the fp16 norm into slot `vrow` (head *
// P + slot) of a page record.
template <int D>
__device__ __forceinline__ void tq4_store(uint8_t* pg, int64_t codes_region, int64_t norm_region,
                                          int kind, int64_t vrow, int lane, uint32_t word,
                                          float rho) {
  constexpr int E = D / 32;
  uint8_t* dst = pg + kind * codes_region + vrow * (D / 2);
  if constexpr (E == 8)
    reinterpret_cast<uint32_t*>(dst)[lane] = word;
  else
    reinterpret_cast<uint16_t*>(dst)[lane] = (uint16_t)word;
  if (lane == 0) {
    const __half h = __float2half_rn(fminf(rho, 65504.f));
    *reinterpret_cast<uint16_t*>(pg + 2 * codes_region + kind * norm_region + vrow * 2) =
        __half_as_ushort(h);
  }
}

template <int D>
__global__ void __launch_bounds__(256) tq4_append_kernel(const Tq4AppendArgs a, const Tq4Params prm) {
  constexpr int E = D / 32;   // elements per lane
  const int lane = threadIdx.x & 31;
  const int64_t vec = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t total = (int64_t)a.n_rows * a.Hkv * 2;
  asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory");
  asm volatile("griddepcontrol.wait;\n" ::: "memory");
  if (vec >= total) return;   // whole warps
  const int64_t row = vec / (2 * a.Hkv);
  const int rem = (int)(vec % (2 * a.Hkv));
  const int kind = rem / a.Hkv;
  const int head = rem % a.Hkv;

  float rho;
  const uint32_t word = tq4_encode<D>((kind ? a.v : a.k) + (row * a.Hkv + head) * D, kind, prm,
                                       lane, rho);

  const int32_t req = a.row_req[row];
  const int32_t pos = a.row_pos[row];
  if (req < 0 || req >= a.num_requests || pos < 0 || pos / a.P >= a.pt_stride) {
    if (lane == 0) flag_error(a.err, JF_DEV_ERR_POSITION);
    return;
  }
  const int32_t page = a.page_table[(int64_t)req * a.pt_stride + pos / a.P];
  if (page < 0 || page >= a.num_pages) {
    if (lane == 0) flag_error(a.err, JF_DEV_ERR_PAGE_ID);
    return;
  }
  tq4_store<D>(a.pool + (int64_t)page * a.page_bytes, a.codes_region, a.norm_region, kind,
               (int64_t)head * a.P + pos % a.P, lane, word, rho);
}

int launch_tq4_append(const Geom& g, const jf_kv_pool& pool, const Tq4Params& prm,
                      const int32_t* page_table, int32_t pt_stride, int32_t num_requests,
                      const int32_t* row_req, const int32_t* row_pos, const void* k,
                      const void* v, int32_t n_rows, int32_t* err, cudaStream_t stream) {
  Tq4AppendArgs a;
  a.pool = static_cast<uint8_t*>(pool.base);
  a.num_pages = g.num_pages;
  a.page_bytes = g.page_bytes;
  a.codes_region = g.codes_region;
  a.norm_region = g.sb_region;
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
  const int64_t blocks = (vectors + 7) / 8;   // 8 warps per CTA, one vector each
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
  const cudaError_t e = (g.D == 256) ? cudaLaunchKernelEx(&cfg, tq4_append_kernel<256>, a, prm)
                                     : cudaLaunchKernelEx(&cfg, tq4_append_kernel<128>, a, prm);
  return e == cudaSuccess ? JF_OK : JF_ERR_CUDA;
}

// ---------------------------------------------------------------------------
// Decode: split kernel
// ---------------------------------------------------------------------------
constexpr int TQ_WARPS = 11;    // one CTA per SM (the centroid table takes 32 KB)
constexpr int TQ_STAGES = 2;    // stages per warp

template <int D>
struct Tq4Smem {
  static constexpr int CB = D / 2;
  static constexpr int CODE_BUF = DTOK * CB;     // one chunk's K (or V) indices
  static constexpr int NORM_BUF = DTOK * 2;      // one chunk's K (or V) norms
  static constexpr int NBUF = TQ_WARPS * TQ_STAGES;
  static constexpr int CODES_BYTES = NBUF * 2 * CODE_BUF;
  static constexpr int LUT_OFF = CODES_BYTES;
  static constexpr int LUT_BYTES = 256 * 32 * 4;
  static constexpr int NORM_OFF = LUT_OFF + LUT_BYTES;
  static constexpr int NORM_BYTES = NBUF * 2 * NORM_BUF;
  // rotated queries (before the first copy is issued) and the combined output
  // (after the last stage is consumed), fp32 [8][D], inside the stage rings
  static constexpr int Q_BYTES = 8 * D * 4;
  static constexpr int Q_OFF = CODES_BYTES - Q_BYTES;
  static constexpr int BAR_OFF = NORM_OFF + NORM_BYTES;
  static constexpr int BAR_BYTES = NBUF * 8;
  static constexpr int MISC_OFF = BAR_OFF + BAR_BYTES;   // plan (4 ints), per-warp |q'| max (8)
  static constexpr int TOTAL = MISC_OFF + 64;
  static constexpr uint32_t STAGE_TX = 2 * CODE_BUF + 2 * NORM_BUF;
  static_assert(TQ_WARPS * 8 * (D + 4) * 4 + TQ_WARPS * 8 * 3 * 4 + 64 <= Q_OFF,
                "combine buffers and the combined output must fit the stage rings");
  static_assert(TOTAL <= 227 * 1024, "shared memory");
};

__device__ __forceinline__ uint32_t lds32(uint32_t addr) {
  uint32_t v;
  asm("ld.shared.b32 %0, [%1];\n" : "=r"(v) : "r"(addr));
  return v;
}

// centroid pair of code byte k of w (f16x2: low nibble's centroid in the low half)
__device__ __forceinline__ uint32_t lut(uint32_t lut_lane, uint32_t w, uint32_t k) {
  return lds32(lut_lane + __byte_perm(w, 0u, 0x4440u + k) * 128u);
}

template <int D>
struct Tq4State {
  float m0, m1, l0, l1;
  float O[D / 64][4][4];   // [64-d block g][d offset e][MMA accumulator]
  __device__ __forceinline__ void init() {
    m0 = m1 = -INFINITY;
    l0 = l1 = 0.f;
#pragma unroll
    for (int g = 0; g < D / 64; ++g)
#pragma unroll
      for (int e = 0; e < 4; ++e)
#pragma unroll
        for (int i = 0; i < 4; ++i) O[g][e][i] = 0.f;
  }
};

__device__ __forceinline__ float h2f(const uint8_t* p) {
  return __half2float(__ushort_as_half(*reinterpret_cast<const uint16_t*>(p)));
}

// One 32-position chunk.  FULL: every position valid and visible to every
// row, no masks.  Otherwise positions >= nvalid get -inf logits and zero
// weights (their bytes are never trusted), and the rows of this thread's
// columns 2c and 2c+1 see only positions < nv0 and < nv1 (the verifier's
// causal limits; both are nvalid for a single query), as plain selects.  The
// chunk loop stays rolled, so the kernel holds two copies of the body (four,
// unrolled by the ring depth, had missed the instruction cache).
template <int D, bool VER, bool FULL>
__device__ __forceinline__ void tq4_chunk(Tq4State<D>& st, const uint32_t (&bq)[D / 32][2][2],
                                          uint32_t kc, const uint8_t* kn, uint32_t lut_lane,
                                          const uint32_t (&koff)[D / 64], float cS, int r,
                                          int nvalid, int nv0, int nv1) {
  constexpr int CB = D / 2;
  constexpr int NJ = DTOK / 16;
  constexpr int NCH = D / 64;
  constexpr float NEG_INF = -INFINITY;
  const uint32_t vc = kc + DTOK * CB;
  const uint8_t* vn = kn + DTOK * 2;

  float sc[NJ][4];
#pragma unroll
  for (int j = 0; j < NJ; ++j) {
    float acc[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
    for (int g = 0; g < NCH; ++g) {
      uint32_t w0, w1, w2, w3;
      ldsm_x4(w0, w1, w2, w3, kc + koff[g] + 16 * j * CB);
      // w0/w1: positions r / r+8, 16-byte chunk 2g; w2/w3: chunk 2g+1
#pragma unroll
      for (int s = 0; s < 2; ++s) {
        mma_f16(acc, lut(lut_lane, w0, 2 * s), lut(lut_lane, w1, 2 * s),
                lut(lut_lane, w0, 2 * s + 1), lut(lut_lane, w1, 2 * s + 1), bq[2 * g][s][0],
                bq[2 * g][s][1]);
      }
#pragma unroll
      for (int s = 0; s < 2; ++s) {
        mma_f16(acc, lut(lut_lane, w2, 2 * s), lut(lut_lane, w3, 2 * s),
                lut(lut_lane, w2, 2 * s + 1), lut(lut_lane, w3, 2 * s + 1), bq[2 * g + 1][s][0],
                bq[2 * g + 1][s][1]);
      }
    }
    const int ta = 16 * j + r, tb = ta + 8;
    const float na = h2f(kn + 2 * ta) * cS, nb = h2f(kn + 2 * tb) * cS;
    if constexpr (FULL) {
      sc[j][0] = acc[0] * na;
      sc[j][1] = acc[1] * na;
      sc[j][2] = acc[2] * nb;
      sc[j][3] = acc[3] * nb;
    } else if constexpr (VER) {
      sc[j][0] = (ta < nv0) ? acc[0] * na : NEG_INF;
      sc[j][1] = (ta < nv1) ? acc[1] * na : NEG_INF;
      sc[j][2] = (tb < nv0) ? acc[2] * nb : NEG_INF;
      sc[j][3] = (tb < nv1) ? acc[3] * nb : NEG_INF;
    } else {
      sc[j][0] = (ta < nvalid) ? acc[0] * na : NEG_INF;
      sc[j][1] = (ta < nvalid) ? acc[1] * na : NEG_INF;
      sc[j][2] = (tb < nvalid) ? acc[2] * nb : NEG_INF;
      sc[j][3] = (tb < nvalid) ? acc[3] * nb : NEG_INF;
    }
  }

  // ---- online softmax with a lazily moved reference maximum -------------
  float mx0 = fmaxf(sc[0][0], sc[0][2]);
  float mx1 = fmaxf(sc[0][1], sc[0][3]);
#pragma unroll
  for (int j = 1; j < NJ; ++j) {
    mx0 = fmaxf(mx0, fmaxf(sc[j][0], sc[j][2]));
    mx1 = fmaxf(mx1, fmaxf(sc[j][1], sc[j][3]));
  }
  if (__any_sync(0xffffffffu, (mx0 > st.m0 + DTAU) || (mx1 > st.m1 + DTAU))) {
#pragma unroll
    for (int o = 4; o < 32; o <<= 1) {
      mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, o));
      mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, o));
    }
    const float nm0 = fmaxf(st.m0, mx0), nm1 = fmaxf(st.m1, mx1);
    const float f0 = (nm0 > st.m0) ? fast_exp2(st.m0 - nm0) : 1.f;
    const float f1 = (nm1 > st.m1) ? fast_exp2(st.m1 - nm1) : 1.f;
#pragma unroll
    for (int g = 0; g < NCH; ++g)
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        st.O[g][e][0] *= f0; st.O[g][e][2] *= f0;
        st.O[g][e][1] *= f1; st.O[g][e][3] *= f1;
      }
    st.l0 *= f0;
    st.l1 *= f1;
    st.m0 = nm0;
    st.m1 = nm1;
  }
  float p[NJ][4];
#pragma unroll
  for (int j = 0; j < NJ; ++j) {
    if constexpr (FULL) {
      p[j][0] = fast_exp2(sc[j][0] - st.m0);
      p[j][1] = fast_exp2(sc[j][1] - st.m1);
      p[j][2] = fast_exp2(sc[j][2] - st.m0);
      p[j][3] = fast_exp2(sc[j][3] - st.m1);
    } else {
      p[j][0] = (sc[j][0] == NEG_INF) ? 0.f : fast_exp2(sc[j][0] - st.m0);
      p[j][1] = (sc[j][1] == NEG_INF) ? 0.f : fast_exp2(sc[j][1] - st.m1);
      p[j][2] = (sc[j][2] == NEG_INF) ? 0.f : fast_exp2(sc[j][2] - st.m0);
      p[j][3] = (sc[j][3] == NEG_INF) ? 0.f : fast_exp2(sc[j][3] - st.m1);
    }
    st.l0 += p[j][0] + p[j][2];
    st.l1 += p[j][1] + p[j][3];
  }

  // ---- PV -----------------------------------------------------------------
#pragma unroll
  for (int j = 0; j < NJ; ++j) {
    const int ta = 16 * j + r, tb = ta + 8;
    const float wa = (FULL || ta < nvalid) ? h2f(vn + 2 * ta) * 0.00390625f : 0.f;
    const float wb = (FULL || tb < nvalid) ? h2f(vn + 2 * tb) * 0.00390625f : 0.f;
    const uint32_t b0 = movm_t(pack_f16x2(wa * p[j][0], wa * p[j][1]));
    const uint32_t b1 = movm_t(pack_f16x2(wb * p[j][2], wb * p[j][3]));
#pragma unroll
    for (int g = 0; g < NCH; ++g) {
      uint32_t v0, v1, v2, v3;
      ldsm_x4_t(v0, v1, v2, v3, vc + koff[g] + 16 * j * CB);
      // v: bytes 0,1 = position 2c (d 4r..4r+3), bytes 2,3 = position 2c+1;
      // v0/v2: positions 0-7 of the tile, chunks 2g / 2g+1; v1/v3: positions 8-15
      const uint32_t L00 = lut(lut_lane, v0, 0), L01 = lut(lut_lane, v0, 1),
                     L02 = lut(lut_lane, v0, 2), L03 = lut(lut_lane, v0, 3);
      const uint32_t L10 = lut(lut_lane, v1, 0), L11 = lut(lut_lane, v1, 1),
                     L12 = lut(lut_lane, v1, 2), L13 = lut(lut_lane, v1, 3);
      const uint32_t L20 = lut(lut_lane, v2, 0), L21 = lut(lut_lane, v2, 1),
                     L22 = lut(lut_lane, v2, 2), L23 = lut(lut_lane, v2, 3);
      const uint32_t L30 = lut(lut_lane, v3, 0), L31 = lut(lut_lane, v3, 1),
                     L32 = lut(lut_lane, v3, 2), L33 = lut(lut_lane, v3, 3);
      // d offset e: (position 2c, position 2c+1) pairs; rows r <-> 64g + 4r + e,
      // r + 8 <-> 64g + 32 + 4r + e
      mma_f16(st.O[g][0], __byte_perm(L00, L02, 0x5410), __byte_perm(L20, L22, 0x5410),
              __byte_perm(L10, L12, 0x5410), __byte_perm(L30, L32, 0x5410), b0, b1);
      mma_f16(st.O[g][1], __byte_perm(L00, L02, 0x7632), __byte_perm(L20, L22, 0x7632),
              __byte_perm(L10, L12, 0x7632), __byte_perm(L30, L32, 0x7632), b0, b1);
      mma_f16(st.O[g][2], __byte_perm(L01, L03, 0x5410), __byte_perm(L21, L23, 0x5410),
              __byte_perm(L11, L13, 0x5410), __byte_perm(L31, L33, 0x5410), b0, b1);
      mma_f16(st.O[g][3], __byte_perm(L01, L03, 0x7632), __byte_perm(L21, L23, 0x7632),
              __byte_perm(L11, L13, 0x7632), __byte_perm(L31, L33, 0x7632), b0, b1);
    }
  }
}

// VER: packed verifier (a.L > 1 query tokens, per-row causal limits; each CTA
// holds 8 of the KV head's G * L (token, head) rows; launched for at most 8
// rows, more go to the warp-pair kernel of tq4_verify.cu); otherwise decode.
// APP: the step's new K/V row is appended first (a.knew, a.vnew).
template <int D, bool VER, bool APP>
__global__ void __launch_bounds__(TQ_WARPS * 32, 1)
tq4_split_kernel(const __grid_constant__ CUtensorMap tmap, const DecodeArgs a,
                 const Tq4Params prm) {
  using L = Tq4Smem<D>;
  constexpr int NCH = D / 64;
  constexpr float NEG_INF = -INFINITY;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* codes = smem_raw;
  uint32_t* lut_w = reinterpret_cast<uint32_t*>(smem_raw + L::LUT_OFF);
  uint8_t* norms = smem_raw + L::NORM_OFF;
  float* qbuf = reinterpret_cast<float*>(smem_raw + L::Q_OFF);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem_raw + L::BAR_OFF);
  int* misc = reinterpret_cast<int*>(smem_raw + L::MISC_OFF);

  const int kvh = VER ? (int)blockIdx.y / a.NT : (int)blockIdx.y;
  const int nt = VER ? (int)blockIdx.y % a.NT : 0;
  const int rows = VER ? min(8, a.G * a.L - 8 * nt) : a.G;
  // row k of this CTA: query token (8 nt + k) / G, head (8 nt + k) % G; its
  // q, out and partial row within the request
  auto row_of = [&](int k) {
    if constexpr (VER) {
      const int gr = 8 * nt + k;
      return (gr / a.G) * a.Hq + kvh * a.G + gr % a.G;
    } else {
      return kvh * a.G + k;
    }
  };
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int r = lane >> 2, c = lane & 3;
  const bool direct = (a.num_splits == 1);
  const bool aligned = (smem_u32(smem_raw) & 1023) == 0;
  // setup that reads only kernel parameters
  if (aligned) {
    if (threadIdx.x == 0) prefetch_tensormap(&tmap);
    if (lane == 0) {
      for (int s = 0; s < TQ_STAGES; ++s) mbar_init(&bars[warp * TQ_STAGES + s], 1);
      fence_barrier_init();
    }
  }
  // centroid table: word b * 32 + lane = f16x2 (c[b & 15], c[b >> 4])
  for (int i = threadIdx.x; i < 256 * 32; i += blockDim.x) {
    const int b = i >> 5;
    lut_w[i] = pack_f16x2(prm.c[b & 15], prm.c[b >> 4]);
  }
  asm volatile("griddepcontrol.wait;\n" ::: "memory");

  int split, b, ctx, nch, cps, nsplit;
  if (a.balanced) {
    if (warp == 0) {
      const BalPlan p = balanced_plan(a, (int)blockIdx.x, -1, lane);
      if (lane == 0) {
        misc[0] = p.b;
        misc[1] = p.split;
        misc[2] = p.nsplit;
        misc[3] = p.cps;
      }
    }
    __syncthreads();
    b = misc[0];
    split = misc[1];
    nsplit = misc[2];
    cps = misc[3];
    if (b < 0) return;
    ctx = checked_ctx(a, b, split);
    nch = (ctx + DTOK - 1) / DTOK;
  } else {
    split = blockIdx.x;
    b = blockIdx.z;
    ctx = checked_ctx(a, b, split);
    split_plan(ctx, a.num_splits, nch, cps, nsplit);
  }
  if (split >= nsplit) {
    if (direct && split == 0) {
      for (int i = threadIdx.x; i < rows * D; i += blockDim.x)
        a.out[((int64_t)b * a.HqL + row_of(i / D)) * D + i % D] = 0;
    }
    return;
  }
  if (!aligned) {
    if (threadIdx.x == 0) flag_error(a.status, JF_DEV_ERR_LAYOUT);
    return;
  }
  const int c_begin = split * cps;
  const int c_end = min(c_begin + cps, nch);
  const int n_cta = c_end - c_begin;
  const int my_n = (n_cta > warp) ? (n_cta - warp + TQ_WARPS - 1) / TQ_WARPS : 0;
  auto chunk_of = [&](int it) { return c_begin + warp + it * TQ_WARPS; };

  if (APP && split == nsplit - 1) {   // owns the last chunk
    // the step's new K (warp 0) and V (warp 1) rows go to position ctx - 1
    // before this split's copies read the page
    if (warp < 2 && ctx > 0) {
      const int pos = ctx - 1;
      float rho;
      const uint32_t word = tq4_encode<D>((warp ? a.vnew : a.knew) + ((int64_t)b * a.Hkv + kvh) * D,
                                          warp, prm, lane, rho);
      const int pidx = pos >> a.log2P;
      const int page = (pidx < a.pt_stride) ? a.page_table[(int64_t)b * a.pt_stride + pidx] : -1;
      if (page < 0 || page >= a.num_pages) {
        if (lane == 0) flag_error(a.status, JF_DEV_ERR_PAGE_ID);
      } else {
        tq4_store<D>(const_cast<uint8_t*>(a.pool) + (int64_t)page * a.page_bytes, a.codes_region,
                     a.sb_region, warp, (int64_t)kvh * a.P + (pos & (a.P - 1)), lane, word, rho);
      }
    }
    fence_proxy_async_global();
    __syncthreads();
    fence_proxy_async_global();
  }

  // ---- rotated queries q' = H S_K q / sqrt(D) (rows >= G stay zero) -------
  // warp h < 8 transforms head row h with shuffles (E elements per lane)
  constexpr int E = D / 32;
  if (warp < 8) {
    float x[E];
#pragma unroll
    for (int e = 0; e < E; ++e) x[e] = 0.f;
    if (warp < rows) {
      load_bf16<E>(a.q + ((int64_t)b * a.HqL + row_of(warp)) * D + lane * E, x);
      const uint32_t sb = prm.sk[(lane * E) >> 5] >> ((lane * E) & 31);
#pragma unroll
      for (int e = 0; e < E; ++e)
        if ((sb >> e) & 1u) x[e] = -x[e];
    }
    warp_fwht<float, E>(x, lane);
    float mx = 0.f;
#pragma unroll
    for (int e = 0; e < E; ++e) {
      qbuf[warp * D + lane * E + e] = x[e];
      mx = fmaxf(mx, fabsf(x[e]));
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    if (lane == 0) misc[8 + warp] = __float_as_int(mx);
  }
  __syncthreads();
  // fp16 range: scale q' by 2^-qe so that max |q'| lies in [2^13, 2^14)
  float qabs = 0.f;
#pragma unroll
  for (int w = 0; w < 8; ++w) qabs = fmaxf(qabs, __int_as_float(misc[8 + w]));
  const float qs0 = a.scale_log2 * rsqrtf((float)D);
  const float qmax = qabs * fabsf(qs0);
  const int qe = (qmax > 0.f && qmax < INFINITY) ? ilogbf(qmax) - 13 : 0;
  const float qmul = qs0 * ldexpf(1.f, -qe);
  const float cS = ldexpf(1.f, qe);
  // B fragments: head r, d = 32 ch + 8 c + 4 s + {0,1} (b0) and {2,3} (b1)
  uint32_t bq[D / 32][2][2];
#pragma unroll
  for (int ch = 0; ch < D / 32; ++ch)
#pragma unroll
    for (int s = 0; s < 2; ++s) {
      const float4 v = *reinterpret_cast<const float4*>(qbuf + r * D + 32 * ch + 8 * c + 4 * s);
      bq[ch][s][0] = pack_f16x2(v.x * qmul, v.y * qmul);
      bq[ch][s][1] = pack_f16x2(v.z * qmul, v.w * qmul);
    }
  __syncthreads();   // the query buffer lies in the stage rings the copies fill

  // ---- page ids and TMA producer (as in the affine decode) ---------------
  auto load_pages = [&](int blk) -> int {
    const int it = blk * 32 + lane;
    int page = -1;
    if (it < my_n) {
      const int pidx = (chunk_of(it) * DTOK) >> a.log2P;
      if (pidx < a.pt_stride) page = __ldg(a.page_table + (int64_t)b * a.pt_stride + pidx);
    }
    return page;
  };
  int pg_cur = load_pages(0);
  int pg_next = load_pages(1);
  // decode reads each page once per call: evict it from L2 first; the
  // verifier's n-tile CTAs read the same pages, so L2 keeps them normally
  const uint64_t l2pol = VER ? l2_evict_normal_policy() : l2_evict_first_policy();
  uint32_t valid = 0;
  auto issue = [&](int it) {
    const int s = it % TQ_STAGES;
    if (it >= 32 && (it & 31) == 0) {
      pg_cur = pg_next;
      pg_next = load_pages((it >> 5) + 1);
    }
    const int page = __shfl_sync(0xffffffffu, pg_cur, it & 31);
    const bool ok = page >= 0 && page < a.num_pages;
    if (lane == 0) {
      const int inp = (chunk_of(it) * DTOK) & (a.P - 1);
      uint64_t* bar = &bars[warp * TQ_STAGES + s];
      if (!ok) {
        flag_error(a.status, JF_DEV_ERR_PAGE_ID);
        mbar_arrive(bar);
      } else {
        uint8_t* kc = codes + (warp * TQ_STAGES + s) * 2 * L::CODE_BUF;
        uint8_t* kn = norms + (warp * TQ_STAGES + s) * 2 * L::NORM_BUF;
        const uint8_t* gn = a.pool + (int64_t)page * a.page_bytes + a.sb_base +
                            ((int64_t)kvh * a.P + inp) * 2;
        mbar_arrive_expect_tx(bar, L::STAGE_TX);
        tma_load_5d_hint(kc, &tmap, 0, inp, kvh, 0, page, bar, l2pol);
        tma_load_5d_hint(kc + L::CODE_BUF, &tmap, 0, inp, kvh, 1, page, bar, l2pol);
        bulk_g2s_hint(kn, gn, L::NORM_BUF, bar, l2pol);
        bulk_g2s_hint(kn + L::NORM_BUF, gn + a.sb_region, L::NORM_BUF, bar, l2pol);
      }
    }
    valid = (valid & ~(1u << s)) | ((uint32_t)ok << s);
  };
  const int npro = my_n < TQ_STAGES ? my_n : TQ_STAGES;
  for (int it = 0; it < npro; ++it) issue(it);

  Tq4State<D> st;
  st.init();
  const int ld_t = (lane & 7) + 8 * ((lane >> 3) & 1);
  const int ld_ch = lane >> 4;
  uint32_t koff[NCH];
#pragma unroll
  for (int g = 0; g < NCH; ++g) koff[g] = swz<L::CB>(ld_t, 2 * g + ld_ch);
  const uint32_t lut_lane = smem_u32(lut_w) + 4u * lane;

  // verifier causal limits: token i of L sees positions < ctx - L + 1 + i
  int lim0 = ctx, lim1 = ctx;
  if constexpr (VER) {
    const int ctx_all = ctx - a.L + 1;
    lim0 = min(ctx, ctx_all + (8 * nt + 2 * c) / a.G);
    lim1 = min(ctx, ctx_all + (8 * nt + 2 * c + 1) / a.G);
  }
  const int ctx_full = VER ? ctx - a.L + 1 : ctx;   // chunks below it: no masks
  int done = 0;
#pragma unroll 1
  for (int it = 0; it < my_n; ++it) {
    const int s = it % TQ_STAGES;
    const uint32_t par = (it / TQ_STAGES) & 1;
    if (!mbar_wait_bounded(&bars[warp * TQ_STAGES + s], par)) {
      if (lane == 0) flag_error(a.status, JF_DEV_ERR_TIMEOUT);
      break;
    }
    done = it + 1;
    const bool ok = (valid >> s) & 1u;
    const int tokbase = chunk_of(it) * DTOK;
    const uint32_t kc = smem_u32(codes + (warp * TQ_STAGES + s) * 2 * L::CODE_BUF);
    const uint8_t* kn = norms + (warp * TQ_STAGES + s) * 2 * L::NORM_BUF;
    if (ok && tokbase + DTOK <= ctx_full) {
      tq4_chunk<D, VER, true>(st, bq, kc, kn, lut_lane, koff, cS, r, DTOK, DTOK, DTOK);
    } else {
      const int nv = ok ? min(ctx - tokbase, DTOK) : 0;
      tq4_chunk<D, VER, false>(st, bq, kc, kn, lut_lane, koff, cS, r, nv,
                               ok ? min(lim0 - tokbase, nv) : 0, ok ? min(lim1 - tokbase, nv) : 0);
    }
    __syncwarp();
    if (it + TQ_STAGES < my_n) {
      fence_proxy_async_smem();
      issue(it + TQ_STAGES);
    }
  }
  if (done < my_n) {
    for (int it = done; it < my_n && it < done + TQ_STAGES; ++it)
      mbar_wait_bounded(&bars[warp * TQ_STAGES + it % TQ_STAGES], (it / TQ_STAGES) & 1, 1u << 16);
  }
  asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory");

  // ---- per-warp finalize and CTA combine -----------------------------------
#pragma unroll
  for (int o = 4; o < 32; o <<= 1) {
    st.l0 += __shfl_xor_sync(0xffffffffu, st.l0, o);
    st.l1 += __shfl_xor_sync(0xffffffffu, st.l1, o);
  }
  __syncthreads();   // every warp is past its last stage: reuse the rings
  constexpr int SROW = D + 4;
  float* so = reinterpret_cast<float*>(codes);            // [TQ_WARPS][8][SROW]
  float* sml = so + TQ_WARPS * 8 * SROW;                  // [TQ_WARPS][8][2]
  float* swt = sml + TQ_WARPS * 8 * 2;                    // [TQ_WARPS][8]
  float* shl = swt + TQ_WARPS * 8;                        // [8][2]
#pragma unroll
  for (int g = 0; g < NCH; ++g)
#pragma unroll
    for (int hf = 0; hf < 2; ++hf)
#pragma unroll
      for (int hh = 0; hh < 2; ++hh) {
        const int i = 2 * hf + hh;
        const float4 v = make_float4(st.O[g][0][i], st.O[g][1][i], st.O[g][2][i], st.O[g][3][i]);
        *reinterpret_cast<float4*>(so + (warp * 8 + 2 * c + hh) * SROW + 64 * g + 32 * hf + 4 * r) = v;
      }
  if (r == 0) {
    sml[(warp * 8 + 2 * c) * 2 + 0] = st.m0;
    sml[(warp * 8 + 2 * c) * 2 + 1] = st.l0;
    sml[(warp * 8 + 2 * c + 1) * 2 + 0] = st.m1;
    sml[(warp * 8 + 2 * c + 1) * 2 + 1] = st.l1;
  }
  __syncthreads();
  if (threadIdx.x < rows) {
    const int h = threadIdx.x;
    float M = NEG_INF;
#pragma unroll
    for (int w = 0; w < TQ_WARPS; ++w) M = fmaxf(M, sml[(w * 8 + h) * 2]);
    float f[TQ_WARPS];
    float Ls = 0.f;
#pragma unroll
    for (int w = 0; w < TQ_WARPS; ++w) {
      const float mw = sml[(w * 8 + h) * 2];
      f[w] = (mw != NEG_INF) ? fast_exp2(mw - M) : 0.f;
      Ls = fmaf(f[w], sml[(w * 8 + h) * 2 + 1], Ls);
    }
    const float inv = direct ? (Ls > 0.f ? 1.f / Ls : 0.f) : 1.f;
#pragma unroll
    for (int w = 0; w < TQ_WARPS; ++w) swt[w * 8 + h] = f[w] * inv;
    shl[h * 2 + 0] = M;
    shl[h * 2 + 1] = Ls;
  }
  __syncthreads();
  // combined rotated-domain output per head -> qbuf [8][D]
  for (int idx = threadIdx.x; idx < rows * (D / 4); idx += blockDim.x) {
    const int h = idx / (D / 4), d = 4 * (idx % (D / 4));
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
    for (int w = 0; w < TQ_WARPS; ++w) {
      const float f = swt[w * 8 + h];
      const float4 v = *reinterpret_cast<const float4*>(so + (w * 8 + h) * SROW + d);
      if (f != 0.f) {
        acc.x = fmaf(f, v.x, acc.x);
        acc.y = fmaf(f, v.y, acc.y);
        acc.z = fmaf(f, v.z, acc.z);
        acc.w = fmaf(f, v.w, acc.w);
      }
    }
    *reinterpret_cast<float4*>(qbuf + h * D + d) = acc;
  }
  __syncthreads();
  // inverse rotation o = S_V H (2^8 acc) / sqrt(D): warp h < rows takes head h
  if (warp < rows) {
    const int h = warp;
    float x[E];
#pragma unroll
    for (int e = 0; e < E; ++e) x[e] = qbuf[h * D + lane * E + e];
    warp_fwht<float, E>(x, lane);
    const float osc = 256.f * rsqrtf((float)D);
    const uint32_t sb = prm.sv[(lane * E) >> 5] >> ((lane * E) & 31);
#pragma unroll
    for (int e = 0; e < E; ++e) x[e] *= ((sb >> e) & 1u) ? -osc : osc;
    const int fr = row_of(h);
    const int d0 = lane * E;
    if (direct) {
      uint32_t w[E / 2];
#pragma unroll
      for (int e = 0; e < E / 2; ++e)
        w[e] = (uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(x[2 * e])) |
               ((uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(x[2 * e + 1])) << 16);
      uint16_t* dst = a.out + ((int64_t)b * a.HqL + fr) * D + d0;
      if constexpr (E == 8)
        *reinterpret_cast<uint4*>(dst) = make_uint4(w[0], w[1], w[2], w[3]);
      else
        *reinterpret_cast<uint2*>(dst) = make_uint2(w[0], w[1]);
    } else {
      const int64_t row = a.balanced ? (int64_t)blockIdx.x * a.HqL + fr
                                     : ((int64_t)b * a.HqL + fr) * a.num_splits + blockIdx.x;
      float* dst = a.part_o + row * D + d0;
#pragma unroll
      for (int e = 0; e < E; e += 4)
        *reinterpret_cast<float4*>(dst + e) = make_float4(x[e], x[e + 1], x[e + 2], x[e + 3]);
      if (lane == 0) {
        a.part_ml[row * 2 + 0] = shl[h * 2 + 0];
        a.part_ml[row * 2 + 1] = shl[h * 2 + 1];
      }
    }
  }
}

template <int D, bool VER, bool APP>
static int launch_tq4_split(const cudaLaunchConfig_t& cfg0, const CUtensorMap& tmap,
                            const DecodeArgs& a, const Tq4Params& prm) {
  if (smem_optin((const void*)tq4_split_kernel<D, VER, APP>, Tq4Smem<D>::TOTAL) != JF_OK)
    return JF_ERR_CUDA;
  cudaLaunchConfig_t cfg = cfg0;
  cfg.dynamicSmemBytes = Tq4Smem<D>::TOTAL;
  return cudaLaunchKernelEx(&cfg, tq4_split_kernel<D, VER, APP>, tmap, a, prm) == cudaSuccess
             ? JF_OK : JF_ERR_CUDA;
}

template <int D>
static int launch_tq4_split_any(const cudaLaunchConfig_t& cfg, const CUtensorMap& tmap,
                                const DecodeArgs& a, const Tq4Params& prm) {
  if (a.L > 1) return launch_tq4_split<D, true, false>(cfg, tmap, a, prm);
  if (a.knew) return launch_tq4_split<D, false, true>(cfg, tmap, a, prm);
  return launch_tq4_split<D, false, false>(cfg, tmap, a, prm);
}

// packed verifier with more than 8 rows per KV head (tq4_verify.cu)
int launch_tq4_verify_pairs(const CUtensorMap& tmap, const DecodeArgs& a, const Tq4Params& prm,
                            int D, int B, cudaStream_t stream);

int launch_tq4_decode(const Geom& g, const jf_kv_pool& pool, const CUtensorMap& tmap,
                      const Tq4Params& prm, const int32_t* page_table, int32_t pt_stride,
                      const int32_t* context_lens, int32_t batch, const void* q, int32_t Hq,
                      float softmax_scale, void* out, void* workspace, int32_t num_splits,
                      cudaStream_t stream, const void* k_new, const void* v_new, int32_t q_len) {
  DecodeArgs a{};
  a.pool = static_cast<const uint8_t*>(pool.base);
  a.num_pages = g.num_pages;
  a.page_bytes = g.page_bytes;
  a.codes_region = g.codes_region;
  a.sb_base = 2 * g.codes_region;
  a.sb_region = g.sb_region;
  a.P = g.P;
  a.log2P = __builtin_ctz((unsigned)g.P);
  a.Hkv = g.Hkv;
  a.Hq = Hq;
  a.G = Hq / g.Hkv;
  a.L = q_len;
  a.NT = (a.G * q_len + 7) / 8;
  a.HqL = q_len * Hq;
  a.page_table = page_table;
  a.pt_stride = pt_stride;
  a.ctx = context_lens;
  a.q = static_cast<const uint16_t*>(q);
  a.knew = static_cast<const uint16_t*>(k_new);
  a.vnew = static_cast<const uint16_t*>(v_new);
  a.out = static_cast<uint16_t*>(out);
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  const int64_t rows = (int64_t)batch * q_len * Hq * num_splits;
  a.status = reinterpret_cast<int32_t*>(ws);
  a.part_ml = reinterpret_cast<float*>(ws + 256);
  a.part_o = reinterpret_cast<float*>(ws + 256 + (rows * 8 + 255) / 256 * 256);
  a.num_splits = num_splits;
  a.plan_splits = num_splits;
  a.span = 0;
  a.scale_log2 = softmax_scale * 1.4426950408889634f;
  a.B = batch;
  a.balanced = (batch > 1 && batch <= 1024 && num_splits > 1) ? 1 : 0;
  a.budget = 1;
  if (q_len > 1 && a.NT >= 2) {
    // warp pairs sharing the centroid lookups: ceil(NT / 3) CTAs per KV head
    // and split, one CTA per SM
    const int ntc = a.NT < 3 ? a.NT : 3;
    const int per_head = g.Hkv * ((a.NT + ntc - 1) / ntc);
    const int vslots = sm_count() / per_head > 1 ? sm_count() / per_head : 1;
    a.plan_splits = num_splits < vslots ? num_splits : vslots;
    if (a.balanced) {
      const int64_t fit = (int64_t)batch * num_splits - batch;
      const int64_t cap = fit < vslots ? fit : vslots;
      a.budget = (int)(cap - batch / 2 > 1 ? cap - batch / 2 : 1);
    }
    return launch_tq4_verify_pairs(tmap, a, prm, g.D, batch, stream);
  }
  if (a.balanced) {   // one CTA per SM in all
    const int slots = (sm_count() + g.Hkv * a.NT - 1) / (g.Hkv * a.NT);
    const int64_t fit = (int64_t)batch * num_splits - batch;
    const int64_t cap = fit < slots ? fit : slots;
    a.budget = (int)(cap - batch / 2 > 1 ? cap - batch / 2 : 1);
  }
  cudaLaunchAttribute pdl[1];
  pdl[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  pdl[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = a.balanced ? dim3((unsigned)(a.budget + batch), (unsigned)(g.Hkv * a.NT), 1u)
                           : dim3((unsigned)num_splits, (unsigned)(g.Hkv * a.NT), (unsigned)batch);
  cfg.blockDim = dim3(TQ_WARPS * 32);
  cfg.stream = stream;
  cfg.attrs = pdl;
  cfg.numAttrs = 1;
  const int st = (g.D == 256) ? launch_tq4_split_any<256>(cfg, tmap, a, prm)
                              : launch_tq4_split_any<128>(cfg, tmap, a, prm);
  if (st) return st;
  if (num_splits > 1) return launch_decode_merge(a, g.D, batch, stream);
  return JF_OK;
}

}  // namespace jfkv
