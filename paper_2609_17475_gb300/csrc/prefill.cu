// Prefill-chunk attention on the 5th-generation tensor cores (tcgen05).
//
// Sec. 3.1 of the paper splits attention into a page-native decode kernel and
// a prefill path that reconstructs K/V from the pool and runs a dense
// attention over a block of queries (Eq. 5: each KV head serves its group of
// query heads).  Here the reconstruction never reaches global memory: it is
// fused into the attention kernel as fp16 shared-memory tiles that feed
// tcgen05.mma directly.
//
// CTA = (tile of QPC = 128 / G queries of one request, KV head); one launch
// may cover the chunks of several requests (each with its own page-table row,
// prefix length and queries).  Its 128 MMA rows are the
// (query, head) pairs r = i * G + j of the G query heads that share the KV
// head, so every dequantized K/V tile is reused by all of them.  Two CTAs on
// two SMs form a pair (a cluster of 2, tcgen05 cta_group::2): the pair runs
// M = 256 MMAs over the same K/V tiles, and each CTA dequantizes only half of
// every tile -- 32 of its 64 K rows (the N half of S = Q K^T it supplies) and
// D/2 of the V columns (its N half of O += P V) -- so the dequantization work
// per SM is halved while each SM's tensor core still does its 128 rows.
// Warp roles (each CTA):
//   warp 0      TMEM allocation (512 columns, pair-wide); in CTA 0, lane 0
//               issues every tcgen05.mma.cta_group::2 of the pair:
//                 S_i  = Q  [K_2i K_2i+1]^T  (A = Q in smem, B = the K halves
//                        of tiles 2i and 2i + 1 in smem, K-major, N = 128)
//                 O   += P_j V_j             (A = P_j in TMEM, B = V_j smem,
//                        MN-major)
//               and commits to the barrier of both CTAs (multicast).
//               TMEM columns: O [0, D), two S/P buffers of a tile pair
//               [D, D + 256); P_j (fp16) overwrites S columns already read.
//               S over two tiles keeps the MMA at N = 128 (an N = 64 pair
//               MMA takes as long as an N = 128 one).
//   warps 1-8   dequantize this CTA's halves of 64-position K/V tiles from
//               the pool (page-table lookup, 4-bit codes -> fp16 integers
//               through the mantissa of fp16 1024, then x = code * scale +
//               bias with one fused multiply-add) into 128B-swizzled
//               buffers, one item (one position's code bytes of a 64-wide
//               block) per thread, loads running two tiles ahead; warps 1-4
//               write K halves into two pair buffers (free again once S of
//               the pair two back is done), warps 5-8 V halves into four
//               tile buffers (free once P V of the tile four back is done),
//               each arriving on CTA 0's K-pair or V-tile barrier.
//   warps 9-12  one thread per row: Q row -> shared memory at the start;
//               online softmax on S (tcgen05.ld), P back to TMEM as fp16
//               over S columns already read (tcgen05.st) and an arrive on
//               CTA 0's P barrier; the running maximum is moved only when it
//               grows by more than 2^8, and then O is rescaled in TMEM;
//               finally O / l -> bf16 output.
// Within every 8 consecutive d the tiles store elements in the order
// 0,4,1,5,2,6,3,7 (the pairs one 32-bit word of codes yields); Q uses the same
// order, so Q K^T is unchanged, and the epilogue undoes it for O.  Q is
// stored pre-multiplied by softmax_scale * log2(e), so S arrives in the log2
// domain.
#include <cmath>

#include "tc.cuh"
#include "tq4.cuh"

namespace jfkv {

constexpr int PF_BM = 128;   // MMA rows per CTA (256 per CTA pair)
constexpr int PF_BN = 64;    // positions per K/V tile
constexpr int PF_DQ_WARPS = 8;
constexpr int PF_SM_WARPS = 4;   // one per TMEM lane quarter, one row per thread
constexpr int PF_THREADS = 32 * (1 + PF_DQ_WARPS + PF_SM_WARPS);
constexpr int PF_KVBUF = 4;     // P V completion barriers, by tile index mod 4
constexpr float PF_TAU = 8.f;   // log2 headroom before the running max moves

// One request's chunk in a launch: its query tiles are CTAs tile0 ..
// tile0 + n_tiles2 - 1 (n_tiles2 even, so a CTA pair never spans requests).
struct PfReq {
  const int32_t* pt;    // its page-table row
  const uint16_t* q;    // its chunk's queries [C, Hq, D]
  uint16_t* out;        // [C, Hq, D]
  int32_t q_start, C, tile0, n_tiles2;
  int32_t row0;         // its first query's row in the launch (split partials)
};

constexpr int PF_MAX_REQ = 64;   // requests per launch

struct PrefillArgs {
  const uint8_t* pool;
  int64_t num_pages;
  int64_t page_bytes;
  int64_t codes_region;
  int64_t sb_base;
  int64_t sb_region;
  int32_t P, Hkv, Hq, G, QPC;
  int32_t causal;
  float scale_log2;
  int32_t* status;
  int32_t num_splits;   // > 1: history ranges per query tile, partials + merge
  float* part_ml;       // [rows * Hq][num_splits][2] (m, l)
  float* part_o;        // [rows * Hq][num_splits][D], unnormalized
  const float* qrot;     // TQ4: rotated queries H S_K q / sqrt(D), fp32 [rows * Hq][D]
  float cent[16];        // TQ4: centroids
  int32_t nreq;
  PfReq req[PF_MAX_REQ];
};

// Each CTA of a pair holds its 128 query rows (fp16, K-major) and half of
// every K/V tile: K positions 32 r .. 32 r + 31 (all of head_dim, K-major)
// and V columns D/2 r .. D/2 (r + 1) (all 64 positions, MN-major), r = its
// rank in the pair.  The K halves of tiles 2i and 2i + 1 share a pair buffer
// (rows 32 (j & 1) + t), so one N = 128 MMA computes S for both.
template <int D, int FMT>
struct PfSmem {
  static constexpr int VB = 4;                           // V tile buffers
  static constexpr int Q_BYTES = PF_BM * D * 2;          // [D/64][128 rows][128 B]
  static constexpr int KP_BYTES = PF_BN * D * 2;         // [D/64][64 rows][128 B]
  static constexpr int VT_BYTES = PF_BN * (D / 2) * 2;   // [D/128][64 rows][128 B]
  static constexpr int OFF_Q = 0;
  static constexpr int OFF_K = Q_BYTES;
  static constexpr int OFF_V = OFF_K + 2 * KP_BYTES;
  static constexpr int OFF_BAR = OFF_V + VB * VT_BYTES;
  static constexpr int OFF_LUT = OFF_BAR + 256;   // TQ4 centroid table (lane-replicated)
  static constexpr int TOTAL = 1024 + OFF_LUT + (FMT == JF_FMT_TQ4 ? 256 * 32 * 4 : 0);
  static_assert(TOTAL <= 227 * 1024, "shared memory per CTA");
};

// packed fp32 pairs (Blackwell f32x2 arithmetic)
__device__ __forceinline__ uint64_t f32x2(float lo, float hi) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};\n" : "=l"(r) : "f"(lo), "f"(hi));
  return r;
}
__device__ __forceinline__ void unpack_f32x2(uint64_t v, float& lo, float& hi) {
  asm("mov.b64 {%0, %1}, %2;\n" : "=f"(lo), "=f"(hi) : "l"(v));
}
__device__ __forceinline__ uint64_t sub_f32x2(uint64_t a, uint64_t b) {
  uint64_t r;
  asm("sub.rn.f32x2 %0, %1, %2;\n" : "=l"(r) : "l"(a), "l"(b));
  return r;
}
__device__ __forceinline__ uint64_t add_f32x2(uint64_t a, uint64_t b) {
  uint64_t r;
  asm("add.rn.f32x2 %0, %1, %2;\n" : "=l"(r) : "l"(a), "l"(b));
  return r;
}

__device__ __forceinline__ uint32_t hmul2(uint32_t a, uint32_t b) {
  uint32_t r;
  asm("mul.rn.f16x2 %0, %1, %2;\n" : "=r"(r) : "r"(a), "r"(b));
  return r;
}

__device__ __forceinline__ uint32_t hadd2(uint32_t a, uint32_t b) {
  uint32_t r;
  asm("add.rn.f16x2 %0, %1, %2;\n" : "=r"(r) : "r"(a), "r"(b));
  return r;
}

__device__ __forceinline__ uint32_t hfma2(uint32_t a, uint32_t b, uint32_t c) {
  uint32_t r;
  asm("fma.rn.f16x2 %0, %1, %2, %3;\n" : "=r"(r) : "r"(a), "r"(b), "r"(c));
  return r;
}

// 8 packed 4-bit codes (d0..d7) -> 8 fp16 values code * scale + bias, stored
// in the order d0,d4,d1,d5,d2,d6,d3,d7.  A nibble OR-ed into the mantissa of
// fp16 1024 (exponent 2^10, unit mantissa step) gives 1024 + n, or 1024 + 16 n
// for a high nibble; subtracting 1024 (or scaling by 1/16 and subtracting 64)
// recovers the integer code exactly, and one fused multiply-add rounds once.
__device__ __forceinline__ uint4 dequant8(uint32_t w, uint32_t s2, uint32_t b2) {
  constexpr uint32_t K1024 = 0x64006400u;    // (1024, 1024)
  constexpr uint32_t KM1024 = 0xE400E400u;   // (-1024, -1024)
  constexpr uint32_t K1_16 = 0x2C002C00u;    // (1/16, 1/16)
  constexpr uint32_t KM64 = 0xD400D400u;     // (-64, -64)
  const uint32_t w8 = __umulhi(w, 0x01000000u);   // w >> 8 on the FMA pipe
  uint4 o;
  o.x = hfma2(hadd2((w & 0x000F000Fu) | K1024, KM1024), s2, b2);           // (d0, d4)
  o.y = hfma2(hfma2((w & 0x00F000F0u) | K1024, K1_16, KM64), s2, b2);      // (d1, d5)
  o.z = hfma2(hadd2((w8 & 0x000F000Fu) | K1024, KM1024), s2, b2);          // (d2, d6)
  o.w = hfma2(hfma2((w8 & 0x00F000F0u) | K1024, K1_16, KM64), s2, b2);     // (d3, d7)
  return o;
}

// bf16 (scale | bias << 16) word -> f16x2 broadcasts of scale and bias
__device__ __forceinline__ void sb_to_h2(uint32_t w, uint32_t& s2, uint32_t& b2) {
  const float s = bf16lo_to_f32(w), b = bf16hi_to_f32(w);
  s2 = pack_f16x2(s, s);
  b2 = pack_f16x2(b, b);
}

// FMT: JF_FMT_AFFINE4_G64, or JF_FMT_TQ4 (centroid table, rotated queries,
// natural d order, partial outputs rotated back by the merge kernel)
template <int D, int FMT>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(PF_THREADS, 1)
prefill_kernel(const __grid_constant__ PrefillArgs a) {
  using L = PfSmem<D, FMT>;
  constexpr bool TQ = FMT == JF_FMT_TQ4;
  constexpr int NKB = D / 64;           // 64-wide d blocks
  constexpr int UPI = (D == 256) ? 2 : 1;   // 16-byte code units per dequant item
  constexpr int SBB = D / 16;
  constexpr int CB = D / 2;
  // 128 K items (32 positions x NKB blocks x 2/UPI units) + 128 V items
  // (64 positions x NKB/2 blocks x 2/UPI units): one per dequant thread
  static_assert((PF_BN / 2) * NKB * 2 / UPI == 128 && PF_BN * (NKB / 2) * 2 / UPI == 128,
                "one item per dequant thread");
  constexpr uint32_t IDQK = tc::idesc_f16_f32(2 * PF_BM, 2 * PF_BN, 0, 0);   // a tile pair
  constexpr uint32_t IDPV = tc::idesc_f16_f32(2 * PF_BM, D, 0, 1);

  extern __shared__ uint8_t smraw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smraw) + 1023) &
                                           ~static_cast<uintptr_t>(1023));
  uint8_t* sK = sm + L::OFF_K;
  uint8_t* sQ = sm + L::OFF_Q;
  uint8_t* sV = sm + L::OFF_V;
  uint64_t* bars = reinterpret_cast<uint64_t*>(sm + L::OFF_BAR);
  uint64_t* k_full = bars + 0;     // [2] on CTA 0: K halves of a tile pair stored
  uint64_t* v_full = bars + 2;     // [VB] on CTA 0: both CTAs' V halves stored (tile j % VB)
  uint64_t* pv_done = bars + 6;    // [4] both CTAs: P V of tile j done (j & 3)
  uint64_t* s_full = bars + 10;    // [2] both CTAs: S of pair i done (i & 1)
  // [4] on CTA 0: both CTAs' P stored (tile j & 3).  S of the next pair is
  // issued before P V of this one, so a CTA's softmax can run up to 3 tiles
  // past the tile P V waits for: four barriers keep one CTA's later arrivals
  // out of the phase the other CTA has not reached.
  uint64_t* p_full = bars + 12;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 16);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = tc::cluster_rank();
  // CTA pairs in launch order: the KV heads of one pair of query tiles are
  // consecutive, so every head's longest tiles start in the first wave
  const int pair = (int)(blockIdx.x >> 1);
  const int kvh = pair % a.Hkv;
  const int tile = (pair / a.Hkv) * 2 + (int)(blockIdx.x & 1);
  // this CTA's request (tile ranges ascend with the request index)
  int ri = 0;
  for (int i = 1; i < a.nreq; ++i)
    if (tile >= a.req[i].tile0) ri = i;
  const PfReq& rq = a.req[ri];
  const int32_t* const pt = rq.pt;
  const int q_start = rq.q_start, C = rq.C;
  const int bx = tile - rq.tile0;
  // query tile of this CTA and of its partner: latest (longest) tiles first
  const int qt = rq.n_tiles2 - 1 - bx;
  const int qt_partner = rq.n_tiles2 - 1 - (bx ^ 1);
  const int q0 = qt * a.QPC;
  const int nq = max(0, min(a.QPC, C - q0));
  const int rows = nq * a.G;
  const int total = q_start + C;
  // positions a query tile attends (0 for the padding tile of an odd count)
  auto kmax_of = [&](int t) {
    const int first = t * a.QPC;
    const int n = max(0, min(a.QPC, C - first));
    return n == 0 ? 0 : (a.causal ? q_start + first + n : total);
  };
  const int kmax = kmax_of(qt);
  const int kmax_pair = max(kmax, kmax_of(qt_partner));
  const int ntiles_all = (kmax_pair + PF_BN - 1) / PF_BN;
  // this CTA pair's contiguous range of history tiles (the whole history when
  // there is one split); both CTAs of the pair walk the same tiles
  const int jb = (int)(((int64_t)ntiles_all * blockIdx.z) / a.num_splits);
  const int je = (int)(((int64_t)ntiles_all * (blockIdx.z + 1)) / a.num_splits);
  const int ntiles = je - jb;

  if (threadIdx.x == 0) {
    for (int i = 0; i < 4; ++i) {
      if (i < L::VB) mbar_init(&v_full[i], PF_DQ_WARPS);   // the 4 V warps of each CTA
      mbar_init(&pv_done[i], 1);
      mbar_init(&p_full[i], 2 * PF_SM_WARPS);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&k_full[i], 2 * PF_DQ_WARPS);    // the 4 K warps of each CTA, twice
      mbar_init(&s_full[i], 1);
    }
    fence_barrier_init();
  }
  if constexpr (TQ) {   // centroid pair of code byte b for lane l: word b * 32 + l
    uint32_t* lut = reinterpret_cast<uint32_t*>(sm + L::OFF_LUT);
    for (int i = threadIdx.x; i < 256 * 32; i += blockDim.x)
      lut[i] = pack_f16x2(a.cent[(i >> 5) & 15], a.cent[i >> 9]);
  }
  if (warp == 0) tc::alloc2(tmem_slot, 512);
  tc::fence_before();
  __syncthreads();
  tc::cluster_sync();   // both CTAs: barriers initialized, TMEM allocated
  tc::fence_after();
  const uint32_t tbase = *tmem_slot;
  const uint32_t tO = tbase;
  const uint32_t tS = tbase + D;               // two S/P buffers of 2 PF_BN columns

  // ---- softmax warps: their Q row -> shared memory (fp16,
  // pre-multiplied by softmax_scale * log2(e), d order 0,4,1,5,2,6,3,7 in
  // every 8; K-major, 128-byte swizzle: the 16-byte chunk m of row r at
  // block m / 8, chunk (m % 8) ^ (r % 8)) -------------------------------------
  const int quarter = warp & 3;                // TMEM lanes this warp may access
  const int r = quarter * 32 + lane;
  const bool row_ok = r < rows;
  const int qi = row_ok ? r / a.G : 0;
  const uint32_t lane_off = (uint32_t)(quarter * 32) << 16;
  int qe = 0;                                  // per-row power of two kept out of fp16
  auto q_chunk = [&](int m) -> uint4* {
    return reinterpret_cast<uint4*>(sQ + (m >> 3) * (PF_BM * 128) + r * 128 +
                                    (((m & 7) ^ (r & 7)) << 4));
  };
  if (TQ && warp > PF_DQ_WARPS) {
    // rotated fp32 query row, natural d order (the centroid pairs are too)
    const float* qrow = a.qrot + ((int64_t)(rq.row0 + q0 + qi) * a.Hq + kvh * a.G + r % a.G) * D;
    float qmax = 0.f;
    if (row_ok) {
      for (int c4 = 0; c4 < D / 4; ++c4) {
        const float4 w = *reinterpret_cast<const float4*>(qrow + 4 * c4);
        qmax = fmaxf(qmax, fmaxf(fmaxf(fabsf(w.x), fabsf(w.y)), fmaxf(fabsf(w.z), fabsf(w.w))));
      }
    }
    qmax *= fabsf(a.scale_log2);
    qe = (qmax >= 16384.f) ? (ilogbf(qmax) - 13) : 0;
    const float qs = ldexpf(a.scale_log2, -qe);
#pragma unroll 4
    for (int m = 0; m < D / 8; ++m) {   // natural d order
      float4 w0 = make_float4(0.f, 0.f, 0.f, 0.f), w1 = w0;
      if (row_ok) {
        w0 = *reinterpret_cast<const float4*>(qrow + 8 * m);
        w1 = *reinterpret_cast<const float4*>(qrow + 8 * m + 4);
      }
      *q_chunk(m) = make_uint4(pack_f16x2(w0.x * qs, w0.y * qs), pack_f16x2(w0.z * qs, w0.w * qs),
                               pack_f16x2(w1.x * qs, w1.y * qs), pack_f16x2(w1.z * qs, w1.w * qs));
    }
    fence_proxy_async_smem();
  } else if (warp > PF_DQ_WARPS) {
    const uint16_t* qrow = rq.q + ((int64_t)(q0 + qi) * a.Hq + kvh * a.G + r % a.G) * D;
    float qmax = 0.f;
    if (row_ok) {
      for (int c8 = 0; c8 < D / 8; ++c8) {
        const uint4 w = *reinterpret_cast<const uint4*>(qrow + 8 * c8);
        const uint32_t ws[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
        for (int k = 0; k < 4; ++k)
          qmax = fmaxf(qmax, fmaxf(fabsf(bf16lo_to_f32(ws[k])), fabsf(bf16hi_to_f32(ws[k]))));
      }
    }
    qmax *= a.scale_log2;
    qe = (qmax >= 16384.f) ? (ilogbf(qmax) - 13) : 0;
    const float qs = ldexpf(a.scale_log2, -qe);
#pragma unroll 4
    for (int m = 0; m < D / 8; ++m) {
      uint4 w = make_uint4(0, 0, 0, 0);
      if (row_ok) w = *reinterpret_cast<const uint4*>(qrow + 8 * m);
      const float e0 = bf16lo_to_f32(w.x) * qs, e1 = bf16hi_to_f32(w.x) * qs;
      const float e2 = bf16lo_to_f32(w.y) * qs, e3 = bf16hi_to_f32(w.y) * qs;
      const float e4 = bf16lo_to_f32(w.z) * qs, e5 = bf16hi_to_f32(w.z) * qs;
      const float e6 = bf16lo_to_f32(w.w) * qs, e7 = bf16hi_to_f32(w.w) * qs;
      *q_chunk(m) = make_uint4(pack_f16x2(e0, e4), pack_f16x2(e1, e5), pack_f16x2(e2, e6),
                               pack_f16x2(e3, e7));
    }
    fence_proxy_async_smem();
  }
  tc::fence_before();
  __syncthreads();
  tc::cluster_sync();   // both CTAs' Q rows are in shared memory before the first MMA
  tc::fence_after();

  if (warp == 0) {
    // ================= MMA issuer (CTA 0 of the pair) =================
    if (rank == 0 && lane == 0) {
      const uint32_t qaddr = smem_u32(sQ), kaddr = smem_u32(sK), vaddr = smem_u32(sV);
      bool ok = true;
      // P_j (fp16, 32 columns) sits in the columns of its pair's S buffer
      // that held S of positions 0..31 of tile j
      auto pv = [&](int j) {   // j: local tile index within this split
        const int kb = j % L::VB;
        if (!tc::wait_cluster(&v_full[kb], (j / L::VB) & 1) ||
            !tc::wait_cluster(&p_full[j & 3], (j >> 2) & 1)) { ok = false; return; }
        tc::fence_after();
        const uint32_t tp = tS + ((j >> 1) & 1) * (2 * PF_BN) + (j & 1) * 32;
#pragma unroll
        for (int k = 0; k < PF_BN / 16; ++k)
          tc::mma2_ts(tO, tp + 8 * k,
                      tc::sdesc_sw128(vaddr + kb * L::VT_BYTES + k * 2048, PF_BN * 128, 1024),
                      IDPV, (j > 0 || k > 0) ? 1u : 0u);
        tc::commit2_both(&pv_done[j & 3]);
      };
      // Pair i: S of tiles 2i, 2i + 1 into S buffer i & 1 (S column n = K row
      // n of CTA 0 for n < 64, row n - 64 of CTA 1 otherwise: position 32 rank
      // + n % 32 of tile 2i + (n % 64) / 32), then P V of the previous pair's
      // tiles; the buffer's last readers (P V of pair i - 2) were issued
      // before it.  One call site each: the issuer's code shares the SM's
      // instruction cache with the other roles.
      const int npairs = (ntiles + 1) >> 1;
      int jn = 0;   // next tile whose P V is due
      for (int i = 0; i <= npairs && ok; ++i) {
        if (i < npairs) {
          if (!tc::wait_cluster(&k_full[i & 1], (i >> 1) & 1)) { ok = false; break; }
          tc::fence_after();
#pragma unroll
          for (int ks = 0; ks < D / 16; ++ks)
            tc::mma2_ss(tS + (i & 1) * (2 * PF_BN),
                        tc::sdesc_sw128(qaddr + (ks >> 2) * (PF_BM * 128) + (ks & 3) * 32, 16, 1024),
                        tc::sdesc_sw128(kaddr + (i & 1) * L::KP_BYTES + (ks >> 2) * (PF_BN * 128) +
                                            (ks & 3) * 32, 16, 1024),
                        IDQK, ks ? 1u : 0u);
          tc::commit2_both(&s_full[i & 1]);
        }
        for (const int upto = i < npairs ? 2 * i : ntiles; jn < upto && ok; ++jn) pv(jn);
      }
      if (!ok) flag_error(a.status, JF_DEV_ERR_TIMEOUT);
    }
    __syncwarp();
  } else if (warp <= PF_DQ_WARPS) {
    // ================= dequantization (this CTA's halves) =================
    // threads 0..127: K item (position 32 rank + t of the tile, block kb, unit u0)
    // threads 128..255: V item (position t, block D/128 * rank + kbl, unit u0)
    const int dt = (int)threadIdx.x - 32;
    const bool is_v = dt >= 128;
    const int e = is_v ? dt - 128 : dt;
    const int t = is_v ? (e % PF_BN) : (e % (PF_BN / 2));
    const int rest = is_v ? (e / PF_BN) : (e / (PF_BN / 2));
    const int kbl = (UPI == 2) ? rest : (is_v ? 0 : rest >> 1);
    const int u0 = (UPI == 2) ? 0 : (is_v ? rest : rest & 1);
    const int kb = is_v ? (NKB / 2) * (int)rank + kbl : kbl;
    const int tpos = is_v ? t : (PF_BN / 2) * (int)rank + t;   // position within the tile
    // V tile buffers [D/128][64 rows][128 B]; K pair buffers [D/64][64 rows][128 B]
    uint8_t* dst_base = (is_v ? sV : sK) + kbl * (PF_BN * 128) + t * 128;
    const int64_t code_off = (is_v ? a.codes_region : 0) + kb * 32 + u0 * 16;
    // affine: the block's scale/bias word; TQ4: the vector's fp16 norm
    const int64_t sb_off = a.sb_base + (is_v ? a.sb_region : 0) + (TQ ? 0 : kb * 4);
    const uint32_t lut_lane = smem_u32(sm + L::OFF_LUT) + 4u * (uint32_t)lane;
    struct Tile {
      uint4 c[UPI];
      uint32_t sbw;
      bool valid;
    };
    // page id of tile j (P >= 64, so a tile lies in one page); it is loaded a
    // step before its tile's code loads need it
    // j: local tile index; the history tile is jb + j
    auto page_of = [&](int j) -> int {
      return j < ntiles ? __ldg(pt + ((jb + j) * PF_BN) / a.P) : -1;
    };
    auto load_tile = [&](int j, int page, Tile& x) {
      const int key0 = (jb + j) * PF_BN;
      const bool pok = page >= 0 && page < a.num_pages;
      if (!pok && dt == 0) flag_error(a.status, JF_DEV_ERR_PAGE_ID);
      x.valid = pok && (key0 + tpos < kmax_pair);
      if (x.valid) {
        const uint8_t* base = a.pool + (int64_t)page * a.page_bytes;
        const int64_t row = (int64_t)kvh * a.P + key0 % a.P + tpos;
        const uint8_t* cp = base + code_off + row * CB;
#pragma unroll
        for (int u = 0; u < UPI; ++u) x.c[u] = __ldg(reinterpret_cast<const uint4*>(cp + 16 * u));
        if constexpr (TQ)
          x.sbw = __ldg(reinterpret_cast<const uint16_t*>(base + sb_off + row * 2));
        else
          x.sbw = __ldg(reinterpret_cast<const uint32_t*>(base + sb_off + row * SBB));
      }
    };
    auto store = [&](uint8_t* tile, const Tile& x) {
      uint4 o[UPI][4];
      if constexpr (TQ) {
        // TQ4: norm * centroid of each index, natural d order (byte i gives
        // d 2i, 2i+1); |c| < 1/4 and norm <= 65504 keep it in fp16 range
        const uint32_t n2 = (x.sbw & 0xFFFFu) | (x.sbw << 16);
#pragma unroll
        for (int u = 0; u < UPI; ++u) {
          const uint32_t cw[4] = {x.c[u].x, x.c[u].y, x.c[u].z, x.c[u].w};
#pragma unroll
          for (int w = 0; w < 4; ++w) {
            uint32_t q4[4];
#pragma unroll
            for (int k = 0; k < 4; ++k) {
              uint32_t v;
              asm("ld.shared.b32 %0, [%1];\n"
                  : "=r"(v) : "r"(lut_lane + __byte_perm(cw[w], 0u, 0x4440u + k) * 128u));
              q4[k] = hmul2(v, n2);
            }
            o[u][w] = make_uint4(q4[0], q4[1], q4[2], q4[3]);
          }
        }
      } else {
        uint32_t s2, b2;
        sb_to_h2(x.sbw, s2, b2);
        // K and V are rebuilt in fp16: a group whose values can leave its
        // range (|bias| + 15 scale >= 65504, or a non-finite word) is reported
        if (x.valid && !(fabsf(bf16hi_to_f32(x.sbw)) + 15.f * bf16lo_to_f32(x.sbw) < 65504.f))
          flag_error(a.status, JF_DEV_ERR_RANGE);
#pragma unroll
        for (int u = 0; u < UPI; ++u) {
          const uint32_t cw[4] = {x.c[u].x, x.c[u].y, x.c[u].z, x.c[u].w};
#pragma unroll
          for (int w = 0; w < 4; ++w) o[u][w] = dequant8(cw[w], s2, b2);
        }
      }
#pragma unroll
      for (int u = 0; u < UPI; ++u)
#pragma unroll
        for (int w = 0; w < 4; ++w) {
          const int cc = (u0 + u) * 4 + w;
          *reinterpret_cast<uint4*>(tile + ((cc ^ (t & 7)) << 4)) =
              x.valid ? o[u][w] : make_uint4(0, 0, 0, 0);
        }
    };
    // Three register tiles rotate by name (the loop is unrolled by 3), so the
    // loads for tile j + 2 stay in flight while tile j is converted.
    Tile ta, tb, tcur;
    bool ok = true;
    int pg_next = page_of(2);
    // K warps: tile j's half goes to rows 32 (j & 1) .. of pair buffer
    // (j / 2) % 2, free once S of the pair two back is done; V warps: tile
    // buffer j % VB, free once P V of tile j - VB is done.  The
    // loads of tile j + 2 are issued after tile j's arrive: a release waits
    // for every earlier access of the warp, so loads still in flight would
    // hold the arrive back by a memory latency.
    // (one call of store per step: the roles share the SM's instruction cache)
    auto step = [&](int j, const Tile& cur, Tile& nxt) {
      const int kbuf = j % L::VB, pb = (j >> 1) & 1;
      uint64_t* const free_bar = is_v ? &pv_done[(j - L::VB) & 3] : &s_full[pb];
      const uint32_t free_par = is_v ? ((j - L::VB) >> 2) & 1 : (((j >> 1) - 2) >> 1) & 1;
      if (j >= (is_v ? L::VB : 4) && !tc::wait_cluster(free_bar, free_par)) { ok = false; return; }
      store(dst_base + (is_v ? kbuf * L::VT_BYTES : pb * L::KP_BYTES + (j & 1) * (32 * 128)), cur);
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) {
        uint64_t* const full_bar = is_v ? &v_full[kbuf] : &k_full[pb];
        tc::arrive_cluster(full_bar, 0);
        // a last K half without a partner tile arrives for it too
        if (!is_v && (j & 1) == 0 && j + 1 == ntiles) tc::arrive_cluster(full_bar, 0);
      }
      if (j + 2 < ntiles) load_tile(j + 2, pg_next, nxt);
      pg_next = page_of(j + 3);
    };
    if (ntiles > 0) load_tile(0, page_of(0), ta);
    if (ntiles > 1) load_tile(1, page_of(1), tb);
    for (int j = 0; j < ntiles && ok; j += 3) {
      step(j, ta, tcur);
      if (j + 1 < ntiles && ok) step(j + 1, tb, ta);
      if (j + 2 < ntiles && ok) step(j + 2, tcur, tb);
    }
    if (!ok && dt == 0) flag_error(a.status, JF_DEV_ERR_TIMEOUT);
  } else {
    // ================= softmax + epilogue (this CTA's 128 rows) =================
    // Rows past the chunk (padding) see every position: their Q rows are zero
    // and their outputs are never stored, and keeping them unmasked keeps the
    // warp on the same (mask-free) path as its real rows.
    const int limit = (row_ok && a.causal) ? q_start + q0 + qi : kmax_pair - 1;
    const float smul = ldexpf(1.f, qe);   // S = (scaled Q) K^T * 2^qe
    float m_ref = -INFINITY, l = 0.f;
    bool ok = true;
    for (int j = 0; j < ntiles; ++j) {
      // tile j's S: positions 0..31 in columns 32 (j & 1) .., 32..63 in
      // columns 64 + 32 (j & 1) .. of its pair's S/P buffer; P_j (fp16)
      // goes to columns 32 (j & 1) .. once both are read
      const int pi = j >> 1;
      if (!tc::wait_cluster(&s_full[pi & 1], (pi >> 1) & 1)) { ok = false; break; }
      tc::fence_after();
      const uint32_t tb = tS + (pi & 1) * (2 * PF_BN);
      uint32_t s0[32], s1[32];
      tc::ld32(tb + (j & 1) * 32 + lane_off, s0);
      tc::ld32(tb + 64 + (j & 1) * 32 + lane_off, s1);
      tc::wait_ld();
      const int key0 = (jb + j) * PF_BN;
      float x[PF_BN];
      float mt;
      {
        float m4[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
        if (key0 + PF_BN - 1 <= limit) {
#pragma unroll
          for (int c = 0; c < 32; ++c) { x[c] = __uint_as_float(s0[c]); x[c + 32] = __uint_as_float(s1[c]); }
        } else {
#pragma unroll
          for (int c = 0; c < 32; ++c) {
            x[c] = (key0 + c <= limit) ? __uint_as_float(s0[c]) : -INFINITY;
            x[c + 32] = (key0 + c + 32 <= limit) ? __uint_as_float(s1[c]) : -INFINITY;
          }
        }
        if (qe != 0) {
#pragma unroll
          for (int c = 0; c < PF_BN; ++c) x[c] *= smul;
        }
#pragma unroll
        for (int c = 0; c < PF_BN; ++c) m4[c & 3] = fmaxf(m4[c & 3], x[c]);
        mt = fmaxf(fmaxf(m4[0], m4[1]), fmaxf(m4[2], m4[3]));
      }
      const bool need = mt > m_ref + PF_TAU;
      if (__any_sync(0xffffffffu, need)) {
        const float nref = need ? mt : m_ref;
        const float f = (need && m_ref != -INFINITY) ? fast_exp2(m_ref - nref) : 1.f;
        if (j > 0) {
          if (!tc::wait_cluster(&pv_done[(j - 1) % PF_KVBUF], ((j - 1) / PF_KVBUF) & 1)) { ok = false; break; }
          tc::fence_after();
#pragma unroll 1
          for (int c0 = 0; c0 < D; c0 += 32) {
            uint32_t o[32];
            tc::ld32(tO + c0 + lane_off, o);
            tc::wait_ld();
#pragma unroll
            for (int c = 0; c < 32; ++c) o[c] = __float_as_uint(__uint_as_float(o[c]) * f);
            tc::st32(tO + c0 + lane_off, o);
          }
        }
        l *= f;
        m_ref = nref;
      }
      uint32_t p[32];
      if (m_ref == -INFINITY) {   // nothing visible yet on this row
#pragma unroll
        for (int c = 0; c < 32; ++c) p[c] = 0u;
      } else {
        // x - m and the running sums on packed fp32 pairs (one instruction
        // per two elements); the exponentials stay on the special-function unit
        const uint64_t mm = f32x2(m_ref, m_ref);
        uint64_t l2[2] = {f32x2(0.f, 0.f), f32x2(0.f, 0.f)};
#pragma unroll
        for (int c = 0; c < 32; ++c) {
          float d0, d1;
          unpack_f32x2(sub_f32x2(f32x2(x[2 * c], x[2 * c + 1]), mm), d0, d1);
          const float p0 = fast_exp2(d0), p1 = fast_exp2(d1);
          l2[c & 1] = add_f32x2(l2[c & 1], f32x2(p0, p1));
          p[c] = pack_f16x2(p0, p1);
        }
        float a0, a1, b0, b1;
        unpack_f32x2(l2[0], a0, a1);
        unpack_f32x2(l2[1], b0, b1);
        l += (a0 + a1) + (b0 + b1);
      }
      tc::st32(tb + (j & 1) * 32 + lane_off, p);
      tc::wait_st();
      tc::fence_before();
      __syncwarp();
      if (lane == 0) tc::arrive_cluster(&p_full[j & 3], 0);
    }
    // epilogue: O / l -> bf16 (one split) or the unnormalized partial
    // (m, l, O) in fp32 (several), undoing the d order 0,4,1,5,2,6,3,7
    const bool split = TQ || a.num_splits > 1;   // TQ4: the merge rotates O back
    const int64_t prow = ((int64_t)(rq.row0 + q0 + qi) * a.Hq + kvh * a.G + r % a.G) *
                         a.num_splits + blockIdx.z;
    if (ntiles == 0) {   // an empty history range: a neutral partial
      if (split && row_ok) {
        a.part_ml[prow * 2 + 0] = -INFINITY;
        a.part_ml[prow * 2 + 1] = 0.f;
        float4* po = reinterpret_cast<float4*>(a.part_o + prow * D);
        for (int c = 0; c < D / 4; ++c) po[c] = make_float4(0.f, 0.f, 0.f, 0.f);
      }
    } else if (ok && tc::wait_cluster(&pv_done[(ntiles - 1) % PF_KVBUF],
                                       ((ntiles - 1) / PF_KVBUF) & 1)) {
      tc::fence_after();
      const float inv = split ? 1.f : (l > 0.f ? 1.f / l : 0.f);
      uint16_t* orow = rq.out + ((int64_t)(q0 + qi) * a.Hq + kvh * a.G + r % a.G) * D;
      float* prow_o = split ? a.part_o + prow * D : nullptr;
      if (split && row_ok) {
        a.part_ml[prow * 2 + 0] = m_ref;
        a.part_ml[prow * 2 + 1] = l;
      }
#pragma unroll 1
      for (int c0 = 0; c0 < D; c0 += 32) {
        uint32_t o[32];
        tc::ld32(tO + c0 + lane_off, o);
        tc::wait_ld();
        if (row_ok && split) {
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            const float* v = reinterpret_cast<const float*>(o + 8 * k);
            float4* dst = reinterpret_cast<float4*>(prow_o + c0 + 8 * k);
            if constexpr (TQ) {
              dst[0] = make_float4(v[0], v[1], v[2], v[3]);
              dst[1] = make_float4(v[4], v[5], v[6], v[7]);
            } else {
              dst[0] = make_float4(v[0], v[2], v[4], v[6]);
              dst[1] = make_float4(v[1], v[3], v[5], v[7]);
            }
          }
        } else if (row_ok) {
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            const float* v = reinterpret_cast<const float*>(o + 8 * k);
            uint4 w;
            w.x = (uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(v[0] * inv)) |
                  ((uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(v[2] * inv)) << 16);
            w.y = (uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(v[4] * inv)) |
                  ((uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(v[6] * inv)) << 16);
            w.z = (uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(v[1] * inv)) |
                  ((uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(v[3] * inv)) << 16);
            w.w = (uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(v[5] * inv)) |
                  ((uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(v[7] * inv)) << 16);
            *reinterpret_cast<uint4*>(orow + c0 + 8 * k) = w;
          }
        }
      }
    } else {
      ok = false;
    }
    if (!ok && lane == 0) flag_error(a.status, JF_DEV_ERR_TIMEOUT);
  }

  // neither CTA may release TMEM or exit while its partner can still reach it
  tc::fence_before();
  __syncthreads();
  tc::cluster_sync();
  if (warp == 0) {
    tc::fence_after();
    tc::dealloc2(tbase, 512);
  }
}

struct SignBits {
  uint32_t w[8];   // bit j set: S_jj = -1
};

// TQ4 prefill: rotated queries q' = H S_K q / sqrt(D) in fp32, one warp per
// (query, head) row (Sec. 3.1 Eq. 4: keys stay in the rotated basis).
template <int D>
__global__ void __launch_bounds__(256)
prefill_rotate_q_kernel(const uint16_t* q, float* qrot, int64_t rows, SignBits sk) {
  constexpr int E = D / 32;
  const int64_t row = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (row >= rows) return;   // whole warps
  const uint16_t* src = q + row * D + lane * E;
  float x[E];
#pragma unroll
  for (int e = 0; e < E; e += 2) {
    const uint32_t w = *reinterpret_cast<const uint32_t*>(src + e);
    x[e] = bf16lo_to_f32(w);
    x[e + 1] = bf16hi_to_f32(w);
  }
  const uint32_t sb = sk.w[(lane * E) >> 5] >> ((lane * E) & 31);
#pragma unroll
  for (int e = 0; e < E; ++e)
    if ((sb >> e) & 1u) x[e] = -x[e];
  warp_fwht<float, E>(x, lane);
  const float r = rsqrtf((float)D);
  float* dst = qrot + row * D + lane * E;
#pragma unroll
  for (int e = 0; e < E; e += 4)
    *reinterpret_cast<float4*>(dst + e) = make_float4(x[e] * r, x[e + 1] * r, x[e + 2] * r,
                                                      x[e + 3] * r);
}

// Merge of a launch's history splits: one warp per (query, head) row combines
// its S partials, o = sum_s 2^(m_s - M) O_s / sum_s 2^(m_s - M) l_s; for TQ4
// (ROT) the result is rotated back, o <- S_V H o / sqrt(D).
template <int D, bool ROT>
__global__ void __launch_bounds__(256)
prefill_merge_kernel(const float* part_ml, const float* part_o, uint16_t* out, int64_t rows,
                     int S, SignBits sv) {
  constexpr int E = D / 32;
  const int64_t row = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (row >= rows) return;   // whole warps
  const float2* ml = reinterpret_cast<const float2*>(part_ml) + row * S;
  float M = -INFINITY;
  for (int s2 = lane; s2 < S; s2 += 32) M = fmaxf(M, ml[s2].x);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, o));
  float acc[E];
#pragma unroll
  for (int e = 0; e < E; ++e) acc[e] = 0.f;
  float L = 0.f;
  if (M != -INFINITY) {
    for (int s2 = 0; s2 < S; ++s2) {
      const float2 v = ml[s2];
      if (v.x == -INFINITY) continue;   // an empty history range
      const float w = fast_exp2(v.x - M);
      L = fmaf(w, v.y, L);
      const float4* po = reinterpret_cast<const float4*>(part_o + (row * S + s2) * D + lane * E);
#pragma unroll
      for (int e = 0; e < E / 4; ++e) {
        const float4 x = po[e];
        acc[4 * e + 0] = fmaf(w, x.x, acc[4 * e + 0]);
        acc[4 * e + 1] = fmaf(w, x.y, acc[4 * e + 1]);
        acc[4 * e + 2] = fmaf(w, x.z, acc[4 * e + 2]);
        acc[4 * e + 3] = fmaf(w, x.w, acc[4 * e + 3]);
      }
    }
  }
  const float inv = L > 0.f ? 1.f / L : 0.f;
  if constexpr (ROT) {
#pragma unroll
    for (int e = 0; e < E; ++e) acc[e] *= inv;
    warp_fwht<float, E>(acc, lane);
    const float r = rsqrtf((float)D);
    const uint32_t sb = sv.w[(lane * E) >> 5] >> ((lane * E) & 31);
#pragma unroll
    for (int e = 0; e < E; ++e) acc[e] *= ((sb >> e) & 1u) ? -r : r;
  } else {
#pragma unroll
    for (int e = 0; e < E; ++e) acc[e] *= inv;
  }
  uint32_t wv[E / 2];
#pragma unroll
  for (int e = 0; e < E / 2; ++e)
    wv[e] = (uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(acc[2 * e])) |
            ((uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(acc[2 * e + 1])) << 16);
  uint16_t* dst = out + row * D + lane * E;
  if constexpr (E == 8)
    *reinterpret_cast<uint4*>(dst) = make_uint4(wv[0], wv[1], wv[2], wv[3]);
  else
    *reinterpret_cast<uint2*>(dst) = make_uint2(wv[0], wv[1]);
}

// Workspace of a prefill launch: status word, then (split launches and every
// TQ4 launch) (m, l) and O partials, then (TQ4) the rotated queries.
size_t prefill_workspace_bytes(int64_t rows, int64_t Hq, int64_t D, int64_t S, int fmt) {
  const bool tq = fmt == JF_FMT_TQ4;
  if (S <= 1 && !tq) return 256;
  const int64_t n = rows * Hq * S;
  const int64_t part = 256 + (n * 8 + 255) / 256 * 256 + n * D * 4;
  return (size_t)(part + (tq ? rows * Hq * D * 4 : 0));
}

// One prefill launch of a given instantiation (its shared-memory opt-in is
// set once per instantiation and device).
template <int D, int FMT>
static int launch_pf(const dim3& grid, const PrefillArgs& a, cudaStream_t stream) {
  if (smem_optin((const void*)prefill_kernel<D, FMT>, PfSmem<D, FMT>::TOTAL) != JF_OK)
    return JF_ERR_CUDA;
  prefill_kernel<D, FMT><<<grid, PF_THREADS, PfSmem<D, FMT>::TOTAL, stream>>>(a);
  return cudaGetLastError() == cudaSuccess ? JF_OK : JF_ERR_CUDA;
}

// One launch over the chunks of `nreq` requests (nreq <= PF_MAX_REQ); requests
// with an empty chunk get no CTAs.  The request with the most attended
// positions goes first, so the longest CTA pairs start earliest.
int launch_prefill_batch(const Geom& g, const jf_kv_pool& pool, const int32_t* const* pt_rows,
                         const int32_t* q_start, const int32_t* chunk_len, const void* q,
                         const int64_t* q_row0, int32_t nreq, int32_t Hq, float softmax_scale,
                         int32_t causal, void* out, void* workspace, cudaStream_t stream,
                         int32_t num_splits, int64_t total_rows, const Tq4Params* tq4) {
  if (nreq < 1 || nreq > PF_MAX_REQ) return JF_ERR_UNSUPPORTED;
  const bool tq = tq4 != nullptr;
  if (num_splits < 1 || num_splits > 65535) return JF_ERR_INVALID_ARG;
  PrefillArgs a;
  a.pool = static_cast<const uint8_t*>(pool.base);
  a.num_pages = g.num_pages;
  a.page_bytes = g.page_bytes;
  a.codes_region = g.codes_region;
  a.sb_base = 2 * g.codes_region;
  a.sb_region = g.sb_region;
  a.P = g.P;
  a.Hkv = g.Hkv;
  a.Hq = Hq;
  a.G = Hq / g.Hkv;
  if (a.G > PF_BM) return JF_ERR_UNSUPPORTED;
  a.QPC = PF_BM / a.G;
  a.causal = causal ? 1 : 0;
  a.scale_log2 = softmax_scale * 1.4426950408889634f;
  a.status = static_cast<int32_t*>(workspace);
  a.num_splits = num_splits;
  SignBits sk{}, sv{};
  {
    uint8_t* ws = static_cast<uint8_t*>(workspace);
    const int64_t n = total_rows * Hq * num_splits;
    a.part_ml = reinterpret_cast<float*>(ws + 256);
    a.part_o = reinterpret_cast<float*>(ws + 256 + (n * 8 + 255) / 256 * 256);
    a.qrot = tq ? reinterpret_cast<const float*>(ws + 256 + (n * 8 + 255) / 256 * 256 +
                                                 n * g.D * 4)
                : nullptr;
    for (int k = 0; k < 16; ++k) a.cent[k] = tq ? tq4->c[k] : 0.f;
    for (int k = 0; k < 8; ++k) {
      sk.w[k] = tq ? tq4->sk[k] : 0u;
      sv.w[k] = tq ? tq4->sv[k] : 0u;
    }
  }
  int order[PF_MAX_REQ];
  int n = 0;
  for (int b = 0; b < nreq; ++b)
    if (chunk_len[b] > 0) order[n++] = b;
  if (n == 0) return JF_OK;
  auto span = [&](int b) { return (int64_t)q_start[b] + chunk_len[b]; };
  for (int i = 1; i < n; ++i)   // longest first (insertion sort, n <= 64)
    for (int j = i; j > 0 && span(order[j]) > span(order[j - 1]); --j) {
      const int t = order[j];
      order[j] = order[j - 1];
      order[j - 1] = t;
    }
  const size_t row_elems = (size_t)Hq * g.D;
  int64_t tiles = 0;
  for (int i = 0; i < n; ++i) {
    const int b = order[i];
    PfReq& r = a.req[i];
    r.pt = pt_rows[b];
    r.q = static_cast<const uint16_t*>(q) + (size_t)q_row0[b] * row_elems;
    r.out = static_cast<uint16_t*>(out) + (size_t)q_row0[b] * row_elems;
    r.q_start = q_start[b];
    r.C = chunk_len[b];
    r.row0 = (int32_t)q_row0[b];
    r.tile0 = (int32_t)tiles;
    const int n_qtiles = (chunk_len[b] + a.QPC - 1) / a.QPC;
    r.n_tiles2 = (n_qtiles + 1) & ~1;   // CTA pairs
    tiles += r.n_tiles2;
  }
  a.nreq = n;
  if (tiles * g.Hkv > 0x7FFFFFFF || g.Hkv > 65535) return JF_ERR_UNSUPPORTED;
  dim3 grid((unsigned)(tiles * g.Hkv), 1u, (unsigned)num_splits);
  const int64_t rows = total_rows * Hq;
  const int64_t rblocks = (rows + 7) / 8;   // 8 warps per CTA, one row each
  if (rblocks > 0x7FFFFFFF) return JF_ERR_UNSUPPORTED;
  if (tq) {   // rotated queries first
    if (g.D == 256)
      prefill_rotate_q_kernel<256><<<(unsigned)rblocks, 256, 0, stream>>>(
          static_cast<const uint16_t*>(q), const_cast<float*>(a.qrot), rows, sk);
    else
      prefill_rotate_q_kernel<128><<<(unsigned)rblocks, 256, 0, stream>>>(
          static_cast<const uint16_t*>(q), const_cast<float*>(a.qrot), rows, sk);
    if (cudaGetLastError() != cudaSuccess) return JF_ERR_CUDA;
  }
  int st;
  if (g.D == 256)
    st = tq ? launch_pf<256, JF_FMT_TQ4>(grid, a, stream)
            : launch_pf<256, JF_FMT_AFFINE4_G64>(grid, a, stream);
  else
    st = tq ? launch_pf<128, JF_FMT_TQ4>(grid, a, stream)
            : launch_pf<128, JF_FMT_AFFINE4_G64>(grid, a, stream);
  if (st) return st;
  if (num_splits > 1 || tq) {
    uint16_t* o = static_cast<uint16_t*>(out);
    if (g.D == 256) {
      if (tq)
        prefill_merge_kernel<256, true><<<(unsigned)rblocks, 256, 0, stream>>>(
            a.part_ml, a.part_o, o, rows, num_splits, sv);
      else
        prefill_merge_kernel<256, false><<<(unsigned)rblocks, 256, 0, stream>>>(
            a.part_ml, a.part_o, o, rows, num_splits, sv);
    } else {
      if (tq)
        prefill_merge_kernel<128, true><<<(unsigned)rblocks, 256, 0, stream>>>(
            a.part_ml, a.part_o, o, rows, num_splits, sv);
      else
        prefill_merge_kernel<128, false><<<(unsigned)rblocks, 256, 0, stream>>>(
            a.part_ml, a.part_o, o, rows, num_splits, sv);
    }
    if (cudaGetLastError() != cudaSuccess) return JF_ERR_CUDA;
  }
  return JF_OK;
}

int launch_prefill(const Geom& g, const jf_kv_pool& pool, const CUtensorMap&,
                   const int32_t* page_table_row, const void* q, int32_t q_start,
                   int32_t chunk_len, int32_t Hq, float softmax_scale, int32_t causal, void* out,
                   void* workspace, cudaStream_t stream) {
  const int64_t row0 = 0;
  return launch_prefill_batch(g, pool, &page_table_row, &q_start, &chunk_len, q, &row0, 1, Hq,
                              softmax_scale, causal, out, workspace, stream, 1, chunk_len,
                              nullptr);
}

}  // namespace jfkv
