// Prefill-chunk attention on the 5th-generation tensor cores (tcgen05).
//
// Sec. 3.1 of the paper splits attention into a page-native decode kernel and
// a prefill path that reconstructs K/V from the pool and runs a dense
// attention over a block of queries (Eq. 5: each KV head serves its group of
// query heads).  Here the reconstruction never reaches global memory: it is
// fused into the attention kernel as fp16 shared-memory tiles that feed
// tcgen05.mma directly.
//
// CTA = (tile of QPC = 128 / G queries, KV head); its 128 MMA rows are the
// (query, head) pairs r = i * G + j of the G query heads that share the KV
// head, so every dequantized K/V tile is reused by all of them.  Warp roles:
//   warp 0      TMEM allocation; lane 0 issues every tcgen05.mma:
//                 S_j  = Q  K_j^T   (A = Q smem, B = K_j smem, both K-major)
//                 O   += P_j V_j    (A = P_j in TMEM, B = V_j smem, MN-major)
//   warps 1-8   dequantize 64-position K/V tiles from the pool (page-table
//               lookup, 4-bit codes -> fp16 via an e4m3 convert, then
//               x = code * scale + bias with one fused multiply-add) into
//               double-buffered 128B-swizzled tiles; each thread owns one
//               position's 32 contiguous code bytes per 64-wide block, loads
//               run two tiles ahead, and the 8 lanes of a quarter-warp store
//               8 different positions (distinct swizzled chunks, no bank
//               conflicts);
//   warps 9-12  one thread per row: online softmax on S (tcgen05.ld), P back
//               to TMEM as fp16 (tcgen05.st); the running maximum is moved
//               only when it grows by more than 2^8, and then O is rescaled
//               in TMEM; finally O / l -> bf16 output.
// Within every 8 consecutive d the tiles store elements in the order
// 0,2,4,6,1,3,5,7 (what the two-nibble convert produces); Q uses the same
// order, so Q K^T is unchanged, and the epilogue undoes it for O.  Q is
// stored pre-multiplied by softmax_scale * log2(e), so S arrives in the log2
// domain.
#include <cmath>

#include "tc.cuh"

namespace jfkv {

constexpr int PF_BM = 128;   // MMA rows per CTA
constexpr int PF_BN = 64;    // positions per K/V tile
constexpr int PF_DQ_WARPS = 8;
constexpr int PF_SM_WARPS = 4;
constexpr int PF_THREADS = 32 * (1 + PF_DQ_WARPS + PF_SM_WARPS);
constexpr float PF_TAU = 8.f;   // log2 headroom before the running max moves

struct PrefillArgs {
  const uint8_t* pool;
  int64_t num_pages;
  int64_t page_bytes;
  int64_t codes_region;
  int64_t sb_base;
  int64_t sb_region;
  int32_t P, Hkv, Hq, G, QPC;
  const int32_t* pt;
  const uint16_t* q;
  uint16_t* out;
  int32_t q_start, C, causal;
  float scale_log2;
  int32_t* status;
  int32_t n_qtiles;
};

template <int D>
struct PfSmem {
  static constexpr int Q_BYTES = PF_BM * D * 2;
  static constexpr int T_BYTES = PF_BN * D * 2;
  static constexpr int OFF_Q = 0;
  static constexpr int OFF_K = Q_BYTES;
  static constexpr int OFF_V = OFF_K + 2 * T_BYTES;
  static constexpr int OFF_BAR = OFF_V + 2 * T_BYTES;
  static constexpr int TOTAL = 1024 + OFF_BAR + 128;
};

__device__ __forceinline__ uint32_t cvt_e4m3x2_f16x2(uint32_t two_bytes) {
  uint32_t r;
  asm("{\n\t.reg .b16 t;\n\tcvt.u16.u32 t, %1;\n\tcvt.rn.f16x2.e4m3x2 %0, t;\n\t}\n"
      : "=r"(r) : "r"(two_bytes));
  return r;
}

__device__ __forceinline__ uint32_t hmul2(uint32_t a, uint32_t b) {
  uint32_t r;
  asm("mul.rn.f16x2 %0, %1, %2;\n" : "=r"(r) : "r"(a), "r"(b));
  return r;
}

__device__ __forceinline__ uint32_t hfma2(uint32_t a, uint32_t b, uint32_t c) {
  uint32_t r;
  asm("fma.rn.f16x2 %0, %1, %2, %3;\n" : "=r"(r) : "r"(a), "r"(b), "r"(c));
  return r;
}

// 8 packed 4-bit codes (d0..d7) -> 8 fp16 values code*scale + bias in the
// order d0,d2,d4,d6,d1,d3,d5,d7.  A byte 0..15 read as e4m3 is exactly
// code * 2^-9 (subnormal for < 8, exponent 1 for >= 8), so the convert plus an
// exact *512 yields the integer code; the fma rounds once.
__device__ __forceinline__ uint4 dequant8(uint32_t w, uint32_t s2, uint32_t b2) {
  const uint32_t lo = w & 0x0F0F0F0Fu;
  const uint32_t hi = (w >> 4) & 0x0F0F0F0Fu;
  const uint32_t k512 = 0x60006000u;   // (512, 512) in f16
  uint4 o;
  o.x = hfma2(hmul2(cvt_e4m3x2_f16x2(lo & 0xFFFFu), k512), s2, b2);
  o.y = hfma2(hmul2(cvt_e4m3x2_f16x2(lo >> 16), k512), s2, b2);
  o.z = hfma2(hmul2(cvt_e4m3x2_f16x2(hi & 0xFFFFu), k512), s2, b2);
  o.w = hfma2(hmul2(cvt_e4m3x2_f16x2(hi >> 16), k512), s2, b2);
  return o;
}

// Same with the *512 folded into the scale (scale * 512 must fit fp16).
__device__ __forceinline__ uint4 dequant8_fast(uint32_t w, uint32_t s512, uint32_t b2) {
  const uint32_t lo = w & 0x0F0F0F0Fu;
  const uint32_t hi = (w >> 4) & 0x0F0F0F0Fu;
  uint4 o;
  o.x = hfma2(cvt_e4m3x2_f16x2(lo & 0xFFFFu), s512, b2);
  o.y = hfma2(cvt_e4m3x2_f16x2(lo >> 16), s512, b2);
  o.z = hfma2(cvt_e4m3x2_f16x2(hi & 0xFFFFu), s512, b2);
  o.w = hfma2(cvt_e4m3x2_f16x2(hi >> 16), s512, b2);
  return o;
}

// bf16 (scale | bias << 16) word -> f16x2 broadcasts of scale (or scale*512
// when that fits fp16: fast = true) and bias
__device__ __forceinline__ void sb_to_h2(uint32_t w, uint32_t& s2, uint32_t& b2, bool& fast) {
  const float s = bf16lo_to_f32(w), b = bf16hi_to_f32(w);
  fast = fabsf(s) <= 120.f;
  const float sc = fast ? s * 512.f : s;
  s2 = pack_f16x2(sc, sc);
  b2 = pack_f16x2(b, b);
}

template <int D>
__global__ void __launch_bounds__(PF_THREADS, 1) prefill_kernel(const PrefillArgs a) {
  using L = PfSmem<D>;
  constexpr int NKB = D / 64;           // 64-wide d blocks
  constexpr int CB = D / 2;
  constexpr int SBB = D / 16;
  constexpr int UPI = (D == 256) ? 2 : 1;   // 16-byte code units per dequant item
  static_assert(PF_BN * NKB * 2 / UPI == 32 * PF_DQ_WARPS, "one item per dequant thread");
  constexpr uint32_t IDQK = tc::idesc_f16_f32(PF_BM, PF_BN, 0, 0);
  constexpr uint32_t IDPV = tc::idesc_f16_f32(PF_BM, D, 0, 1);

  extern __shared__ uint8_t smraw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smraw) + 1023) &
                                           ~static_cast<uintptr_t>(1023));
  uint8_t* sQ = sm + L::OFF_Q;
  uint8_t* sK = sm + L::OFF_K;
  uint8_t* sV = sm + L::OFF_V;
  uint64_t* bars = reinterpret_cast<uint64_t*>(sm + L::OFF_BAR);
  uint64_t* kv_full = bars + 0;
  uint64_t* s_full = bars + 2;
  uint64_t* p_full = bars + 4;
  uint64_t* pv_done = bars + 6;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 8);
  uint32_t* qmax_slot = tmem_slot + 1;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int qt = a.n_qtiles - 1 - (int)blockIdx.x;   // latest (longest) query tiles first
  const int kvh = blockIdx.y;
  const int q0 = qt * a.QPC;
  const int nq = min(a.QPC, a.C - q0);
  const int rows = nq * a.G;
  const int total = a.q_start + a.C;
  const int kmax = a.causal ? a.q_start + q0 + nq : total;
  const int ntiles = (kmax + PF_BN - 1) / PF_BN;

  if (warp == 0) tc::alloc(tmem_slot, 512);
  if (threadIdx.x == 0) {
    for (int i = 0; i < 2; ++i) {
      mbar_init(&kv_full[i], PF_DQ_WARPS);
      mbar_init(&s_full[i], 1);
      mbar_init(&p_full[i], PF_SM_WARPS);
      mbar_init(&pv_done[i], 1);
    }
    *qmax_slot = 0;
    fence_barrier_init();
  }
  __syncthreads();

  // ---- Q tile -> fp16, 128B-swizzled K-major, d order 0,2,4,6,1,3,5,7 ------
  const int ltid = (int)threadIdx.x - 32;          // 0..383 for warps 1..12
  constexpr int QTHREADS = PF_THREADS - 32;
  constexpr int QITEMS = PF_BM * (D / 8);
  auto q_src = [&](int r) -> const uint16_t* {
    return a.q + ((int64_t)(q0 + r / a.G) * a.Hq + kvh * a.G + r % a.G) * D;
  };
  if (warp > 0) {
    float mx = 0.f;
    for (int it = ltid; it < QITEMS; it += QTHREADS) {
      const int r = it / (D / 8), c8 = it % (D / 8);
      if (r < rows) {
        const uint4 w = *reinterpret_cast<const uint4*>(q_src(r) + 8 * c8);
        const uint32_t ws[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
        for (int i = 0; i < 4; ++i)
          mx = fmaxf(mx, fmaxf(fabsf(bf16lo_to_f32(ws[i])), fabsf(bf16hi_to_f32(ws[i]))));
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    if (lane == 0) atomicMax(qmax_slot, __float_as_uint(mx));
  }
  __syncthreads();
  // Q enters fp16 pre-multiplied by softmax_scale * log2(e); a power of two
  // keeps it below 2^14 and is multiplied back onto S.
  const float qmax = __uint_as_float(*qmax_slot) * a.scale_log2;
  const int qe = (qmax >= 16384.f) ? (ilogbf(qmax) - 13) : 0;
  if (warp > 0) {
    const float qs = ldexpf(a.scale_log2, -qe);
    for (int it = ltid; it < QITEMS; it += QTHREADS) {
      const int r = it / (D / 8), c8 = it % (D / 8);
      uint4 o = make_uint4(0, 0, 0, 0);
      if (r < rows) {
        const uint4 w = *reinterpret_cast<const uint4*>(q_src(r) + 8 * c8);
        float e[8];
        e[0] = bf16lo_to_f32(w.x) * qs; e[1] = bf16hi_to_f32(w.x) * qs;
        e[2] = bf16lo_to_f32(w.y) * qs; e[3] = bf16hi_to_f32(w.y) * qs;
        e[4] = bf16lo_to_f32(w.z) * qs; e[5] = bf16hi_to_f32(w.z) * qs;
        e[6] = bf16lo_to_f32(w.w) * qs; e[7] = bf16hi_to_f32(w.w) * qs;
        o.x = pack_f16x2(e[0], e[2]);
        o.y = pack_f16x2(e[4], e[6]);
        o.z = pack_f16x2(e[1], e[3]);
        o.w = pack_f16x2(e[5], e[7]);
      }
      const int kb = c8 / 8, cc = c8 % 8;
      *reinterpret_cast<uint4*>(sQ + kb * (PF_BM * 128) + r * 128 + ((cc ^ (r & 7)) << 4)) = o;
    }
    fence_proxy_async_smem();
  }
  tc::fence_before();
  __syncthreads();
  tc::fence_after();
  const uint32_t tbase = *tmem_slot;
  const uint32_t tO = tbase;
  const uint32_t tS = tbase + D;
  const uint32_t tP = tbase + D + 2 * PF_BN;

  if (warp == 0) {
    // ================= MMA issuer =================
    if (lane == 0) {
      const uint32_t qaddr = smem_u32(sQ), kaddr = smem_u32(sK), vaddr = smem_u32(sV);
      bool ok = true;
      auto pv = [&](int j) {
        const int b = j & 1;
        if (!mbar_wait_bounded(&p_full[b], (j >> 1) & 1)) { ok = false; return; }
        tc::fence_after();
#pragma unroll
        for (int k = 0; k < PF_BN / 16; ++k)
          tc::mma_ts(tO, tP + b * (PF_BN / 2) + 8 * k,
                     tc::sdesc_sw128(vaddr + b * L::T_BYTES + k * 2048, PF_BN * 128, 1024), IDPV,
                     (j > 0 || k > 0) ? 1u : 0u);
        tc::commit(&pv_done[b]);
      };
      for (int j = 0; j < ntiles && ok; ++j) {
        const int b = j & 1;
        if (!mbar_wait_bounded(&kv_full[b], (j >> 1) & 1)) { ok = false; break; }
        tc::fence_after();
#pragma unroll
        for (int kb = 0; kb < NKB; ++kb)
#pragma unroll
          for (int k = 0; k < 4; ++k)
            tc::mma_ss(tS + b * PF_BN,
                       tc::sdesc_sw128(qaddr + kb * (PF_BM * 128) + 32 * k, 16, 1024),
                       tc::sdesc_sw128(kaddr + b * L::T_BYTES + kb * (PF_BN * 128) + 32 * k, 16,
                                       1024),
                       IDQK, (kb | k) ? 1u : 0u);
        tc::commit(&s_full[b]);
        if (j >= 1) pv(j - 1);
      }
      if (ok) pv(ntiles - 1);
      if (!ok) flag_error(a.status, JF_DEV_ERR_TIMEOUT);
    }
    __syncwarp();
  } else if (warp <= PF_DQ_WARPS) {
    // ================= dequantization =================
    // item = (position t, 64-wide block kb[, half u]): UPI 16-byte code units
    const int dt = (int)threadIdx.x - 32;   // 0 .. 32*PF_DQ_WARPS-1
    const int t = dt % PF_BN;
    const int rest = dt / PF_BN;
    const int kb = (UPI == 2) ? rest : rest >> 1;
    const int u0 = (UPI == 2) ? 0 : (rest & 1);
    struct Tile {
      uint4 k[UPI], v[UPI];
      uint32_t ks, vs;
      bool valid;
    };
    auto load_tile = [&](int j, Tile& x) {
      const int key0 = j * PF_BN;
      const int page = __ldg(a.pt + key0 / a.P);
      const bool pok = page >= 0 && page < a.num_pages;
      if (!pok && dt == 0) flag_error(a.status, JF_DEV_ERR_PAGE_ID);
      x.valid = pok && (key0 + t < kmax);
      if (x.valid) {
        const uint8_t* base = a.pool + (int64_t)page * a.page_bytes;
        const int64_t row = (int64_t)kvh * a.P + key0 % a.P + t;
        const uint8_t* kp = base + row * CB + kb * 32 + u0 * 16;
#pragma unroll
        for (int u = 0; u < UPI; ++u) {
          x.k[u] = __ldg(reinterpret_cast<const uint4*>(kp + 16 * u));
          x.v[u] = __ldg(reinterpret_cast<const uint4*>(kp + a.codes_region + 16 * u));
        }
        const uint8_t* sp = base + a.sb_base + row * SBB + kb * 4;
        x.ks = __ldg(reinterpret_cast<const uint32_t*>(sp));
        x.vs = __ldg(reinterpret_cast<const uint32_t*>(sp + a.sb_region));
      }
    };
    auto store_half = [&](uint8_t* tile, const uint4 (&codes)[UPI], uint32_t sbw, bool valid) {
      uint32_t s2, b2;
      bool fast;
      sb_to_h2(sbw, s2, b2, fast);
      uint4 o[UPI][4];
#pragma unroll
      for (int u = 0; u < UPI; ++u) {
        const uint32_t cw[4] = {codes[u].x, codes[u].y, codes[u].z, codes[u].w};
        if (fast) {
#pragma unroll
          for (int w = 0; w < 4; ++w) o[u][w] = dequant8_fast(cw[w], s2, b2);
        } else {
#pragma unroll
          for (int w = 0; w < 4; ++w) o[u][w] = dequant8(cw[w], s2, b2);
        }
      }
#pragma unroll
      for (int u = 0; u < UPI; ++u)
#pragma unroll
        for (int w = 0; w < 4; ++w) {
          const int cc = (u0 + u) * 4 + w;
          *reinterpret_cast<uint4*>(tile + kb * (PF_BN * 128) + t * 128 + ((cc ^ (t & 7)) << 4)) =
              valid ? o[u][w] : make_uint4(0, 0, 0, 0);
        }
    };
    Tile cur, nxt, nn;
    load_tile(0, cur);
    if (ntiles > 1) load_tile(1, nxt);
    bool ok = true;
    for (int j = 0; j < ntiles; ++j) {
      if (j + 2 < ntiles) load_tile(j + 2, nn);
      if (j >= 2 && !mbar_wait_bounded(&pv_done[j & 1], ((j - 2) >> 1) & 1)) { ok = false; break; }
      store_half(sK + (j & 1) * L::T_BYTES, cur.k, cur.ks, cur.valid);
      store_half(sV + (j & 1) * L::T_BYTES, cur.v, cur.vs, cur.valid);
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) mbar_arrive(&kv_full[j & 1]);
      cur = nxt;
      nxt = nn;
    }
    if (!ok && dt == 0) flag_error(a.status, JF_DEV_ERR_TIMEOUT);
  } else {
    // ================= softmax + epilogue =================
    const int quarter = warp & 3;                 // TMEM lanes this warp may access
    const int r = quarter * 32 + lane;
    const bool row_ok = r < rows;
    const int qi = row_ok ? r / a.G : 0;
    const int limit = !row_ok ? -1 : (a.causal ? a.q_start + q0 + qi : total - 1);
    const uint32_t lane_off = (uint32_t)(quarter * 32) << 16;
    const float smul = ldexpf(1.f, qe);   // S = (scaled Q) K^T * 2^qe
    float m_ref = -INFINITY, l = 0.f;
    bool ok = true;
    for (int j = 0; j < ntiles; ++j) {
      const int b = j & 1;
      if (!mbar_wait_bounded(&s_full[b], (j >> 1) & 1)) { ok = false; break; }
      tc::fence_after();
      uint32_t s0[32], s1[32];
      tc::ld32(tS + b * PF_BN + lane_off, s0);
      tc::ld32(tS + b * PF_BN + 32 + lane_off, s1);
      tc::wait_ld();
      const int key0 = j * PF_BN;
      float x[PF_BN];
      float mt = -INFINITY;
      if (key0 + PF_BN - 1 <= limit) {       // every position of the tile visible
#pragma unroll
        for (int c = 0; c < 32; ++c) {
          x[c] = __uint_as_float(s0[c]) * smul;
          x[c + 32] = __uint_as_float(s1[c]) * smul;
          mt = fmaxf(mt, fmaxf(x[c], x[c + 32]));
        }
      } else {
#pragma unroll
        for (int c = 0; c < 32; ++c) {
          x[c] = (key0 + c <= limit) ? __uint_as_float(s0[c]) * smul : -INFINITY;
          x[c + 32] = (key0 + c + 32 <= limit) ? __uint_as_float(s1[c]) * smul : -INFINITY;
          mt = fmaxf(mt, fmaxf(x[c], x[c + 32]));
        }
      }
      const bool need = mt > m_ref + PF_TAU;
      if (__any_sync(0xffffffffu, need)) {
        const float nref = need ? mt : m_ref;
        const float f = (need && m_ref != -INFINITY) ? fast_exp2(m_ref - nref) : 1.f;
        if (j > 0) {
          if (!mbar_wait_bounded(&pv_done[(j - 1) & 1], ((j - 1) >> 1) & 1)) { ok = false; break; }
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
#pragma unroll
      for (int c = 0; c < 32; ++c) {
        const float p0 = (x[2 * c] == -INFINITY) ? 0.f : fast_exp2(x[2 * c] - m_ref);
        const float p1 = (x[2 * c + 1] == -INFINITY) ? 0.f : fast_exp2(x[2 * c + 1] - m_ref);
        l += p0 + p1;
        p[c] = pack_f16x2(p0, p1);
      }
      tc::st32(tP + b * (PF_BN / 2) + lane_off, p);
      tc::wait_st();
      tc::fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&p_full[b]);
    }
    // epilogue: O / l -> bf16, undoing the d order 0,2,4,6,1,3,5,7
    if (ok && mbar_wait_bounded(&pv_done[(ntiles - 1) & 1], ((ntiles - 1) >> 1) & 1)) {
      tc::fence_after();
      const float inv = l > 0.f ? 1.f / l : 0.f;
      uint16_t* orow = a.out + ((int64_t)(q0 + qi) * a.Hq + kvh * a.G + r % a.G) * D;
#pragma unroll 1
      for (int c0 = 0; c0 < D; c0 += 32) {
        uint32_t o[32];
        tc::ld32(tO + c0 + lane_off, o);
        tc::wait_ld();
        if (row_ok) {
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            const float* v = reinterpret_cast<const float*>(o + 8 * k);
            uint4 w;
            w.x = (uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(v[0] * inv)) |
                  ((uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(v[4] * inv)) << 16);
            w.y = (uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(v[1] * inv)) |
                  ((uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(v[5] * inv)) << 16);
            w.z = (uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(v[2] * inv)) |
                  ((uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(v[6] * inv)) << 16);
            w.w = (uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(v[3] * inv)) |
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

  tc::fence_before();
  __syncthreads();
  if (warp == 0) {
    tc::fence_after();
    tc::dealloc(tbase, 512);
  }
}

int launch_prefill(const Geom& g, const jf_kv_pool& pool, const CUtensorMap&,
                   const int32_t* page_table_row, const void* q, int32_t q_start,
                   int32_t chunk_len, int32_t Hq, float softmax_scale, int32_t causal, void* out,
                   void* workspace, cudaStream_t stream) {
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
  a.pt = page_table_row;
  a.q = static_cast<const uint16_t*>(q);
  a.out = static_cast<uint16_t*>(out);
  a.q_start = q_start;
  a.C = chunk_len;
  a.causal = causal ? 1 : 0;
  a.scale_log2 = softmax_scale * 1.4426950408889634f;
  a.status = static_cast<int32_t*>(workspace);
  a.n_qtiles = (chunk_len + a.QPC - 1) / a.QPC;
  if (g.Hkv > 65535) return JF_ERR_UNSUPPORTED;
  dim3 grid((unsigned)a.n_qtiles, (unsigned)g.Hkv);
  if (g.D == 256) {
    static bool attr = false;
    if (!attr) {
      if (cudaFuncSetAttribute(prefill_kernel<256>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               PfSmem<256>::TOTAL) != cudaSuccess)
        return JF_ERR_CUDA;
      attr = true;
    }
    prefill_kernel<256><<<grid, PF_THREADS, PfSmem<256>::TOTAL, stream>>>(a);
  } else {
    static bool attr = false;
    if (!attr) {
      if (cudaFuncSetAttribute(prefill_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               PfSmem<128>::TOTAL) != cudaSuccess)
        return JF_ERR_CUDA;
      attr = true;
    }
    prefill_kernel<128><<<grid, PF_THREADS, PfSmem<128>::TOTAL, stream>>>(a);
  }
  return cudaGetLastError() == cudaSuccess ? JF_OK : JF_ERR_CUDA;
}

}  // namespace jfkv
