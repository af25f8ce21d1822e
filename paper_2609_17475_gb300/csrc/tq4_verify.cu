// Packed verifier over TQ4 pages (Sec. 3.1: 2-4 proposed tokens verified in
// one pass over the pages; Eq. 4: K and V rebuilt from centroid indices and a
// norm in the rotated domain; App. A.1: causal among the query tokens).
//
// The warp-pair scheme of the affine verifier (verify.cu) on the TQ4 format:
// a CTA holds up to NTC n-tiles of 8 (token, head) rows of one KV head, and
// the two warps of a pair take the same 32-position chunk, each for half of
// the head dimension.  A warp looks up the centroids of its half's K indices
// once (the lane-replicated table of the TQ4 decode kernel, one code byte ->
// an f16x2 pair) and multiplies them with every n-tile's rotated queries; the
// partners swap these partial dot products through shared memory (one named
// barrier per chunk) and both scale the sums by the position's norm, so both
// run the same online softmax; each warp then looks up its half's V
// centroids once and accumulates the rotated-domain O of every n-tile.  At
// the end the pairs are combined and each row is rotated back,
// o = S_V H (sum_t p_t rho_t c[z_t]) / sqrt(D), and written as output or as
// a split partial for the decode's merge kernel.
#include <cmath>
#include <cfloat>

#include "decode.cuh"
#include "decode_frag.cuh"
#include "pair_sync.cuh"
#include "tq4.cuh"

namespace jfkv {
namespace {

// warps per CTA (one CTA per SM) and stages per pair: two n-tiles fit 168
// registers with 12 warps; three take more and run 8
template <int NTC>
constexpr int tv_warps() { return NTC <= 2 ? 12 : 8; }
template <int NTC>
constexpr int tv_stages() { return NTC <= 2 ? 2 : 3; }

template <int D, int NTC>
struct TvSmem {
  static constexpr int NW = tv_warps<NTC>();
  static constexpr int VST = tv_stages<NTC>();
  static constexpr int NP = NW / 2;
  static constexpr int CB = D / 2;
  static constexpr int NCK = D / 32;              // 16-byte code chunks per vector
  static constexpr int CODE_BUF = DTOK * CB;      // one chunk's K (or V) indices
  static constexpr int NORM_BUF = DTOK * 2;       // one chunk's K (or V) norms
  static constexpr int XK = NTC * 2;              // float4 exchange slots per lane
  // pair region: VST x (K, V indices) | VST x (K, V norms) | exchange
  static constexpr int RING_CODES = VST * 2 * CODE_BUF;
  static constexpr int RING_NORM = VST * 2 * NORM_BUF;
  static constexpr int XBUF = 2 * 2 * XK * 32 * 16;
  static constexpr int PAIR = (RING_CODES + RING_NORM + XBUF + 1023) / 1024 * 1024;
  static constexpr int LUT_OFF = NP * PAIR;
  static constexpr int LUT_BYTES = 256 * 32 * 4;
  static constexpr int QF_OFF = LUT_OFF + LUT_BYTES;
  static constexpr int QF_BYTES = NTC * NCK * 32 * 16;   // [n-tile][chunk][lane] uint4
  static constexpr int BAR_OFF = QF_OFF + QF_BYTES;
  static constexpr int BAR_BYTES = NP * VST * 8;
  static constexpr int MISC_OFF = BAR_OFF + BAR_BYTES;
  // plan (4 ints) | per-warp |q'| maxima (NW) | per-row (M, L) (NTC * 8 x 2)
  static constexpr int MISC_BYTES = 16 + NW * 4 + NTC * 8 * 8;
  static constexpr int TOTAL = MISC_OFF + MISC_BYTES;
  static constexpr uint32_t STAGE_TX = 2 * CODE_BUF + 2 * NORM_BUF;
  static constexpr int SROW = D + 4;
  static constexpr int ML_OFF = NTC * 8 * SROW * 4;
  static_assert(ML_OFF + NTC * 8 * 2 * 4 <= PAIR, "combine rows fit a pair region");
  // rotated queries (before the first copy) live in the pair regions, the
  // combined rotated-domain rows (after the loop) in the centroid table
  static_assert(NTC * 8 * D * 4 <= NP * PAIR && NTC * 8 * D * 4 <= LUT_BYTES, "row buffers");
  static_assert(TOTAL <= 227 * 1024, "shared memory per CTA");
};

__device__ __forceinline__ uint32_t tv_lds32(uint32_t addr) {
  uint32_t v;
  asm("ld.shared.b32 %0, [%1];\n" : "=r"(v) : "r"(addr));
  return v;
}

// centroid pair of code byte k of w (f16x2: low nibble's centroid in the low half)
__device__ __forceinline__ uint32_t tv_lut(uint32_t lut_lane, uint32_t w, uint32_t k) {
  return tv_lds32(lut_lane + __byte_perm(w, 0u, 0x4440u + k) * 128u);
}

__device__ __forceinline__ float tv_h2f(const uint8_t* p) {
  return __half2float(__ushort_as_half(*reinterpret_cast<const uint16_t*>(p)));
}

// rotated-domain state of one n-tile for this warp's half of d; thread (r, c)
// owns columns 2c, 2c+1 and the d-rows {64 g + 4 r + e, 64 g + 32 + 4 r + e}
template <int NGH>
struct TvState {
  float m0, m1, l0, l1;
  float O[NGH][4][4];
  __device__ __forceinline__ void init() {
    m0 = m1 = -INFINITY;
    l0 = l1 = 0.f;
#pragma unroll
    for (int g = 0; g < NGH; ++g)
#pragma unroll
      for (int e = 0; e < 4; ++e)
#pragma unroll
        for (int i = 0; i < 4; ++i) O[g][e][i] = 0.f;
  }
};

// Partial dot products <q', c[z_t]> over this warp's 64-element blocks
// g = h NGH .. h NGH + NGH - 1, for every n-tile.
template <int D, int NTC>
__device__ __forceinline__ void tv_qk(float (&acc)[NTC][2][4], const uint4* qf, uint32_t kc,
                                      uint32_t lut_lane, const uint32_t (&koff)[D / 128]) {
  constexpr int NGH = D / 128, NCK = D / 32, CB = D / 2;
#pragma unroll
  for (int j = 0; j < 2; ++j) {
#pragma unroll
    for (int t = 0; t < NTC; ++t) acc[t][j][0] = acc[t][j][1] = acc[t][j][2] = acc[t][j][3] = 0.f;
#pragma unroll
    for (int gg = 0; gg < NGH; ++gg) {
      uint32_t w0, w1, w2, w3;
      ldsm_x4(w0, w1, w2, w3, kc + koff[gg] + 16 * j * CB);
      // w0/w1: positions r / r+8, 16-byte chunk 2g; w2/w3: chunk 2g+1
      uint32_t A[2][2][4];   // [chunk][k-step][fragment register]
#pragma unroll
      for (int s = 0; s < 2; ++s) {
        A[0][s][0] = tv_lut(lut_lane, w0, 2 * s);
        A[0][s][1] = tv_lut(lut_lane, w1, 2 * s);
        A[0][s][2] = tv_lut(lut_lane, w0, 2 * s + 1);
        A[0][s][3] = tv_lut(lut_lane, w1, 2 * s + 1);
        A[1][s][0] = tv_lut(lut_lane, w2, 2 * s);
        A[1][s][1] = tv_lut(lut_lane, w3, 2 * s);
        A[1][s][2] = tv_lut(lut_lane, w2, 2 * s + 1);
        A[1][s][3] = tv_lut(lut_lane, w3, 2 * s + 1);
      }
#pragma unroll
      for (int t = 0; t < NTC; ++t) {
#pragma unroll
        for (int hc = 0; hc < 2; ++hc) {
          const uint4 q = qf[(t * NCK + 2 * gg + hc) * 32];
          mma_f16(acc[t][j], A[hc][0][0], A[hc][0][1], A[hc][0][2], A[hc][0][3], q.x, q.y);
          mma_f16(acc[t][j], A[hc][1][0], A[hc][1][1], A[hc][1][2], A[hc][1][3], q.z, q.w);
        }
      }
    }
  }
}

// Online softmax of every n-tile (identical in both warps of a pair) and PV
// over this warp's half of d.  FULL: every position of the chunk is valid and
// visible to every row, so no mask is built (a separate instance: the masked
// body on every chunk measured 16-21 % slower).  Otherwise positions >= nvalid
// hold no data and column 2c (2c+1) of n-tile t sees only positions < nv0[t]
// (nv1[t]).
template <int D, int NTC, bool FULL>
__device__ __forceinline__ void tv_softmax_pv(TvState<D / 128> (&st)[NTC], float (&sc)[NTC][2][4],
                                              uint32_t vc, const uint8_t* vn, uint32_t lut_lane,
                                              const uint32_t (&koff)[D / 128], int r, int nvalid,
                                              const int (&nv0)[NTC], const int (&nv1)[NTC]) {
  constexpr int NGH = D / 128, CB = D / 2;
  constexpr float NEG_INF = -INFINITY;
  float p[NTC][2][4];
#pragma unroll
  for (int t = 0; t < NTC; ++t) {
    if constexpr (!FULL) {
#pragma unroll
      for (int j = 0; j < 2; ++j) {
        const int ta = 16 * j + r, tb = ta + 8;
        if (ta >= nv0[t]) sc[t][j][0] = NEG_INF;
        if (ta >= nv1[t]) sc[t][j][1] = NEG_INF;
        if (tb >= nv0[t]) sc[t][j][2] = NEG_INF;
        if (tb >= nv1[t]) sc[t][j][3] = NEG_INF;
      }
    }
    float mx0 = fmaxf(fmaxf(sc[t][0][0], sc[t][0][2]), fmaxf(sc[t][1][0], sc[t][1][2]));
    float mx1 = fmaxf(fmaxf(sc[t][0][1], sc[t][0][3]), fmaxf(sc[t][1][1], sc[t][1][3]));
    TvState<NGH>& s = st[t];
    if (__any_sync(0xffffffffu, (mx0 > s.m0 + DTAU) || (mx1 > s.m1 + DTAU))) {
#pragma unroll
      for (int o = 4; o < 32; o <<= 1) {
        mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, o));
        mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, o));
      }
      const float nm0 = fmaxf(s.m0, mx0), nm1 = fmaxf(s.m1, mx1);
      const float f0 = (nm0 > s.m0) ? fast_exp2(s.m0 - nm0) : 1.f;
      const float f1 = (nm1 > s.m1) ? fast_exp2(s.m1 - nm1) : 1.f;
      const f2 ff = mk2(f0, f1);
#pragma unroll
      for (int g = 0; g < NGH; ++g)
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          un2(mul2(mk2(s.O[g][e][0], s.O[g][e][1]), ff), s.O[g][e][0], s.O[g][e][1]);
          un2(mul2(mk2(s.O[g][e][2], s.O[g][e][3]), ff), s.O[g][e][2], s.O[g][e][3]);
        }
      un2(mul2(mk2(s.l0, s.l1), ff), s.l0, s.l1);
      s.m0 = nm0;
      s.m1 = nm1;
    }
#pragma unroll
    for (int j = 0; j < 2; ++j) {
      if constexpr (FULL) {
        const f2 m2 = mk2(s.m0, s.m1);
        float d0, d1, d2, d3;
        un2(sub2(mk2(sc[t][j][0], sc[t][j][1]), m2), d0, d1);
        un2(sub2(mk2(sc[t][j][2], sc[t][j][3]), m2), d2, d3);
        p[t][j][0] = fast_exp2(d0);
        p[t][j][1] = fast_exp2(d1);
        p[t][j][2] = fast_exp2(d2);
        p[t][j][3] = fast_exp2(d3);
      } else {
        p[t][j][0] = (sc[t][j][0] == NEG_INF) ? 0.f : fast_exp2(sc[t][j][0] - s.m0);
        p[t][j][1] = (sc[t][j][1] == NEG_INF) ? 0.f : fast_exp2(sc[t][j][1] - s.m1);
        p[t][j][2] = (sc[t][j][2] == NEG_INF) ? 0.f : fast_exp2(sc[t][j][2] - s.m0);
        p[t][j][3] = (sc[t][j][3] == NEG_INF) ? 0.f : fast_exp2(sc[t][j][3] - s.m1);
      }
      un2(add2(mk2(s.l0, s.l1), add2(mk2(p[t][j][0], p[t][j][1]), mk2(p[t][j][2], p[t][j][3]))),
          s.l0, s.l1);
    }
  }

#pragma unroll
  for (int j = 0; j < 2; ++j) {
    const int ta = 16 * j + r, tb = ta + 8;
    // B = p_t rho_t 2^-8 (the 2^8 comes back in the inverse rotation)
    const float wa = (FULL || ta < nvalid) ? tv_h2f(vn + 2 * ta) * 0.00390625f : 0.f;
    const float wb = (FULL || tb < nvalid) ? tv_h2f(vn + 2 * tb) * 0.00390625f : 0.f;
    uint32_t bo[NTC][2];
#pragma unroll
    for (int t = 0; t < NTC; ++t) {
      bo[t][0] = movm_t(pack_f16x2(wa * p[t][j][0], wa * p[t][j][1]));
      bo[t][1] = movm_t(pack_f16x2(wb * p[t][j][2], wb * p[t][j][3]));
    }
#pragma unroll
    for (int gg = 0; gg < NGH; ++gg) {
      uint32_t v0, v1, v2, v3;
      ldsm_x4_t(v0, v1, v2, v3, vc + koff[gg] + 16 * j * CB);
      // v: bytes 0,1 = position 2c (d 4r..4r+3), bytes 2,3 = position 2c+1;
      // v0/v2: positions 0-7 of the tile, chunks 2g / 2g+1; v1/v3: positions 8-15
      const uint32_t L00 = tv_lut(lut_lane, v0, 0), L01 = tv_lut(lut_lane, v0, 1),
                     L02 = tv_lut(lut_lane, v0, 2), L03 = tv_lut(lut_lane, v0, 3);
      const uint32_t L10 = tv_lut(lut_lane, v1, 0), L11 = tv_lut(lut_lane, v1, 1),
                     L12 = tv_lut(lut_lane, v1, 2), L13 = tv_lut(lut_lane, v1, 3);
      const uint32_t L20 = tv_lut(lut_lane, v2, 0), L21 = tv_lut(lut_lane, v2, 1),
                     L22 = tv_lut(lut_lane, v2, 2), L23 = tv_lut(lut_lane, v2, 3);
      const uint32_t L30 = tv_lut(lut_lane, v3, 0), L31 = tv_lut(lut_lane, v3, 1),
                     L32 = tv_lut(lut_lane, v3, 2), L33 = tv_lut(lut_lane, v3, 3);
      // d offset e: (position 2c, position 2c+1) pairs
      uint32_t E[4][4];
      E[0][0] = __byte_perm(L00, L02, 0x5410); E[0][1] = __byte_perm(L20, L22, 0x5410);
      E[0][2] = __byte_perm(L10, L12, 0x5410); E[0][3] = __byte_perm(L30, L32, 0x5410);
      E[1][0] = __byte_perm(L00, L02, 0x7632); E[1][1] = __byte_perm(L20, L22, 0x7632);
      E[1][2] = __byte_perm(L10, L12, 0x7632); E[1][3] = __byte_perm(L30, L32, 0x7632);
      E[2][0] = __byte_perm(L01, L03, 0x5410); E[2][1] = __byte_perm(L21, L23, 0x5410);
      E[2][2] = __byte_perm(L11, L13, 0x5410); E[2][3] = __byte_perm(L31, L33, 0x5410);
      E[3][0] = __byte_perm(L01, L03, 0x7632); E[3][1] = __byte_perm(L21, L23, 0x7632);
      E[3][2] = __byte_perm(L11, L13, 0x7632); E[3][3] = __byte_perm(L31, L33, 0x7632);
#pragma unroll
      for (int t = 0; t < NTC; ++t)
#pragma unroll
        for (int e = 0; e < 4; ++e)
          mma_f16(st[t].O[gg][e], E[e][0], E[e][1], E[e][2], E[e][3], bo[t][0], bo[t][1]);
    }
  }
}

template <int D, int NTC>
__global__ void __launch_bounds__(tv_warps<NTC>() * 32, 1)
tq4_verify_pair_kernel(const __grid_constant__ CUtensorMap tmap, const DecodeArgs a,
                       const Tq4Params prm) {
  using L = TvSmem<D, NTC>;
  constexpr int NW = L::NW, NP = L::NP, VST = L::VST, NCK = L::NCK, SROW = L::SROW;
  constexpr int NGH = D / 128;
  constexpr int E = D / 32;   // elements per lane of a row vector
  constexpr float NEG_INF = -INFINITY;

  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* pairs = smem_raw;
  uint32_t* lut_w = reinterpret_cast<uint32_t*>(smem_raw + L::LUT_OFF);
  uint4* qsm = reinterpret_cast<uint4*>(smem_raw + L::QF_OFF);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem_raw + L::BAR_OFF);
  int* misc = reinterpret_cast<int*>(smem_raw + L::MISC_OFF);
  float* wmax = reinterpret_cast<float*>(misc + 4);          // [NW]
  float* rowml = reinterpret_cast<float*>(misc + 4 + NW);    // [NTC * 8][2]

  const int ncta = (a.NT + NTC - 1) / NTC;
  const int kvh = (int)blockIdx.y / ncta;
  const int nt0 = ((int)blockIdx.y % ncta) * NTC;
  const int GL = a.G * a.L;
  const int rows = min(8 * NTC, GL - 8 * nt0);
  auto row_of = [&](int k) {
    const int gr = 8 * nt0 + k;
    return (gr / a.G) * a.Hq + kvh * a.G + gr % a.G;
  };
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int r = lane >> 2, c = lane & 3;
  const int pr = warp >> 1, h = warp & 1;
  const bool direct = (a.plan_splits == 1 && !a.balanced);
  uint8_t* preg = pairs + pr * L::PAIR;
  uint8_t* rcodes = preg;
  uint8_t* rnorm = preg + L::RING_CODES;
  float4* xbuf = reinterpret_cast<float4*>(preg + L::RING_CODES + L::RING_NORM);
  uint64_t* pbars = bars + pr * VST;

  const bool aligned = (smem_u32(smem_raw) & 1023) == 0;
  if (aligned) {
    if (threadIdx.x == 0) prefetch_tensormap(&tmap);
    if (h == 0 && lane == 0) {
      for (int s = 0; s < VST; ++s) mbar_init(&pbars[s], 1);
      fence_barrier_init();
    }
  }
  // centroid table: word b * 32 + lane = f16x2 (c[b & 15], c[b >> 4])
  for (int i = threadIdx.x; i < 256 * 32; i += blockDim.x) {
    const int bb = i >> 5;
    lut_w[i] = pack_f16x2(prm.c[bb & 15], prm.c[bb >> 4]);
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
    split_plan(ctx, a.plan_splits, nch, cps, nsplit);
  }
  if (split >= nsplit) {
    if (direct && split == 0) {   // empty context: zero output
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
  const int my_n = (n_cta > pr) ? (n_cta - pr + NP - 1) / NP : 0;
  auto chunk_of = [&](int it) { return c_begin + pr + it * NP; };

  // ---- rotated queries q' = H S_K q (unnormalised), fp32 rows in the pair
  // regions; rows past the CTA's last stay zero --------------------------------
  float* qrot = reinterpret_cast<float*>(pairs);   // [NTC * 8][D]
  {
    float mx = 0.f;
    for (int k = warp; k < 8 * NTC; k += NW) {
      float x[E];
#pragma unroll
      for (int e = 0; e < E; ++e) x[e] = 0.f;
      if (k < rows) {
        const uint16_t* src = a.q + ((int64_t)b * a.HqL + row_of(k)) * D + lane * E;
        if constexpr (E == 8) {
          const uint4 w = *reinterpret_cast<const uint4*>(src);
          const uint32_t ws[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            x[2 * i] = bf16lo_to_f32(ws[i]);
            x[2 * i + 1] = bf16hi_to_f32(ws[i]);
          }
        } else {
          const uint2 w = *reinterpret_cast<const uint2*>(src);
          x[0] = bf16lo_to_f32(w.x); x[1] = bf16hi_to_f32(w.x);
          x[2] = bf16lo_to_f32(w.y); x[3] = bf16hi_to_f32(w.y);
        }
        const uint32_t sb = prm.sk[(lane * E) >> 5] >> ((lane * E) & 31);
#pragma unroll
        for (int e = 0; e < E; ++e)
          if ((sb >> e) & 1u) x[e] = -x[e];
      }
      warp_fwht<float, E>(x, lane);
#pragma unroll
      for (int e = 0; e < E; ++e) {
        qrot[k * D + lane * E + e] = x[e];
        mx = fmaxf(mx, fabsf(x[e]));
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    if (lane == 0) wmax[warp] = mx;
  }
  __syncthreads();
  // fp16 range: scale q' by 2^-qe so that max |q'| lies in [2^13, 2^14)
  float qabs = 0.f;
#pragma unroll
  for (int w = 0; w < NW; ++w) qabs = fmaxf(qabs, wmax[w]);
  const float qs0 = a.scale_log2 * rsqrtf((float)D);
  const float qmax = qabs * fabsf(qs0);
  const int qe = (qmax > 0.f && qmax < INFINITY) ? ilogbf(qmax) - 13 : 0;
  const float qmul = qs0 * ldexpf(1.f, -qe);
  const float cS = ldexpf(1.f, qe);
  // B fragments: n-tile t, 16-byte chunk ch, lane (r, c): column r of the
  // tile, d = 32 ch + 8 c + {0,1 | 2,3} (k-step 0) and {4,5 | 6,7} (k-step 1)
  for (int i = threadIdx.x; i < NTC * NCK * 32; i += blockDim.x) {
    const int t = i / (NCK * 32), ch = (i / 32) % NCK, ln = i % 32;
    const float* v = qrot + (8 * t + (ln >> 2)) * D + 32 * ch + 8 * (ln & 3);
    const float4 x0 = *reinterpret_cast<const float4*>(v);
    const float4 x1 = *reinterpret_cast<const float4*>(v + 4);
    qsm[i] = make_uint4(pack_f16x2(x0.x * qmul, x0.y * qmul), pack_f16x2(x0.z * qmul, x0.w * qmul),
                        pack_f16x2(x1.x * qmul, x1.y * qmul), pack_f16x2(x1.z * qmul, x1.w * qmul));
  }
  __syncthreads();   // the rotated rows lie in the rings the copies fill

  // ---- page ids and the pair's TMA producer (as in verify.cu) -------------
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
  const uint64_t l2pol = (ncta > 1) ? l2_evict_normal_policy() : l2_evict_first_policy();
  uint32_t valid = 0;
  int issued = 0;
  auto issue = [&](int it) {
    const int s = it % VST;
    if (it >= 32 && (it & 31) == 0) {
      pg_cur = pg_next;
      pg_next = load_pages((it >> 5) + 1);
    }
    const int page = __shfl_sync(0xffffffffu, pg_cur, it & 31);
    const bool ok = page >= 0 && page < a.num_pages;
    if (h == 0 && lane == 0) {
      const int inp = (chunk_of(it) * DTOK) & (a.P - 1);
      uint64_t* bar = &pbars[s];
      if (!ok) {
        flag_error(a.status, JF_DEV_ERR_PAGE_ID);
        mbar_arrive(bar);
      } else {
        uint8_t* kc = rcodes + s * 2 * L::CODE_BUF;
        uint8_t* kn = rnorm + s * 2 * L::NORM_BUF;
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
    issued = it + 1;
  };
  {
    const int npro = my_n < VST ? my_n : VST;
    for (int it = 0; it < npro; ++it) issue(it);
  }

  const uint4* qf = qsm + h * NGH * 2 * 32 + lane;   // this warp's chunks 2g, 2g+1
  const uint32_t lut_lane = smem_u32(lut_w) + 4u * lane;
  uint32_t koff[NGH];
  {
    const int ld_t = (lane & 7) + 8 * ((lane >> 3) & 1);
    const int ld_ch = lane >> 4;
#pragma unroll
    for (int gg = 0; gg < NGH; ++gg) koff[gg] = swz<L::CB>(ld_t, 2 * (h * NGH + gg) + ld_ch);
  }
  TvState<NGH> st[NTC];
#pragma unroll
  for (int t = 0; t < NTC; ++t) st[t].init();
  const int ctx_all = ctx - a.L + 1;

  const int bar_id = 1 + pr;
  int done = 0;
  bool gave_up = false;
  // two n-tiles: unrolled by 2 (the exchange buffer's parity a constant)
  constexpr int UNR = NTC <= 2 ? 2 : 1;
#pragma unroll UNR
  for (int it = 0; it < my_n; ++it) {
    const int s = it % VST;
    const uint32_t par = (it / VST) & 1;
    const bool got = mbar_wait_bounded(&pbars[s], par);
    const bool ok = (valid >> s) & 1u;
    const int tokbase = chunk_of(it) * DTOK;
    const uint32_t kc = smem_u32(rcodes + s * 2 * L::CODE_BUF);
    const uint8_t* kn = rnorm + s * 2 * L::NORM_BUF;
    float sc[NTC][2][4];
    if (got) {
      tv_qk<D, NTC>(sc, qf, kc, lut_lane, koff);
    } else {
#pragma unroll
      for (int t = 0; t < NTC; ++t)
#pragma unroll
        for (int j = 0; j < 2; ++j) sc[t][j][0] = sc[t][j][1] = sc[t][j][2] = sc[t][j][3] = 0.f;
    }
    float4* xme = xbuf + (((it & 1) * 2 + h) * L::XK) * 32 + lane;
    const float4* xot = xbuf + (((it & 1) * 2 + (h ^ 1)) * L::XK) * 32 + lane;
#pragma unroll
    for (int t = 0; t < NTC; ++t)
#pragma unroll
      for (int j = 0; j < 2; ++j)
        xme[(t * 2 + j) * 32] = make_float4(sc[t][j][0], sc[t][j][1], sc[t][j][2], sc[t][j][3]);
    if (!pair_sync_and(bar_id, got)) {   // both warps leave together
      if (lane == 0 && !got) flag_error(a.status, JF_DEV_ERR_TIMEOUT);
      gave_up = true;
      break;
    }
    done = it + 1;
    // logits: the summed dot products times the position's norm
#pragma unroll
    for (int j = 0; j < 2; ++j) {
      const int ta = 16 * j + r, tb = ta + 8;
      const float na = tv_h2f(kn + 2 * ta) * cS, nb = tv_h2f(kn + 2 * tb) * cS;
#pragma unroll
      for (int t = 0; t < NTC; ++t) {
        const float4 o = xot[(t * 2 + j) * 32];
        sc[t][j][0] = (sc[t][j][0] + o.x) * na;
        sc[t][j][1] = (sc[t][j][1] + o.y) * na;
        sc[t][j][2] = (sc[t][j][2] + o.z) * nb;
        sc[t][j][3] = (sc[t][j][3] + o.w) * nb;
      }
    }
    // the partner is past chunk it - 1: its stage can be refilled
    if (it >= 1 && it - 1 + VST < my_n) {
      if (h == 0) fence_proxy_async_smem();
      issue(it - 1 + VST);
    }
    if (ok && tokbase + DTOK <= ctx_all) {   // every position visible to every row
      const int none[NTC] = {};
      tv_softmax_pv<D, NTC, true>(st, sc, kc + L::CODE_BUF, kn + L::NORM_BUF, lut_lane, koff, r,
                                  DTOK, none, none);
    } else {
      const int nvalid = ok ? min(ctx - tokbase, DTOK) : 0;
      int nv0[NTC], nv1[NTC];
#pragma unroll
      for (int t = 0; t < NTC; ++t) {
        const int col = 8 * (nt0 + t) + 2 * c;
        nv0[t] = ok ? min(min(ctx, ctx_all + col / a.G) - tokbase, nvalid) : 0;
        nv1[t] = ok ? min(min(ctx, ctx_all + (col + 1) / a.G) - tokbase, nvalid) : 0;
      }
      tv_softmax_pv<D, NTC, false>(st, sc, kc + L::CODE_BUF, kn + L::NORM_BUF, lut_lane, koff, r,
                                   nvalid, nv0, nv1);
    }
    __syncwarp();
  }
  if (gave_up) {
    for (int it = done; it < issued; ++it)
      mbar_wait_bounded(&pbars[it % VST], (it / VST) & 1, 1u << 16);
  }
  asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory");

  // ---- per-warp finalize: rotated-domain O rows of this warp's half ---------
  pair_sync(bar_id);   // the partner is done with the ring and the exchange buffers
  float* so = reinterpret_cast<float*>(preg);                 // [NTC * 8][SROW]
  float* sml = reinterpret_cast<float*>(preg + L::ML_OFF);    // [NTC * 8][2]
#pragma unroll
  for (int t = 0; t < NTC; ++t) {
    float l0 = st[t].l0, l1 = st[t].l1;
#pragma unroll
    for (int o = 4; o < 32; o <<= 1) {
      l0 += __shfl_xor_sync(0xffffffffu, l0, o);
      l1 += __shfl_xor_sync(0xffffffffu, l1, o);
    }
#pragma unroll
    for (int gg = 0; gg < NGH; ++gg) {
      const int g = h * NGH + gg;
#pragma unroll
      for (int hf = 0; hf < 2; ++hf)
#pragma unroll
        for (int hh = 0; hh < 2; ++hh) {
          const int k = 8 * t + 2 * c + hh;
          const int i = 2 * hf + hh;
          if (k < rows)
            *reinterpret_cast<float4*>(so + k * SROW + 64 * g + 32 * hf + 4 * r) =
                make_float4(st[t].O[gg][0][i], st[t].O[gg][1][i], st[t].O[gg][2][i],
                            st[t].O[gg][3][i]);
        }
    }
    if (h == 0 && r == 0) {
      const int k = 8 * t + 2 * c;
      sml[k * 2 + 0] = st[t].m0;
      sml[k * 2 + 1] = l0;
      sml[(k + 1) * 2 + 0] = st[t].m1;
      sml[(k + 1) * 2 + 1] = l1;
    }
  }
  __syncthreads();

  // ---- combine the pairs: rotated-domain rows into the (idle) table --------
  float* crow = reinterpret_cast<float*>(lut_w);   // [NTC * 8][D]
  for (int idx = threadIdx.x; idx < rows * (D / 4); idx += blockDim.x) {
    const int k = idx / (D / 4), d = 4 * (idx % (D / 4));
    float mw[NP], lw[NP];
    float M = NEG_INF;
#pragma unroll
    for (int q = 0; q < NP; ++q) {
      const float2 v = *reinterpret_cast<const float2*>(pairs + q * L::PAIR + L::ML_OFF + k * 8);
      mw[q] = v.x;
      lw[q] = v.y;
      M = fmaxf(M, v.x);
    }
    float f[NP];
    float Lsum = 0.f;
#pragma unroll
    for (int q = 0; q < NP; ++q) {
      f[q] = (mw[q] != NEG_INF) ? fast_exp2(mw[q] - M) : 0.f;
      Lsum = fmaf(f[q], lw[q], Lsum);
    }
    const float inv = direct ? (Lsum > 0.f ? 1.f / Lsum : 0.f) : 1.f;
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
    for (int q = 0; q < NP; ++q) {
      const float fw = f[q] * inv;
      if (fw != 0.f) {
        const float4 v = *reinterpret_cast<const float4*>(
            reinterpret_cast<const float*>(pairs + q * L::PAIR) + k * SROW + d);
        acc.x = fmaf(fw, v.x, acc.x);
        acc.y = fmaf(fw, v.y, acc.y);
        acc.z = fmaf(fw, v.z, acc.z);
        acc.w = fmaf(fw, v.w, acc.w);
      }
    }
    *reinterpret_cast<float4*>(crow + k * D + d) = acc;
    if (d == 0) {
      rowml[k * 2 + 0] = M;
      rowml[k * 2 + 1] = Lsum;
    }
  }
  __syncthreads();

  // ---- inverse rotation o = S_V H (2^8 row) / sqrt(D), one warp per row ----
  const float osc = 256.f * rsqrtf((float)D);
  const uint32_t svb = prm.sv[(lane * E) >> 5] >> ((lane * E) & 31);
  for (int k = warp; k < rows; k += NW) {
    float x[E];
#pragma unroll
    for (int e = 0; e < E; ++e) x[e] = crow[k * D + lane * E + e];
    warp_fwht<float, E>(x, lane);
#pragma unroll
    for (int e = 0; e < E; ++e) x[e] *= ((svb >> e) & 1u) ? -osc : osc;
    const int fr = row_of(k);
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
        a.part_ml[row * 2 + 0] = rowml[k * 2 + 0];
        a.part_ml[row * 2 + 1] = rowml[k * 2 + 1];
      }
    }
  }
}

template <int D, int NTC>
int launch_tv(const CUtensorMap& tmap, const DecodeArgs& a, const Tq4Params& prm, int B,
              cudaStream_t stream) {
  using L = TvSmem<D, NTC>;
  const void* kernel = (const void*)tq4_verify_pair_kernel<D, NTC>;
  if (smem_optin(kernel, L::TOTAL) != JF_OK) return JF_ERR_CUDA;
  cudaLaunchAttribute pdl[1];
  pdl[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  pdl[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t cfg = {};
  const int ncta = (a.NT + NTC - 1) / NTC;
  cfg.gridDim = a.balanced ? dim3((unsigned)(a.budget + B), (unsigned)(a.Hkv * ncta), 1u)
                           : dim3((unsigned)a.plan_splits, (unsigned)(a.Hkv * ncta), (unsigned)B);
  cfg.blockDim = dim3(L::NW * 32);
  cfg.dynamicSmemBytes = L::TOTAL;
  cfg.stream = stream;
  cfg.attrs = pdl;
  cfg.numAttrs = 1;
  if (cudaLaunchKernelEx(&cfg, tq4_verify_pair_kernel<D, NTC>, tmap, a, prm) != cudaSuccess)
    return JF_ERR_CUDA;
  if (a.balanced || a.plan_splits > 1) return launch_decode_merge(a, D, B, stream);
  return JF_OK;
}

}  // namespace

// TQ4 packed verifier for NT >= 2 n-tiles per KV head (split launch + merge);
// the caller has filled `a` (plan_splits, balanced and budget included).
int launch_tq4_verify_pairs(const CUtensorMap& tmap, const DecodeArgs& a, const Tq4Params& prm,
                            int D, int B, cudaStream_t stream) {
  const int ntc = a.NT < 3 ? a.NT : 3;
  if (D == 256)
    return ntc == 2 ? launch_tv<256, 2>(tmap, a, prm, B, stream)
                    : launch_tv<256, 3>(tmap, a, prm, B, stream);
  return ntc == 2 ? launch_tv<128, 2>(tmap, a, prm, B, stream)
                  : launch_tv<128, 3>(tmap, a, prm, B, stream);
}

}  // namespace jfkv
