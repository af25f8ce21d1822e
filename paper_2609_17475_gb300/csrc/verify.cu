// Packed verifier over paged 4-bit KV (Sec. 3.1: the 2-4 proposed tokens of a
// speculative step are verified in one pass over the pages; App. A.1: the
// query tokens are causal among themselves).  Split phase only: the split
// partials use the decode's workspace rows and merge kernel.
//
// A KV head carries G * L (token, head) rows, more than the 8 columns of one
// m16n8 MMA tile once G * L > 8.  One CTA holds up to NTC such n-tiles (every
// row of the KV head while G * L <= 8 NTC) and its warps work in pairs on the
// same 32-position chunk, each warp for half of the head dimension (its own
// 64-element groups):
//  * QK^T: a warp unpacks the K codes of its groups once (the fp16-subnormal
//    reading of a nibble, as in the decode kernel) and multiplies each
//    fragment with the query fragments of every n-tile, giving logits partial
//    over its groups (with the per-group affine fix-up);
//  * the two warps swap their partial logits through shared memory (one
//    named barrier per chunk) and add them in the same order, so both hold
//    identical logits and run an identical online softmax;
//  * PV: a warp unpacks the V codes of its groups once and accumulates O for
//    its half of d and every n-tile.
// Each code is therefore unpacked once per chunk, however many rows share it.
// The pair's shared ring of stages is fed by TMA (the decode's tensor map);
// the first warp refills a stage once both warps are past it, which the next
// chunk's barrier shows.
#include <cmath>
#include <cfloat>

#include "decode.cuh"
#include "decode_frag.cuh"
#include "pair_sync.cuh"

namespace jfkv {

constexpr int VSTAGES = 3;   // stages per pair

// warps per CTA (one CTA per SM): 12 (6 pairs) for two n-tiles (168
// registers); 8 (4 pairs) for three, whose softmax state and O take ~250
// registers (capped at 168 they spill and run 10 % slower)
template <int NTC>
constexpr int verify_warps() { return NTC <= 2 ? 12 : 8; }

template <int D, int NTC>
struct VerifySmem {
  static constexpr int VNW = verify_warps<NTC>();
  static constexpr int CB = D / 2;
  static constexpr int NG = D / 64;
  static constexpr int SBB = 4 * NG;
  static constexpr int NP = VNW / 2;
  static constexpr int CODE_BUF = DTOK * CB;
  static constexpr int SB_BUF = DTOK * SBB;
  static constexpr int XK = NTC * 2;   // float4 exchange slots per lane: (n-tile, 16-position tile)
  // pair region: VSTAGES x (K codes, V codes) | VSTAGES x (K, V scale/bias) |
  // exchange [parity][warp of pair][XK][lane] float4
  static constexpr int RING_CODES = VSTAGES * 2 * CODE_BUF;
  static constexpr int RING_SB = VSTAGES * 2 * SB_BUF;
  static constexpr int XBUF = 2 * 2 * XK * 32 * 16;
  static constexpr int PAIR = (RING_CODES + RING_SB + XBUF + 1023) / 1024 * 1024;
  static constexpr int QF_BYTES = NTC * NG * 2 * 32 * 16;   // [n-tile][g][half][lane] uint4
  static constexpr int BQ_BYTES = NTC * 2 * 32 * 4;         // [n-tile][warp of pair][lane]
  static constexpr int CA_BYTES = 16;
  static constexpr int BAR_BYTES = NP * VSTAGES * 8;
  static constexpr int PLAN_BYTES = 16;
  static constexpr int TOTAL =
      NP * PAIR + QF_BYTES + BQ_BYTES + CA_BYTES + BAR_BYTES + PLAN_BYTES;
  static constexpr uint32_t STAGE_TX = 2 * CODE_BUF + 2 * SB_BUF;
  // after the loop a pair region holds its O rows (padded by 4 floats) and (m, l)
  static constexpr int SROW = D + 4;
  static constexpr int ML_OFF = NTC * 8 * SROW * 4;
  static_assert(ML_OFF + NTC * 8 * 2 * 4 <= PAIR, "combine rows fit a pair region");
  static_assert(NTC <= 3, "n-tiles per CTA (also bounds the softmax state in registers)");
  static_assert(TOTAL <= 227 * 1024, "shared memory per CTA");
};

// online-softmax state of one n-tile for this warp's half of d; thread (r, c)
// owns the n-tile's columns 2c, 2c+1 and, for PV, the d-rows
// {64 g + 4 r + e, 64 g + 32 + 4 r + e} of its groups g
template <int NGH>
struct PairState {
  float m0, m1, l0, l1;
  float O[NGH][4][4];
  float Bs[NGH][2];   // this thread's positions' share of sum_t bias_{t,g} p_t, columns 2c, 2c+1
  __device__ __forceinline__ void init() {
    m0 = m1 = -INFINITY;
    l0 = l1 = 0.f;
#pragma unroll
    for (int g = 0; g < NGH; ++g) Bs[g][0] = Bs[g][1] = 0.f;
#pragma unroll
    for (int g = 0; g < NGH; ++g)
#pragma unroll
      for (int e = 0; e < 4; ++e)
#pragma unroll
        for (int i = 0; i < 4; ++i) O[g][e][i] = 0.f;
  }
};

template <int D, int NTC>
struct PairCtx {
  const uint4* qf;       // this lane's query fragments of this warp's first group
  const uint32_t* bq;    // QK bias B fragments (other groups' Q zeroed), [n-tile] x 64
  const float* cA;       // logit scale of the MMA term per n-tile (2^24 / q scaling)
  float cB;
  int r, c, h;
  uint32_t koff[D / 128];   // ldmatrix row offsets of this warp's groups
  int sbo;                  // byte offset of this warp's scale/bias words in a position's row
};

// scale/bias words of this warp's groups for position row p
template <int NGH>
__device__ __forceinline__ void load_my_sb(const uint8_t* p, uint32_t (&w)[NGH]) {
  if constexpr (NGH == 2) {
    const uint2 x = *reinterpret_cast<const uint2*>(p);
    w[0] = x.x;
    w[1] = x.y;
  } else {
    w[0] = *reinterpret_cast<const uint32_t*>(p);
  }
}

// Partial logits over this warp's groups for every n-tile (the decode's QK^T
// and affine fix-up restricted to groups h NGH .. h NGH + NGH - 1).
template <int D, int NTC>
__device__ __forceinline__ void pair_qk(float (&sc)[NTC][2][4], const PairCtx<D, NTC>& cc,
                                        uint32_t kc, const uint8_t* ksb) {
  constexpr int NG = D / 64, NGH = NG / 2, CB = D / 2, SBB = 4 * NG;
#pragma unroll
  for (int j = 0; j < 2; ++j) {
    const int ta = 16 * j + cc.r, tb = ta + 8;
    uint32_t wa[NGH], wb[NGH];
    load_my_sb<NGH>(ksb + ta * SBB + cc.sbo, wa);
    load_my_sb<NGH>(ksb + tb * SBB + cc.sbo, wb);
    f2 t1a[NTC], t1b[NTC];
#pragma unroll
    for (int t = 0; t < NTC; ++t) t1a[t] = t1b[t] = mk2(0.f, 0.f);
#pragma unroll
    for (int gg = 0; gg < NGH; ++gg) {
      uint32_t w0, w1, w2, w3;
      ldsm_x4(w0, w1, w2, w3, kc + cc.koff[gg] + 16 * j * CB);
      const uint32_t h0 = shr8(w0), h1 = shr8(w1), h2 = shr8(w2), h3 = shr8(w3);
      const uint32_t a00 = nib0(w0), a01 = nib0(w1), a02 = nib1(w0), a03 = nib1(w1);
      const uint32_t a10 = nib0(h0), a11 = nib0(h1), a12 = nib1(h0), a13 = nib1(h1);
      const uint32_t a20 = nib0(w2), a21 = nib0(w3), a22 = nib1(w2), a23 = nib1(w3);
      const uint32_t a30 = nib0(h2), a31 = nib0(h3), a32 = nib1(h2), a33 = nib1(h3);
      const float sa = bf16lo_to_f32(wa[gg]), sbv = bf16lo_to_f32(wb[gg]);
#pragma unroll
      for (int t = 0; t < NTC; ++t) {
        const uint4 qa = cc.qf[((t * NG + gg) * 2) * 32];
        const uint4 qb = cc.qf[((t * NG + gg) * 2 + 1) * 32];
        float acc[4];
        mma_f16_zc(acc, a00, a01, a02, a03, qa.x, qa.y);
        mma_f16(acc, a10, a11, a12, a13, qa.z, qa.w);
        mma_f16(acc, a20, a21, a22, a23, qb.x, qb.y);
        mma_f16(acc, a30, a31, a32, a33, qb.z, qb.w);
        t1a[t] = fma2(mk2(sa, sa), mk2(acc[0], acc[1]), t1a[t]);
        t1b[t] = fma2(mk2(sbv, sbv), mk2(acc[2], acc[3]), t1b[t]);
      }
    }
    // bias term over this warp's groups: A rows = positions, k-slots as in
    // decode (groups x (Q high, Q low)); the slots of the partner's groups
    // are zero in A and in B
    uint32_t aa, ab;
    if constexpr (NG == 4) {
      const bool mine = (cc.c & 1) == cc.h;
      aa = mine ? hi_halves(wa[0], wa[1]) : 0u;
      ab = mine ? hi_halves(wb[0], wb[1]) : 0u;
    } else {
      aa = (cc.c < 2) ? (cc.h ? hi_halves(0u, wa[0]) : hi_halves(wa[0], 0u)) : 0u;
      ab = (cc.c < 2) ? (cc.h ? hi_halves(0u, wb[0]) : hi_halves(wb[0], 0u)) : 0u;
    }
    const f2 cB2 = mk2(cc.cB, cc.cB);
#pragma unroll
    for (int t = 0; t < NTC; ++t) {
      float t2[4];
      mma_bf16_zc(t2, aa, ab, 0u, 0u, cc.bq[t * 64], 0u);
      const f2 cA2 = mk2(cc.cA[t], cc.cA[t]);
      un2(fma2(t1a[t], cA2, mul2(mk2(t2[0], t2[1]), cB2)), sc[t][j][0], sc[t][j][1]);
      un2(fma2(t1b[t], cA2, mul2(mk2(t2[2], t2[3]), cB2)), sc[t][j][2], sc[t][j][3]);
    }
  }
}

// Online softmax of one n-tile (identical in both warps of a pair) and PV for
// this warp's groups.  FULL: every position valid and visible to every row;
// otherwise positions >= nvalid hold no data and column 2c (2c+1) sees only
// positions < nv0 (nv1).
template <int D, int NTC, bool FULL>
__device__ __forceinline__ void pair_softmax_pv(PairState<D / 128> (&st)[NTC],
                                                float (&sc)[NTC][2][4],
                                                const PairCtx<D, NTC>& cc, uint32_t vc,
                                                const uint8_t* vsb, int nvalid,
                                                const int (&nv0)[NTC], const int (&nv1)[NTC]) {
  constexpr int NG = D / 64, NGH = NG / 2, CB = D / 2, SBB = 4 * NG;
  constexpr float NEG_INF = -INFINITY;
  const int r = cc.r;
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
    PairState<NGH>& s = st[t];
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
#pragma unroll
      for (int g = 0; g < NGH; ++g) un2(mul2(mk2(s.Bs[g][0], s.Bs[g][1]), ff), s.Bs[g][0], s.Bs[g][1]);
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

  // ---- PV over this warp's groups ------------------------------------------
#pragma unroll
  for (int j = 0; j < 2; ++j) {
    const int ta = 16 * j + r, tb = ta + 8;
    uint32_t wa[NGH], wb[NGH];
    load_my_sb<NGH>(vsb + ta * SBB + cc.sbo, wa);
    load_my_sb<NGH>(vsb + tb * SBB + cc.sbo, wb);
    bool va = true, vb = true;
    if constexpr (!FULL) {
      va = ta < nvalid;
      vb = tb < nvalid;
    }
    // bias term sum_t bias_{t,g} p_t in fp32: this thread's positions ta, tb
    // (summed over the lanes of a column at the end)
#pragma unroll
    for (int gg = 0; gg < NGH; ++gg) {
      float ba = bf16hi_to_f32(wa[gg]), bb = bf16hi_to_f32(wb[gg]);
      if constexpr (!FULL) {
        if (!va) ba = 0.f;
        if (!vb) bb = 0.f;
      }
      const f2 ba2 = mk2(ba, ba), bb2 = mk2(bb, bb);
#pragma unroll
      for (int t = 0; t < NTC; ++t)
        un2(fma2(bb2, mk2(p[t][j][2], p[t][j][3]),
                 fma2(ba2, mk2(p[t][j][0], p[t][j][1]), mk2(st[t].Bs[gg][0], st[t].Bs[gg][1]))),
            st[t].Bs[gg][0], st[t].Bs[gg][1]);
    }
#pragma unroll
    for (int gg = 0; gg < NGH; ++gg) {
      float sva = bf16lo_to_f32(wa[gg]);
      float svb = bf16lo_to_f32(wb[gg]);
      if constexpr (!FULL) {
        if (!va) sva = 0.f;
        if (!vb) svb = 0.f;
      }
      uint32_t v0, v1, v2, v3;
      ldsm_x4_t(v0, v1, v2, v3, vc + cc.koff[gg] + 16 * j * CB);
      const uint32_t h0 = shr8(v0), h1 = shr8(v1), h2 = shr8(v2), h3 = shr8(v3);
      const uint32_t e00 = nib0(v0), e01 = nib0(v2), e02 = nib0(v1), e03 = nib0(v3);
      const uint32_t e10 = nib1(v0), e11 = nib1(v2), e12 = nib1(v1), e13 = nib1(v3);
      const uint32_t e20 = nib0(h0), e21 = nib0(h2), e22 = nib0(h1), e23 = nib0(h3);
      const uint32_t e30 = nib1(h0), e31 = nib1(h2), e32 = nib1(h1), e33 = nib1(h3);
      const f2 sa2 = mk2(sva, sva), sb2 = mk2(svb, svb);
#pragma unroll
      for (int t = 0; t < NTC; ++t) {
        float b00, b01, b10, b11;
        un2(mul2(sa2, mk2(p[t][j][0], p[t][j][1])), b00, b01);
        un2(mul2(sb2, mk2(p[t][j][2], p[t][j][3])), b10, b11);
        const uint32_t b0 = movm_t(pack_f16x2(b00, b01));
        const uint32_t b1 = movm_t(pack_f16x2(b10, b11));
        mma_f16(st[t].O[gg][0], e00, e01, e02, e03, b0, b1);
        mma_f16(st[t].O[gg][1], e10, e11, e12, e13, b0, b1);
        mma_f16(st[t].O[gg][2], e20, e21, e22, e23, b0, b1);
        mma_f16(st[t].O[gg][3], e30, e31, e32, e33, b0, b1);
      }
    }
  }
}

template <int D, int NTC>
__global__ void __launch_bounds__(verify_warps<NTC>() * 32, 1)
verify_pair_kernel(const __grid_constant__ CUtensorMap tmap, const DecodeArgs a) {
  using L = VerifySmem<D, NTC>;
  constexpr int NG = L::NG;
  constexpr int NGH = NG / 2;
  constexpr int SBB = L::SBB;
  constexpr int NP = L::NP;
  constexpr int SROW = L::SROW;
  constexpr float NEG_INF = -INFINITY;

  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* pairs = smem_raw;
  uint4* qsm = reinterpret_cast<uint4*>(smem_raw + NP * L::PAIR);
  uint32_t* bqsm = reinterpret_cast<uint32_t*>(smem_raw + NP * L::PAIR + L::QF_BYTES);
  float* casm = reinterpret_cast<float*>(smem_raw + NP * L::PAIR + L::QF_BYTES + L::BQ_BYTES);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem_raw + NP * L::PAIR + L::QF_BYTES +
                                               L::BQ_BYTES + L::CA_BYTES);
  int* plan_sh = reinterpret_cast<int*>(smem_raw + NP * L::PAIR + L::QF_BYTES + L::BQ_BYTES +
                                        L::CA_BYTES + L::BAR_BYTES);

  // CTA (split, KV head x n-tile group, request): n-tiles nt0 .. nt0 + NTC - 1
  // of the KV head's G * L rows; local row k is (token, head) row 8 nt0 + k
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
  uint8_t* rsb = preg + L::RING_CODES;
  float4* xbuf = reinterpret_cast<float4*>(preg + L::RING_CODES + L::RING_SB);
  uint64_t* pbars = bars + pr * VSTAGES;

  const bool aligned = (smem_u32(smem_raw) & 1023) == 0;
  if (aligned) {
    if (threadIdx.x == 0) prefetch_tensormap(&tmap);
    if (h == 0 && lane == 0) {
      for (int s = 0; s < VSTAGES; ++s) mbar_init(&pbars[s], 1);
      fence_barrier_init();
    }
  }
  asm volatile("griddepcontrol.wait;\n" ::: "memory");

  int split, b, ctx, nch, cps, nsplit;
  if (a.balanced) {
    if (warp == 0) {
      const BalPlan p = balanced_plan(a, (int)blockIdx.x, -1, lane);
      if (lane == 0) {
        plan_sh[0] = p.b;
        plan_sh[1] = p.split;
        plan_sh[2] = p.nsplit;
        plan_sh[3] = p.cps;
      }
    }
    __syncthreads();
    b = plan_sh[0];
    split = plan_sh[1];
    nsplit = plan_sh[2];
    cps = plan_sh[3];
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

  // ---- query fragments: warp t < NTC builds n-tile t ------------------------
  if (warp < NTC) {
    const int rows_t = GL - 8 * (nt0 + warp);   // may be <= 0 for a padding n-tile
    const bool head_ok = r < rows_t;
    const uint16_t* qrow = a.q + ((int64_t)b * a.HqL + row_of(head_ok ? 8 * warp + r : 0)) * D;
    uint4 qlo[NG], qhi[NG];
    float qmax = 0.f;
#pragma unroll
    for (int g = 0; g < NG; ++g) {
      if (head_ok) {
        qlo[g] = *reinterpret_cast<const uint4*>(qrow + 64 * g + 8 * c);
        qhi[g] = *reinterpret_cast<const uint4*>(qrow + 64 * g + 32 + 8 * c);
      } else {
        qlo[g] = make_uint4(0, 0, 0, 0);
        qhi[g] = make_uint4(0, 0, 0, 0);
      }
      const uint32_t ws[8] = {qlo[g].x, qlo[g].y, qlo[g].z, qlo[g].w,
                              qhi[g].x, qhi[g].y, qhi[g].z, qhi[g].w};
#pragma unroll
      for (int i = 0; i < 8; ++i)
        qmax = fmaxf(qmax, fmaxf(fabsf(bf16lo_to_f32(ws[i])), fabsf(bf16hi_to_f32(ws[i]))));
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) qmax = fmaxf(qmax, __shfl_xor_sync(0xffffffffu, qmax, o));
    // keep |q| * 2^-qe < 2^14 so the fp16 operand cannot overflow
    const int qe = (qmax >= 16384.f) ? (ilogbf(qmax) - 13) : 0;
    const float qs = ldexpf(1.f, -qe);
    const float qs16 = qs * 0.0625f;
    float Qg[NG];
#pragma unroll
    for (int g = 0; g < NG; ++g) {
      float e[16];
      const uint32_t ws[8] = {qlo[g].x, qlo[g].y, qlo[g].z, qlo[g].w,
                              qhi[g].x, qhi[g].y, qhi[g].z, qhi[g].w};
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        e[2 * i] = bf16lo_to_f32(ws[i]);
        e[2 * i + 1] = bf16hi_to_f32(ws[i]);
      }
      // the k-slot order of the unpacked code words (see the decode kernel):
      // word W of d = base..base+7 gives (base, base+4), (base+1, base+5) x16,
      // (base+2, base+6), (base+3, base+7) x16
      uint32_t f[8];
#pragma unroll
      for (int hf = 0; hf < 2; ++hf) {
        const float* x = e + 8 * hf;
        f[4 * hf + 0] = pack_f16x2(x[0] * qs, x[4] * qs);
        f[4 * hf + 1] = pack_f16x2(x[1] * qs16, x[5] * qs16);
        f[4 * hf + 2] = pack_f16x2(x[2] * qs, x[6] * qs);
        f[4 * hf + 3] = pack_f16x2(x[3] * qs16, x[7] * qs16);
      }
      qsm[((warp * NG + g) * 2) * 32 + lane] = make_uint4(f[0], f[1], f[2], f[3]);
      qsm[((warp * NG + g) * 2 + 1) * 32 + lane] = make_uint4(f[4], f[5], f[6], f[7]);
      float sum = 0.f;
#pragma unroll
      for (int i = 0; i < 16; ++i) sum += e[i];
      sum += __shfl_xor_sync(0xffffffffu, sum, 1);
      sum += __shfl_xor_sync(0xffffffffu, sum, 2);
      Qg[g] = sum;
    }
    // QK bias B fragment of column r, one per warp of a pair (the partner's
    // groups zeroed): k-slots as in the decode kernel
#pragma unroll
    for (int hh = 0; hh < 2; ++hh) {
      float hi[NG], lo[NG];
#pragma unroll
      for (int g = 0; g < NG; ++g) {
        const float qg = (g / NGH == hh) ? Qg[g] : 0.f;
        hi[g] = __bfloat162float(__float2bfloat16_rn(qg));
        lo[g] = qg - hi[g];
      }
      uint32_t bq;
      if constexpr (NG == 4) {
        if (c == 0) bq = pack_bf16x2(hi[0], hi[1]);
        else if (c == 1) bq = pack_bf16x2(hi[2], hi[3]);
        else if (c == 2) bq = pack_bf16x2(lo[0], lo[1]);
        else bq = pack_bf16x2(lo[2], lo[3]);
      } else {
        if (c == 0) bq = pack_bf16x2(hi[0], hi[1]);
        else if (c == 1) bq = pack_bf16x2(lo[0], lo[1]);
        else bq = 0;
      }
      bqsm[(warp * 2 + hh) * 32 + lane] = bq;
    }
    if (lane == 0) casm[warp] = a.scale_log2 * 16777216.f * ldexpf(1.f, qe);
  }

  // ---- page ids: lane i holds the page of this pair's iteration 32k + i -----
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

  // ---- TMA producer: lane 0 of the pair's first warp; both warps keep the
  // page bookkeeping (which stages hold valid data) ---------------------------
  // one n-tile group per KV head reads each page once: evict it from L2 first
  const uint64_t l2pol = (ncta > 1) ? l2_evict_normal_policy() : l2_evict_first_policy();
  uint32_t valid = 0;
  int issued = 0;
  auto issue = [&](int it) {
    const int s = it % VSTAGES;
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
        uint8_t* ks = rsb + s * 2 * L::SB_BUF;
        const uint8_t* gsb = a.pool + (int64_t)page * a.page_bytes + a.sb_base +
                             ((int64_t)kvh * a.P + inp) * SBB;
        mbar_arrive_expect_tx(bar, L::STAGE_TX);
        tma_load_5d_hint(kc, &tmap, 0, inp, kvh, 0, page, bar, l2pol);
        tma_load_5d_hint(kc + L::CODE_BUF, &tmap, 0, inp, kvh, 1, page, bar, l2pol);
        bulk_g2s_hint(ks, gsb, L::SB_BUF, bar, l2pol);
        bulk_g2s_hint(ks + L::SB_BUF, gsb + a.sb_region, L::SB_BUF, bar, l2pol);
      }
    }
    valid = (valid & ~(1u << s)) | ((uint32_t)ok << s);
    issued = it + 1;
  };
  __syncthreads();   // barriers initialised, query fragments written
  {
    const int npro = my_n < VSTAGES ? my_n : VSTAGES;
    for (int it = 0; it < npro; ++it) issue(it);
  }

  PairCtx<D, NTC> cc;
  cc.qf = qsm + h * NGH * 2 * 32 + lane;
  cc.bq = bqsm + h * 32 + lane;
  cc.cA = casm;
  cc.cB = a.scale_log2;
  cc.r = r;
  cc.c = c;
  cc.h = h;
  {
    const int ld_t = (lane & 7) + 8 * ((lane >> 3) & 1);
    const int ld_ch = lane >> 4;
#pragma unroll
    for (int gg = 0; gg < NGH; ++gg) cc.koff[gg] = swz<L::CB>(ld_t, 2 * (h * NGH + gg) + ld_ch);
  }
  cc.sbo = h * NGH * 4;

  PairState<NGH> st[NTC];
#pragma unroll
  for (int t = 0; t < NTC; ++t) st[t].init();

  // causal limits: token i of the L sees positions < ctx - L + 1 + i; a chunk
  // below ctx_all is visible to every row
  const int ctx_all = ctx - a.L + 1;

  const int bar_id = 1 + pr;
  int done = 0;
  bool gave_up = false;
  // two n-tiles: unrolled by 2, so the exchange buffer's parity is a
  // constant (3 % faster at q_len 2); three: rolled (the unrolled body was
  // 0.5 % slower)
  constexpr int UNR = NTC <= 2 ? 2 : 1;
#pragma unroll UNR
  for (int it = 0; it < my_n; ++it) {
    const int s = it % VSTAGES;
    const uint32_t par = (it / VSTAGES) & 1;
    const bool got = mbar_wait_bounded(&pbars[s], par);
    const bool ok = (valid >> s) & 1u;
    const int tokbase = chunk_of(it) * DTOK;
    const uint32_t kc = smem_u32(rcodes + s * 2 * L::CODE_BUF);
    const uint8_t* ksb = rsb + s * 2 * L::SB_BUF;
    float sc[NTC][2][4];
    if (got) {
      pair_qk<D, NTC>(sc, cc, kc, ksb);
    } else {
#pragma unroll
      for (int t = 0; t < NTC; ++t)
#pragma unroll
        for (int j = 0; j < 2; ++j) sc[t][j][0] = sc[t][j][1] = sc[t][j][2] = sc[t][j][3] = 0.f;
    }
    // swap partial logits with the partner warp (buffers alternate by chunk)
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
#pragma unroll
    for (int t = 0; t < NTC; ++t)
#pragma unroll
      for (int j = 0; j < 2; ++j) {
        const float4 o = xot[(t * 2 + j) * 32];
        un2(add2(mk2(sc[t][j][0], sc[t][j][1]), mk2(o.x, o.y)), sc[t][j][0], sc[t][j][1]);
        un2(add2(mk2(sc[t][j][2], sc[t][j][3]), mk2(o.z, o.w)), sc[t][j][2], sc[t][j][3]);
      }
    // the partner is past chunk it - 1: its stage can be refilled
    if (it >= 1 && it - 1 + VSTAGES < my_n) {
      if (h == 0) fence_proxy_async_smem();
      issue(it - 1 + VSTAGES);
    }
    const uint32_t vc = kc + L::CODE_BUF;
    const uint8_t* vsb = ksb + L::SB_BUF;
    if (ok && tokbase + DTOK <= ctx_all) {
      const int none[NTC] = {};
      pair_softmax_pv<D, NTC, true>(st, sc, cc, vc, vsb, 0, none, none);
    } else {
      int nv0[NTC], nv1[NTC];
#pragma unroll
      for (int t = 0; t < NTC; ++t) {
        const int col = 8 * (nt0 + t) + 2 * c;
        nv0[t] = ok ? min(ctx, ctx_all + col / a.G) - tokbase : 0;
        nv1[t] = ok ? min(ctx, ctx_all + (col + 1) / a.G) - tokbase : 0;
      }
      pair_softmax_pv<D, NTC, false>(st, sc, cc, vc, vsb, ok ? ctx - tokbase : 0, nv0, nv1);
    }
    __syncwarp();
  }
  if (gave_up) {
    // give copies still in flight a bounded chance to land before the ring
    // is reused below
    for (int it = done; it < issued; ++it)
      mbar_wait_bounded(&pbars[it % VSTAGES], (it / VSTAGES) & 1, 1u << 16);
  }

  asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory");

  // ---- per-warp finalize: O rows of this warp's half of d, (m, l) ----------
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
    // bias sums over the 8 lanes of each column pair
    float Bs[NGH][2];
#pragma unroll
    for (int gg = 0; gg < NGH; ++gg) {
      Bs[gg][0] = st[t].Bs[gg][0];
      Bs[gg][1] = st[t].Bs[gg][1];
#pragma unroll
      for (int o = 4; o < 32; o <<= 1) {
        Bs[gg][0] += __shfl_xor_sync(0xffffffffu, Bs[gg][0], o);
        Bs[gg][1] += __shfl_xor_sync(0xffffffffu, Bs[gg][1], o);
      }
    }
#pragma unroll
    for (int gg = 0; gg < NGH; ++gg) {
      const int g = h * NGH + gg;
#pragma unroll
      for (int hf = 0; hf < 2; ++hf) {
#pragma unroll
        for (int hh = 0; hh < 2; ++hh) {
          const int k = 8 * t + 2 * c + hh;
          if (k < rows) {
            float4 v;
            // 2^24 undoes the fp16 subnormal codes (2^20 for the hi nibbles)
            v.x = fmaf(st[t].O[gg][0][2 * hf + hh], 16777216.f, Bs[gg][hh]);
            v.y = fmaf(st[t].O[gg][1][2 * hf + hh], 1048576.f, Bs[gg][hh]);
            v.z = fmaf(st[t].O[gg][2][2 * hf + hh], 16777216.f, Bs[gg][hh]);
            v.w = fmaf(st[t].O[gg][3][2 * hf + hh], 1048576.f, Bs[gg][hh]);
            *reinterpret_cast<float4*>(so + k * SROW + 64 * g + 32 * hf + 4 * r) = v;
          }
        }
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

  // ---- combine the pairs of this CTA ------------------------------------------
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
    const int fr = row_of(k);
    if (direct) {
      uint2 o;
      o.x = (uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(acc.x)) |
            ((uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(acc.y)) << 16);
      o.y = (uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(acc.z)) |
            ((uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(acc.w)) << 16);
      *reinterpret_cast<uint2*>(a.out + ((int64_t)b * a.HqL + fr) * D + d) = o;
    } else {
      const int64_t row = a.balanced ? (int64_t)blockIdx.x * a.HqL + fr
                                     : ((int64_t)b * a.HqL + fr) * a.num_splits + blockIdx.x;
      *reinterpret_cast<float4*>(a.part_o + row * D + d) = acc;
      if (d == 0) {
        a.part_ml[row * 2 + 0] = M;
        a.part_ml[row * 2 + 1] = Lsum;
      }
    }
  }
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------
int verify_pair_ntc(int NT) { return NT < 3 ? NT : 3; }

int verify_pair_ctas(int NT) {
  const int ntc = verify_pair_ntc(NT);
  return (NT + ntc - 1) / ntc;
}

template <int D, int NTC>
static int launch_verify_t(const CUtensorMap& tmap, const DecodeArgs& a, int B,
                           cudaStream_t stream) {
  using L = VerifySmem<D, NTC>;
  const void* kernel = (const void*)verify_pair_kernel<D, NTC>;
  if (smem_optin(kernel, L::TOTAL) != JF_OK) return JF_ERR_CUDA;
  cudaLaunchAttribute pdl[1];
  pdl[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  pdl[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t cfg = {};
  const int ncta = verify_pair_ctas(a.NT);
  cfg.gridDim = a.balanced ? dim3((unsigned)(a.budget + B), (unsigned)(a.Hkv * ncta), 1u)
                           : dim3((unsigned)a.plan_splits, (unsigned)(a.Hkv * ncta), (unsigned)B);
  cfg.blockDim = dim3(L::VNW * 32);
  cfg.dynamicSmemBytes = L::TOTAL;
  cfg.stream = stream;
  cfg.attrs = pdl;
  cfg.numAttrs = 1;
  if (cudaLaunchKernelEx(&cfg, verify_pair_kernel<D, NTC>, tmap, a) != cudaSuccess)
    return JF_ERR_CUDA;
  if (a.balanced || a.plan_splits > 1) return launch_decode_merge(a, D, B, stream);
  return JF_OK;
}

int launch_verify_pairs(const CUtensorMap& tmap, const DecodeArgs& a, int D, int B,
                        cudaStream_t stream) {
  const int ntc = verify_pair_ntc(a.NT);
  if (D == 256)
    return ntc == 2 ? launch_verify_t<256, 2>(tmap, a, B, stream)
                    : launch_verify_t<256, 3>(tmap, a, B, stream);
  return ntc == 2 ? launch_verify_t<128, 2>(tmap, a, B, stream)
                  : launch_verify_t<128, 3>(tmap, a, B, stream);
}

}  // namespace jfkv
