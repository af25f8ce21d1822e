// Paged 4-bit decode attention with a fixed split-K workspace (Sec. 3.1:
// decode reads the compressed pages where they are used; Sec. 2, Eq. 3: never
// size temporaries by the history length; Eq. 5: contiguous GQA head groups).
//
// Kernel 1 (split phase).  CTA = (split s, KV head, request b), 6 warps.  A
// split takes a contiguous range of the context's 32-position chunks and
// deals them round-robin to its warps; each warp owns
// a private ring of DSTAGES shared-memory stages that it refills itself with
// TMA: a 5-D tiled copy (128-byte swizzle) for the K and V code rows of the
// chunk and two 1-D bulk copies for their scale/bias words.
//
// Dequantization never leaves registers and never builds bf16 K/V:
//  * A 4-bit code n placed in the low bits of an fp16 is the subnormal
//    n * 2^-24 exactly (the hi nibble of a byte gives 16 n * 2^-24), so
//    `w & 0x000F000F` turns two packed codes into an f16x2 MMA operand.
//  * QK^T: A = K codes [16 positions x 16 d] (ldmatrix), B = q [16 d x 8 heads]
//    (the G <= 8 heads of the KV head share every K fragment).  Each k-step
//    stays inside one 64-element group, so a group's partial dot product
//    acc_g = 2^-24 sum_d q_d n_d is kept apart and the affine fix-up is exact:
//        s_t = sum_g scale_{t,g} 2^24 acc_g + sum_g bias_{t,g} Q_g,
//    Q_g = sum_{d in g} q_d; the bias term is a bf16 MMA of the bias words
//    against Q_g split into bf16 high and low parts.
//  * PV: A = V codes transposed [16 d x 16 positions] (ldmatrix.trans gives the
//    position pairs), B = p_t * scale_{t,g} as f16 [16 positions x 8 heads]
//    (the QK accumulator transposed with movmatrix); the bias term
//    sum_t bias_{t,g} p_t is accumulated in fp32 by each thread over its own
//    positions and summed over the lanes of a head pair at the end.
//  * Online softmax in the log2 domain.  The reference maximum moves only when
//    a logit exceeds it by more than 2^DTAU, so the common chunk needs no
//    cross-lane reduction; the accumulators are rescaled only then.
// The four warps' states are combined in shared memory and written as one
// split partial (m, l, O) to the workspace, or straight to the output when
// num_splits == 1.
//
// Kernel 2 (merge).  CTAs over (32-wide d slice, query head, request) combine:
//   o = sum_s 2^{m_s - m*} O_s / sum_s 2^{m_s - m*} l_s.
#include <cmath>
#include <cfloat>
#include <mutex>
#include <utility>
#include <vector>

#include "decode.cuh"
#include "decode_frag.cuh"
#include "quant.cuh"

namespace jfkv {

// Warps per split CTA (NW, a template parameter): 6 (two CTAs per SM) or 12
// (one CTA per SM, the same warps per SM in one block).
constexpr int DSTAGES = 2;    // stages per warp

template <int D, int NW>
struct DecodeSmem {
  static constexpr int CB = D / 2;
  static constexpr int NG = D / 64;
  static constexpr int SBB = 4 * NG;
  static constexpr int CODE_BUF = DTOK * CB;
  static constexpr int SB_BUF = DTOK * SBB;
  static constexpr int NBUF = NW * DSTAGES;
  static constexpr int CODES_BYTES = NBUF * 2 * CODE_BUF;
  static constexpr int SB_BYTES = NBUF * 2 * SB_BUF;
  static constexpr int QF_BYTES = NG * 2 * 32 * 16;   // query fragments [g][half][lane][4]
  static constexpr int BAR_BYTES = NBUF * 8;
  // The dynamic shared window starts 1024-byte aligned (checked at run time),
  // which the 128-byte TMA swizzle of the code buffers needs.
  static constexpr int PLAN_BYTES = 16;                // batch plan broadcast
  static constexpr int TOTAL = CODES_BYTES + SB_BYTES + QF_BYTES + BAR_BYTES + PLAN_BYTES;
  static constexpr uint32_t STAGE_TX = 2 * CODE_BUF + 2 * SB_BUF;
  static_assert(NW * 8 * (D + 4) * 4 <= CODES_BYTES, "combine buffer must fit");
  static_assert((NW * 8 * 3 + 16) * 4 <= SB_BYTES, "combine (m, l), weights must fit");
  static_assert(TOTAL <= 227 * 1024, "shared memory per CTA");
};

// Per-warp online-softmax state.  Thread (r, c) of the warp owns query heads
// 2c and 2c+1 (columns of the m16n8 accumulators) and, for PV, the d-rows
// {64g + 4r + e, 64g + 32 + 4r + e}.
template <int NG>
struct DecodeState {
  float m0, m1, l0, l1;
  float O[NG][4][4];
  float Bs[NG][2];   // this thread's positions' share of sum_t bias_{t,g} p_t, heads 2c, 2c+1
  __device__ __forceinline__ void init() {
    m0 = m1 = -INFINITY;
    l0 = l1 = 0.f;
#pragma unroll
    for (int g = 0; g < NG; ++g) Bs[g][0] = Bs[g][1] = 0.f;
#pragma unroll
    for (int g = 0; g < NG; ++g) {
#pragma unroll
      for (int e = 0; e < 4; ++e)
#pragma unroll
        for (int i = 0; i < 4; ++i) O[g][e][i] = 0.f;
    }
  }
};

template <int NG>
struct ChunkCtx {
  const uint4* qf;   // this lane's query fragments: qf[2 g + half] = k-steps 2 half, 2 half + 1
  uint32_t bq;   // B fragment of the QK bias MMA: (Q_g high | low parts) for head r
  float cA, cB;
  int r, c;
  // this lane's ldmatrix row address within a stage buffer for group g's two
  // 16-byte chunks (16-position tile 0; tile j adds 16 j rows, which keeps
  // the swizzle phase)
  uint32_t koff[NG];
};

// One 32-position chunk (two 16-position MMA tiles).  FULL: every position is
// valid and visible to every row, so no masking work is done; otherwise
// positions >= nvalid hold no data (their logits become -inf and their
// scale/bias words are never used, so whatever bytes sit in unused slots
// cannot leak into the result), and the rows of this thread's columns 2c and
// 2c+1 see only positions < nv0 and < nv1 (causal limits of the verifier's
// query tokens; both are nvalid for a single query).
template <int D, bool FULL>
__device__ __forceinline__ void process_chunk(DecodeState<D / 64>& st, const ChunkCtx<D / 64>& cc,
                                              uint32_t kc, const uint8_t* ksb, int nvalid,
                                              int nv0, int nv1) {
  constexpr int NG = D / 64;
  constexpr int CB = D / 2;
  constexpr int SBB = 4 * NG;
  constexpr int SB_BUF = DTOK * SBB;
  constexpr float NEG_INF = -INFINITY;
  const uint32_t vc = kc + DTOK * CB;
  const uint8_t* vsb = ksb + SB_BUF;
  constexpr int NJ = DTOK / 16;   // 16-position MMA tiles per chunk
  const int r = cc.r;

  float sc[NJ][4];
#pragma unroll
  for (int j = 0; j < NJ; ++j) {
    const int ta = 16 * j + r, tb = ta + 8;
    float acc[NG][4];
#pragma unroll
    for (int g = 0; g < NG; ++g) {
      const uint4 qa = cc.qf[(2 * g) * 32], qb = cc.qf[(2 * g + 1) * 32];
      uint32_t w0, w1, w2, w3;
      ldsm_x4(w0, w1, w2, w3, kc + cc.koff[g] + 16 * j * CB);
      const uint32_t h0 = shr8(w0), h1 = shr8(w1), h2 = shr8(w2), h3 = shr8(w3);
      mma_f16_zc(acc[g], nib0(w0), nib0(w1), nib1(w0), nib1(w1), qa.x, qa.y);
      mma_f16(acc[g], nib0(h0), nib0(h1), nib1(h0), nib1(h1), qa.z, qa.w);
      mma_f16(acc[g], nib0(w2), nib0(w3), nib1(w2), nib1(w3), qb.x, qb.y);
      mma_f16(acc[g], nib0(h2), nib0(h3), nib1(h2), nib1(h3), qb.z, qb.w);
    }
    uint32_t wa[NG], wb[NG];
    load_sb_words<NG>(ksb + ta * SBB, wa);
    load_sb_words<NG>(ksb + tb * SBB, wb);
    // bias term sum_g bias_{t,g} Q_g: A rows = positions, k-slots = groups x (Q high, Q low)
    float t2[4];
    {
      uint32_t aa, ab;
      if constexpr (NG == 4) {
        aa = (cc.c & 1) ? hi_halves(wa[2], wa[3]) : hi_halves(wa[0], wa[1]);
        ab = (cc.c & 1) ? hi_halves(wb[2], wb[3]) : hi_halves(wb[0], wb[1]);
      } else {
        aa = (cc.c < 2) ? hi_halves(wa[0], wa[1]) : 0u;
        ab = (cc.c < 2) ? hi_halves(wb[0], wb[1]) : 0u;
      }
      mma_bf16_zc(t2, aa, ab, 0u, 0u, cc.bq, 0u);
    }
    // t1 = sum_g scale_g acc_g on (head 2c, 2c+1) pairs
    f2 t1a = mk2(0.f, 0.f), t1b = mk2(0.f, 0.f);
#pragma unroll
    for (int g = 0; g < NG; ++g) {
      const float sa = bf16lo_to_f32(wa[g]), sbv = bf16lo_to_f32(wb[g]);
      t1a = fma2(mk2(sa, sa), mk2(acc[g][0], acc[g][1]), t1a);
      t1b = fma2(mk2(sbv, sbv), mk2(acc[g][2], acc[g][3]), t1b);
    }
    const f2 cA2 = mk2(cc.cA, cc.cA), cB2 = mk2(cc.cB, cc.cB);
    un2(fma2(t1a, cA2, mul2(mk2(t2[0], t2[1]), cB2)), sc[j][0], sc[j][1]);
    un2(fma2(t1b, cA2, mul2(mk2(t2[2], t2[3]), cB2)), sc[j][2], sc[j][3]);
    if constexpr (!FULL) {
      if (ta >= nv0) sc[j][0] = NEG_INF;
      if (ta >= nv1) sc[j][1] = NEG_INF;
      if (tb >= nv0) sc[j][2] = NEG_INF;
      if (tb >= nv1) sc[j][3] = NEG_INF;
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
    for (int g = 0; g < NG; ++g) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        st.O[g][e][0] *= f0; st.O[g][e][2] *= f0;
        st.O[g][e][1] *= f1; st.O[g][e][3] *= f1;
      }
    }
#pragma unroll
    for (int g = 0; g < NG; ++g) {
      st.Bs[g][0] *= f0;
      st.Bs[g][1] *= f1;
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
      const f2 m2 = mk2(st.m0, st.m1);
      float d0, d1, d2, d3;
      un2(sub2(mk2(sc[j][0], sc[j][1]), m2), d0, d1);
      un2(sub2(mk2(sc[j][2], sc[j][3]), m2), d2, d3);
      p[j][0] = fast_exp2(d0);
      p[j][1] = fast_exp2(d1);
      p[j][2] = fast_exp2(d2);
      p[j][3] = fast_exp2(d3);
    } else {
      p[j][0] = (sc[j][0] == NEG_INF) ? 0.f : fast_exp2(sc[j][0] - st.m0);
      p[j][1] = (sc[j][1] == NEG_INF) ? 0.f : fast_exp2(sc[j][1] - st.m1);
      p[j][2] = (sc[j][2] == NEG_INF) ? 0.f : fast_exp2(sc[j][2] - st.m0);
      p[j][3] = (sc[j][3] == NEG_INF) ? 0.f : fast_exp2(sc[j][3] - st.m1);
    }
    float l0n, l1n;
    un2(add2(mk2(st.l0, st.l1), add2(mk2(p[j][0], p[j][1]), mk2(p[j][2], p[j][3]))), l0n, l1n);
    st.l0 = l0n;
    st.l1 = l1n;
  }

  // ---- PV ---------------------------------------------------------------
#pragma unroll
  for (int j = 0; j < NJ; ++j) {
    const int ta = 16 * j + r, tb = ta + 8;
    uint32_t wa[NG], wb[NG];
    load_sb_words<NG>(vsb + ta * SBB, wa);
    load_sb_words<NG>(vsb + tb * SBB, wb);
    bool va = true, vb = true;
    if constexpr (!FULL) {
      va = ta < nvalid;
      vb = tb < nvalid;
    }
    // bias term sum_t bias_{t,g} p_t in fp32: this thread's positions ta, tb
    // (summed over the lanes of a head pair at the end)
#pragma unroll
    for (int g = 0; g < NG; ++g) {
      float ba = bf16hi_to_f32(wa[g]), bb = bf16hi_to_f32(wb[g]);
      if constexpr (!FULL) {
        if (!va) ba = 0.f;
        if (!vb) bb = 0.f;
      }
      un2(fma2(mk2(bb, bb), mk2(p[j][2], p[j][3]),
               fma2(mk2(ba, ba), mk2(p[j][0], p[j][1]), mk2(st.Bs[g][0], st.Bs[g][1]))),
          st.Bs[g][0], st.Bs[g][1]);
    }
#pragma unroll
    for (int g = 0; g < NG; ++g) {
      float sva = bf16lo_to_f32(wa[g]);
      float svb = bf16lo_to_f32(wb[g]);
      if constexpr (!FULL) {
        if (!va) sva = 0.f;
        if (!vb) svb = 0.f;
      }
      float b00, b01, b10, b11;
      un2(mul2(mk2(sva, sva), mk2(p[j][0], p[j][1])), b00, b01);
      un2(mul2(mk2(svb, svb), mk2(p[j][2], p[j][3])), b10, b11);
      const uint32_t b0 = movm_t(pack_f16x2(b00, b01));
      const uint32_t b1 = movm_t(pack_f16x2(b10, b11));
      uint32_t v0, v1, v2, v3;
      ldsm_x4_t(v0, v1, v2, v3, vc + cc.koff[g] + 16 * j * CB);
      const uint32_t h0 = shr8(v0), h1 = shr8(v1), h2 = shr8(v2), h3 = shr8(v3);
      mma_f16(st.O[g][0], nib0(v0), nib0(v2), nib0(v1), nib0(v3), b0, b1);
      mma_f16(st.O[g][1], nib1(v0), nib1(v2), nib1(v1), nib1(v3), b0, b1);
      mma_f16(st.O[g][2], nib0(h0), nib0(h2), nib0(h1), nib0(h3), b0, b1);
      mma_f16(st.O[g][3], nib1(h0), nib1(h2), nib1(h1), nib1(h3), b0, b1);
    }
  }
}

// Fused append: the split that owns position pos of request b quantizes the
// step's new K and V vectors of its KV head (one vector per D/8 lanes, the
// quantizer the append kernel uses) and stores them before any of its reads.
template <int D>
__device__ __forceinline__ void append_new_row(const DecodeArgs& a, int b, int kvh, int pos,
                                               int warp, int lane) {
  constexpr int LPV = D / 8;        // lanes per vector
  constexpr int VPW = 32 / LPV;     // vectors per warp
  if (warp * VPW >= 2) return;      // warp-uniform: the K and V vectors only
  const int vec = warp * VPW + lane / LPV;   // 0: K, 1: V
  const int li = lane % LPV;
  const bool active = vec < 2;
  float x[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
  if (active) load8_bf16((vec ? a.vnew : a.knew) + ((int64_t)b * a.Hkv + kvh) * D + li * 8, x);
  __nv_bfloat16 sh, bh;
  const uint32_t word = quantize8(x, sh, bh);
  if (!active) return;
  const int pidx = pos >> a.log2P;
  const int page = (pidx < a.pt_stride) ? a.page_table[(int64_t)b * a.pt_stride + pidx] : -1;
  if (page < 0 || page >= a.num_pages) {
    if (li == 0) flag_error(a.status, JF_DEV_ERR_PAGE_ID);
    return;
  }
  store_quantized<D>(const_cast<uint8_t*>(a.pool) + (int64_t)page * a.page_bytes,
                     a.codes_region, a.sb_region, a.P, kvh, pos & (a.P - 1), vec, li, word, sh,
                     bh);
}

template <int D, bool VER, int NW>
__global__ void __launch_bounds__(NW * 32, 12 / NW)
decode_split_kernel(const __grid_constant__ CUtensorMap tmap, const DecodeArgs a) {
  // VER: packed verifier (a.L > 1, per-row causal limits); otherwise decode
  using L = DecodeSmem<D, NW>;
  constexpr int NG = L::NG;
  constexpr int SBB = L::SBB;
  constexpr float NEG_INF = -INFINITY;

  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* codes = smem_raw;
  uint8_t* sbuf = codes + L::CODES_BYTES;
  uint4* qsm = reinterpret_cast<uint4*>(sbuf + L::SB_BYTES);
  uint64_t* bars = reinterpret_cast<uint64_t*>(sbuf + L::SB_BYTES + L::QF_BYTES);

  // decode: one CTA per KV head holds its G query heads; verifier: NT CTAs
  // each hold 8 of its G * L (token, head) rows (launched for NT = 1; more
  // rows go to the warp-pair kernel of verify.cu)
  const int kvh = VER ? (int)blockIdx.y / a.NT : (int)blockIdx.y;
  const int nt = VER ? (int)blockIdx.y % a.NT : 0;
  const int rows = VER ? min(8, a.G * a.L - 8 * nt) : a.G;
  // row k of this CTA: query token i = (8 nt + k) / G, head h = (8 nt + k) % G;
  // its q, out and partial row within the request is i * Hq + kvh * G + h
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
  const bool direct = (a.plan_splits == 1 && !a.balanced);
  int* plan_sh = reinterpret_cast<int*>(sbuf + L::SB_BYTES + L::QF_BYTES + L::BAR_BYTES);
  // the swizzled TMA boxes need a 1024-byte aligned window
  const bool aligned = (smem_u32(smem_raw) & 1023) == 0;
  if (aligned) {   // setup that reads nothing a previous kernel writes
    if (threadIdx.x == 0) prefetch_tensormap(&tmap);
    if (lane == 0) {
      for (int s = 0; s < DSTAGES; ++s) mbar_init(&bars[warp * DSTAGES + s], 1);
      fence_barrier_init();
    }
  }
  // launched with programmatic dependent launch: wait for the previous
  // kernel (e.g. the append that wrote the newest position) before any read
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
    if (b < 0) return;   // past the batch's last split
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
  const int c_begin = split * cps;
  const int c_end = min(c_begin + cps, nch);
  const int n_cta = c_end - c_begin;
  const int my_n = (n_cta > warp) ? (n_cta - warp + NW - 1) / NW : 0;
  auto chunk_of = [&](int it) { return c_begin + warp + it * NW; };

  if (!aligned) {
    if (threadIdx.x == 0) flag_error(a.status, JF_DEV_ERR_LAYOUT);
    return;
  }
  if (a.knew != nullptr && split == nsplit - 1) {   // owns the last chunk
    // the new row goes to the pool before this split's TMA reads it
    append_new_row<D>(a, b, kvh, ctx - 1, warp, lane);
    fence_proxy_async_global();
    __syncthreads();
    fence_proxy_async_global();
  }
  __syncwarp();

  // ---- query fragments (B operand of QK^T) ---------------------------------
  const bool head_ok = r < rows;
  const uint16_t* qrow = a.q + ((int64_t)b * a.HqL + row_of(head_ok ? r : 0)) * D;
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

  uint32_t qf[NG][4][2];
  float Qg[NG];
#pragma unroll
  for (int g = 0; g < NG; ++g) {
    float e[16];
    const uint32_t ws[8] = {qlo[g].x, qlo[g].y, qlo[g].z, qlo[g].w,
                            qhi[g].x, qhi[g].y, qhi[g].z, qhi[g].w};
#pragma unroll
    for (int i = 0; i < 8; ++i) { e[2 * i] = bf16lo_to_f32(ws[i]); e[2 * i + 1] = bf16hi_to_f32(ws[i]); }
    // word W covers d = base..base+7; nib0 -> (base, base+4), nib1 -> (base+1, base+5) x16,
    // nib0 of W>>8 -> (base+2, base+6), nib1 of W>>8 -> (base+3, base+7) x16
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const float* x = e + 8 * h;
      qf[g][2 * h + 0][0] = pack_f16x2(x[0] * qs, x[4] * qs);
      qf[g][2 * h + 0][1] = pack_f16x2(x[1] * qs16, x[5] * qs16);
      qf[g][2 * h + 1][0] = pack_f16x2(x[2] * qs, x[6] * qs);
      qf[g][2 * h + 1][1] = pack_f16x2(x[3] * qs16, x[7] * qs16);
    }
    float sum = 0.f;
#pragma unroll
    for (int i = 0; i < 16; ++i) sum += e[i];
    sum += __shfl_xor_sync(0xffffffffu, sum, 1);
    sum += __shfl_xor_sync(0xffffffffu, sum, 2);
    Qg[g] = sum;
  }
  // QK bias B fragment for head r: k-slot k < NG is Q_k high, NG <= k < 2 NG
  // is Q_{k-NG} low (the bf16 residual); thread c holds slots 2c, 2c+1.
  uint32_t bq = 0;
  {
    float hi[NG], lo[NG];
#pragma unroll
    for (int g = 0; g < NG; ++g) {
      hi[g] = __bfloat162float(__float2bfloat16_rn(Qg[g]));
      lo[g] = Qg[g] - hi[g];
    }
    if constexpr (NG == 4) {
      if (c == 0) bq = pack_bf16x2(hi[0], hi[1]);
      else if (c == 1) bq = pack_bf16x2(hi[2], hi[3]);
      else if (c == 2) bq = pack_bf16x2(lo[0], lo[1]);
      else bq = pack_bf16x2(lo[2], lo[3]);
    } else {
      if (c == 0) bq = pack_bf16x2(hi[0], hi[1]);
      else if (c == 1) bq = pack_bf16x2(lo[0], lo[1]);
    }
  }
  const float cA = a.scale_log2 * 16777216.f * ldexpf(1.f, qe);
  const float cB = a.scale_log2;

  // ---- page ids: lane i holds the page of this warp's iteration 32k + i ------
  // (two blocks of 32 in flight so the dependent load never stalls an issue)
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

  // ---- TMA producer (lane 0 of each warp feeds its own ring) -------------
  // decode reads each page once per call: evict it from L2 first; the
  // verifier's n-tile CTAs read the same pages, so L2 keeps them normally
  const uint64_t l2pol = VER ? l2_evict_normal_policy() : l2_evict_first_policy();
  uint32_t valid = 0;
  auto issue = [&](int it) {
    const int s = it % DSTAGES;
    if (it >= 32 && (it & 31) == 0) {
      pg_cur = pg_next;
      pg_next = load_pages((it >> 5) + 1);
    }
    const int page = __shfl_sync(0xffffffffu, pg_cur, it & 31);
    const bool ok = page >= 0 && page < a.num_pages;
    if (lane == 0) {
      const int inp = (chunk_of(it) * DTOK) & (a.P - 1);
      uint64_t* bar = &bars[warp * DSTAGES + s];
      if (!ok) {
        flag_error(a.status, JF_DEV_ERR_PAGE_ID);
        mbar_arrive(bar);
      } else {
        uint8_t* kc = codes + (warp * DSTAGES + s) * 2 * L::CODE_BUF;
        uint8_t* ks = sbuf + (warp * DSTAGES + s) * 2 * L::SB_BUF;
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
  };

  const int npro = my_n < DSTAGES ? my_n : DSTAGES;
  for (int it = 0; it < npro; ++it) issue(it);

  // ---- running state ---------------------------------------------------
  DecodeState<NG> st;
  st.init();

  // ldmatrix row address pieces: matrix m = lane>>3 -> (position half, chunk)
  const int ld_t = (lane & 7) + 8 * ((lane >> 3) & 1);
  const int ld_ch = lane >> 4;
  if (warp == 0) {
#pragma unroll
    for (int g = 0; g < NG; ++g) {
      qsm[(2 * g) * 32 + lane] = make_uint4(qf[g][0][0], qf[g][0][1], qf[g][1][0], qf[g][1][1]);
      qsm[(2 * g + 1) * 32 + lane] = make_uint4(qf[g][2][0], qf[g][2][1], qf[g][3][0], qf[g][3][1]);
    }
  }
  __syncthreads();
  ChunkCtx<NG> cc{qsm + lane, bq, cA, cB, r, c, {}};
#pragma unroll
  for (int g = 0; g < NG; ++g) cc.koff[g] = swz<L::CB>(ld_t, 2 * g + ld_ch);

  // verifier causal limits: query token i of L sees positions < ctx - L + 1 + i;
  // a chunk below ctx_all is visible to every row (decode: ctx_all = ctx)
  int ctx_all = ctx, lim0 = ctx, lim1 = ctx;
  if constexpr (VER) {
    ctx_all = ctx - a.L + 1;
    lim0 = min(ctx, ctx_all + (8 * nt + 2 * c) / a.G);
    lim1 = min(ctx, ctx_all + (8 * nt + 2 * c + 1) / a.G);
  }
  int done = 0;
  // unrolled by the ring depth, so every stage address is a constant offset
#pragma unroll DSTAGES
  for (int it = 0; it < my_n; ++it) {
    const int s = it % DSTAGES;
    const uint32_t par = (it / DSTAGES) & 1;
    if (!mbar_wait_bounded(&bars[warp * DSTAGES + s], par)) {
      if (lane == 0) flag_error(a.status, JF_DEV_ERR_TIMEOUT);
      break;
    }
    done = it + 1;
    const bool ok = (valid >> s) & 1u;
    const int tokbase = chunk_of(it) * DTOK;
    const uint32_t kc = smem_u32(codes + (warp * DSTAGES + s) * 2 * L::CODE_BUF);
    const uint8_t* ksb = sbuf + (warp * DSTAGES + s) * 2 * L::SB_BUF;
    if (ok && tokbase + DTOK <= (VER ? ctx_all : ctx)) {
      process_chunk<D, true>(st, cc, kc, ksb, 0, 0, 0);
    } else if constexpr (VER) {
      process_chunk<D, false>(st, cc, kc, ksb, ok ? ctx - tokbase : 0,
                              ok ? lim0 - tokbase : 0, ok ? lim1 - tokbase : 0);
    } else {
      const int nv = ok ? ctx - tokbase : 0;
      process_chunk<D, false>(st, cc, kc, ksb, nv, nv, nv);
    }

    __syncwarp();
    if (it + DSTAGES < my_n) {
      fence_proxy_async_smem();
      issue(it + DSTAGES);
    }
  }
  if (done < my_n) {
    // a wait gave up: give copies still in flight a bounded chance to land
    for (int it = done; it < my_n && it < done + DSTAGES; ++it)
      mbar_wait_bounded(&bars[warp * DSTAGES + it % DSTAGES], (it / DSTAGES) & 1, 1u << 16);
  }
  float& m0 = st.m0;
  float& m1 = st.m1;
  float& l0 = st.l0;
  float& l1 = st.l1;
  auto& O = st.O;

  // the merge kernel may start launching; it waits for this grid to finish
  asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory");

  // ---- per-warp finalize ---------------------------------------------------
#pragma unroll
  for (int o = 4; o < 32; o <<= 1) {
    l0 += __shfl_xor_sync(0xffffffffu, l0, o);
    l1 += __shfl_xor_sync(0xffffffffu, l1, o);
  }
  // bias sums over the 8 lanes of each head pair
  float Bs[NG][2];
#pragma unroll
  for (int g = 0; g < NG; ++g) {
    Bs[g][0] = st.Bs[g][0];
    Bs[g][1] = st.Bs[g][1];
#pragma unroll
    for (int o = 4; o < 32; o <<= 1) {
      Bs[g][0] += __shfl_xor_sync(0xffffffffu, Bs[g][0], o);
      Bs[g][1] += __shfl_xor_sync(0xffffffffu, Bs[g][1], o);
    }
  }
  // This warp's ring is idle now (each of its copies has landed and been
  // read), so its O rows (padded by 4 floats: the 128-bit stores of one
  // quarter-warp hit 8 distinct bank groups) and (m, l) per head go into its
  // own stage buffers at once, without waiting for the other warps.
  constexpr int SROW = D + 4;
  constexpr int WCODES = DSTAGES * 2 * L::CODE_BUF;   // one warp's code ring (bytes)
  constexpr int WSB = DSTAGES * 2 * L::SB_BUF;        // one warp's scale/bias ring
  static_assert(8 * SROW * 4 <= WCODES && 8 * 2 * 4 <= WSB, "combine rows fit a warp's ring");
  {
    float* so = reinterpret_cast<float*>(codes + warp * WCODES);   // [8][SROW]
    float* sml = reinterpret_cast<float*>(sbuf + warp * WSB);      // [8][2]
#pragma unroll
    for (int g = 0; g < NG; ++g) {
#pragma unroll
      for (int hf = 0; hf < 2; ++hf) {          // d block 64g + 32 hf + 4r + e
#pragma unroll
        for (int hh = 0; hh < 2; ++hh) {        // head 2c + hh
          if (2 * c + hh < rows) {
            float4 v;
            // 2^24 undoes the fp16 subnormal codes (2^20 for the hi nibbles)
            v.x = fmaf(O[g][0][2 * hf + hh], 16777216.f, Bs[g][hh]);
            v.y = fmaf(O[g][1][2 * hf + hh], 1048576.f, Bs[g][hh]);
            v.z = fmaf(O[g][2][2 * hf + hh], 16777216.f, Bs[g][hh]);
            v.w = fmaf(O[g][3][2 * hf + hh], 1048576.f, Bs[g][hh]);
            *reinterpret_cast<float4*>(so + (2 * c + hh) * SROW + 64 * g + 32 * hf + 4 * r) = v;
          }
        }
      }
    }
    if (r == 0) {
      sml[(2 * c) * 2 + 0] = m0;
      sml[(2 * c) * 2 + 1] = l0;
      sml[(2 * c + 1) * 2 + 0] = m1;
      sml[(2 * c + 1) * 2 + 1] = l1;
    }
  }
  __syncthreads();

  // ---- combine the warps of this CTA --------------------------------------
  // per head: M = max_w m_w, weights 2^(m_w - M) (divided by L when this CTA
  // writes the final output), L = sum_w 2^(m_w - M) l_w; every thread works
  // out the weights of its own head.
  for (int idx = threadIdx.x; idx < rows * (D / 4); idx += blockDim.x) {
    const int h = idx / (D / 4), d = 4 * (idx % (D / 4));
    float mw[NW], lw[NW];
    float M = NEG_INF;
#pragma unroll
    for (int w = 0; w < NW; ++w) {
      const float2 v = *reinterpret_cast<const float2*>(sbuf + w * WSB + h * 8);
      mw[w] = v.x;
      lw[w] = v.y;
      M = fmaxf(M, v.x);
    }
    float f[NW];
    float Lsum = 0.f;
#pragma unroll
    for (int w = 0; w < NW; ++w) {
      f[w] = (mw[w] != NEG_INF) ? fast_exp2(mw[w] - M) : 0.f;
      Lsum = fmaf(f[w], lw[w], Lsum);
    }
    const float inv = direct ? (Lsum > 0.f ? 1.f / Lsum : 0.f) : 1.f;
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
    for (int w = 0; w < NW; ++w) {
      const float fw = f[w] * inv;
      const float4 v = *reinterpret_cast<const float4*>(
          reinterpret_cast<const float*>(codes + w * WCODES) + h * SROW + d);
      if (fw != 0.f) {
        acc.x = fmaf(fw, v.x, acc.x);
        acc.y = fmaf(fw, v.y, acc.y);
        acc.z = fmaf(fw, v.z, acc.z);
        acc.w = fmaf(fw, v.w, acc.w);
      }
    }
    const int fr = row_of(h);
    if (direct) {
      uint2 o;
      o.x = (uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(acc.x)) |
            ((uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(acc.y)) << 16);
      o.y = (uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(acc.z)) |
            ((uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(acc.w)) << 16);
      *reinterpret_cast<uint2*>(a.out + ((int64_t)blockIdx.z * a.HqL + fr) * D + d) = o;
    } else {
      // partial row: global split x (batch plan) or (b, split) per request
      // without the batch plan (b, split) = (blockIdx.z, blockIdx.x)
      const int64_t row = a.balanced
          ? (int64_t)blockIdx.x * a.HqL + fr
          : ((int64_t)blockIdx.z * a.HqL + fr) * a.num_splits + blockIdx.x;
      *reinterpret_cast<float4*>(a.part_o + row * D + d) = acc;
      if (d == 0) {
        a.part_ml[row * 2 + 0] = M;
        a.part_ml[row * 2 + 1] = Lsum;
      }
    }
  }
}

// Decode of a batch under the span plan (decode.cuh): the same per-split
// work as decode_split_kernel (one 12-warp CTA per SM), run over the
// segments in which this CTA's piece meets the batch's requests.  A separate
// kernel, so that the single-request kernel keeps its straight-line code
// (the same body as a lambda there measured 1.3 us slower per 256K call).
template <int D>
__global__ void __launch_bounds__(12 * 32, 1)
decode_span_kernel(const __grid_constant__ CUtensorMap tmap, const DecodeArgs a) {
  constexpr bool VER = false;
  constexpr int NW = 12;
  using L = DecodeSmem<D, NW>;
  constexpr int NG = L::NG;
  constexpr int SBB = L::SBB;
  constexpr float NEG_INF = -INFINITY;

  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* codes = smem_raw;
  uint8_t* sbuf = codes + L::CODES_BYTES;
  uint4* qsm = reinterpret_cast<uint4*>(sbuf + L::SB_BYTES);
  uint64_t* bars = reinterpret_cast<uint64_t*>(sbuf + L::SB_BYTES + L::QF_BYTES);

  // decode: one CTA per KV head holds its G query heads; verifier: NT CTAs
  // each hold 8 of its G * L (token, head) rows
  const int kvh = VER ? (int)blockIdx.y / a.NT : (int)blockIdx.y;
  const int nt = VER ? (int)blockIdx.y % a.NT : 0;
  const int rows = VER ? min(8, a.G * a.L - 8 * nt) : a.G;
  // row k of this CTA: query token i = (8 nt + k) / G, head h = (8 nt + k) % G;
  // its q, out and partial row within the request is i * Hq + kvh * G + h
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
  int* plan_sh = reinterpret_cast<int*>(sbuf + L::SB_BYTES + L::QF_BYTES + L::BAR_BYTES);
  // the swizzled TMA boxes need a 1024-byte aligned window
  const bool aligned = (smem_u32(smem_raw) & 1023) == 0;
  if (aligned) {   // setup that reads nothing a previous kernel writes
    if (threadIdx.x == 0) prefetch_tensormap(&tmap);
    if (lane == 0) {
      for (int s = 0; s < DSTAGES; ++s) mbar_init(&bars[warp * DSTAGES + s], 1);
      fence_barrier_init();
    }
  }
  // launched with programmatic dependent launch: wait for the previous
  // kernel (e.g. the append that wrote the newest position) before any read
  asm volatile("griddepcontrol.wait;\n" ::: "memory");

  // this warp's ring: bit s holds the parity of the next wait on stage s
  // (a CTA of the span plan runs its ring through several splits)
  uint32_t ph = 0;
  // One split: chunks [c_begin, c_end) of request b (context ctx); its
  // partial rows are prow0 + prow_step * (row within the request), or the
  // output rows when `direct`; owns_last: it holds the request's last chunk
  // (where the fused append stores the step's row).  False when a bounded
  // wait gave up.
  auto run_split = [&](const int b, const int ctx, const int c_begin, const int c_end,
                       const int64_t prow0, const int64_t prow_step, const bool direct,
                       const bool owns_last) -> bool {
    const int n_cta = c_end - c_begin;
    const int my_n = (n_cta > warp) ? (n_cta - warp + NW - 1) / NW : 0;
    auto chunk_of = [&](int it) { return c_begin + warp + it * NW; };

    if (a.knew != nullptr && owns_last) {   // the split holding the last chunk
      // the new row goes to the pool before this split's TMA reads it
      append_new_row<D>(a, b, kvh, ctx - 1, warp, lane);
      fence_proxy_async_global();
      __syncthreads();
      fence_proxy_async_global();
    }
    __syncwarp();

    // ---- query fragments (B operand of QK^T) ---------------------------------
    const bool head_ok = r < rows;
    const uint16_t* qrow = a.q + ((int64_t)b * a.HqL + row_of(head_ok ? r : 0)) * D;
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

    uint32_t qf[NG][4][2];
    float Qg[NG];
  #pragma unroll
    for (int g = 0; g < NG; ++g) {
      float e[16];
      const uint32_t ws[8] = {qlo[g].x, qlo[g].y, qlo[g].z, qlo[g].w,
                              qhi[g].x, qhi[g].y, qhi[g].z, qhi[g].w};
  #pragma unroll
      for (int i = 0; i < 8; ++i) { e[2 * i] = bf16lo_to_f32(ws[i]); e[2 * i + 1] = bf16hi_to_f32(ws[i]); }
      // word W covers d = base..base+7; nib0 -> (base, base+4), nib1 -> (base+1, base+5) x16,
      // nib0 of W>>8 -> (base+2, base+6), nib1 of W>>8 -> (base+3, base+7) x16
  #pragma unroll
      for (int h = 0; h < 2; ++h) {
        const float* x = e + 8 * h;
        qf[g][2 * h + 0][0] = pack_f16x2(x[0] * qs, x[4] * qs);
        qf[g][2 * h + 0][1] = pack_f16x2(x[1] * qs16, x[5] * qs16);
        qf[g][2 * h + 1][0] = pack_f16x2(x[2] * qs, x[6] * qs);
        qf[g][2 * h + 1][1] = pack_f16x2(x[3] * qs16, x[7] * qs16);
      }
      float sum = 0.f;
  #pragma unroll
      for (int i = 0; i < 16; ++i) sum += e[i];
      sum += __shfl_xor_sync(0xffffffffu, sum, 1);
      sum += __shfl_xor_sync(0xffffffffu, sum, 2);
      Qg[g] = sum;
    }
    // QK bias B fragment for head r: k-slot k < NG is Q_k high, NG <= k < 2 NG
    // is Q_{k-NG} low (the bf16 residual); thread c holds slots 2c, 2c+1.
    uint32_t bq = 0;
    {
      float hi[NG], lo[NG];
  #pragma unroll
      for (int g = 0; g < NG; ++g) {
        hi[g] = __bfloat162float(__float2bfloat16_rn(Qg[g]));
        lo[g] = Qg[g] - hi[g];
      }
      if constexpr (NG == 4) {
        if (c == 0) bq = pack_bf16x2(hi[0], hi[1]);
        else if (c == 1) bq = pack_bf16x2(hi[2], hi[3]);
        else if (c == 2) bq = pack_bf16x2(lo[0], lo[1]);
        else bq = pack_bf16x2(lo[2], lo[3]);
      } else {
        if (c == 0) bq = pack_bf16x2(hi[0], hi[1]);
        else if (c == 1) bq = pack_bf16x2(lo[0], lo[1]);
      }
    }
    const float cA = a.scale_log2 * 16777216.f * ldexpf(1.f, qe);
    const float cB = a.scale_log2;

    // ---- page ids: lane i holds the page of this warp's iteration 32k + i ------
    // (two blocks of 32 in flight so the dependent load never stalls an issue)
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

    // ---- TMA producer (lane 0 of each warp feeds its own ring) -------------
    // decode reads each page once per call: evict it from L2 first; the
    // verifier's n-tile CTAs read the same pages, so L2 keeps them normally
    const uint64_t l2pol = VER ? l2_evict_normal_policy() : l2_evict_first_policy();
    uint32_t valid = 0;
    auto issue = [&](int it) {
      const int s = it % DSTAGES;
      if (it >= 32 && (it & 31) == 0) {
        pg_cur = pg_next;
        pg_next = load_pages((it >> 5) + 1);
      }
      const int page = __shfl_sync(0xffffffffu, pg_cur, it & 31);
      const bool ok = page >= 0 && page < a.num_pages;
      if (lane == 0) {
        const int inp = (chunk_of(it) * DTOK) & (a.P - 1);
        uint64_t* bar = &bars[warp * DSTAGES + s];
        if (!ok) {
          flag_error(a.status, JF_DEV_ERR_PAGE_ID);
          mbar_arrive(bar);
        } else {
          uint8_t* kc = codes + (warp * DSTAGES + s) * 2 * L::CODE_BUF;
          uint8_t* ks = sbuf + (warp * DSTAGES + s) * 2 * L::SB_BUF;
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
    };

    const int npro = my_n < DSTAGES ? my_n : DSTAGES;
    for (int it = 0; it < npro; ++it) issue(it);

    // ---- running state ---------------------------------------------------
    DecodeState<NG> st;
    st.init();

    // ldmatrix row address pieces: matrix m = lane>>3 -> (position half, chunk)
    const int ld_t = (lane & 7) + 8 * ((lane >> 3) & 1);
    const int ld_ch = lane >> 4;
    if (warp == 0) {
  #pragma unroll
      for (int g = 0; g < NG; ++g) {
        qsm[(2 * g) * 32 + lane] = make_uint4(qf[g][0][0], qf[g][0][1], qf[g][1][0], qf[g][1][1]);
        qsm[(2 * g + 1) * 32 + lane] = make_uint4(qf[g][2][0], qf[g][2][1], qf[g][3][0], qf[g][3][1]);
      }
    }
    __syncthreads();
    ChunkCtx<NG> cc{qsm + lane, bq, cA, cB, r, c, {}};
  #pragma unroll
    for (int g = 0; g < NG; ++g) cc.koff[g] = swz<L::CB>(ld_t, 2 * g + ld_ch);

    // verifier causal limits: query token i of L sees positions < ctx - L + 1 + i;
    // a chunk below ctx_all is visible to every row (decode: ctx_all = ctx)
    int ctx_all = ctx, lim0 = ctx, lim1 = ctx;
    if constexpr (VER) {
      ctx_all = ctx - a.L + 1;
      lim0 = min(ctx, ctx_all + (8 * nt + 2 * c) / a.G);
      lim1 = min(ctx, ctx_all + (8 * nt + 2 * c + 1) / a.G);
    }
    int done = 0;
    // unrolled by the ring depth, so every stage address is a constant offset
  #pragma unroll DSTAGES
    for (int it = 0; it < my_n; ++it) {
      const int s = it % DSTAGES;
      if (!mbar_wait_bounded(&bars[warp * DSTAGES + s], (ph >> s) & 1u)) {
        if (lane == 0) flag_error(a.status, JF_DEV_ERR_TIMEOUT);
        break;
      }
      ph ^= 1u << s;
      done = it + 1;
      const bool ok = (valid >> s) & 1u;
      const int tokbase = chunk_of(it) * DTOK;
      const uint32_t kc = smem_u32(codes + (warp * DSTAGES + s) * 2 * L::CODE_BUF);
      const uint8_t* ksb = sbuf + (warp * DSTAGES + s) * 2 * L::SB_BUF;
      if (ok && tokbase + DTOK <= (VER ? ctx_all : ctx)) {
        process_chunk<D, true>(st, cc, kc, ksb, 0, 0, 0);
      } else if constexpr (VER) {
        process_chunk<D, false>(st, cc, kc, ksb, ok ? ctx - tokbase : 0,
                                ok ? lim0 - tokbase : 0, ok ? lim1 - tokbase : 0);
      } else {
        const int nv = ok ? ctx - tokbase : 0;
        process_chunk<D, false>(st, cc, kc, ksb, nv, nv, nv);
      }

      __syncwarp();
      if (it + DSTAGES < my_n) {
        fence_proxy_async_smem();
        issue(it + DSTAGES);
      }
    }
    const bool gave_up = done < my_n;
    if (gave_up) {
      // a wait gave up: give copies still in flight a bounded chance to land
      for (int it = done; it < my_n && it < done + DSTAGES; ++it)
        mbar_wait_bounded(&bars[warp * DSTAGES + it % DSTAGES], (ph >> (it % DSTAGES)) & 1u,
                          1u << 16);
    }
    float& m0 = st.m0;
    float& m1 = st.m1;
    float& l0 = st.l0;
    float& l1 = st.l1;
    auto& O = st.O;

    // the merge kernel may start launching; it waits for this grid to finish
    asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory");

    // ---- per-warp finalize ---------------------------------------------------
  #pragma unroll
    for (int o = 4; o < 32; o <<= 1) {
      l0 += __shfl_xor_sync(0xffffffffu, l0, o);
      l1 += __shfl_xor_sync(0xffffffffu, l1, o);
    }
    // bias sums over the 8 lanes of each head pair
    float Bs[NG][2];
  #pragma unroll
    for (int g = 0; g < NG; ++g) {
      Bs[g][0] = st.Bs[g][0];
      Bs[g][1] = st.Bs[g][1];
  #pragma unroll
      for (int o = 4; o < 32; o <<= 1) {
        Bs[g][0] += __shfl_xor_sync(0xffffffffu, Bs[g][0], o);
        Bs[g][1] += __shfl_xor_sync(0xffffffffu, Bs[g][1], o);
      }
    }
    // This warp's ring is idle now (each of its copies has landed and been
    // read), so its O rows (padded by 4 floats: the 128-bit stores of one
    // quarter-warp hit 8 distinct bank groups) and (m, l) per head go into its
    // own stage buffers at once, without waiting for the other warps.
    constexpr int SROW = D + 4;
    constexpr int WCODES = DSTAGES * 2 * L::CODE_BUF;   // one warp's code ring (bytes)
    constexpr int WSB = DSTAGES * 2 * L::SB_BUF;        // one warp's scale/bias ring
    static_assert(8 * SROW * 4 <= WCODES && 8 * 2 * 4 <= WSB, "combine rows fit a warp's ring");
    {
      float* so = reinterpret_cast<float*>(codes + warp * WCODES);   // [8][SROW]
      float* sml = reinterpret_cast<float*>(sbuf + warp * WSB);      // [8][2]
  #pragma unroll
      for (int g = 0; g < NG; ++g) {
  #pragma unroll
        for (int hf = 0; hf < 2; ++hf) {          // d block 64g + 32 hf + 4r + e
  #pragma unroll
          for (int hh = 0; hh < 2; ++hh) {        // head 2c + hh
            if (2 * c + hh < rows) {
              float4 v;
              // 2^24 undoes the fp16 subnormal codes (2^20 for the hi nibbles)
              v.x = fmaf(O[g][0][2 * hf + hh], 16777216.f, Bs[g][hh]);
              v.y = fmaf(O[g][1][2 * hf + hh], 1048576.f, Bs[g][hh]);
              v.z = fmaf(O[g][2][2 * hf + hh], 16777216.f, Bs[g][hh]);
              v.w = fmaf(O[g][3][2 * hf + hh], 1048576.f, Bs[g][hh]);
              *reinterpret_cast<float4*>(so + (2 * c + hh) * SROW + 64 * g + 32 * hf + 4 * r) = v;
            }
          }
        }
      }
      if (r == 0) {
        sml[(2 * c) * 2 + 0] = m0;
        sml[(2 * c) * 2 + 1] = l0;
        sml[(2 * c + 1) * 2 + 0] = m1;
        sml[(2 * c + 1) * 2 + 1] = l1;
      }
    }
    __syncthreads();

    // ---- combine the warps of this CTA --------------------------------------
    // per head: M = max_w m_w, weights 2^(m_w - M) (divided by L when this CTA
    // writes the final output), L = sum_w 2^(m_w - M) l_w; every thread works
    // out the weights of its own head.
    for (int idx = threadIdx.x; idx < rows * (D / 4); idx += blockDim.x) {
      const int h = idx / (D / 4), d = 4 * (idx % (D / 4));
      float mw[NW], lw[NW];
      float M = NEG_INF;
  #pragma unroll
      for (int w = 0; w < NW; ++w) {
        const float2 v = *reinterpret_cast<const float2*>(sbuf + w * WSB + h * 8);
        mw[w] = v.x;
        lw[w] = v.y;
        M = fmaxf(M, v.x);
      }
      float f[NW];
      float Lsum = 0.f;
  #pragma unroll
      for (int w = 0; w < NW; ++w) {
        f[w] = (mw[w] != NEG_INF) ? fast_exp2(mw[w] - M) : 0.f;
        Lsum = fmaf(f[w], lw[w], Lsum);
      }
      const float inv = direct ? (Lsum > 0.f ? 1.f / Lsum : 0.f) : 1.f;
      float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
  #pragma unroll
      for (int w = 0; w < NW; ++w) {
        const float fw = f[w] * inv;
        const float4 v = *reinterpret_cast<const float4*>(
            reinterpret_cast<const float*>(codes + w * WCODES) + h * SROW + d);
        if (fw != 0.f) {
          acc.x = fmaf(fw, v.x, acc.x);
          acc.y = fmaf(fw, v.y, acc.y);
          acc.z = fmaf(fw, v.z, acc.z);
          acc.w = fmaf(fw, v.w, acc.w);
        }
      }
      const int fr = row_of(h);
      if (direct) {
        uint2 o;
        o.x = (uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(acc.x)) |
              ((uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(acc.y)) << 16);
        o.y = (uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(acc.z)) |
              ((uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(acc.w)) << 16);
        *reinterpret_cast<uint2*>(a.out + ((int64_t)b * a.HqL + fr) * D + d) = o;
      } else {
        const int64_t row = prow0 + prow_step * fr;   // this split's partial row
        *reinterpret_cast<float4*>(a.part_o + row * D + d) = acc;
        if (d == 0) {
          a.part_ml[row * 2 + 0] = M;
          a.part_ml[row * 2 + 1] = Lsum;
        }
      }
    }
    // one CTA-wide answer (and the barrier after which a span plan's next
    // split may reuse the rings and query fragments)
    return __syncthreads_or(gave_up ? 1 : 0) == 0;
  };

  if (!aligned) {
    if (threadIdx.x == 0) flag_error(a.status, JF_DEV_ERR_LAYOUT);
    return;
  }
  // pieces of W chunks cut from the batch's chunks laid end to end; piece
  // x meets requests in segments, each a split with partial row x + b
  const long long T = span_total(a, lane);
  const int W = span_width(T, a.budget);
  long long pos = (long long)blockIdx.x * W;
  const long long end = min(pos + W, T);
  while (pos < end) {
    const SpanHit h = span_find(a, pos, lane);
    if (h.b < 0) break;
    // offsets in the request's sequence range: its first SPAN_HDR places stand
    // for the segment setup, then come its chunks
    const int v0 = (int)(pos - h.start);
    const int v1 = (int)(min(end, h.start + h.nch) - h.start);
    const int c0 = max(v0 - SPAN_HDR, 0), c1 = max(v1 - SPAN_HDR, 0);
    const int ctx = checked_ctx(a, h.b, v0);
    if (!run_split(h.b, ctx, c0, c1, ((int64_t)blockIdx.x + h.b) * a.HqL, 1, false,
                   v1 == h.nch))
      return;   // a bounded wait gave up (reported); the CTA stops
    pos = h.start + v1;
  }
}


// Merge for one or a few requests: one CTA per (32-wide slice of head_dim,
// query row, request); its 8 warps take interleaved splits and reduce through
// shared memory, so even one request's merge is spread over the whole GPU.
// The kernel is a chain of dependent loads, so it issues them all at once:
// the context length, every (m, l) row and this thread's partial outputs for
// up to MERGE_SG_BATCH splits are loaded before any is used; rows past the
// split plan are loaded (the workspace holds num_splits rows) and then
// ignored.
constexpr int MERGE_THREADS = 256;
constexpr int MERGE_DSLICE = 32;
constexpr int MERGE_NSG = MERGE_THREADS / MERGE_DSLICE;   // split groups
constexpr int MERGE_SG_BATCH = 16;                        // splits per thread per batch
constexpr int MERGE_MLB = MERGE_SG_BATCH * MERGE_NSG / 32;   // (m, l) rows per lane per batch

template <int D, bool SPAN>
__global__ void __launch_bounds__(MERGE_THREADS) decode_merge_sg_kernel(const DecodeArgs a) {
  // SPAN: partial rows of the span plan.  A template parameter: the span
  // branch in the single-request instance, though never taken, had slowed
  // the 256K call by ~1.2 us.
  __shared__ float red[MERGE_NSG][MERGE_DSLICE];
  // the next kernel in the stream may be scheduled now; it waits for this
  // grid to complete before it reads anything
  asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory");
  // the split kernel's partials must be complete and visible
  asm volatile("griddepcontrol.wait;\n" ::: "memory");
  const int d0 = blockIdx.x * MERGE_DSLICE, hq = blockIdx.y, b = blockIdx.z;
  const int t = threadIdx.x, dd = t % MERGE_DSLICE, sg = t / MERGE_DSLICE;
  const int lane = t & 31;
  // partials of split s: row row0 + s * rs.  Per-request plans put them at
  // ((b Hq + hq) num_splits + s) and are known only after the context is
  // read, so the plan's plan_splits rows are loaded speculatively; the batch
  // plan numbers splits globally (row (g0 + s) Hq + hq) and is worked out
  // first.
  __shared__ int plan_sh[2];
  int S = a.plan_splits;
  int64_t row0 = ((int64_t)b * a.HqL + hq) * a.num_splits;
  int64_t rs = 1;
  int nsplit_bal = 0;
  if (a.balanced) {
    if (t < 32) {
      const BalPlan p = balanced_plan(a, -1, b, lane);
      if (lane == 0) {
        plan_sh[0] = p.g0;
        plan_sh[1] = p.nsplit;
      }
    }
    __syncthreads();
    row0 = (int64_t)plan_sh[0] * a.HqL + hq;
    rs = a.HqL;
    nsplit_bal = plan_sh[1];
    S = nsplit_bal;
  } else if constexpr (SPAN) {
    if (t < 32) {
      const SpanRows sr = span_rows(a, b, lane);
      if (lane == 0) {
        plan_sh[0] = sr.row;
        plan_sh[1] = sr.n;
      }
    }
    __syncthreads();
    row0 = (int64_t)plan_sh[0] * a.HqL + hq;
    rs = a.HqL;
    nsplit_bal = plan_sh[1];
    S = nsplit_bal;
  }
  const float2* ml = reinterpret_cast<const float2*>(a.part_ml) + row0;
  const float* po = a.part_o + row0 * D + d0 + dd;

  const int ctx_raw = a.ctx[b];
  float2 mlv[MERGE_MLB];
  float ov[MERGE_SG_BATCH], mv[MERGE_SG_BATCH];
#pragma unroll
  for (int k = 0; k < MERGE_MLB; ++k) {
    const int s = lane + 32 * k;
    mlv[k] = (s < S) ? ml[s * rs] : make_float2(-INFINITY, 0.f);
  }
#pragma unroll
  for (int u = 0; u < MERGE_SG_BATCH; ++u) {
    const int s = sg + MERGE_NSG * u;
    ov[u] = (s < S) ? po[s * rs * D] : 0.f;
    mv[u] = (s < S) ? ml[s * rs].x : -INFINITY;
  }
  int ctx = ctx_raw;
  const int64_t cap = (int64_t)a.pt_stride * a.P;
  if ((ctx < 0 || ctx > cap) && t == 0 && blockIdx.x == 0 && hq == 0)
    flag_error(a.status, JF_DEV_ERR_POSITION);   // also covers requests with no split
  if (ctx < 0) ctx = 0;
  if (ctx > cap) ctx = (int)cap;
  int nch, cps, nsplit;
  split_plan(ctx, a.plan_splits, nch, cps, nsplit);
  if (a.balanced || SPAN) nsplit = nsplit_bal;
  uint16_t* orow = a.out + ((int64_t)b * a.HqL + hq) * D + d0;
  if (nsplit == 0) {
    if (t < MERGE_DSLICE) orow[t] = 0;
    return;
  }

  // global maximum (every warp finds it itself)
  float M = -INFINITY;
#pragma unroll
  for (int k = 0; k < MERGE_MLB; ++k)
    if (lane + 32 * k < nsplit) M = fmaxf(M, mlv[k].x);
  for (int s = lane + 32 * MERGE_MLB; s < nsplit; s += 32) M = fmaxf(M, ml[s * rs].x);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, o));

  float L = 0.f, acc = 0.f;
  if (M != -INFINITY) {
#pragma unroll
    for (int k = 0; k < MERGE_MLB; ++k)
      if (lane + 32 * k < nsplit && mlv[k].x != -INFINITY)
        L = fmaf(fast_exp2(mlv[k].x - M), mlv[k].y, L);
    for (int s = lane + 32 * MERGE_MLB; s < nsplit; s += 32) {
      const float2 v = ml[s * rs];
      if (v.x != -INFINITY) L = fmaf(fast_exp2(v.x - M), v.y, L);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) L += __shfl_xor_sync(0xffffffffu, L, o);
#pragma unroll
    for (int u = 0; u < MERGE_SG_BATCH; ++u)
      if (sg + MERGE_NSG * u < nsplit && mv[u] != -INFINITY)
        acc = fmaf(fast_exp2(mv[u] - M), ov[u], acc);
    // more splits than one batch covers
    for (int s0 = sg + MERGE_NSG * MERGE_SG_BATCH; s0 < nsplit; s0 += MERGE_NSG * MERGE_SG_BATCH) {
#pragma unroll
      for (int u = 0; u < MERGE_SG_BATCH; ++u) {
        const int s = s0 + MERGE_NSG * u;
        ov[u] = (s < nsplit) ? po[s * rs * D] : 0.f;
        mv[u] = (s < nsplit) ? ml[s * rs].x : -INFINITY;
      }
#pragma unroll
      for (int u = 0; u < MERGE_SG_BATCH; ++u)
        if (mv[u] != -INFINITY) acc = fmaf(fast_exp2(mv[u] - M), ov[u], acc);
    }
  }
  red[sg][dd] = acc;
  __syncthreads();
  if (t < MERGE_DSLICE) {
    float o = 0.f;
#pragma unroll
    for (int k = 0; k < MERGE_NSG; ++k) o += red[k][t];
    orow[t] = __bfloat16_as_ushort(__float2bfloat16_rn(L > 0.f ? o / L : 0.f));
  }
}

// Merge for batches (one CTA per query row and request).  D / 2 threads,
// each owning two adjacent columns of the output row.  Every warp works out the row's
// reference maximum M itself from the splits' (m, l) pairs (lane j holds
// splits j and j + 32 of a batch), and each thread sums its two columns over
// the splits in split order, the weights 2^(m_s - M) passed along by
// shuffles:
//   o = sum_s 2^{m_s - M} O_s / sum_s 2^{m_s - M} l_s.
// A batch's loads are all issued before any is used.  Per-request plans are
// known only once the context length is read, so the first batch of their
// rows is loaded speculatively and rows past the plan are ignored (whatever
// the workspace holds there).
constexpr int MERGE_BATCH = 64;   // splits per batch: two per lane for the weights

template <int D, bool SPAN>
__global__ void __launch_bounds__(D / 2) decode_merge_kernel(const DecodeArgs a) {
  // the next kernel in the stream may be scheduled now; it waits for this
  // grid to complete before it reads anything
  asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory");
  // the split kernel's partials must be complete and visible
  asm volatile("griddepcontrol.wait;\n" ::: "memory");
  const int hq = blockIdx.x, b = blockIdx.y;
  const int t = threadIdx.x, lane = t & 31;
  int64_t row0, rs;   // partials of split s: row row0 + s * rs
  int S, nsplit_bal = 0;
  if (a.balanced) {   // every warp works the plan out itself
    const BalPlan p = balanced_plan(a, -1, b, lane);
    row0 = (int64_t)p.g0 * a.HqL + hq;
    rs = a.HqL;
    nsplit_bal = p.nsplit;
    S = p.nsplit;
  } else if constexpr (SPAN) {
    const SpanRows sr = span_rows(a, b, lane);
    row0 = (int64_t)sr.row * a.HqL + hq;
    rs = a.HqL;
    nsplit_bal = sr.n;
    S = sr.n;
  } else {
    row0 = ((int64_t)b * a.HqL + hq) * a.num_splits;
    rs = 1;
    S = a.plan_splits;
  }
  const float2* ml = reinterpret_cast<const float2*>(a.part_ml) + row0;
  const float2* po = reinterpret_cast<const float2*>(a.part_o + row0 * D) + t;
  const int64_t ostride = rs * (D / 2);   // float2 elements between split rows

  const int ctx_raw = a.ctx[b];
  float2 ml0 = (lane < S) ? ml[lane * rs] : make_float2(-INFINITY, 0.f);
  float2 ml1 = (lane + 32 < S) ? ml[(lane + 32) * rs] : make_float2(-INFINITY, 0.f);
  float2 ov[MERGE_BATCH];
#pragma unroll
  for (int j = 0; j < MERGE_BATCH; ++j)
    ov[j] = (j < S) ? po[j * ostride] : make_float2(0.f, 0.f);

  int ctx = ctx_raw;
  const int64_t cap = (int64_t)a.pt_stride * a.P;
  if ((ctx < 0 || ctx > cap) && t == 0 && hq == 0)
    flag_error(a.status, JF_DEV_ERR_POSITION);   // also covers requests with no split
  if (ctx < 0) ctx = 0;
  if (ctx > cap) ctx = (int)cap;
  int nch, cps, nsplit;
  split_plan(ctx, a.plan_splits, nch, cps, nsplit);
  if (a.balanced || SPAN) nsplit = nsplit_bal;
  uint32_t* orow = reinterpret_cast<uint32_t*>(a.out + ((int64_t)b * a.HqL + hq) * D) + t;
  if (nsplit == 0) {
    *orow = 0u;
    return;
  }

  // reference maximum over every split (each warp on its own)
  float M = fmaxf(lane < nsplit ? ml0.x : -INFINITY, lane + 32 < nsplit ? ml1.x : -INFINITY);
  for (int s = lane + MERGE_BATCH; s < nsplit; s += 32) M = fmaxf(M, ml[s * rs].x);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, o));

  float L = 0.f;
  float2 acc = make_float2(0.f, 0.f);
  for (int s0 = 0; s0 < nsplit; s0 += MERGE_BATCH) {
    if (s0 > 0) {   // the next batch (more splits than one batch covers)
      ml0 = (s0 + lane < nsplit) ? ml[(s0 + lane) * rs] : make_float2(-INFINITY, 0.f);
      ml1 = (s0 + lane + 32 < nsplit) ? ml[(s0 + lane + 32) * rs]
                                      : make_float2(-INFINITY, 0.f);
#pragma unroll
      for (int j = 0; j < MERGE_BATCH; ++j)
        ov[j] = (s0 + j < nsplit) ? po[(s0 + j) * ostride] : make_float2(0.f, 0.f);
    }
    const float w0 = (s0 + lane < nsplit && ml0.x != -INFINITY) ? fast_exp2(ml0.x - M) : 0.f;
    const float w1 =
        (s0 + lane + 32 < nsplit && ml1.x != -INFINITY) ? fast_exp2(ml1.x - M) : 0.f;
    if (w0 != 0.f) L = fmaf(w0, ml0.y, L);   // rows past the plan hold anything
    if (w1 != 0.f) L = fmaf(w1, ml1.y, L);
#pragma unroll
    for (int j = 0; j < MERGE_BATCH; ++j) {
      const float w = __shfl_sync(0xffffffffu, j < 32 ? w0 : w1, j & 31);
      if (s0 + j < nsplit && w != 0.f) {
        acc.x = fmaf(w, ov[j].x, acc.x);
        acc.y = fmaf(w, ov[j].y, acc.y);
      }
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) L += __shfl_xor_sync(0xffffffffu, L, o);
  const float inv = L > 0.f ? 1.f / L : 0.f;
  *orow = (uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(acc.x * inv)) |
          ((uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(acc.y * inv)) << 16);
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------
constexpr int BAL_MAX_B = 1024;   // batch plan limit (each plan reads every context length)

// SMs of the current device (cached per device)
int sm_count() {
  static int cache[256] = {0};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 256) return 152;
  if (cache[dev] == 0) {
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0)
      n = 152;
    cache[dev] = n;
  }
  return cache[dev];
}

int smem_optin(const void* kernel, int bytes) {
  static std::mutex mu;
  static std::vector<std::pair<const void*, int>> done;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return JF_ERR_CUDA;
  std::lock_guard<std::mutex> lock(mu);
  for (const auto& e : done)
    if (e.first == kernel && e.second == dev) return JF_OK;
  if (cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes) !=
      cudaSuccess)
    return JF_ERR_CUDA;
  done.emplace_back(kernel, dev);
  return JF_OK;
}

// rows (positions) of one TMA box of the decode code tensor map
int decode_box_rows() { return DTOK; }

size_t decode_workspace_bytes(int64_t B, int64_t Hq, int64_t D, int64_t S) {
  const int64_t rows = B * Hq * S;
  const int64_t ml = (rows * 8 + 255) / 256 * 256;
  return (size_t)(256 + ml + rows * D * 4);
}

// Merge phase, launched with programmatic dependent launch after the split
// kernel.
int launch_decode_merge(const DecodeArgs& a, int D, int B, cudaStream_t stream) {
  cudaLaunchAttribute pdl[1];
  pdl[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  pdl[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t mc = {};
  // a few rows: 32-column slices with 8 split groups each (more CTAs, fewer
  // loads per thread); a batch: one CTA per row
  const bool sg = (int64_t)B * a.HqL * (D / MERGE_DSLICE) <= 4 * (int64_t)sm_count();
  mc.gridDim = sg ? dim3((unsigned)(D / MERGE_DSLICE), (unsigned)a.HqL, (unsigned)B)
                  : dim3((unsigned)a.HqL, (unsigned)B, 1u);
  mc.blockDim = dim3(sg ? (unsigned)MERGE_THREADS : (unsigned)(D / 2));
  mc.dynamicSmemBytes = 0;
  mc.stream = stream;
  mc.attrs = pdl;
  mc.numAttrs = 1;
  cudaError_t e;
  if (sg) {
    if (a.span)
      e = (D == 256) ? cudaLaunchKernelEx(&mc, decode_merge_sg_kernel<256, true>, a)
                     : cudaLaunchKernelEx(&mc, decode_merge_sg_kernel<128, true>, a);
    else
      e = (D == 256) ? cudaLaunchKernelEx(&mc, decode_merge_sg_kernel<256, false>, a)
                     : cudaLaunchKernelEx(&mc, decode_merge_sg_kernel<128, false>, a);
  } else {
    if (a.span)
      e = (D == 256) ? cudaLaunchKernelEx(&mc, decode_merge_kernel<256, true>, a)
                     : cudaLaunchKernelEx(&mc, decode_merge_kernel<128, true>, a);
    else
      e = (D == 256) ? cudaLaunchKernelEx(&mc, decode_merge_kernel<256, false>, a)
                     : cudaLaunchKernelEx(&mc, decode_merge_kernel<128, false>, a);
  }
  return e == cudaSuccess ? JF_OK : JF_ERR_CUDA;
}

template <int D, bool VER, int NW, bool SPAN>
static int launch_decode_t(const CUtensorMap& tmap, const DecodeArgs& a, int B,
                           cudaStream_t stream) {
  using L = DecodeSmem<D, NW>;
  static_assert(!SPAN || (NW == 12 && !VER), "the span kernel is the 12-warp decode");
  const void* kernel = SPAN ? (const void*)decode_span_kernel<D>
                            : (const void*)decode_split_kernel<D, VER, NW>;
  if (smem_optin(kernel, L::TOTAL) != JF_OK) return JF_ERR_CUDA;
  // Both kernels use programmatic dependent launch: each may be scheduled
  // while the previous kernel in the stream drains, and waits (griddepcontrol)
  // before it reads anything that kernel wrote.
  cudaLaunchAttribute pdl[1];
  pdl[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  pdl[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t cfg = {};
  // span plan: budget pieces per KV head; batch plan: a.budget + B CTAs per
  // KV head cover every split (sum_b n_b <= T / cps + B <= budget + B);
  // per-request plans: plan_splits per request
  cfg.gridDim = SPAN ? dim3((unsigned)a.budget, (unsigned)a.Hkv, 1u)
              : a.balanced ? dim3((unsigned)(a.budget + B), (unsigned)(a.Hkv * a.NT), 1u)
                           : dim3((unsigned)a.plan_splits, (unsigned)(a.Hkv * a.NT), (unsigned)B);
  cfg.blockDim = dim3(NW * 32);
  cfg.dynamicSmemBytes = L::TOTAL;
  cfg.stream = stream;
  cfg.attrs = pdl;
  cfg.numAttrs = 1;
  cudaError_t e;
  if constexpr (SPAN)
    e = cudaLaunchKernelEx(&cfg, decode_span_kernel<D>, tmap, a);
  else
    e = cudaLaunchKernelEx(&cfg, decode_split_kernel<D, VER, NW>, tmap, a);
  if (e != cudaSuccess) return JF_ERR_CUDA;
  if (a.span || a.balanced || a.plan_splits > 1) return launch_decode_merge(a, D, B, stream);
  return JF_OK;
}

// Warps per split CTA (the NW template parameter) and the plan.  Two 6-warp
// CTAs on one SM do not share it evenly: the CTA placed first keeps issue
// priority and ends its share ~4 us (of ~50) before the other, so decode runs
// one 12-warp CTA per SM: a single request with per-request splits, a batch
// with the span plan (equal pieces, so the longer pieces of 12-warp CTAs
// leave no unevenness).  The packed verifier with at most 8 rows per KV head
// (one n-tile) keeps 6-warp CTAs (measured faster) and the batch plan of
// whole-request pieces (more rows go to the warp-pair kernel, verify.cu);
// many requests that do not fit one wave of 12-warp CTAs use 6-warp CTAs.
static int decode_warps(int batch, int num_splits, int Hkv, int NT) {
  if (NT > 1) return 6;
  if (batch > 1 && batch <= BAL_MAX_B && num_splits > 1) return 12;   // span plan
  return (batch == 1 || (int64_t)batch * Hkv * NT * num_splits <= sm_count()) ? 12 : 6;
}

int launch_decode(const Geom& g, const jf_kv_pool& pool, const CUtensorMap& tmap,
                  const int32_t* page_table, int32_t pt_stride, const int32_t* context_lens,
                  int32_t batch, const void* q, int32_t Hq, float softmax_scale, void* out,
                  void* workspace, int32_t num_splits, cudaStream_t stream, const void* k_new,
                  const void* v_new, int32_t q_len) {
  DecodeArgs a;
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
  a.scale_log2 = softmax_scale * 1.4426950408889634f;
  a.B = batch;
  const int nw = decode_warps(batch, num_splits, g.Hkv, a.NT);
  const int per_sm = 12 / nw;   // split CTAs resident per SM
  const int slots = (per_sm * sm_count() + g.Hkv * a.NT - 1) / (g.Hkv * a.NT);
  // per-request plans: one CTA wave (12-warp CTAs) or the caller's cap
  a.plan_splits = (nw == 12 && num_splits > slots) ? slots : num_splits;
  // Batches of up to BAL_MAX_B requests size their splits for the whole
  // batch: decode with the span plan (one piece per CTA slot, within the
  // workspace's B * num_splits rows: budget <= B (num_splits - 1) + 1), the
  // verifier with balanced_plan (whole-request pieces, fewer than
  // B * num_splits minus B/2 for rounding).
  const bool batch_plan = batch > 1 && batch <= BAL_MAX_B && num_splits > 1;
  a.span = (batch_plan && q_len == 1) ? 1 : 0;
  a.balanced = (batch_plan && q_len > 1) ? 1 : 0;
  a.budget = 1;
  if (a.span) {
    const int64_t fit = (int64_t)batch * (num_splits - 1) + 1;
    a.budget = (int)(fit < slots ? fit : slots);
  } else if (a.balanced) {
    const int64_t fit = (int64_t)batch * num_splits - batch;
    const int64_t cap = fit < slots ? fit : slots;
    a.budget = (int)(cap - batch / 2 > 1 ? cap - batch / 2 : 1);
  }
  const bool d256 = g.D == 256;
  if (q_len > 1 && a.NT >= 2) {
    // packed verifier with more than 8 rows per KV head: warp pairs share the
    // unpacking (verify.cu), one 8-warp CTA per SM, ncta CTAs per KV head
    const int per_head = g.Hkv * verify_pair_ctas(a.NT);
    const int vslots = sm_count() / per_head > 1 ? sm_count() / per_head : 1;
    a.plan_splits = num_splits < vslots ? num_splits : vslots;
    if (a.balanced) {
      const int64_t fit = (int64_t)batch * num_splits - batch;
      const int64_t cap = fit < vslots ? fit : vslots;
      a.budget = (int)(cap - batch / 2 > 1 ? cap - batch / 2 : 1);
    }
    return launch_verify_pairs(tmap, a, g.D, batch, stream);
  }
  if (q_len > 1)
    return d256 ? launch_decode_t<256, true, 6, false>(tmap, a, batch, stream)
                : launch_decode_t<128, true, 6, false>(tmap, a, batch, stream);
  if (a.span)
    return d256 ? launch_decode_t<256, false, 12, true>(tmap, a, batch, stream)
                : launch_decode_t<128, false, 12, true>(tmap, a, batch, stream);
  if (nw == 12)
    return d256 ? launch_decode_t<256, false, 12, false>(tmap, a, batch, stream)
                : launch_decode_t<128, false, 12, false>(tmap, a, batch, stream);
  return d256 ? launch_decode_t<256, false, 6, false>(tmap, a, batch, stream)
              : launch_decode_t<128, false, 6, false>(tmap, a, batch, stream);
}

}  // namespace jfkv
