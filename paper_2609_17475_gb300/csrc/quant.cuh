// Affine 4-bit group-64 quantizer shared by the append kernel and the fused
// append-then-attend decode (Sec. 3.3 pending cache writes; App. A.1 Table 3:
// midpoint thresholds, a value above a midpoint by a strict > takes the upper
// code).  All arithmetic is IEEE fp32 with explicit rounding intrinsics (no
// contraction) so the codes match the CPU oracle bit for bit.
#pragma once
#include "common.cuh"

namespace jfkv {

// One vector of D bf16 elements is spread over D/8 consecutive lanes; lane li
// holds elements 8 li .. 8 li + 7 in x.  A 64-element group spans 8 lanes and
// its min/max is reduced with three xor-shuffles, so every lane of the warp
// must call this (inactive lanes pass zeros).  Returns this lane's 8 codes
// (element 8 li + i in bits 4i .. 4i + 3) and the group's bf16 scale and bias.
__device__ __forceinline__ uint32_t quantize8(const float (&x)[8], __nv_bfloat16& scale_h,
                                              __nv_bfloat16& bias_h) {
  float mn = x[0], mx = x[0];
#pragma unroll
  for (int i = 1; i < 8; ++i) { mn = fminf(mn, x[i]); mx = fmaxf(mx, x[i]); }
#pragma unroll
  for (int o = 1; o < 8; o <<= 1) {
    mn = fminf(mn, __shfl_xor_sync(0xffffffffu, mn, o));
    mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
  }
  const float bias = __fadd_rn(mn, 0.0f);                 // -0 -> +0
  const float range = __fsub_rn(mx, mn);
  scale_h = __float2bfloat16_rn(__fdiv_rn(range, 15.0f));
  bias_h = __float2bfloat16_rn(bias);
  const float scale = __bfloat162float(scale_h);
  uint32_t word = 0;
  if (scale != 0.0f) {
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const float r = __fdiv_rn(__fsub_rn(x[i], bias), scale);
      // code = number of thresholds k + 1/2 (k = 0..14) that r strictly exceeds
      int c = (int)ceilf(__fsub_rn(r, 0.5f));
      c = min(max(c, 0), 15);
      word |= (uint32_t)c << (4 * i);
    }
  }
  return word;
}

// 8 bf16 elements (16 bytes) -> floats
__device__ __forceinline__ void load8_bf16(const uint16_t* src, float (&x)[8]) {
  const uint4 w = *reinterpret_cast<const uint4*>(src);
  x[0] = bf16lo_to_f32(w.x); x[1] = bf16hi_to_f32(w.x);
  x[2] = bf16lo_to_f32(w.y); x[3] = bf16hi_to_f32(w.y);
  x[4] = bf16lo_to_f32(w.z); x[5] = bf16hi_to_f32(w.z);
  x[6] = bf16lo_to_f32(w.w); x[7] = bf16hi_to_f32(w.w);
}

// Store lane li's code word and (first lane of each group) the group's
// scale/bias word into slot `slot` of KV head `head` of a page record.
template <int D>
__device__ __forceinline__ void store_quantized(uint8_t* page_base, int64_t codes_region,
                                                int64_t sb_region, int P, int head, int slot,
                                                int kind, int li, uint32_t word,
                                                __nv_bfloat16 scale_h, __nv_bfloat16 bias_h) {
  constexpr int CB = D / 2;
  constexpr int SBB = D / 16;   // 4 bytes per 64-group
  const int64_t vrow = (int64_t)head * P + slot;
  *reinterpret_cast<uint32_t*>(page_base + kind * codes_region + vrow * CB + li * 4) = word;
  if ((li & 7) == 0) {
    const uint32_t sb = (uint32_t)__bfloat16_as_ushort(scale_h) |
                        ((uint32_t)__bfloat16_as_ushort(bias_h) << 16);
    *reinterpret_cast<uint32_t*>(page_base + 2 * codes_region + kind * sb_region + vrow * SBB +
                                 (li >> 3) * 4) = sb;
  }
}

}  // namespace jfkv
