// TQ4 codec parameters as the kernels receive them (by value): the fp32
// centroids, their fp32 midpoints, and the random-sign diagonals as bit masks
// (Sec. 3.1 Eq. 4; App. A.1 Table 3); and the warp-wide Hadamard transform
// the TQ4 kernels share.
#pragma once
#include "common.cuh"

namespace jfkv {

struct Tq4Params {
  float c[16];      // centroids, ascending
  float t[15];      // fp32 midpoints t_k = fp32(fp32(c_k + c_{k+1}) * 0.5)
  float tq[15];     // fp32(sqrt(d) t_k): thresholds in units of rho (fast path)
  uint32_t sk[8];   // sign bits of S for K: bit j set <=> S_jj = -1
  uint32_t sv[8];   // ... for V
  int32_t exact_all;   // thresholds closer than 2^-12 rho apart: every index takes the fp64 path
};

// In-place unnormalized Walsh-Hadamard transform (Sylvester order) of a
// vector spread over a warp, lane l holding elements E l .. E l + E - 1.
template <typename T, int E>
__device__ __forceinline__ void warp_fwht(T (&u)[E], int lane) {
#pragma unroll
  for (int h = 1; h < E; h <<= 1) {
#pragma unroll
    for (int i = 0; i < E; ++i) {
      if (!(i & h)) {
        const T a = u[i], b = u[i + h];
        u[i] = a + b;
        u[i + h] = a - b;
      }
    }
  }
#pragma unroll
  for (int m = 1; m < 32; m <<= 1) {
    // lower lane: u + o; upper lane: o - u (one rounding either way)
    const T sg = (lane & m) ? T(-1) : T(1);
#pragma unroll
    for (int i = 0; i < E; ++i) {
      const T o = __shfl_xor_sync(0xffffffffu, u[i], m);
      u[i] = fma(u[i], sg, o);
    }
  }
}

}  // namespace jfkv
