// TQ4 codec parameters as the kernels receive them (by value): the fp32
// centroids, their fp32 midpoints, and the random-sign diagonals as bit masks
// (Sec. 3.1 Eq. 4; App. A.1 Table 3).
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

}  // namespace jfkv
