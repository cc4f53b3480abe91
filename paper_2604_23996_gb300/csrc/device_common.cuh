// device_common.cuh -- small device helpers shared by several kernels.
#pragma once

#include <cstdint>

#include "smoes_internal.cuh"

namespace smoes {

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ double warp_sum_d(double v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Coefficients of one feature of the Gaussian log-likelihood difference of eq. (8),
//   dLL(x) = LL_v - LL_t = sum_d ga[d] x_d^2 + gb[d] x_d + gc,
//   ga = (var_v - var_t) / (2 var_v var_t),  gb = (mu_v var_t - mu_t var_v) / (var_v var_t),
//   gc = -1/2 sum_d [ log(var_v / var_t) + (mu_v^2 var_t - mu_t^2 var_v) / (var_v var_t) ];
// c receives the feature's term of the sum in gc. Differences are formed before the (fast,
// 2-ulp) reciprocals so that nearly equal statistics lose no accuracy. Returns false for
// non-positive or non-finite statistics.
__device__ __forceinline__ bool gauss_coef_feature(float mv, float mt, float vv, float vt, float& a,
                                                   float& b, float& c) {
  const float ivv = __fdividef(1.f, vv), ivt = __fdividef(1.f, vt);
  const float ip = ivv * ivt;
  a = 0.5f * (vv - vt) * ip;
  b = fmaf(mv, vt, -mt * vv) * ip;
  c = log1pf((vv - vt) * ivt) + fmaf(mv * mv, vt, -(mt * mt) * vv) * ip;
  return vv > 0.f && vt > 0.f && isfinite(vv) && isfinite(vt) && isfinite(mv) && isfinite(mt);
}

// Constant term gc of the Gaussian log-likelihood difference from the coefficient kernel's
// per-block partials, summed in block order.
__device__ __forceinline__ float gauss_gc(const float* gcoef, int dcoef) {
  const float* part = gcoef + 2 * static_cast<size_t>(dcoef);
  float t = 0.f;
  for (int b = 0; b < dcoef / 256; ++b) t += part[b];
  return -0.5f * t;
}

__device__ __forceinline__ float sigmoid_acc(float y) {
  if (y >= 0.f) return 1.f / (1.f + expf(-y));
  const float e = expf(y);
  return e / (1.f + e);
}

// Transpose-reduce of 32 values per lane: afterwards v[0] of lane l holds the sum over the 32
// lanes of their v[l] (a fixed butterfly tree, 31 shuffles).
__device__ __forceinline__ float warp_transpose_sum(float (&v)[32]) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int s = 16; s >= 1; s >>= 1) {
    const bool upper = (lane & s) != 0;
#pragma unroll
    for (int i = 0; i < s; ++i) {
      const float send = upper ? v[i] : v[i + s];
      const float keep = upper ? v[i + s] : v[i];
      v[i] = keep + __shfl_xor_sync(0xffffffffu, send, s);
    }
  }
  return v[0];
}

}  // namespace smoes
