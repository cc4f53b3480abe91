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

// Coefficients of the log-likelihood difference dLL(x) = LL_v - LL_t of eq. (8):
//   dLL = sum_d ga[d] x_d^2 + gb[d] x_d + gc,
//   ga = (var_v - var_t) / (2 var_v var_t), gb = (mu_v var_t - mu_t var_v) / (var_v var_t),
//   gc = -1/2 sum_d [ log(var_v / var_t) + (mu_v^2 var_t - mu_t^2 var_v) / (var_v var_t) ].
// Writing the difference directly avoids subtracting two log-likelihoods of size ~d.
// Entries d..dpad-1 are zero. Returns gc; `red` needs (blockDim/32 + 1) floats.
__device__ inline float gauss_coefficients(const float* __restrict__ mu, const float* __restrict__ var,
                                    int d, int dpad, float* ga, float* gb, float* red,
                                    uint32_t* status) {
  float part = 0.f;
  bool bad = false;
  for (int i = threadIdx.x; i < dpad; i += blockDim.x) {
    float a = 0.f, b = 0.f;
    if (i < d) {
      const float vv = var[i], vt = var[d + i], mv = mu[i], mt = mu[d + i];
      if (!(vv > 0.f) || !(vt > 0.f) || !isfinite(vv) || !isfinite(vt) || !isfinite(mv) ||
          !isfinite(mt))
        bad = true;
      const float pv = vv * vt;
      a = (vv - vt) / (2.f * pv);
      b = (mv * vt - mt * vv) / pv;
      part += log1pf((vv - vt) / vt) + (mv * mv * vt - mt * mt * vv) / pv;
    }
    ga[i] = a;
    gb[i] = b;
  }
  if (bad) atomicOr(status, kStatusData);
  part = warp_sum(part);
  const int nw = blockDim.x >> 5;
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = part;
  __syncthreads();
  if (threadIdx.x == 0) {
    float t = 0.f;
    for (int w = 0; w < nw; ++w) t += red[w];
    red[nw] = -0.5f * t;
  }
  __syncthreads();
  return red[nw];
}

__device__ __forceinline__ float sigmoid_acc(float y) {
  if (y >= 0.f) return 1.f / (1.f + expf(-y));
  const float e = expf(y);
  return e / (1.f + e);
}

}  // namespace smoes
