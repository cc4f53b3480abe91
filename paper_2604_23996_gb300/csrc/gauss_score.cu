// gauss_score.cu -- standalone Gaussian-statistics modality score, eqs. (8)-(9).
//
// M[j] = softmax over {vision, text} of LL[j, m] / tau. For two modalities this is
// M_v = sigmoid((LL_v - LL_t) / tau), with the log-likelihood difference evaluated directly as
// sum_d ga[d] x_d^2 + gb[d] x_d + gc (coefficients in shared memory). One warp per token row,
// 16-byte vector loads; the kernel is bound by the read of X.
#include <cuda_bf16.h>

#include "device_common.cuh"
#include "smoes_internal.cuh"

namespace smoes {
namespace {

template <bool kBf16>
__global__ void __launch_bounds__(256) k_gauss_score(const GaussParams p) {
  extern __shared__ float gsm[];
  const int dpad = round_up(p.d, 256);
  float* ga = gsm;
  float* gb = ga + dpad;
  float* red = gb + dpad;
  const float gc = gauss_coefficients(p.mu, p.var, p.d, dpad, ga, gb, red, p.status);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int per = kBf16 ? 8 : 4;                      // elements per 16-byte load
  constexpr int kU = 4;                               // 16-byte loads in flight per lane
  for (int j = blockIdx.x * 8 + warp; j < p.T; j += gridDim.x * 8) {
    float acc = 0.f;
    if (kBf16) {
      const __nv_bfloat16* row = static_cast<const __nv_bfloat16*>(p.X) + static_cast<size_t>(j) * p.d;
      for (int c0 = lane * per; c0 < p.d; c0 += 32 * per * kU) {
        uint4 u[kU];
#pragma unroll
        for (int q = 0; q < kU; ++q) {
          const int c = c0 + q * 32 * per;
          u[q] = c < p.d ? __ldg(reinterpret_cast<const uint4*>(row + c)) : make_uint4(0, 0, 0, 0);
        }
#pragma unroll
        for (int q = 0; q < kU; ++q) {
          const int c = c0 + q * 32 * per;
          if (c >= p.d) break;
          const uint32_t w[4] = {u[q].x, u[q].y, u[q].z, u[q].w};
#pragma unroll
          for (int r = 0; r < 4; ++r) {
            const float x0 = __uint_as_float(w[r] << 16), x1 = __uint_as_float(w[r] & 0xffff0000u);
            acc = fmaf(x0, fmaf(ga[c + 2 * r], x0, gb[c + 2 * r]), acc);
            acc = fmaf(x1, fmaf(ga[c + 2 * r + 1], x1, gb[c + 2 * r + 1]), acc);
          }
        }
      }
    } else {
      const float* row = static_cast<const float*>(p.X) + static_cast<size_t>(j) * p.d;
      for (int c0 = lane * per; c0 < p.d; c0 += 32 * per * kU) {
        float4 u[kU];
#pragma unroll
        for (int q = 0; q < kU; ++q) {
          const int c = c0 + q * 32 * per;
          u[q] = c < p.d ? __ldg(reinterpret_cast<const float4*>(row + c)) : make_float4(0.f, 0.f, 0.f, 0.f);
        }
#pragma unroll
        for (int q = 0; q < kU; ++q) {
          const int c = c0 + q * 32 * per;
          if (c >= p.d) break;
          acc = fmaf(u[q].x, fmaf(ga[c], u[q].x, gb[c]), acc);
          acc = fmaf(u[q].y, fmaf(ga[c + 1], u[q].y, gb[c + 1]), acc);
          acc = fmaf(u[q].z, fmaf(ga[c + 2], u[q].z, gb[c + 2]), acc);
          acc = fmaf(u[q].w, fmaf(ga[c + 3], u[q].w, gb[c + 3]), acc);
        }
      }
    }
    acc = warp_sum(acc);
    if (lane == 0) {
      const float y = (acc + gc) * p.inv_tau;
      *reinterpret_cast<float2*>(p.M + 2 * static_cast<size_t>(j)) = make_float2(sigmoid_acc(y), sigmoid_acc(-y));
    }
  }
}

}  // namespace

cudaError_t launch_gauss_score(const GaussParams& p, smoes_dtype dt, int n_sms, cudaStream_t s) {
  const int dpad = round_up(p.d, 256);
  const size_t smem = sizeof(float) * (2 * dpad + 16);
  int grid = (p.T + 7) / 8;
  if (grid > 4 * n_sms) grid = 4 * n_sms;
  if (grid < 1) grid = 1;
  if (dt == SMOES_BF16) {
    cudaError_t e = cudaFuncSetAttribute(k_gauss_score<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    k_gauss_score<true><<<grid, 256, smem, s>>>(p);
  } else {
    cudaError_t e = cudaFuncSetAttribute(k_gauss_score<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    k_gauss_score<false><<<grid, 256, smem, s>>>(p);
  }
  return cudaGetLastError();
}

}  // namespace smoes
