// gauss_score.cu -- Gaussian-statistics modality score, eqs. (8)-(9).
//
// The log-likelihood difference of token x between the vision and text Gaussians is written
// directly as a quadratic in x (gauss_coef_feature), avoiding the difference of two
// log-likelihoods of size ~d. k_gauss_coef evaluates the coefficients once per call (one thread
// per feature) for the standalone score kernel below and the fp32 forward; the bf16 forward
// evaluates its own copy. For two modalities the softmax of eq. (9) is
// M_v = sigmoid(dLL / tau), M_t = sigmoid(-dLL / tau).
#include <cuda_bf16.h>

#include "device_common.cuh"
#include "ptx.cuh"
#include "smoes_internal.cuh"

namespace smoes {
namespace {

// coef = ga[dcoef] | gb[dcoef] | part[dcoef / 256]; entries d..dcoef-1 of ga, gb are zero and
// part[b] is the fixed-order sum of block b's constant terms (gc = -part_total / 2).
__global__ void __launch_bounds__(256) k_gauss_coef(const float* __restrict__ mu,
                                                    const float* __restrict__ var, int d, int dcoef,
                                                    float* __restrict__ coef, uint32_t* status) {
  __shared__ float red[8];
  pdl_wait();
  pdl_trigger();                            // the consumer may start its own prologue now
  const int i = blockIdx.x * 256 + threadIdx.x;
  float a = 0.f, b = 0.f, c = 0.f;
  if (i < d && !gauss_coef_feature(mu[i], mu[d + i], var[i], var[d + i], a, b, c))
    atomicOr(status, kStatusData);
  coef[i] = a;
  coef[dcoef + i] = b;
  c = warp_sum(c);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = c;
  __syncthreads();
  if (threadIdx.x == 0) {
    float t = 0.f;
    for (int w = 0; w < 8; ++w) t += red[w];
    coef[2 * dcoef + blockIdx.x] = t;
  }
}

template <bool kBf16>
__global__ void __launch_bounds__(256) k_gauss_score(const GaussParams p) {
  extern __shared__ float gsm[];
  const int dpad = round_up(p.d, 256);
  float* ga = gsm;
  float* gb = ga + dpad;
  pdl_wait();                               // coefficients of the kernel launched just before
  pdl_trigger();
  for (int i = threadIdx.x; i < dpad; i += 256) {
    ga[i] = p.gcoef[i];
    gb[i] = p.gcoef[p.dcoef + i];
  }
  const float gc = gauss_gc(p.gcoef, p.dcoef);
  __syncthreads();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int per = kBf16 ? 8 : 4;                      // elements per 16-byte load
  constexpr int kU = 4;                               // 16-byte loads in flight per lane
  for (int j = blockIdx.x * 8 + warp; j < p.T; j += gridDim.x * 8) {
    float acc[2] = {0.f, 0.f};
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
            acc[0] = fmaf(x0, fmaf(ga[c + 2 * r], x0, gb[c + 2 * r]), acc[0]);
            acc[1] = fmaf(x1, fmaf(ga[c + 2 * r + 1], x1, gb[c + 2 * r + 1]), acc[1]);
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
          acc[0] = fmaf(u[q].x, fmaf(ga[c], u[q].x, gb[c]), acc[0]);
          acc[1] = fmaf(u[q].y, fmaf(ga[c + 1], u[q].y, gb[c + 1]), acc[1]);
          acc[0] = fmaf(u[q].z, fmaf(ga[c + 2], u[q].z, gb[c + 2]), acc[0]);
          acc[1] = fmaf(u[q].w, fmaf(ga[c + 3], u[q].w, gb[c + 3]), acc[1]);
        }
      }
    }
    const float t = warp_sum(acc[0] + acc[1]);
    if (lane == 0) {
      const float y = (t + gc) * p.inv_tau;
      *reinterpret_cast<float2*>(p.M + 2 * static_cast<size_t>(j)) = make_float2(sigmoid_acc(y), sigmoid_acc(-y));
    }
  }
}

}  // namespace

cudaError_t launch_gauss_coef(const float* mu, const float* var, int d, int dcoef, float* coef,
                              uint32_t* status, cudaStream_t s) {
  return launch_pdl(k_gauss_coef, dim3(dcoef / 256), dim3(256), 0, s, mu, var, d, dcoef, coef, status);
}

cudaError_t launch_gauss_score(const GaussParams& p, smoes_dtype dt, int n_sms, cudaStream_t s) {
  const int dpad = round_up(p.d, 256);
  const size_t smem = sizeof(float) * 2 * dpad;
  int grid = (p.T + 7) / 8;
  if (grid > 4 * n_sms) grid = 4 * n_sms;
  if (grid < 1) grid = 1;
  auto k = (dt == SMOES_BF16) ? k_gauss_score<true> : k_gauss_score<false>;
  cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  return launch_pdl(k, dim3(grid), dim3(256), smem, s, p);
}

}  // namespace smoes
