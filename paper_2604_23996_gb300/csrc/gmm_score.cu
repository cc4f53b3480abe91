// gmm_score.cu -- soft modality score with the Gaussian-mixture estimator (the paper's
// supplementary extension of eqs. 8-9: each modality's features modelled by C diagonal Gaussians
// with weights pi).
//
//   LL_m(x) = log sum_c pi_mc N(x; mu_mc, var_mc),   M_v = sigmoid((LL_v - LL_t) / tau).
// Every component's log-density q_mc is taken relative to a reference component (text, 0):
//   D_mc(x) = q_mc(x) - q_t0(x) = sum_d (a_d x_d^2 + b_d x_d) + K_mc,
// a difference formed from per-feature coefficients (gauss_coef_feature, as for the single
// Gaussian), so the O(d)-sized log-densities never meet in a subtraction. Then
//   LL_v - LL_t = logsumexp_c D_vc - logsumexp_c D_tc   (D_t0 = 0).
// The F = 2C - 1 forms are accumulated in one pass over X (warp per token, 16-byte loads); with
// C = 1 this is the arithmetic of the Gaussian score.
#include <cuda_bf16.h>
#include <math_constants.h>

#include "device_common.cuh"
#include "ptx.cuh"
#include "smoes_internal.cuh"

namespace smoes {
namespace {

// Form f of C components: f < C -> (vision, f); otherwise (text, f - C + 1).
__device__ __forceinline__ void form_component(int f, int C, int& m, int& c) {
  m = f < C ? 0 : 1;
  c = f < C ? f : f - C + 1;
}

// coef: [F][a | b][dcoef] then part [F][dcoef / 256] (block sums of the constant terms).
__global__ void __launch_bounds__(256) k_gmm_coef(const GmmParams p) {
  __shared__ float red[8];
  pdl_wait();
  pdl_trigger();
  const int f = blockIdx.y, C = p.C, d = p.d;
  int m, c;
  form_component(f, C, m, c);
  const int i = blockIdx.x * 256 + threadIdx.x;
  float a = 0.f, b = 0.f, cc = 0.f;
  if (i < d) {
    const size_t mc = (static_cast<size_t>(m) * C + c) * d + i;
    const size_t t0 = static_cast<size_t>(C) * d + i;             // (text, 0)
    if (!gauss_coef_feature(p.mu[mc], p.mu[t0], p.var[mc], p.var[t0], a, b, cc))
      atomicOr(p.status, kStatusData);
  }
  float* cf = p.coef + static_cast<size_t>(f) * 2 * p.dcoef;
  cf[i] = a;
  cf[p.dcoef + i] = b;
  cc = warp_sum(cc);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = cc;
  __syncthreads();
  if (threadIdx.x == 0) {
    float t = 0.f;
    for (int w = 0; w < 8; ++w) t += red[w];
    p.coef[static_cast<size_t>(p.F) * 2 * p.dcoef + static_cast<size_t>(f) * (p.dcoef / 256) + blockIdx.x] = t;
  }
}

// Coefficients in shared memory with one padding float after every 8 features, so that the lanes
// of a warp, each reading its own 8 consecutive features, hit distinct banks.
__device__ __forceinline__ int cpad(int c) { return c + (c >> 3); }

template <bool kBf16>
__global__ void __launch_bounds__(256) k_gmm_score(const GmmParams p) {
  extern __shared__ float gsm[];
  const int dpad = round_up(p.d, 256);
  const int dps = cpad(dpad);                      // padded length of one coefficient vector
  const int F = p.F, C = p.C;
  pdl_wait();                                     // the coefficients of the kernel just before
  pdl_trigger();
  for (int f = 0; f < F; ++f)
    for (int i = threadIdx.x; i < dpad; i += 256) {
      gsm[(2 * f) * dps + cpad(i)] = p.coef[static_cast<size_t>(f) * 2 * p.dcoef + i];
      gsm[(2 * f + 1) * dps + cpad(i)] = p.coef[static_cast<size_t>(f) * 2 * p.dcoef + p.dcoef + i];
    }
  float K[kGmmMaxForms];
  bool bad = false;
#pragma unroll
  for (int f = 0; f < kGmmMaxForms; ++f) {
    K[f] = 0.f;
    if (f < F) {
      int m, c;
      form_component(f, C, m, c);
      const float* part = p.coef + static_cast<size_t>(F) * 2 * p.dcoef + static_cast<size_t>(f) * (p.dcoef / 256);
      float t = 0.f;
      for (int b = 0; b < p.dcoef / 256; ++b) t += part[b];
      K[f] = (p.log_pi[m * C + c] - p.log_pi[C]) - 0.5f * t;
      bad = bad || !isfinite(K[f]);
    }
  }
  if (bad && blockIdx.x == 0 && threadIdx.x == 0) atomicOr(p.status, kStatusData);
  __syncthreads();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  constexpr int per = kBf16 ? 8 : 4;              // features per 16-byte load
  constexpr int kIn = 8;                          // 16-byte loads of a row in flight per lane
  for (int j = blockIdx.x * 8 + warp; j < p.T; j += gridDim.x * 8) {
    float acc[kGmmMaxForms];
#pragma unroll
    for (int f = 0; f < kGmmMaxForms; ++f) acc[f] = 0.f;
    for (int cb = 0; cb < p.d; cb += 32 * per * kIn) {
      uint4 raw[kIn];
#pragma unroll
      for (int u = 0; u < kIn; ++u) {
        const int c0 = cb + u * 32 * per + lane * per;
        raw[u] = c0 < p.d ? __ldg(reinterpret_cast<const uint4*>(static_cast<const char*>(p.X) +
                                                                 (static_cast<size_t>(j) * p.d + c0) * (kBf16 ? 2 : 4)))
                          : make_uint4(0u, 0u, 0u, 0u);
      }
#pragma unroll
      for (int u = 0; u < kIn; ++u) {
        const int c0 = cb + u * 32 * per + lane * per;
        if (c0 >= p.d) break;
        float x[8];
        const uint32_t w[4] = {raw[u].x, raw[u].y, raw[u].z, raw[u].w};
        if (kBf16) {
#pragma unroll
          for (int r = 0; r < 4; ++r) {
            x[2 * r] = __uint_as_float(w[r] << 16);
            x[2 * r + 1] = __uint_as_float(w[r] & 0xffff0000u);
          }
        } else {
#pragma unroll
          for (int r = 0; r < 4; ++r) x[r] = __uint_as_float(w[r]);
        }
        const int cp = cpad(c0);
#pragma unroll
        for (int f = 0; f < kGmmMaxForms; ++f) {
          if (f < F) {
            const float* ga = gsm + (2 * f) * dps + cp;
            const float* gb = gsm + (2 * f + 1) * dps + cp;
#pragma unroll
            for (int q = 0; q < per; ++q) acc[f] = fmaf(x[q], fmaf(ga[q], x[q], gb[q]), acc[f]);
          }
        }
      }
    }
    float D[kGmmMaxForms];
#pragma unroll
    for (int f = 0; f < kGmmMaxForms; ++f) D[f] = f < F ? warp_sum(acc[f]) + K[f] : 0.f;
    if (lane == 0) {
      // logsumexp over the vision forms (f < C) and over {0 (text, 0)} + the text forms (f >= C)
      float mv = -CUDART_INF_F, mt = 0.f;
#pragma unroll
      for (int f = 0; f < kGmmMaxForms; ++f) {
        if (f < C) mv = fmaxf(mv, D[f]);
        else if (f < F) mt = fmaxf(mt, D[f]);
      }
      float sv = 0.f, st = expf(-mt);
#pragma unroll
      for (int f = 0; f < kGmmMaxForms; ++f) {
        if (f < C) sv += expf(D[f] - mv);
        else if (f < F) st += expf(D[f] - mt);
      }
      const float dll = (mv + logf(sv)) - (mt + logf(st));
      const float y = dll * p.inv_tau;
      *reinterpret_cast<float2*>(p.M + 2 * static_cast<size_t>(j)) = make_float2(sigmoid_acc(y), sigmoid_acc(-y));
    }
  }
}

}  // namespace

cudaError_t launch_gmm_score(const GmmParams& p, smoes_dtype dt, int n_sms, cudaStream_t s) {
  if (p.C < 1 || p.F > kGmmMaxForms) return cudaErrorInvalidValue;
  cudaError_t e = launch_pdl(k_gmm_coef, dim3(p.dcoef / 256, p.F), dim3(256), 0, s, p);
  if (e != cudaSuccess) return e;
  const int dpad = round_up(p.d, 256);
  const size_t smem = sizeof(float) * 2 * static_cast<size_t>(p.F) * (dpad + dpad / 8);
  if (smem > 227u * 1024u) return cudaErrorInvalidConfiguration;
  int grid = (p.T + 7) / 8;
  if (grid > 4 * n_sms) grid = 4 * n_sms;
  if (grid < 1) grid = 1;
  auto k = (dt == SMOES_BF16) ? k_gmm_score<true> : k_gmm_score<false>;
  e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  return launch_pdl(k, dim3(grid), dim3(256), smem, s, p);
}

}  // namespace smoes
