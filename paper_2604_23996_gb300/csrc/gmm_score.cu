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
// The F = 2C - 1 forms are accumulated in one pass over X (batches of rows per block, 16-byte
// loads); with C = 1 this is the arithmetic of the Gaussian score.
#include <cuda_bf16.h>
#include <math_constants.h>

#include <type_traits>

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

// Rows in batches: thread t of a block owns features 8t .. 8t + 7 of every 2048-feature pass,
// reads their coefficients from shared memory once per batch of R rows (two 16-byte loads per
// vector, consecutive threads at consecutive addresses), and keeps R x F running sums; a batch's
// sums are reduced over the block once (a lane-transposing butterfly per warp, then the eight
// warps in order). Reading the coefficients per row instead (one warp per token) made the
// shared-memory traffic twelve times the bytes of X. The R rows' loads are issued together.
template <int F>
struct GmmRows {
  static constexpr int R = F <= 3 ? 8 : (F == 5 ? 6 : 4);    // R x F <= 32 sums per thread
};

template <bool kBf16, int F>
__global__ void __launch_bounds__(256, 2) k_gmm_score(const GmmParams p) {
  extern __shared__ float gsm[];
  constexpr int R = GmmRows<F>::R;
  constexpr int NV = R * F;
  constexpr int W = kBf16 ? 1 : 2;                 // 16-byte words per thread and row
  __shared__ float red[8][32];
  __shared__ float Dsm[32];
  const int dpad = p.dcoef;
  const int C = p.C;
  pdl_wait();                                     // the coefficients of the kernel just before
  pdl_trigger();
  for (int f = 0; f < F; ++f)
    for (int i = threadIdx.x; i < dpad; i += 256) {
      gsm[(2 * f) * dpad + i] = p.coef[static_cast<size_t>(f) * 2 * p.dcoef + i];
      gsm[(2 * f + 1) * dpad + i] = p.coef[static_cast<size_t>(f) * 2 * p.dcoef + p.dcoef + i];
    }
  __shared__ float Ks[F];                         // constant term of each form
  if (threadIdx.x < F) {
    const int f = threadIdx.x;
    int m, c;
    form_component(f, C, m, c);
    const float* part = p.coef + static_cast<size_t>(F) * 2 * p.dcoef + static_cast<size_t>(f) * (p.dcoef / 256);
    float t = 0.f;
    for (int b = 0; b < p.dcoef / 256; ++b) t += part[b];
    Ks[f] = (p.log_pi[m * C + c] - p.log_pi[C]) - 0.5f * t;
    if (!isfinite(Ks[f]) && blockIdx.x == 0) atomicOr(p.status, kStatusData);
  }
  __syncthreads();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int j0 = blockIdx.x * R; j0 < p.T; j0 += gridDim.x * R) {
    float acc[R][F];
#pragma unroll
    for (int r = 0; r < R; ++r)
#pragma unroll
      for (int f = 0; f < F; ++f) acc[r][f] = 0.f;
    for (int cc = 0; cc < p.d; cc += 2048) {
      const int c0 = cc + 8 * threadIdx.x;
      const bool act = c0 < p.d;
      uint4 raw[R][W];
#pragma unroll
      for (int r = 0; r < R; ++r) {
        const bool in = act && j0 + r < p.T;
        const char* src = static_cast<const char*>(p.X) +
                          (static_cast<size_t>(in ? j0 + r : 0) * p.d + (in ? c0 : 0)) * (kBf16 ? 2 : 4);
#pragma unroll
        for (int w = 0; w < W; ++w)
          raw[r][w] = in ? __ldg(reinterpret_cast<const uint4*>(src) + w) : make_uint4(0u, 0u, 0u, 0u);
      }
      if (!act) continue;
#pragma unroll
      for (int f = 0; f < F; ++f) {
        const float4* ga = reinterpret_cast<const float4*>(gsm + (2 * f) * dpad + c0);
        const float4* gb = reinterpret_cast<const float4*>(gsm + (2 * f + 1) * dpad + c0);
        const float4 a0 = ga[0], a1 = ga[1], b0 = gb[0], b1 = gb[1];
        const float a[8] = {a0.x, a0.y, a0.z, a0.w, a1.x, a1.y, a1.z, a1.w};
        const float b[8] = {b0.x, b0.y, b0.z, b0.w, b1.x, b1.y, b1.z, b1.w};
#pragma unroll
        for (int r = 0; r < R; ++r) {
          float x[8];
          if (kBf16) {
            const uint32_t w4[4] = {raw[r][0].x, raw[r][0].y, raw[r][0].z, raw[r][0].w};
#pragma unroll
            for (int q = 0; q < 4; ++q) {
              x[2 * q] = __uint_as_float(w4[q] << 16);
              x[2 * q + 1] = __uint_as_float(w4[q] & 0xffff0000u);
            }
          } else {
            const uint32_t w8[8] = {raw[r][0].x, raw[r][0].y, raw[r][0].z, raw[r][0].w,
                                    raw[r][W - 1].x, raw[r][W - 1].y, raw[r][W - 1].z, raw[r][W - 1].w};
#pragma unroll
            for (int q = 0; q < 8; ++q) x[q] = __uint_as_float(w8[q]);
          }
#pragma unroll
          for (int q = 0; q < 8; ++q) acc[r][f] = fmaf(x[q], fmaf(a[q], x[q], b[q]), acc[r][f]);
        }
      }
    }
    // block sums of the R x F values: per warp a transposing butterfly (lane v gets value v),
    // then the warps in order
    float v[32];
#pragma unroll
    for (int q = 0; q < 32; ++q) v[q] = q < NV ? acc[q / F][q % F] : 0.f;
    const float ws = warp_transpose_sum(v);
    red[warp][lane] = ws;
    __syncthreads();
    if (threadIdx.x < NV) {
      float t = 0.f;
#pragma unroll
      for (int w = 0; w < 8; ++w) t += red[w][threadIdx.x];
      Dsm[threadIdx.x] = t + Ks[threadIdx.x % F];
    }
    __syncthreads();
    if (threadIdx.x < R && j0 + threadIdx.x < p.T) {
      const float* D = Dsm + threadIdx.x * F;
      // logsumexp over the vision forms (f < C) and over {0 (text, 0)} + the text forms (f >= C)
      float mv = -CUDART_INF_F, mt = 0.f;
#pragma unroll
      for (int f = 0; f < F; ++f) {
        if (f < C) mv = fmaxf(mv, D[f]);
        else mt = fmaxf(mt, D[f]);
      }
      float sv = 0.f, st = expf(-mt);
#pragma unroll
      for (int f = 0; f < F; ++f) {
        if (f < C) sv += expf(D[f] - mv);
        else st += expf(D[f] - mt);
      }
      const float dll = (mv + logf(sv)) - (mt + logf(st));
      const float y = dll * p.inv_tau;
      const size_t j = static_cast<size_t>(j0 + threadIdx.x);
      *reinterpret_cast<float2*>(p.M + 2 * j) = make_float2(sigmoid_acc(y), sigmoid_acc(-y));
    }
    __syncthreads();                              // red and Dsm are rewritten by the next batch
  }
}

}  // namespace

cudaError_t launch_gmm_score(const GmmParams& p, smoes_dtype dt, int n_sms, cudaStream_t s) {
  if (p.C < 1 || p.F != 2 * p.C - 1 || p.F > kGmmMaxForms) return cudaErrorInvalidValue;
  cudaError_t e = launch_pdl(k_gmm_coef, dim3(p.dcoef / 256, p.F), dim3(256), 0, s, p);
  if (e != cudaSuccess) return e;
  const size_t smem = sizeof(float) * 2 * static_cast<size_t>(p.F) * p.dcoef;
  if (smem > 200u * 1024u) return cudaErrorInvalidConfiguration;
  const bool bf = dt == SMOES_BF16;
  auto pick = [&](auto fc) {
    constexpr int F = decltype(fc)::value;
    return bf ? k_gmm_score<true, F> : k_gmm_score<false, F>;
  };
  auto k = p.F == 1 ? pick(std::integral_constant<int, 1>())
         : p.F == 3 ? pick(std::integral_constant<int, 3>())
         : p.F == 5 ? pick(std::integral_constant<int, 5>())
                    : pick(std::integral_constant<int, 7>());
  const int R = p.F <= 3 ? 8 : (p.F == 5 ? 6 : 4);
  int grid = (p.T + R - 1) / R;
  if (grid > 2 * n_sms) grid = 2 * n_sms;
  if (grid < 1) grid = 1;
  e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  return launch_pdl(k, dim3(grid), dim3(256), smem, s, p);
}

}  // namespace smoes
