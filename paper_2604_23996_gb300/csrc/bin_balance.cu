// bin_balance.cu -- bin-level load-balance loss of Sec. 3.5, eq. (16), from the forward's saved
// softmax, and the table its gradient needs in the backward.
//
//   L_bal = sum_k N_B sum_{e in B_k} f_e P_e,
// read as: U_k = tokens with at least one top-k expert in bin B_k; f_e = selections of e /
// selections of B_k's experts; P_e = mean over U_k of h_je = g_je / G_jk with G_jk = sum_{e' in
// B_k} g_je' (the gate renormalised inside the bin; the softmax normaliser cancels, so h is formed
// from the saved exp(z - max)). A bin no token selects contributes 0.
//
// With f held constant (they are counts) the gradient at the logits is, for e in B_k, k in U_j,
//   dL/dz_je = N_B / |U_k| * h_je * (f_e - sum_{e' in B_k} f_e' h_je')
// (the softmax's own term sum_e' g_je' dL/dg_je' vanishes because h sums to 1 over a bin), and 0
// elsewhere. k_bal_partial: one warp per token at a time (lane l holds experts l, l+32, ...),
// per-bin sums by fixed warp reductions, per-lane running sums, then the block's warps added in
// warp order. k_bal_finalize: the blocks added in a fixed order (fp64), f, P, the loss, and the
// backward table (f_e, a_k = scale N_B / |U_k|) with its arming flag.
#include "device_common.cuh"
#include "ptx.cuh"
#include "smoes_internal.cuh"

namespace smoes {
namespace {

constexpr int kBalThreads = 256;
constexpr int kBalWarps = kBalThreads / 32;

// PL experts per lane (E <= 32 PL); each warp walks the block's tokens kR at a time with all of
// their loads issued first.
constexpr int kR = 4;

template <int PL>
__global__ void __launch_bounds__(kBalThreads) k_bal_partial(const BalParams p) {
  __shared__ float hs[kBalWarps][kMaxExperts];
  __shared__ int ss[kBalWarps][kMaxExperts];
  __shared__ int us[kBalWarps][kMaxBins];
  pdl_wait();                                       // the forward's saved scores and top-k
  pdl_trigger();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int E = p.E, k = p.k, K = p.K;
  const int G = gridDim.x, b = blockIdx.x;
  const int r0 = static_cast<int>(static_cast<long long>(b) * p.T / G);
  const int r1 = static_cast<int>(static_cast<long long>(b + 1) * p.T / G);
  int my_bin[PL];
#pragma unroll
  for (int i = 0; i < PL; ++i) {
    const int e = lane + 32 * i;
    my_bin[i] = e < E ? __ldg(p.expert_bin + e) : -1;
  }
  float hacc[PL];
  int sacc[PL];
#pragma unroll
  for (int i = 0; i < PL; ++i) { hacc[i] = 0.f; sacc[i] = 0; }
  int uacc = 0;                                     // lane k: tokens of this warp routed to bin k
  for (int j0 = r0 + warp; j0 < r1; j0 += kR * kBalWarps) {
    float ev[kR][PL];
    int sel[kR];
#pragma unroll
    for (int r = 0; r < kR; ++r) {
      const int j = j0 + r * kBalWarps;
      const bool in = j < r1;
      const float* grow = p.gsave + static_cast<size_t>(in ? j : r0) * E;
#pragma unroll
      for (int i = 0; i < PL; ++i) {
        const int e = lane + 32 * i;
        ev[r][i] = (in && e < E) ? __ldcg(grow + e) : 0.f;
      }
      sel[r] = (in && lane < k) ? __ldcg(p.topk_idx + static_cast<size_t>(j) * k + lane) : -1;
    }
#pragma unroll
    for (int r = 0; r < kR; ++r) {
      const int sbin = (sel[r] >= 0 && sel[r] < E) ? __ldg(p.expert_bin + sel[r]) : -1;
      const uint32_t ubins = __reduce_or_sync(0xffffffffu, sbin >= 0 ? (1u << sbin) : 0u);
      // selections of this lane's experts (a token selects an expert at most once)
      for (int q = 0; q < k; ++q) {
        const int sq = __shfl_sync(0xffffffffu, sel[r], q);
#pragma unroll
        for (int i = 0; i < PL; ++i) sacc[i] += (sq == lane + 32 * i) ? 1 : 0;
      }
      if (lane < K) uacc += (ubins >> lane) & 1u;
      // h_je for the token's bins (set bits of ubins, in bin order): bin sums by a fixed butterfly
      for (uint32_t bm = ubins; bm != 0u; bm &= bm - 1u) {     // warp-uniform
        const int kb = __ffs(bm) - 1;
        float v = 0.f;
#pragma unroll
        for (int i = 0; i < PL; ++i) v += my_bin[i] == kb ? ev[r][i] : 0.f;
        const float iS = 1.f / warp_sum(v);
#pragma unroll
        for (int i = 0; i < PL; ++i)
          if (my_bin[i] == kb) hacc[i] = fmaf(ev[r][i], iS, hacc[i]);
      }
    }
  }
#pragma unroll
  for (int i = 0; i < PL; ++i) {
    const int e = lane + 32 * i;
    if (e < E) {
      hs[warp][e] = hacc[i];
      ss[warp][e] = sacc[i];
    }
  }
  if (lane < K) us[warp][lane] = uacc;
  __syncthreads();
  for (int e = threadIdx.x; e < E; e += kBalThreads) {
    float h = 0.f;
    int c = 0;
    for (int w = 0; w < kBalWarps; ++w) {
      h += hs[w][e];
      c += ss[w][e];
    }
    p.part_h[static_cast<size_t>(b) * E + e] = h;
    p.part_s[static_cast<size_t>(b) * E + e] = c;
  }
  if (threadIdx.x < K) {
    int c = 0;
    for (int w = 0; w < kBalWarps; ++w) c += us[w][threadIdx.x];
    p.part_u[static_cast<size_t>(b) * K + threadIdx.x] = c;
  }
}

// Four slices of the block partials per expert (1024 threads), each with 16 loads in flight, the
// slices added in slice order; the bin map staged in shared memory.
constexpr int kFinSl = 4;
constexpr int kFinU = 16;

__global__ void __launch_bounds__(kFinSl * kMaxExperts) k_bal_finalize(const BalParams p) {
  __shared__ double f_s[kMaxExperts], P_s[kMaxExperts], h_sl[kFinSl][kMaxExperts];
  __shared__ long long sel_s[kMaxExperts], s_sl[kFinSl][kMaxExperts];
  __shared__ long long bin_sel[kMaxBins], bin_u[kMaxBins];
  __shared__ int eb_s[kMaxExperts];
  pdl_wait();                                       // the block partials
  pdl_trigger();
  const int e = threadIdx.x % kMaxExperts, sl = threadIdx.x / kMaxExperts;
  const int E = p.E, K = p.K, G = p.G;
  if (sl == 0 && e < E) eb_s[e] = __ldg(p.expert_bin + e);
  double H = 0.0;
  long long S = 0;
  if (e < E) {
    const int g0 = sl * G / kFinSl, g1 = (sl + 1) * G / kFinSl;
    for (int g = g0; g < g1; g += kFinU) {
      float hv[kFinU];
      int sv[kFinU];
#pragma unroll
      for (int u = 0; u < kFinU; ++u) {
        const bool in = g + u < g1;
        hv[u] = in ? __ldcg(p.part_h + static_cast<size_t>(g + u) * E + e) : 0.f;
        sv[u] = in ? __ldcg(p.part_s + static_cast<size_t>(g + u) * E + e) : 0;
      }
#pragma unroll
      for (int u = 0; u < kFinU; ++u) {
        H += static_cast<double>(hv[u]);
        S += sv[u];
      }
    }
  }
  h_sl[sl][e] = H;
  s_sl[sl][e] = S;
  if (sl == 1 && e < K) {
    long long u = 0;
    for (int g = 0; g < G; g += kFinU) {
      int uv[kFinU];
#pragma unroll
      for (int q = 0; q < kFinU; ++q) uv[q] = g + q < G ? __ldcg(p.part_u + static_cast<size_t>(g + q) * K + e) : 0;
#pragma unroll
      for (int q = 0; q < kFinU; ++q) u += uv[q];
    }
    bin_u[e] = u;
  }
  __syncthreads();
  if (sl == 0) {
    H = 0.0;
    S = 0;
    for (int t = 0; t < kFinSl; ++t) {
      H += h_sl[t][e];
      S += s_sl[t][e];
    }
    if (e < E) sel_s[e] = S;
  }
  __syncthreads();
  if (sl == 0 && e < K) {                           // selections of each bin's experts, in expert order
    long long t = 0;
    for (int x = 0; x < E; ++x) t += eb_s[x] == e ? sel_s[x] : 0;
    bin_sel[e] = t;
  }
  __syncthreads();
  const double NB = static_cast<double>(p.N_B);
  if (sl == 0 && e < E) {
    const int kb = eb_s[e];
    const double f = bin_sel[kb] > 0 ? static_cast<double>(S) / static_cast<double>(bin_sel[kb]) : 0.0;
    const double P = bin_u[kb] > 0 ? H / static_cast<double>(bin_u[kb]) : 0.0;
    f_s[e] = f;
    P_s[e] = P;
    p.tab_f[e] = static_cast<float>(f);
    if (p.f_out) p.f_out[e] = static_cast<float>(f);
    if (p.P_out) p.P_out[e] = static_cast<float>(P);
  }
  if (sl == 0 && e < K)
    p.tab_a[e] = bin_u[e] > 0 ? static_cast<float>(p.scale * NB / static_cast<double>(bin_u[e])) : 0.f;
  __syncthreads();
  if (threadIdx.x == 0) {
    double L = 0.0;                                 // eq. (16), bins in order, experts in order
    for (int kb = 0; kb < K; ++kb) {
      double t = 0.0;
      for (int x = 0; x < E; ++x)
        if (eb_s[x] == kb) t += f_s[x] * P_s[x];
      L += NB * t;
    }
    *p.loss = static_cast<float>(L);
    __threadfence();
    *p.flag = 1u;                                   // the next backward adds the gradient
  }
}

}  // namespace

cudaError_t launch_bin_balance(const BalParams& p, cudaStream_t s) {
  if (p.E < 1 || p.E > kMaxExperts || p.K < 1 || p.K > kMaxBins) return cudaErrorInvalidValue;
  auto kp = p.E <= 32 ? k_bal_partial<1> : p.E <= 64 ? k_bal_partial<2> : p.E <= 128 ? k_bal_partial<4>
                                                                             : k_bal_partial<8>;
  cudaError_t e = launch_pdl(kp, dim3(p.G), dim3(kBalThreads), 0, s, p);
  if (e != cudaSuccess) return e;
  return launch_pdl(k_bal_finalize, dim3(1), dim3(kFinSl * kMaxExperts), 0, s, p);
}

}  // namespace smoes
