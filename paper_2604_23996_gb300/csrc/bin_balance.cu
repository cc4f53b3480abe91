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
// warp order (k_bal_partial_pow2: the same for bins that are power-of-two runs of consecutive
// experts, every bin's sum from one butterfly). k_bal_finalize: the blocks added in a fixed order
// (fp32), f, P, the loss, and the backward table (f_e, a_k = scale N_B / |U_k|) with its arming
// flag.
#include "device_common.cuh"
#include "ptx.cuh"
#include "smoes_internal.cuh"

namespace smoes {
namespace {

constexpr int kBalThreads = 256;
constexpr int kBalWarps = kBalThreads / 32;

// PL experts per lane (E <= 32 PL, E <= 128); each warp walks the block's tokens kR at a time with all of
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

// The same partials for bins that are runs of N_B consecutive experts with N_B a power of two
// (the usual map): lane l holds experts l + 32i, so for N_B <= 32 the experts of a bin sit in
// N_B adjacent lanes at the same i, and every bin's sum of the token's saved scores comes out of
// one xor butterfly over log2(N_B) lane distances, all bins at once (for N_B = 64 the two halves
// at i and i + 1 are added as well). Selections are counted by shared-memory integer atomics.
constexpr int kR2 = 8;                        // tokens per warp with their loads in flight

template <int PL>
__global__ void __launch_bounds__(kBalThreads) k_bal_partial_pow2(const BalParams p, const int lnb) {
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
  const int span = lnb < 5 ? 1 << lnb : 32;         // lanes per bin run
  for (int e = lane; e < E; e += 32) ss[warp][e] = 0;
  __syncwarp();
  float hacc[PL];
#pragma unroll
  for (int i = 0; i < PL; ++i) hacc[i] = 0.f;
  int uacc = 0;                                     // lane k: tokens of this warp routed to bin k
  for (int j0 = r0 + warp; j0 < r1; j0 += kR2 * kBalWarps) {
    float ev[kR2][PL];
    int sel[kR2];
#pragma unroll
    for (int r = 0; r < kR2; ++r) {
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
    for (int r = 0; r < kR2; ++r) {
      const bool ok = sel[r] >= 0 && sel[r] < E;
      if (ok) atomicAdd(&ss[warp][sel[r]], 1);
      const uint32_t ubins = __reduce_or_sync(0xffffffffu, ok ? (1u << (sel[r] >> lnb)) : 0u);
      if (lane < K) uacc += (ubins >> lane) & 1u;
      float gs[PL];
#pragma unroll
      for (int i = 0; i < PL; ++i) gs[i] = ev[r][i];
#pragma unroll
      for (int d = 1; d < 32; d <<= 1) {            // log2(span) levels (warp-uniform)
        if (d < span) {
#pragma unroll
          for (int i = 0; i < PL; ++i) gs[i] += __shfl_xor_sync(0xffffffffu, gs[i], d);
        }
      }
      if (lnb == 6) {                               // 64-expert bins: experts at i and i ^ 1
#pragma unroll
        for (int i = 0; i + 1 < PL; i += 2) {
          const float t = gs[i] + gs[i + 1];
          gs[i] = t;
          gs[i + 1] = t;
        }
      }
#pragma unroll
      for (int i = 0; i < PL; ++i) {
        const int kb = (lane + 32 * i) >> lnb;
        if (lane + 32 * i < E && ((ubins >> kb) & 1u)) hacc[i] += __fdividef(ev[r][i], gs[i]);
      }
    }
  }
#pragma unroll
  for (int i = 0; i < PL; ++i) {
    const int e = lane + 32 * i;
    if (e < E) hs[warp][e] = hacc[i];
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

// One block of 1024 threads (plans hold E <= 128), all in fp32 and integers. The block partials
// of each expert are summed in eight slices of the blocks, each slice with its loads issued
// together and added in block order, then the slices in slice order; the per-bin token counts the
// same way in integers. Every later step runs one thread per expert or per bin. (The sums are
// fixed-order and so bitwise reproducible; fp64 is avoided because on GB300 each fp64 operation
// in these short dependent chains costs far more than the fp32 one, and the fp32 rounding of
// sums over a few hundred partials is far inside the 2e-3 tolerance of the outputs.)
constexpr int kFinThreads = 1024;
constexpr int kFinRow = 128;                        // threads per expert row of a slice
constexpr int kFinSl = kFinThreads / kFinRow;       // slices of the blocks
constexpr int kFinU = 8;                            // loads in flight per thread and round (64 registers)

__global__ void __launch_bounds__(kFinThreads) k_bal_finalize(const BalParams p) {
  __shared__ float h_sl[kFinSl][kFinRow];
  __shared__ int s_sl[kFinSl][kFinRow];
  __shared__ int u_sl[kFinSl][kMaxBins];
  __shared__ float f_s[kFinRow], P_s[kFinRow], H_s[kFinRow], term_s[kMaxBins];
  __shared__ int sel_s[kFinRow], bin_sel[kMaxBins], bin_u[kMaxBins];
  __shared__ int eb_s[kFinRow];
  pdl_wait();                                       // the block partials
  pdl_trigger();
  const int E = p.E, K = p.K, G = p.G;
  const int tid = threadIdx.x;
  const int e = tid % kFinRow, sl = tid / kFinRow;
  if (tid < E) eb_s[tid] = __ldg(p.expert_bin + tid);
  {
    const int g0 = sl * G / kFinSl, g1 = (sl + 1) * G / kFinSl;
    float H = 0.f;
    int S = 0, U = 0;
    for (int g = g0; g < g1; g += kFinU) {
      float hv[kFinU];
      int sv[kFinU], uv[kFinU];
#pragma unroll
      for (int u = 0; u < kFinU; ++u) {
        const bool in = g + u < g1;
        hv[u] = (in && e < E) ? __ldcg(p.part_h + static_cast<size_t>(g + u) * E + e) : 0.f;
        sv[u] = (in && e < E) ? __ldcg(p.part_s + static_cast<size_t>(g + u) * E + e) : 0;
        uv[u] = (in && e < K) ? __ldcg(p.part_u + static_cast<size_t>(g + u) * K + e) : 0;
      }
#pragma unroll
      for (int u = 0; u < kFinU; ++u) {
        H += hv[u];
        S += sv[u];
        U += uv[u];
      }
    }
    h_sl[sl][e] = H;
    s_sl[sl][e] = S;
    if (e < K) u_sl[sl][e] = U;
  }
  __syncthreads();
  if (tid < E) {
    float H = 0.f;
    int S = 0;
    for (int t = 0; t < kFinSl; ++t) {
      H += h_sl[t][tid];
      S += s_sl[t][tid];
    }
    H_s[tid] = H;
    sel_s[tid] = S;
  }
  if (tid < K) {
    int u = 0;
    for (int t = 0; t < kFinSl; ++t) u += u_sl[t][tid];
    bin_u[tid] = u;
  }
  __syncthreads();
  if (tid < K) {                                    // selections of each bin's experts (counts < 2^24)
    int t = 0;
    for (int x = 0; x < E; ++x) t += eb_s[x] == tid ? sel_s[x] : 0;
    bin_sel[tid] = t;
  }
  __syncthreads();
  const float NB = static_cast<float>(p.N_B);
  if (tid < E) {
    const int kb = eb_s[tid];
    const float f = bin_sel[kb] > 0 ? static_cast<float>(sel_s[tid]) / static_cast<float>(bin_sel[kb]) : 0.f;
    const float P = bin_u[kb] > 0 ? H_s[tid] / static_cast<float>(bin_u[kb]) : 0.f;
    f_s[tid] = f;
    P_s[tid] = P;
    p.tab_f[tid] = f;
    if (p.f_out) p.f_out[tid] = f;
    if (p.P_out) p.P_out[tid] = P;
  }
  if (tid < K)
    p.tab_a[tid] = bin_u[tid] > 0 ? static_cast<float>(p.scale) * NB / static_cast<float>(bin_u[tid]) : 0.f;
  __syncthreads();
  if (tid < K) {                                    // eq. (16): bin tid's term, its experts in order
    float t = 0.f;
    for (int x = 0; x < E; ++x)
      if (eb_s[x] == tid) t = fmaf(f_s[x], P_s[x], t);
    term_s[tid] = NB * t;
  }
  __syncthreads();
  if (tid == 0) {
    float L = 0.f;                                  // the bins' terms in bin order
    for (int kb = 0; kb < K; ++kb) L += term_s[kb];
    *p.loss = L;
    __threadfence();
    *p.flag = 1u;                                   // the next backward adds the gradient
  }
}

}  // namespace

cudaError_t launch_bin_balance(const BalParams& p, cudaStream_t s) {
  if (p.E < 1 || p.E > kFinRow || p.K < 1 || p.K > kMaxBins) return cudaErrorInvalidValue;
  // bins that are runs of a power-of-two number of consecutive experts: the butterfly kernel
  bool runs = (p.N_B & (p.N_B - 1)) == 0 && p.N_B <= 64 && p.N_B * p.K == p.E && p.E <= 128;
  for (int x = 0; runs && x < p.E; ++x) runs = p.expert_bin_host[x] == x / p.N_B;
  cudaError_t e;
  if (runs) {
    int lnb = 0;
    while ((1 << lnb) < p.N_B) ++lnb;
    auto kp = p.E <= 32 ? k_bal_partial_pow2<1> : p.E <= 64 ? k_bal_partial_pow2<2> : k_bal_partial_pow2<4>;
    e = launch_pdl(kp, dim3(p.G), dim3(kBalThreads), 0, s, p, lnb);
  } else {
    auto kp = p.E <= 32 ? k_bal_partial<1> : p.E <= 64 ? k_bal_partial<2> : k_bal_partial<4>;
    e = launch_pdl(kp, dim3(p.G), dim3(kBalThreads), 0, s, p);
  }
  if (e != cudaSuccess) return e;
  return launch_pdl(k_bal_finalize, dim3(1), dim3(kFinThreads), 0, s, p);
}

}  // namespace smoes
