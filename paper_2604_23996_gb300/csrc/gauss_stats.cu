// gauss_stats.cu -- online statistics of the Gaussian modality score (Sec. 3.2, eqs. 5-7) and
// momentum-adaptive binning (Sec. 3.3, eqs. 10-11).
//
// Statistics update. The state (N_m, S_mu,m, S_var,m) of each modality m is kept in fp64 on the
// device. One pass over X forms, per feature and hard modality, the shifted sums
//   s1 = sum_{x in T_m} (x - c),   s2 = sum_{x in T_m} (x - c)^2,
// with the shift c = S_mu,m,t-1 / N_m,t-1 rounded to fp32 (0 for an empty state): the previous
// mean is close to the batch mean, so the centred second moment
//   sum (x - mu_T)^2 = s2 - s1^2 / n,   mu_T = c + s1 / n,
// loses nothing to cancellation. k_stats_partial streams X once (16-byte loads, 8 features per
// thread, fp32 sums over a contiguous run of rows per block) and writes one partial per block;
// k_stats_finalize sums the partials in block order (runs of 8 in fp32, then fp64) and applies
// eqs. (5)-(7) in fp64. Both are deterministic.
//
// Adaptive binning. k_adaptive_bins (one block, E <= 256 threads) updates the EMA expert loads
// of eq. (10) from this step's per-modality selection counts, forms the text bias f_spec of
// eq. (11), and ranks the experts by ascending f_spec (equal values in expert-index order); the
// rank cut into runs of N_B experts is the new expert -> bin map. All of it is fp64 with the
// rounding of separate multiplies, adds and a correctly rounded division, so the order, and
// with it the bin map, is reproducible bit for bit.
#include <cuda_bf16.h>

#include "device_common.cuh"
#include "ptx.cuh"
#include "smoes_internal.cuh"

namespace smoes {
namespace {

constexpr int kStatThreads = 256;
constexpr int kStatCols = 8 * kStatThreads;      // features per pass of a block (8 per thread)
constexpr int kStatRowsInFlight = 8;             // rows loaded ahead per thread

// Shift of feature i of modality m: the previous mean (fp32), or 0 for an empty state.
__device__ __forceinline__ float stat_shift(const double* N0, const double* S_mu0, int d, int m, int i) {
  const double n = N0[m];
  return n > 0.0 ? static_cast<float>(S_mu0[static_cast<size_t>(m) * d + i] / n) : 0.f;
}

// Eight consecutive features of a row: raw 16-byte words (bf16: one, fp32: two), loaded ahead
// and widened to floats when they are used.
template <bool kBf16>
struct Raw8 {
  uint4 w[kBf16 ? 1 : 2];
};

template <bool kBf16>
__device__ __forceinline__ void load_raw8(const void* X, size_t off, Raw8<kBf16>& r) {
  if (kBf16) {
    r.w[0] = __ldg(reinterpret_cast<const uint4*>(static_cast<const __nv_bfloat16*>(X) + off));
  } else {
    const uint4* p = reinterpret_cast<const uint4*>(static_cast<const float*>(X) + off);
    r.w[0] = __ldg(p);
    r.w[kBf16 ? 0 : 1] = __ldg(p + 1);
  }
}

template <bool kBf16>
__device__ __forceinline__ void widen8(const Raw8<kBf16>& r, float (&v)[8]) {
  if (kBf16) {
    const uint32_t w[4] = {r.w[0].x, r.w[0].y, r.w[0].z, r.w[0].w};
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      v[2 * q] = __uint_as_float(w[q] << 16);
      v[2 * q + 1] = __uint_as_float(w[q] & 0xffff0000u);
    }
  } else {
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const uint4 u = r.w[kBf16 ? 0 : h];
      v[4 * h] = __uint_as_float(u.x);
      v[4 * h + 1] = __uint_as_float(u.y);
      v[4 * h + 2] = __uint_as_float(u.z);
      v[4 * h + 3] = __uint_as_float(u.w);
    }
  }
}

// Block b sums rows [b T / G, (b+1) T / G). part: [G][4][d] = (s1_v, s2_v, s1_t, s2_t);
// nvis: [G] vision rows of the block; block 0 also keeps a copy of N_{t-1} for the finalize
// kernel (which overwrites N).
template <bool kBf16>
__global__ void __launch_bounds__(kStatThreads) k_stats_partial(const StatsParams p) {
  pdl_wait();                                     // X and the state may be written just before
  pdl_trigger();
  const int G = gridDim.x, b = blockIdx.x;
  const int r0 = static_cast<int>(static_cast<long long>(b) * p.T / G);
  const int r1 = static_cast<int>(static_cast<long long>(b + 1) * p.T / G);
  int nv = 0;
  for (int c0 = 0; c0 < p.d; c0 += kStatCols) {
    const int c = c0 + threadIdx.x * 8;
    const bool act = c < p.d;
    float sh[2][8];
#pragma unroll
    for (int q = 0; q < 8; ++q) {
      sh[0][q] = act ? stat_shift(p.N, p.S_mu, p.d, 0, c + q) : 0.f;
      sh[1][q] = act ? stat_shift(p.N, p.S_mu, p.d, 1, c + q) : 0.f;
    }
    float s1[2][8], s2[2][8];
#pragma unroll
    for (int q = 0; q < 8; ++q) s1[0][q] = s1[1][q] = s2[0][q] = s2[1][q] = 0.f;
    for (int j0 = r0; j0 < r1; j0 += kStatRowsInFlight) {
      Raw8<kBf16> raw[kStatRowsInFlight];
      int lab[kStatRowsInFlight];
#pragma unroll
      for (int u = 0; u < kStatRowsInFlight; ++u) {
        const int j = j0 + u;
        lab[u] = j < r1 ? (__ldg(p.is_vision + j) ? 0 : 1) : -1;
        if (act && j < r1) load_raw8<kBf16>(p.X, static_cast<size_t>(j) * p.d + c, raw[u]);
      }
#pragma unroll
      for (int u = 0; u < kStatRowsInFlight; ++u) {
        if (lab[u] < 0 || !act) continue;
        if (c0 == 0 && threadIdx.x == 0 && lab[u] == 0) ++nv;
        const int m = lab[u];
        float v[8];
        widen8<kBf16>(raw[u], v);
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          const float dv = v[q] - (m ? sh[1][q] : sh[0][q]);
          if (m) {
            s1[1][q] += dv;
            s2[1][q] = fmaf(dv, dv, s2[1][q]);
          } else {
            s1[0][q] += dv;
            s2[0][q] = fmaf(dv, dv, s2[0][q]);
          }
        }
      }
    }
    if (act) {
      float* out = p.part + static_cast<size_t>(b) * 4 * p.d + c;
#pragma unroll
      for (int m = 0; m < 2; ++m) {
        float* o1 = out + static_cast<size_t>(2 * m) * p.d;
        float* o2 = out + static_cast<size_t>(2 * m + 1) * p.d;
        *reinterpret_cast<float4*>(o1) = make_float4(s1[m][0], s1[m][1], s1[m][2], s1[m][3]);
        *reinterpret_cast<float4*>(o1 + 4) = make_float4(s1[m][4], s1[m][5], s1[m][6], s1[m][7]);
        *reinterpret_cast<float4*>(o2) = make_float4(s2[m][0], s2[m][1], s2[m][2], s2[m][3]);
        *reinterpret_cast<float4*>(o2 + 4) = make_float4(s2[m][4], s2[m][5], s2[m][6], s2[m][7]);
      }
    }
  }
  if (threadIdx.x == 0) {
    p.nvis[b] = nv;
    if (b == 0) {
      p.N0[0] = p.N[0];
      p.N0[1] = p.N[1];
    }
  }
}

// One (modality, feature) column per (block column, 8 slices): slice t sums the partials of
// blocks [t G / 8, (t+1) G / 8) in order (runs of 8 in fp32, the runs in fp64), the slices are
// added in slice order in fp64; then eqs. (5)-(7) in fp64. The counts |T_m| are integer sums of
// nvis.
constexpr int kFinSlices = 8;
constexpr int kFinCols = 32;

__global__ void __launch_bounds__(kFinSlices * kFinCols) k_stats_finalize(const StatsParams p) {
  __shared__ double red[2][kFinSlices][kFinCols];
  __shared__ long long cnt_s;
  pdl_wait();                                     // the partials of k_stats_partial
  pdl_trigger();
  const int col = threadIdx.x % kFinCols, sl = threadIdx.x / kFinCols;
  const int i2 = blockIdx.x * kFinCols + col;     // m * d + i
  const int m = i2 < 2 * p.d ? i2 / p.d : 0;
  const int i = i2 < 2 * p.d ? i2 % p.d : 0;
  const int G = p.G;
  if (threadIdx.x < 32) {                         // |T_v|: integer counts, lanes stride the blocks
    long long nvis = 0;
    for (int g = threadIdx.x; g < G; g += 32) nvis += p.nvis[g];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) nvis += __shfl_xor_sync(0xffffffffu, nvis, o);
    if (threadIdx.x == 0) cnt_s = nvis;
  }
  // runs of 8 block partials added in fp32 (their loads issued together), the runs in fp64: GB300's
  // fp64 rate is a small fraction of its fp32 rate, and one fp64 add per partial set this
  // kernel's time
  double a1 = 0.0, a2 = 0.0;
  if (i2 < 2 * p.d) {
    const int g0 = sl * G / kFinSlices, g1 = (sl + 1) * G / kFinSlices;
    for (int g = g0; g < g1; g += 8) {
      float v1[8], v2[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const bool in = g + u < g1;
        const float* base = p.part + static_cast<size_t>(in ? g + u : g0) * 4 * p.d;
        v1[u] = in ? __ldcg(base + static_cast<size_t>(2 * m) * p.d + i) : 0.f;
        v2[u] = in ? __ldcg(base + static_cast<size_t>(2 * m + 1) * p.d + i) : 0.f;
      }
      float r1 = 0.f, r2 = 0.f;
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        r1 += v1[u];
        r2 += v2[u];
      }
      a1 += static_cast<double>(r1);
      a2 += static_cast<double>(r2);
    }
  }
  red[0][sl][col] = a1;
  red[1][sl][col] = a2;
  __syncthreads();
  if (sl != 0 || i2 >= 2 * p.d) return;
  double s1 = 0.0, s2 = 0.0;
  for (int t = 0; t < kFinSlices; ++t) {
    s1 += red[0][t][col];
    s2 += red[1][t][col];
  }
  const double n = m == 0 ? static_cast<double>(cnt_s) : static_cast<double>(p.T - cnt_s);
  const double beta = p.beta;
  const double N0 = p.N0[m];
  const size_t at = static_cast<size_t>(m) * p.d + i;
  const double Smu0 = p.S_mu[at], Svar0 = p.S_var[at];
  const double N1 = beta * N0 + n;                                    // eq. (5)
  double Smu1 = beta * Smu0, Svar1 = beta * Svar0;
  if (n > 0.0) {
    const double c = N0 > 0.0 ? static_cast<double>(static_cast<float>(Smu0 / N0)) : 0.0;
    const double mu_b = c + s1 / n;                                   // batch mean
    const double m2 = fmax(s2 - s1 * (s1 / n), 0.0);                  // sum (x - mu_b)^2
    Smu1 += n * mu_b;                                                 // eq. (6)
    Svar1 += m2;                                                      // eq. (7)
    if (N0 > 0.0) {
      const double dm = (c - Smu0 / N0) + s1 / n;                     // mu_b - S_mu,t-1 / N_t-1
      Svar1 += dm * dm * (beta * N0 * n / (beta * N0 + n));
    }
  }
  p.S_mu[at] = Smu1;
  p.S_var[at] = Svar1;
  if (i == 0) p.N[m] = N1;
  if (p.mu_out) p.mu_out[at] = static_cast<float>(Smu1 / N1);
  if (p.var_out) p.var_out[at] = static_cast<float>(Svar1 / N1);
}

// Eqs. (10)-(11) and the stable ascending rank of f_spec; one thread per expert.
__global__ void __launch_bounds__(kMaxExperts) k_adaptive_bins(const BinsParams p) {
  __shared__ double f_s[kMaxExperts];
  pdl_wait();                                     // this step's counts
  pdl_trigger();
  const int e = threadIdx.x;
  double f = 0.5;
  if (e < p.E) {
    const double w_old = p.beta, w_new = 1.0 - p.beta;
    const double cv = __dadd_rn(__dmul_rn(w_old, p.C_bar[e]),
                                __dmul_rn(w_new, static_cast<double>(p.counts[e])));
    const double ct = __dadd_rn(__dmul_rn(w_old, p.C_bar[p.E + e]),
                                __dmul_rn(w_new, static_cast<double>(p.counts[p.E + e])));
    p.C_bar[e] = cv;                                                  // eq. (10)
    p.C_bar[p.E + e] = ct;
    const double tot = __dadd_rn(ct, cv);
    f = tot > 0.0 ? __ddiv_rn(ct, tot) : 0.5;                        // eq. (11); 0/0 -> neutral
    f_s[e] = f;
    if (p.f_spec) p.f_spec[e] = f;
  }
  __syncthreads();
  if (e < p.E) {
    int rank = 0;
    for (int o = 0; o < p.E; ++o) {
      const double g = f_s[o];
      rank += (g < f || (g == f && o < e)) ? 1 : 0;
    }
    p.expert_bin[e] = rank / p.N_B;
  }
}

}  // namespace

cudaError_t launch_stats_update(const StatsParams& p, bool bf16, cudaStream_t s) {
  auto k = bf16 ? k_stats_partial<true> : k_stats_partial<false>;
  cudaError_t e = launch_pdl(k, dim3(p.G), dim3(kStatThreads), 0, s, p);
  if (e != cudaSuccess) return e;
  const int blocks = (2 * p.d + kFinCols - 1) / kFinCols;
  return launch_pdl(k_stats_finalize, dim3(blocks), dim3(kFinSlices * kFinCols), 0, s, p);
}

cudaError_t launch_adaptive_bins(const BinsParams& p, cudaStream_t s) {
  if (p.E < 1 || p.E > kMaxExperts) return cudaErrorInvalidValue;
  return launch_pdl(k_adaptive_bins, dim3(1), dim3(kMaxExperts), 0, s, p);
}

}  // namespace smoes
