// router_fwd.cu -- SMoES router forward on sm_103a.
//
// One pass over X computes, per token: the gate logits z = W x (Sec. 3.1) on tcgen05 tensor
// cores (TMA-fed, accumulators in TMEM), the Gaussian modality score of eqs. (8)-(9) from the
// same shared-memory X tiles, softmax, top-k, bin sums p_k = sum_{e in B_k} g_e, and the
// per-(128-token tile, sample) partial sums of the joint table of eq. (12). The epilogue group
// that completes the last partial of a sample reduces that sample's joint to P (eq. 13),
// I (eq. 14) and the backward coefficient table; the one that completes the last sample writes
// the loss of eq. (15). All reductions run in a fixed order: results are bitwise reproducible.
#include <cuda_bf16.h>
#include <math_constants.h>

#include "device_common.cuh"
#include "ptx.cuh"
#include "smoes_internal.cuh"

namespace smoes {
namespace {

constexpr float kLog2e = 1.4426950408889634f;
constexpr int kTileRows = kPieceTokens;      // 128 tokens per tile and per partial-sum piece
constexpr int kPsStride = kTileRows + 1;     // padded row of the per-bin probability table

// Top-k selection key: the logit's bits mapped to an unsigned order-preserving integer, with
// the low `ib` bits replaced by (2^ib - 1 - e). Keys order by logit (to 23 - ib mantissa bits,
// at least 15) and, among equal logits, by ascending expert index.
__device__ __forceinline__ uint32_t topk_key(float z, int e, uint32_t imask) {
  const uint32_t u = __float_as_uint(z);
  const uint32_t o = (u & 0x80000000u) ? ~u : (u | 0x80000000u);
  return (o & ~imask) | (imask - static_cast<uint32_t>(e));
}

// Sorted (descending) insertion of key q into tk[0..KM): new[i] = max(tk[i], min(tk[i-1], q)).
template <int KM>
__device__ __forceinline__ void topk_push(uint32_t (&tk)[KM], uint32_t q) {
#pragma unroll
  for (int i = KM - 1; i > 0; --i) tk[i] = max(tk[i], min(tk[i - 1], q));
  tk[0] = max(tk[0], q);
}

// Reduces sample s (called by the one warp that completed its last piece): fixed-order sums of
// the pieces, then eqs. (12)-(14) and the backward coefficients
//   a_k = dI/dSbar_vk / (N_B A_v), b_k = dI/dSbar_tk / (N_B A_t), h_k = (a_k + b_k) / 2,
//   dI/dSbar_mk = (log(P_mk / (P_m P_k)) - I) / Z,
// so that dI/dg_je = M_jv a_b(e) + M_jt b_b(e) = h_b(e) + (M_jv - 1/2) a_b(e) + (M_jt - 1/2) b_b(e).
//
// Evaluation (fp32, no cancellation): with q_k = Q_k / sum_k Q_k, write N_B Sbar_mk = q_k rho_mk,
// rho_mk = 1 + eps_mk. For a modality holding at least a quarter of the mass the centred sums give
// eps_mk = (x_mk - y_m) / (1 + y_m), x_mk = 2 R_mk / Q_k, y_m = 2 D_m / n; otherwise
// eps_mk = N_mk n / (Q_k A_m) - 1. With s_m = sum_k q_k eps_mk (so N_B sum_k Sbar_mk = 1 + s_m),
//   P_mk = q_k (1 + eps_mk) / (2 + s_v + s_t),
//   log(P_mk / (P_m P_k)) = log1p(eps_mk) - log1p((eps_vk + eps_tk)/2) + log1p((s_v + s_t)/2) - log1p(s_m),
// every term a log1p of a small, directly computed quantity; h_k is formed from second-order
// differences directly as well (see below).
constexpr int kReduceRound = 16;             // pieces loaded per round before they are summed

__device__ void sample_reduce(const FwdParams& p, int s) {
  const Dims& dm = p.dm;
  const int K = dm.K;
  const int NV = piece_values(K);
  const int lane = threadIdx.x & 31;
  const int pb = p.ws.sample_pieces[s], pe = p.ws.sample_pieces[s + 1];
  float acc[6];
#pragma unroll
  for (int t = 0; t < 6; ++t) acc[t] = 0.f;
  const int nval = (NV + 31) / 32;            // values per lane (<= 6)
  for (int q0 = pb; q0 < pe; q0 += kReduceRound) {
    const int nq = min(kReduceRound, pe - q0);
    if (nval <= 3) {
      float v[kReduceRound][3];
#pragma unroll
      for (int u = 0; u < kReduceRound; ++u)
#pragma unroll
        for (int t = 0; t < 3; ++t) {
          const int c = lane + 32 * t;
          v[u][t] = (u < nq && c < NV) ? __ldcg(p.ws.pieces + static_cast<size_t>(q0 + u) * dm.pstride + c) : 0.f;
        }
#pragma unroll
      for (int u = 0; u < kReduceRound; ++u)
#pragma unroll
        for (int t = 0; t < 3; ++t) acc[t] += v[u][t];
    } else {
      for (int u = 0; u < nq; ++u)
#pragma unroll
        for (int t = 0; t < 6; ++t) {
          const int c = lane + 32 * t;
          if (c < NV) acc[t] += __ldcg(p.ws.pieces + static_cast<size_t>(q0 + u) * dm.pstride + c);
        }
    }
  }
  auto fetch = [&](int v) -> float {
    float r = 0.f;
#pragma unroll
    for (int t = 0; t < 6; ++t) {
      const float x = __shfl_sync(0xffffffffu, acc[t], v & 31);
      if ((v >> 5) == t) r = x;
    }
    return r;
  };
  const bool act = lane < K;
  const int kk = act ? lane : 0;
  const float Qall = fetch(kk);                // every lane takes part in the shuffles
  const float Q = act ? Qall : 0.f;
  const float Rv = fetch(K + kk), Rt = fetch(2 * K + kk);
  const float Nv = fetch(3 * K + kk), Nt = fetch(4 * K + kk);
  const float Dv = fetch(5 * K), Dt = fetch(5 * K + 1), Avd = fetch(5 * K + 2), Atd = fetch(5 * K + 3);
  const float n = static_cast<float>(p.ws.offsets[s + 1] - p.ws.offsets[s]);
  const float sumQ = warp_sum(Q);
  const float q = act ? Q / sumQ : 0.f;
  // per-modality mass and deviation of rho from 1
  const bool cv = Avd >= 0.25f * n, ct = Atd >= 0.25f * n;
  const float Av = cv ? 0.5f * n + Dv : Avd;
  const float At = ct ? 0.5f * n + Dt : Atd;
  const bool has_v = Av > 1e-12f, has_t = At > 1e-12f;   // absent modality: Sbar row = 0
  float ev = 0.f, et = 0.f;
  if (act && has_v) {
    if (cv) { const float y = 2.f * Dv / n; ev = (2.f * Rv / Q - y) / (1.f + y); }
    else    { ev = Nv * n / (Q * Av) - 1.f; }
  }
  if (act && has_t) {
    if (ct) { const float y = 2.f * Dt / n; et = (2.f * Rt / Q - y) / (1.f + y); }
    else    { et = Nt * n / (Q * At) - 1.f; }
  }
  const float sv = warp_sum(q * ev), st = warp_sum(q * et);
  const float NB = static_cast<float>(dm.N_B);
  float Pv = 0.f, Pt = 0.f, a = 0.f, b = 0.f, h = 0.f, I = 0.f;
  if (has_v && has_t) {
    const float nbz = 2.f + sv + st;                               // N_B * Z
    Pv = q * (1.f + ev) / nbz;                                     // eq. (13)
    Pt = q * (1.f + et) / nbz;
    const float lk = log1pf(0.5f * (ev + et)), lz = log1pf(0.5f * (sv + st));
    const float Lv = act ? log1pf(ev) - lk + lz - log1pf(sv) : 0.f;
    const float Lt = act ? log1pf(et) - lk + lz - log1pf(st) : 0.f;
    I = warp_sum(Pv * Lv + Pt * Lt);                               // eq. (14)
    const float Z = nbz / NB;
    a = act ? (Lv - I) / Z / (NB * Av) : 0.f;
    b = act ? (Lt - I) / Z / (NB * At) : 0.f;
    if (cv && ct && act) {
      // h = (a + b) / 2 is second order (a ~ -b): form L_v + L_t and 1/A_v - 1/A_t directly,
      //   L_v + L_t = log1p(-(d/(1+m))^2) - log1p(-(d_s/(1+m_s))^2),
      // with m, d the half-sum and half-difference of (eps_v, eps_t) and m_s, d_s those of (s_v, s_t).
      const float yv = 2.f * Dv / n, yt = 2.f * Dt / n;
      const float m = 0.5f * (ev + et), dd = 0.5f * (ev - et);
      const float ms = 0.5f * (sv + st), ds = 0.5f * (sv - st);
      const float rk = dd / (1.f + m), rs = ds / (1.f + ms);
      const float S2 = log1pf(-rk * rk) - log1pf(-rs * rs);
      h = ((S2 - 2.f * I) / (1.f + yv) + (Lt - I) * (yv - yt) / ((1.f + yv) * (1.f + yt))) / (Z * NB * n);
    } else {
      h = 0.5f * (a + b);
    }
  } else if (has_v || has_t) {                                     // one modality only: I = 0
    const float e1 = has_v ? ev : et, s1 = has_v ? sv : st;
    const float P1 = q * (1.f + e1) / (1.f + s1);
    Pv = has_v ? P1 : 0.f;
    Pt = has_t ? P1 : 0.f;
  }
  if (act) {
    float* tb = p.ws.tabs + static_cast<size_t>(s) * 3 * K;
    tb[lane] = a;
    tb[K + lane] = b;
    tb[2 * K + lane] = h;
    if (p.joint) {
      p.joint[(static_cast<size_t>(s) * 2 + 0) * K + lane] = Pv;
      p.joint[(static_cast<size_t>(s) * 2 + 1) * K + lane] = Pt;
    }
  }
  if (lane == 0) {
    p.mi[s] = I;
    p.ws.mi32[s] = I;
    const uint32_t absent = (has_v ? 0u : 1u) + (has_t ? 0u : 1u);
    if (absent) atomicAdd(p.ws.status + 1, absent);
    if (!isfinite(I) || !(sumQ > 0.f)) atomicOr(p.ws.status, kStatusData);
    p.ws.sample_ticket[s] = 0u;                       // ready for the next call
  }
  __threadfence();
  __syncwarp();
  uint32_t last = 0;
  if (lane == 0) last = (atomicAdd(p.ws.loss_ticket, 1u) + 1u == static_cast<uint32_t>(dm.B));
  last = __shfl_sync(0xffffffffu, last, 0);
  if (last) {                                         // eq. (15) for one layer
    __threadfence();
    float t = 0.f;
    for (int i = lane; i < dm.B; i += 32) t += __ldcg(p.ws.mi32 + i);
    t = warp_sum(t);
    if (lane == 0) {
      *p.loss = -t / static_cast<float>(dm.B);
      *p.ws.loss_ticket = 0u;
    }
  }
}

// Shared memory used by the per-tile epilogue group (128 threads, one token row each).
struct EpiSmem {
  float* p_s;            // [2][K][kPsStride] bin probabilities of the tile's rows
  float* m_s;            // [2][4][128] (M_v - 1/2, M_t - 1/2, M_v, M_t) of the tile's rows
  uint64_t* bar_in;      // count 128: the tile's rows are in p_s / m_s
  uint64_t* bar_out;     // count 128: the tile's pieces are written
  const int* s_bin;      // [E]
};

// Per-tile epilogue. Provider::load32(c, v) returns logits [32c, 32c+32) of this thread's row
// (warp-collective; Provider::ncols = logits available, a multiple of 16); release() is called
// after the last logit read. row: token row in the tile; etid: 0..127 inside the group;
// lt: index of the tile among those this group processes (selects buffers and phases).
template <int KM, class Provider, class Release>
__device__ void epilogue_tile(const FwdParams& p, const Provider& prov, const Release& release,
                              int tile, int row, int etid, int lt, float dll, const EpiSmem& es,
                              const WaitCtx& wc) {
  const Dims& dm = p.dm;
  const int E = dm.E, K = dm.K, k = dm.k;
  const int j = tile * kTileRows + row;
  const bool valid = j < dm.T;
  const int buf = lt & 1;
  float* p_s = es.p_s + buf * K * kPsStride;
  float* m_s = es.m_s + buf * 4 * kTileRows;
  const uint32_t imask = (E <= 2) ? 1u : ((1u << (32 - __clz(E - 1))) - 1u);
  const int nch = (prov.ncols + 31) / 32;

  // pass 1: softmax max and top-k keys
  uint32_t tk[KM];
#pragma unroll
  for (int i = 0; i < KM; ++i) tk[i] = 0u;
  float mx = -CUDART_INF_F;
  for (int c = 0; c < nch; ++c) {
    float v[32];
    prov.load32(c, v);
#pragma unroll
    for (int t = 0; t < 32; ++t) {
      const int e = c * 32 + t;
      if (e < E) {
        mx = fmaxf(mx, v[t]);
        topk_push<KM>(tk, topk_key(v[t], e, imask));
      }
    }
  }
  // pass 2: softmax denominator
  float sum = 0.f;
  for (int c = 0; c < nch; ++c) {
    float v[32];
    prov.load32(c, v);
#pragma unroll
    for (int t = 0; t < 32; ++t)
      if (c * 32 + t < E) sum += exp2f((v[t] - mx) * kLog2e);
  }
  const float inv = 1.f / sum;
  if (valid && !(isfinite(mx) && isfinite(sum) && sum > 0.f)) atomicOr(p.ws.status, kStatusData);
  // pass 3: g, saved g, bin sums (accumulated over runs of experts sharing a bin)
  for (int kb = 0; kb < K; ++kb) p_s[kb * kPsStride + row] = 0.f;
  float* grow = p.ws.gsave + static_cast<size_t>(valid ? j : 0) * E;
  const bool vec = (E & 3) == 0;
  float run = 0.f;
  int run_bin = es.s_bin[0];
  for (int c = 0; c < nch; ++c) {
    float v[32];
    prov.load32(c, v);
#pragma unroll
    for (int t = 0; t < 32; ++t) v[t] = (c * 32 + t < E) ? exp2f((v[t] - mx) * kLog2e) * inv : 0.f;
    if (valid) {
      if (vec && c * 32 + 32 <= E) {
#pragma unroll
        for (int t = 0; t < 32; t += 4)
          *reinterpret_cast<float4*>(grow + c * 32 + t) = make_float4(v[t], v[t + 1], v[t + 2], v[t + 3]);
      } else {
#pragma unroll
        for (int t = 0; t < 32; ++t)
          if (c * 32 + t < E) grow[c * 32 + t] = v[t];
      }
    }
#pragma unroll
    for (int t = 0; t < 32; ++t) {
      const int e = c * 32 + t;
      if (e < E) {
        const int b = es.s_bin[e];                 // warp-uniform
        if (b != run_bin) {
          p_s[run_bin * kPsStride + row] += run;
          run = 0.f;
          run_bin = b;
        }
        run += v[t];
      }
    }
  }
  p_s[run_bin * kPsStride + row] += run;
  release();

  // modality score of this token (eq. 9 for two modalities, or the provided scores)
  float Mv = 0.f, Mt = 0.f, dv = 0.f, dt = 0.f;
  if (valid) {
    if (p.M_in) {
      const float2 m = __ldg(reinterpret_cast<const float2*>(p.M_in) + j);
      Mv = m.x;
      Mt = m.y;
      dv = Mv - 0.5f;
      dt = Mt - 0.5f;
    } else {
      const float y = dll * p.inv_tau;
      Mv = sigmoid_acc(y);
      Mt = sigmoid_acc(-y);
      dv = 0.5f * tanhf(0.5f * y);
      dt = -dv;
      if (p.M_out) reinterpret_cast<float2*>(p.M_out)[j] = make_float2(Mv, Mt);
    }
    // top-k outputs: indices from the keys, weights = the exact saved scores
    float w[KM];
    float wsum = 0.f;
#pragma unroll
    for (int i = 0; i < KM; ++i) {
      w[i] = 0.f;
      if (i < k) {
        const int e = static_cast<int>(imask - (tk[i] & imask));
        p.topk_idx[static_cast<size_t>(j) * k + i] = e;
        w[i] = grow[e];
        wsum += w[i];
      }
    }
    const float ws = dm.renorm ? 1.f / wsum : 1.f;
#pragma unroll
    for (int i = 0; i < KM; ++i)
      if (i < k) p.topk_w[static_cast<size_t>(j) * k + i] = w[i] * ws;
    if (p.bin_prob)
      for (int kb = 0; kb < K; ++kb) p.bin_prob[static_cast<size_t>(j) * K + kb] = p_s[kb * kPsStride + row];
  }
  m_s[0 * kTileRows + row] = dv;
  m_s[1 * kTileRows + row] = dt;
  m_s[2 * kTileRows + row] = Mv;
  m_s[3 * kTileRows + row] = Mt;
  mbar_arrive(es.bar_in);
  if (!mbar_wait(es.bar_in, static_cast<uint32_t>(lt & 1), wc)) return;

  // partial sums of the joint table: one piece per (tile, sample), fixed row order
  const int t0 = tile * kTileRows;
  const int s0 = p.ws.token_sample[t0];
  const int s1 = p.ws.token_sample[min(t0 + kTileRows - 1, dm.T - 1)];
  const int NV = piece_values(K);
  const int pbase = p.ws.piece_base[tile];
  for (int s = s0; s <= s1; ++s) {
    const int r0 = max(p.ws.offsets[s] - t0, 0);
    const int r1 = min(p.ws.offsets[s + 1] - t0, kTileRows);
    float* piece = p.ws.pieces + static_cast<size_t>(pbase + (s - s0)) * dm.pstride;
    for (int v = etid; v < NV; v += 128) {
      float acc = 0.f;
      if (v < 5 * K) {
        const int kind = v / K, kb = v - kind * K;
        const float* pr = p_s + kb * kPsStride;
        if (kind == 0) {
          for (int r = r0; r < r1; ++r) acc += pr[r];
        } else {
          const float* wr = m_s + (kind - 1) * kTileRows;
          for (int r = r0; r < r1; ++r) acc = fmaf(wr[r], pr[r], acc);
        }
      } else {
        const float* wr = m_s + (v - 5 * K) * kTileRows;
        for (int r = r0; r < r1; ++r) acc += wr[r];
      }
      piece[v] = acc;
    }
  }
  __threadfence();
  mbar_arrive(es.bar_out);
  if (etid < 32) {                        // one warp announces the pieces and reduces samples
    const int lane = threadIdx.x & 31;
    bool ok = true;
    if (lane == 0) ok = mbar_wait(es.bar_out, static_cast<uint32_t>(lt & 1), wc);
    ok = __shfl_sync(0xffffffffu, ok, 0);
    if (!ok) return;
    for (int s = s0; s <= s1; ++s) {
      uint32_t last = 0;
      if (lane == 0) {
        const uint32_t need = static_cast<uint32_t>(p.ws.sample_pieces[s + 1] - p.ws.sample_pieces[s]);
        last = (atomicAdd(p.ws.sample_ticket + s, 1u) + 1u == need);
      }
      last = __shfl_sync(0xffffffffu, last, 0);
      if (last) {
        __threadfence();
        sample_reduce(p, s);
      }
    }
  }
}

// Gaussian coefficients computed by the 128 threads of the Gaussian group (gtid 0..127), with
// the group synchronised through `bar` (count 128). Returns gc in every thread.
__device__ float gauss_coef_group(const FwdParams& p, int dpad, float* ga, float* gb, float* red,
                                  uint64_t* bar, int gtid, const WaitCtx& wc) {
  const int d = p.dm.d;
  constexpr int kU = 8;                      // elements per thread and round, loads first
  float part = 0.f;
  bool bad = false;
  for (int i0 = gtid; i0 < dpad; i0 += 128 * kU) {
    float vv[kU], vt[kU], mv[kU], mt[kU];
#pragma unroll
    for (int u = 0; u < kU; ++u) {
      const int i = i0 + 128 * u;
      const bool in = i < d;
      vv[u] = in ? __ldg(p.var + i) : 1.f;
      vt[u] = in ? __ldg(p.var + d + i) : 1.f;
      mv[u] = in ? __ldg(p.mu + i) : 0.f;
      mt[u] = in ? __ldg(p.mu + d + i) : 0.f;
    }
#pragma unroll
    for (int u = 0; u < kU; ++u) {
      const int i = i0 + 128 * u;
      if (i >= dpad) break;
      if (!(vv[u] > 0.f) || !(vt[u] > 0.f) || !isfinite(vv[u]) || !isfinite(vt[u]) ||
          !isfinite(mv[u]) || !isfinite(mt[u]))
        bad = true;
      const float pv = vv[u] * vt[u];
      ga[i] = (vv[u] - vt[u]) / (2.f * pv);
      gb[i] = (mv[u] * vt[u] - mt[u] * vv[u]) / pv;
      if (i < d) part += log1pf((vv[u] - vt[u]) / vt[u]) + (mv[u] * mv[u] * vt[u] - mt[u] * mt[u] * vv[u]) / pv;
    }
  }
  if (bad) atomicOr(p.ws.status, kStatusData);
  part = warp_sum(part);
  if ((gtid & 31) == 0) red[gtid >> 5] = part;
  mbar_arrive(bar);
  mbar_wait(bar, 0, wc);
  return -0.5f * (((red[0] + red[1]) + red[2]) + red[3]);
}

// ------------------------------------------------------------------ tcgen05 forward (bf16)

__host__ __device__ inline size_t fwd_stage_bytes(int N) { return 16384u + static_cast<size_t>(N) * 128u; }

__host__ __device__ inline size_t epi_smem_floats(int K) {
  return 2u * static_cast<size_t>(K) * kPsStride + 2u * 4u * kTileRows;
}

__host__ __device__ inline size_t fwd_smem_bytes(int N, int n_stages, int d, int K, int E, bool gauss) {
  size_t b = static_cast<size_t>(n_stages) * fwd_stage_bytes(N);
  if (gauss) b += 2u * sizeof(float) * static_cast<size_t>(round_up(d, kFwdBK));
  b += sizeof(float) * (epi_smem_floats(K) + 256u + 8u);
  b += sizeof(int) * static_cast<size_t>(round_up(E, 4));
  b += sizeof(uint64_t) * (2u * n_stages + 12u);
  b += 16u;
  return b + 1024u;   // alignment slack
}

template <bool kGauss, int KM>
__global__ void __launch_bounds__(kGauss ? 320 : 192, 1)
k_router_fwd_tc(const __grid_constant__ CUtensorMap tmX, const __grid_constant__ CUtensorMap tmW,
                const FwdParams p, const int N, const int n_stages) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const Dims& dm = p.dm;
  const int dpad = round_up(dm.d, kFwdBK);
  const int n_kb = dpad / kFwdBK;
  const size_t sbytes = fwd_stage_bytes(N);

  uint8_t* q = base;
  uint8_t* stage = q;                             q += n_stages * sbytes;
  float* ga = reinterpret_cast<float*>(q);        q += kGauss ? sizeof(float) * dpad : 0;
  float* gb = reinterpret_cast<float*>(q);        q += kGauss ? sizeof(float) * dpad : 0;
  float* epi = reinterpret_cast<float*>(q);       q += sizeof(float) * epi_smem_floats(dm.K);
  float* dll_s = reinterpret_cast<float*>(q);     q += sizeof(float) * 256;
  float* red = reinterpret_cast<float*>(q);       q += sizeof(float) * 8;
  int* s_bin = reinterpret_cast<int*>(q);         q += sizeof(int) * round_up(dm.E, 4);
  q = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(q) + 7) & ~uintptr_t(7));
  uint64_t* full = reinterpret_cast<uint64_t*>(q);      q += 8 * n_stages;
  uint64_t* empty = reinterpret_cast<uint64_t*>(q);     q += 8 * n_stages;
  uint64_t* acc_full = reinterpret_cast<uint64_t*>(q);  q += 16;
  uint64_t* acc_empty = reinterpret_cast<uint64_t*>(q); q += 16;
  uint64_t* g_full = reinterpret_cast<uint64_t*>(q);    q += 16;
  uint64_t* g_empty = reinterpret_cast<uint64_t*>(q);   q += 16;
  uint64_t* drain = reinterpret_cast<uint64_t*>(q);     q += 8;
  uint64_t* bar_in = reinterpret_cast<uint64_t*>(q);    q += 8;
  uint64_t* bar_out = reinterpret_cast<uint64_t*>(q);   q += 8;
  uint64_t* coef_bar = reinterpret_cast<uint64_t*>(q);  q += 8;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(q); q += 4;
  int* abort_flag = reinterpret_cast<int*>(q);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  WaitCtx wc{abort_flag, p.ws.status, p.limit_ns};

  if (threadIdx.x == 0) {
    *abort_flag = 0;
    for (int i = 0; i < n_stages; ++i) {
      mbar_init(full + i, 1);
      mbar_init(empty + i, 1 + (kGauss ? 4 : 0));
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(acc_full + i, 1);
      mbar_init(acc_empty + i, 128);
      mbar_init(g_full + i, 128);
      mbar_init(g_empty + i, 128);
    }
    mbar_init(drain, 1);
    mbar_init(bar_in, 128);
    mbar_init(bar_out, 128);
    mbar_init(coef_bar, 128);
    fence_mbar_init();
    tma_prefetch_desc(&tmX);
    tma_prefetch_desc(&tmW);
  }
  for (int e = threadIdx.x; e < dm.E; e += blockDim.x) s_bin[e] = p.ws.expert_bin[e];
  const uint32_t tmem_cols = (2 * N <= 32) ? 32u : (2 * N <= 64) ? 64u : (2 * N <= 128) ? 128u
                                                 : (2 * N <= 256) ? 256u : 512u;
  if (warp == 1) tmem_alloc(tmem_slot, tmem_cols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  if (warp == 0) {
    // ---------------------------------------------------------------- TMA producer
    if (lane == 0) {
      int st = 0;
      uint32_t ph = 0;
      long issued = 0;
      bool ok = true;
      const uint32_t tx = static_cast<uint32_t>(sbytes);
      for (int tile = blockIdx.x; tile < p.n_tiles && ok; tile += gridDim.x) {
        for (int kb = 0; kb < n_kb; ++kb) {
          if (!mbar_wait(empty + st, ph ^ 1u, wc)) { ok = false; break; }
          uint8_t* xs = stage + st * sbytes;
          mbar_arrive_expect_tx(full + st, tx);
          tma_load_2d(xs, &tmX, full + st, kb * kFwdBK, tile * kFwdBM);
          tma_load_2d(xs + 16384, &tmW, full + st, kb * kFwdBK, 0);
          ++issued;
          if (++st == n_stages) { st = 0; ph ^= 1u; }
        }
      }
      if (!ok) {            // every issued copy must land before the CTA may exit
        WaitCtx wd = wc;
        int dummy = 0;
        wd.abort_flag = &dummy;
        for (long qn = (issued > n_stages ? issued - n_stages : 0); qn < issued; ++qn)
          mbar_wait(full + (qn % n_stages), static_cast<uint32_t>((qn / n_stages) & 1), wd);
      }
    }
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA issuer
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16(kFwdBM, N, false, false);
      int st = 0;
      uint32_t ph = 0;
      int lt = 0;
      bool ok = true;
      for (int tile = blockIdx.x; tile < p.n_tiles && ok; tile += gridDim.x, ++lt) {
        const int buf = lt & 1;
        const uint32_t use = static_cast<uint32_t>(lt >> 1);
        if (!mbar_wait(acc_empty + buf, (use & 1u) ^ 1u, wc)) { ok = false; break; }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(buf * N);
        for (int kb = 0; kb < n_kb; ++kb) {
          if (!mbar_wait(full + st, ph, wc)) { ok = false; break; }
          tc_fence_after();
          const uint8_t* xs = stage + st * sbytes;
          const uint64_t da = sdesc_sw128(smem_u32(xs), 16, 1024);
          const uint64_t db = sdesc_sw128(smem_u32(xs + 16384), 16, 1024);
#pragma unroll
          for (int kk = 0; kk < kFwdBK / 16; ++kk)   // K = 16 per instruction: +32 bytes
            umma_bf16(d_tmem, da + 2u * kk, db + 2u * kk, idesc, (kb | kk) != 0 ? 1u : 0u);
          umma_commit(empty + st);
          if (++st == n_stages) { st = 0; ph ^= 1u; }
        }
        if (ok) umma_commit(acc_full + buf);
      }
      umma_commit(drain);   // every issued MMA completes before TMEM is released
      WaitCtx wd = wc;
      int dummy = 0;
      wd.abort_flag = &dummy;
      mbar_wait(drain, 0, wd);
    }
  } else if (warp < 6) {
    // ---------------------------------------------------------------- epilogue (4 warps)
    const int lg = warp & 3;                 // TMEM lane group accessible to this warp
    const int row = lg * 32 + lane;          // tile row == TMEM lane == token offset
    const int etid = threadIdx.x - 64;
    EpiSmem es{epi, epi + 2 * dm.K * kPsStride, bar_in, bar_out, s_bin};
    int lt = 0;
    for (int tile = blockIdx.x; tile < p.n_tiles; tile += gridDim.x, ++lt) {
      const int buf = lt & 1;
      const uint32_t use = static_cast<uint32_t>(lt >> 1);
      if (!mbar_wait(acc_full + buf, use & 1u, wc)) break;
      tc_fence_after();
      float dll = 0.f;
      if (kGauss) {
        if (!mbar_wait(g_full + buf, use & 1u, wc)) break;
        dll = dll_s[buf * 128 + row];
        mbar_arrive(g_empty + buf);
      }
      struct Prov {
        uint32_t base;
        int ncols;
        __device__ void load32(int c, float (&v)[32]) const {
          if (32 * c + 32 <= ncols) {
            tmem_ld32(base + 32u * c, v);
          } else {
            float h[16];
            tmem_ld16(base + 32u * c, h);
#pragma unroll
            for (int i = 0; i < 16; ++i) { v[i] = h[i]; v[16 + i] = 0.f; }
          }
        }
      } prov{tmem_base + (static_cast<uint32_t>(lg * 32) << 16) + static_cast<uint32_t>(buf * N), N};
      struct Rel {                  // hand the accumulator buffer back to the MMA warp
        uint64_t* bar;
        __device__ void operator()() const { tc_fence_before(); mbar_arrive(bar); }
      } rel{acc_empty + buf};
      epilogue_tile<KM>(p, prov, rel, tile, row, etid, lt, dll, es, wc);
    }
  } else {
    // ---------------------------------------------------------------- Gaussian warps (4)
    if (kGauss) {
      const int row = (warp - 6) * 32 + lane;
      const float gc = gauss_coef_group(p, dpad, ga, gb, red, coef_bar, row, wc);
      int st = 0;
      uint32_t ph = 0;
      int lt = 0;
      bool ok = true;
      for (int tile = blockIdx.x; tile < p.n_tiles && ok; tile += gridDim.x, ++lt) {
        const int buf = lt & 1;
        const uint32_t use = static_cast<uint32_t>(lt >> 1);
        if (!mbar_wait(g_empty + buf, (use & 1u) ^ 1u, wc)) break;
        float acc = 0.f;
        for (int kb = 0; kb < n_kb; ++kb) {
          if (!mbar_wait(full + st, ph, wc)) { ok = false; break; }
          const uint8_t* xr = stage + st * sbytes + row * 128;
          const float* a = ga + kb * kFwdBK;
          const float* b = gb + kb * kFwdBK;
#pragma unroll
          for (int c = 0; c < 8; ++c) {
            const uint4 u = *reinterpret_cast<const uint4*>(xr + ((c ^ (row & 7)) << 4));
            const float4 a0 = *reinterpret_cast<const float4*>(a + c * 8);
            const float4 a1 = *reinterpret_cast<const float4*>(a + c * 8 + 4);
            const float4 b0 = *reinterpret_cast<const float4*>(b + c * 8);
            const float4 b1 = *reinterpret_cast<const float4*>(b + c * 8 + 4);
            const float x0 = __uint_as_float(u.x << 16), x1 = __uint_as_float(u.x & 0xffff0000u);
            const float x2 = __uint_as_float(u.y << 16), x3 = __uint_as_float(u.y & 0xffff0000u);
            const float x4 = __uint_as_float(u.z << 16), x5 = __uint_as_float(u.z & 0xffff0000u);
            const float x6 = __uint_as_float(u.w << 16), x7 = __uint_as_float(u.w & 0xffff0000u);
            acc = fmaf(x0, fmaf(a0.x, x0, b0.x), acc);
            acc = fmaf(x1, fmaf(a0.y, x1, b0.y), acc);
            acc = fmaf(x2, fmaf(a0.z, x2, b0.z), acc);
            acc = fmaf(x3, fmaf(a0.w, x3, b0.w), acc);
            acc = fmaf(x4, fmaf(a1.x, x4, b1.x), acc);
            acc = fmaf(x5, fmaf(a1.y, x5, b1.y), acc);
            acc = fmaf(x6, fmaf(a1.z, x6, b1.z), acc);
            acc = fmaf(x7, fmaf(a1.w, x7, b1.w), acc);
          }
          __syncwarp();
          if (lane == 0) mbar_arrive(empty + st);
          if (++st == n_stages) { st = 0; ph ^= 1u; }
        }
        if (!ok) break;
        dll_s[buf * 128 + row] = acc + gc;
        mbar_arrive(g_full + buf);
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem_base, tmem_cols);
}

// ------------------------------------------------------------------ FFMA forward (fp32)
// 128 tokens per block, 512 threads: thread (row r = t/4, quarter q = t%4) accumulates the
// logits of experts e = q + 4i over d and a quarter of the Gaussian sum; threads 0..127 then
// run the same epilogue as the tensor-core path (logits read from shared memory).
constexpr int kF32MaxE = 64;

__host__ __device__ inline size_t f32_smem_floats(const Dims& dm) {
  const int E16 = round_up(dm.E, 16);
  const int dpad = round_up(dm.d, 32);
  return 128 * 33 + static_cast<size_t>(dm.E) * 33 + 128 * static_cast<size_t>(E16 + 1) + 2 * dpad +
         epi_smem_floats(dm.K) + 128 + 24;
}

template <bool kGauss, int KM>
__global__ void __launch_bounds__(512)
k_router_fwd_f32(const FwdParams p) {
  extern __shared__ float fs[];
  const Dims& dm = p.dm;
  const int E = dm.E, d = dm.d;
  const int E16 = round_up(E, 16);
  const int dpad = round_up(d, 32);
  float* xs = fs;                          // [128][33]
  float* wsm = xs + 128 * 33;              // [E][33]
  float* zs = wsm + E * 33;                // [128][E16 + 1]
  float* ga = zs + 128 * (E16 + 1);        // [dpad]
  float* gb = ga + dpad;                   // [dpad]
  float* epi = gb + dpad;                  // epilogue tables
  float* dll_s = epi + epi_smem_floats(dm.K);   // [128]
  float* red = dll_s + 128;                // [17]
  uint64_t* bars = reinterpret_cast<uint64_t*>(
      (reinterpret_cast<uintptr_t>(red + 17) + 7) & ~uintptr_t(7));   // [2]
  int* abort_flag = reinterpret_cast<int*>(bars + 2);
  int* s_bin = abort_flag + 1;

  const int t = threadIdx.x, r = t >> 2, qd = t & 3;
  const int tile = blockIdx.x;
  const int j0 = tile * kTileRows;
  if (t == 0) {
    *abort_flag = 0;
    mbar_init(bars + 0, 128);
    mbar_init(bars + 1, 128);
    fence_mbar_init();
  }
  for (int e = t; e < E; e += 512) s_bin[e] = p.ws.expert_bin[e];
  float gc = 0.f;
  if (kGauss) gc = gauss_coefficients(p.mu, p.var, d, dpad, ga, gb, red, p.ws.status);
  float acc[kF32MaxE / 4];
#pragma unroll
  for (int i = 0; i < kF32MaxE / 4; ++i) acc[i] = 0.f;
  float gacc = 0.f;
  const float* X = static_cast<const float*>(p.X);
  const float* W = static_cast<const float*>(p.W);
  __syncthreads();
  for (int d0 = 0; d0 < d; d0 += 32) {
    for (int i = t; i < 128 * 32; i += 512) {
      const int rr = i >> 5, cc = i & 31;
      xs[rr * 33 + cc] = (j0 + rr < dm.T && d0 + cc < d) ? X[static_cast<size_t>(j0 + rr) * d + d0 + cc] : 0.f;
    }
    for (int i = t; i < E * 32; i += 512) {
      const int e = i >> 5, cc = i & 31;
      wsm[e * 33 + cc] = (d0 + cc < d) ? W[static_cast<size_t>(e) * d + d0 + cc] : 0.f;
    }
    __syncthreads();
#pragma unroll 4
    for (int cc = 0; cc < 32; ++cc) {
      const float x = xs[r * 33 + cc];
#pragma unroll
      for (int i = 0; i < kF32MaxE / 4; ++i) {
        const int e = qd + 4 * i;
        if (e < E) acc[i] = fmaf(x, wsm[e * 33 + cc], acc[i]);
      }
      if (kGauss && (cc & 3) == qd) gacc = fmaf(x, fmaf(ga[d0 + cc], x, gb[d0 + cc]), gacc);
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < kF32MaxE / 4; ++i) {
    const int e = qd + 4 * i;
    if (e < E16) zs[r * (E16 + 1) + e] = (e < E) ? acc[i] : 0.f;
  }
  gacc += __shfl_xor_sync(0xffffffffu, gacc, 1);
  gacc += __shfl_xor_sync(0xffffffffu, gacc, 2);
  if (qd == 0) dll_s[r] = gacc + gc;
  __syncthreads();
  if (t < 128) {
    struct Prov {
      const float* z;
      int ncols;
      __device__ void load32(int c, float (&v)[32]) const {
#pragma unroll
        for (int i = 0; i < 32; ++i) v[i] = (32 * c + i < ncols) ? z[32 * c + i] : 0.f;
      }
    } prov{zs + t * (E16 + 1), E16};
    struct Rel {
      __device__ void operator()() const {}
    } rel;
    WaitCtx wc{abort_flag, p.ws.status, p.limit_ns};
    EpiSmem es{epi, epi + 2 * dm.K * kPsStride, bars + 0, bars + 1, s_bin};
    epilogue_tile<KM>(p, prov, rel, tile, t, t, 0, kGauss ? dll_s[t] : 0.f, es, wc);
  }
}

template <bool kGauss>
cudaError_t launch_tc(const FwdParams& p, const CUtensorMap& tmX, const CUtensorMap& tmW, int grid,
                      int threads, size_t smem, int N, int n_stages, cudaStream_t s) {
  auto k = (p.dm.k <= 8) ? k_router_fwd_tc<kGauss, 8> : k_router_fwd_tc<kGauss, 16>;
  cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  k<<<grid, threads, smem, s>>>(tmX, tmW, p, N, n_stages);
  return cudaGetLastError();
}

template <bool kGauss>
cudaError_t launch_f32(const FwdParams& p, size_t smem, cudaStream_t s) {
  auto k = (p.dm.k <= 8) ? k_router_fwd_f32<kGauss, 8> : k_router_fwd_f32<kGauss, 16>;
  cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  k<<<p.n_tiles, 512, smem, s>>>(p);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_router_fwd_bf16(const FwdParams& p, const CUtensorMap& tmX,
                                   const CUtensorMap& tmW, int n_sms, cudaStream_t s) {
  const int N = round_up(p.dm.E, 16);
  const bool gauss = p.M_in == nullptr;
  // as many pipeline stages as fit next to the epilogue's shared memory
  int n_stages = 8;
  while (n_stages > 2 && fwd_smem_bytes(N, n_stages, p.dm.d, p.dm.K, p.dm.E, gauss) > 227u * 1024u)
    --n_stages;
  const size_t smem = fwd_smem_bytes(N, n_stages, p.dm.d, p.dm.K, p.dm.E, gauss);
  if (smem > 227u * 1024u) return cudaErrorInvalidConfiguration;
  const int grid = p.n_tiles < n_sms ? p.n_tiles : n_sms;
  return gauss ? launch_tc<true>(p, tmX, tmW, grid, 320, smem, N, n_stages, s)
               : launch_tc<false>(p, tmX, tmW, grid, 192, smem, N, n_stages, s);
}

cudaError_t launch_router_fwd_f32(const FwdParams& p, cudaStream_t s) {
  if (p.dm.E > kF32MaxE) return cudaErrorInvalidValue;
  const size_t smem = sizeof(float) * f32_smem_floats(p.dm) + sizeof(int) * round_up(p.dm.E, 4) + 64;
  if (smem > 227u * 1024u) return cudaErrorInvalidConfiguration;
  return (p.M_in == nullptr) ? launch_f32<true>(p, smem, s) : launch_f32<false>(p, smem, s);
}

}  // namespace smoes
