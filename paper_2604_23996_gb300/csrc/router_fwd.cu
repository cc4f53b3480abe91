// router_fwd.cu -- SMoES router forward on sm_103a.
//
// One pass over X computes, per token: the gate logits z = W x (Sec. 3.1) on tcgen05 tensor
// cores (TMA-fed, accumulators in TMEM), the Gaussian modality score of eqs. (8)-(9) from the
// same shared-memory X tiles, softmax, top-k, bin sums p_k = sum_{e in B_k} g_e, and the
// per-32-token partial sums of the joint table of eq. (12). The warp that completes the last
// partial of a sample reduces that sample's joint to P (eq. 13), I (eq. 14) and the backward
// coefficient table; the warp that completes the last sample writes the loss of eq. (15).
// All reductions run in a fixed order, so results are bitwise reproducible.
#include <cuda_bf16.h>
#include <math_constants.h>

#include "device_common.cuh"
#include "ptx.cuh"
#include "smoes_internal.cuh"

namespace smoes {
namespace {

constexpr float kLog2e = 1.4426950408889634f;

// Insert (z, e) into the descending list tv[0..k). Strictly-greater comparisons keep the lower
// expert index first among equal logits (experts are offered in ascending order).
__device__ __forceinline__ void topk_insert(float (&tv)[kMaxTopK], int (&ti)[kMaxTopK], int k,
                                            float z, int e) {
#pragma unroll
  for (int i = kMaxTopK - 1; i >= 0; --i) {
    if (i < k) {
      const bool above = (i > 0) && (z > tv[i > 0 ? i - 1 : 0]);
      if (above) {
        tv[i] = tv[i - 1 >= 0 ? i - 1 : 0];
        ti[i] = ti[i - 1 >= 0 ? i - 1 : 0];
      } else if (z > tv[i]) {
        tv[i] = z;
        ti[i] = e;
      }
    }
  }
}

// Reduces sample s (called by the one warp that completed its last piece): fixed-order fp64
// sums of the pieces, then eqs. (12)-(14) and the backward coefficients
//   a_k = dI/dSbar_vk / (N_B A_v), b_k = dI/dSbar_tk / (N_B A_t), h_k = (a_k + b_k) / 2,
//   dI/dSbar_mk = (log(P_mk / (P_m P_k)) - I) / Z,
// so that dI/dg_je = M_jv a_b(e) + M_jt b_b(e) = h_b(e) + (M_jv - 1/2) a_b(e) + (M_jt - 1/2) b_b(e).
__device__ void sample_reduce(const FwdParams& p, int s) {
  const Dims& dm = p.dm;
  const int K = dm.K;
  const int NV = piece_values(K);
  const int lane = threadIdx.x & 31;
  const int pb = p.ws.sample_pieces[s], pe = p.ws.sample_pieces[s + 1];
  double acc[6];
#pragma unroll
  for (int t = 0; t < 6; ++t) acc[t] = 0.0;
  for (int q = pb; q < pe; ++q) {
    const float* pc = p.ws.pieces + static_cast<size_t>(q) * dm.pstride;
#pragma unroll
    for (int t = 0; t < 6; ++t) {
      const int v = lane + 32 * t;
      if (v < NV) acc[t] += static_cast<double>(__ldcg(pc + v));
    }
  }
  auto fetch = [&](int v) -> double {
    double r = 0.0;
#pragma unroll
    for (int t = 0; t < 6; ++t) {
      const double x = __shfl_sync(0xffffffffu, acc[t], v & 31);
      if ((v >> 5) == t) r = x;
    }
    return r;
  };
  const bool act = lane < K;
  const int kk = act ? lane : 0;
  const double Q = fetch(kk), Rv = fetch(K + kk), Rt = fetch(2 * K + kk);
  const double Nvd = fetch(3 * K + kk), Ntd = fetch(4 * K + kk);
  const double Dv = fetch(5 * K), Dt = fetch(5 * K + 1), Avd = fetch(5 * K + 2), Atd = fetch(5 * K + 3);
  const double n = static_cast<double>(p.ws.offsets[s + 1] - p.ws.offsets[s]);
  // centred sums when the modality holds at least a quarter of the sample's mass
  const bool cv = Avd >= 0.25 * n, ct = Atd >= 0.25 * n;
  const double Av = cv ? 0.5 * n + Dv : Avd;
  const double At = ct ? 0.5 * n + Dt : Atd;
  const double Nv = cv ? 0.5 * Q + Rv : Nvd;
  const double Nt = ct ? 0.5 * Q + Rt : Ntd;
  const bool has_v = Av > 1e-12, has_t = At > 1e-12;   // absent modality: Sbar row = 0
  const double NB = static_cast<double>(dm.N_B);
  const double Sv = (act && has_v) ? Nv / (NB * Av) : 0.0;          // eq. (12)
  const double St = (act && has_t) ? Nt / (NB * At) : 0.0;
  const double Z = warp_sum_d(Sv + St);
  const double Pv = Sv / Z, Pt = St / Z;                            // eq. (13)
  const double PV = warp_sum_d(Pv), PT = warp_sum_d(Pt);
  const double Pk = Pv + Pt;
  const double lv = (Pv > 0.0) ? log(Pv / (PV * Pk)) : 0.0;
  const double lt = (Pt > 0.0) ? log(Pt / (PT * Pk)) : 0.0;
  const double I = warp_sum_d(Pv * lv + Pt * lt);                   // eq. (14)
  const double Gv = (Pv > 0.0) ? (lv - I) / Z : 0.0;
  const double Gt = (Pt > 0.0) ? (lt - I) / Z : 0.0;
  const double a = has_v ? Gv / (NB * Av) : 0.0;
  const double b = has_t ? Gt / (NB * At) : 0.0;
  if (act) {
    float* tb = p.ws.tabs + static_cast<size_t>(s) * 3 * K;
    tb[lane] = static_cast<float>(a);
    tb[K + lane] = static_cast<float>(b);
    tb[2 * K + lane] = static_cast<float>(0.5 * (a + b));
    if (p.joint) {
      p.joint[(static_cast<size_t>(s) * 2 + 0) * K + lane] = static_cast<float>(Pv);
      p.joint[(static_cast<size_t>(s) * 2 + 1) * K + lane] = static_cast<float>(Pt);
    }
  }
  if (lane == 0) {
    p.mi[s] = static_cast<float>(I);
    p.ws.mi64[s] = I;
    const uint32_t absent = (has_v ? 0u : 1u) + (has_t ? 0u : 1u);
    if (absent) atomicAdd(p.ws.status + 1, absent);
    if (!(Z > 0.0) || !isfinite(I)) atomicOr(p.ws.status, kStatusData);
    p.ws.sample_ticket[s] = 0u;                       // ready for the next call
  }
  __threadfence();
  __syncwarp();
  uint32_t last = 0;
  if (lane == 0) last = (atomicAdd(p.ws.loss_ticket, 1u) + 1u == static_cast<uint32_t>(dm.B));
  last = __shfl_sync(0xffffffffu, last, 0);
  if (last) {                                         // eq. (15) for one layer
    __threadfence();
    double t = 0.0;
    for (int i = lane; i < dm.B; i += 32) t += __ldcg(p.ws.mi64 + i);
    t = warp_sum_d(t);
    if (lane == 0) {
      *p.loss = static_cast<float>(-t / dm.B);
      *p.ws.loss_ticket = 0u;
    }
  }
}

// Per-token epilogue, executed by one warp for 32 consecutive tokens (lane = token offset).
// Provider::load16(c, v) returns logits [16c, 16c+16) of this lane's token (warp-collective);
// release() is called once the logits have been read for the last time.
// row: this thread's column in p_s (p_s is [K][p_rows]); wg: the 32-token group index.
template <class Provider, class Release>
__device__ void router_epilogue(const FwdParams& p, const Provider& prov, const Release& release,
                                int nchunk16, int row, int j, int wg, float dll, float* p_s,
                                int p_rows, const int* s_bin) {
  const Dims& dm = p.dm;
  const int lane = threadIdx.x & 31;
  const bool valid = j < dm.T;
  const int E = dm.E, K = dm.K, k = dm.k;

  float tv[kMaxTopK];
  int ti[kMaxTopK];
#pragma unroll
  for (int i = 0; i < kMaxTopK; ++i) { tv[i] = -CUDART_INF_F; ti[i] = 0; }
  float mx = -CUDART_INF_F;
  for (int c = 0; c < nchunk16; ++c) {                       // pass 1: max, top-k
    float v[16];
    prov.load16(c, v);
#pragma unroll
    for (int t = 0; t < 16; ++t) {
      const int e = c * 16 + t;
      if (e < E) {
        mx = fmaxf(mx, v[t]);
        topk_insert(tv, ti, k, v[t], e);
      }
    }
  }
  float sum = 0.f;
  for (int c = 0; c < nchunk16; ++c) {                       // pass 2: softmax denominator
    float v[16];
    prov.load16(c, v);
#pragma unroll
    for (int t = 0; t < 16; ++t)
      if (c * 16 + t < E) sum += exp2f((v[t] - mx) * kLog2e);
  }
  const float inv = 1.f / sum;
  if (valid && !(isfinite(mx) && isfinite(sum) && sum > 0.f)) atomicOr(p.ws.status, kStatusData);
  for (int kb = 0; kb < K; ++kb) p_s[kb * p_rows + row] = 0.f;
  float* grow = p.ws.gsave + static_cast<size_t>(valid ? j : 0) * E;
  for (int c = 0; c < nchunk16; ++c) {                       // pass 3: g, saved g, bin sums
    float v[16];
    prov.load16(c, v);
    float g[16];
#pragma unroll
    for (int t = 0; t < 16; ++t) g[t] = (c * 16 + t < E) ? exp2f((v[t] - mx) * kLog2e) * inv : 0.f;
    if (valid) {
      if ((E & 3) == 0 && c * 16 + 16 <= E) {
#pragma unroll
        for (int t = 0; t < 16; t += 4)
          *reinterpret_cast<float4*>(grow + c * 16 + t) = make_float4(g[t], g[t + 1], g[t + 2], g[t + 3]);
      } else {
#pragma unroll
        for (int t = 0; t < 16; ++t)
          if (c * 16 + t < E) grow[c * 16 + t] = g[t];
      }
    }
#pragma unroll
    for (int t = 0; t < 16; ++t) {
      const int e = c * 16 + t;
      if (e < E) p_s[s_bin[e] * p_rows + row] += g[t];
    }
  }
  release();                                                 // logits no longer needed

  // modality score of this token
  float Mv = 0.f, Mt = 0.f, dv = 0.f, dt = 0.f;
  if (valid) {
    if (p.M_in) {
      Mv = __ldg(p.M_in + 2 * static_cast<size_t>(j));
      Mt = __ldg(p.M_in + 2 * static_cast<size_t>(j) + 1);
      dv = Mv - 0.5f;
      dt = Mt - 0.5f;
    } else {
      const float y = dll * p.inv_tau;                     // eq. (9) for two modalities
      Mv = sigmoid_acc(y);
      Mt = sigmoid_acc(-y);
      dv = 0.5f * tanhf(0.5f * y);
      dt = -dv;
      if (p.M_out) {
        *reinterpret_cast<float2*>(p.M_out + 2 * static_cast<size_t>(j)) = make_float2(Mv, Mt);
      }
    }
    // routing outputs
    float wsum = 0.f;
#pragma unroll
    for (int i = 0; i < kMaxTopK; ++i)
      if (i < k) wsum += exp2f((tv[i] - mx) * kLog2e) * inv;
    const float wscale = dm.renorm ? 1.f / wsum : 1.f;
#pragma unroll
    for (int i = 0; i < kMaxTopK; ++i) {
      if (i < k) {
        p.topk_idx[static_cast<size_t>(j) * k + i] = ti[i];
        p.topk_w[static_cast<size_t>(j) * k + i] = exp2f((tv[i] - mx) * kLog2e) * inv * wscale;
      }
    }
    if (p.bin_prob) {
      for (int kb = 0; kb < K; ++kb) p.bin_prob[static_cast<size_t>(j) * K + kb] = p_s[kb * p_rows + row];
    }
  }

  // partial sums of the joint table, one piece per (32-token group, sample) pair
  if (wg >= dm.n_groups) return;
  const int jg0 = wg * kPieceTokens;
  const int s_first = p.ws.token_sample[jg0];
  const int s_last = p.ws.token_sample[min(jg0 + kPieceTokens - 1, dm.T - 1)];
  const int s_j = valid ? p.ws.token_sample[j] : -1;
  const int pbase = p.ws.piece_base[wg];
  for (int s = s_first; s <= s_last; ++s) {
    const bool in = (s_j == s);
    const float mv = in ? Mv : 0.f, mt = in ? Mt : 0.f, xv = in ? dv : 0.f, xt = in ? dt : 0.f;
    float* piece = p.ws.pieces + static_cast<size_t>(pbase + (s - s_first)) * dm.pstride;
    for (int kb = 0; kb < K; ++kb) {
      const float pk = in ? p_s[kb * p_rows + row] : 0.f;
      const float q = warp_sum(pk);
      const float rv = warp_sum(xv * pk);
      const float rt = warp_sum(xt * pk);
      const float nv = warp_sum(mv * pk);
      const float nt = warp_sum(mt * pk);
      if (lane == 0) {
        piece[kb] = q;
        piece[K + kb] = rv;
        piece[2 * K + kb] = rt;
        piece[3 * K + kb] = nv;
        piece[4 * K + kb] = nt;
      }
    }
    const float sdv = warp_sum(xv), sdt = warp_sum(xt), sav = warp_sum(mv), sat = warp_sum(mt);
    uint32_t last = 0;
    if (lane == 0) {
      piece[5 * K] = sdv;
      piece[5 * K + 1] = sdt;
      piece[5 * K + 2] = sav;
      piece[5 * K + 3] = sat;
      __threadfence();
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

// ------------------------------------------------------------------ tcgen05 forward (bf16)

struct FwdSmem {
  uint8_t* stage;        // n_stages x (X tile 16 KB | W tile N x 128 B), 1024-aligned
  float* ga;
  float* gb;
  float* p_s;            // [K][128]
  float* dll;            // [2][128]
  int* s_bin;            // [E]
  uint64_t* full;        // [n_stages]
  uint64_t* empty;       // [n_stages]
  uint64_t* acc_full;    // [2]
  uint64_t* acc_empty;   // [2]
  uint64_t* g_full;      // [2]
  uint64_t* g_empty;     // [2]
  uint64_t* drain;       // [1]
  uint32_t* tmem_slot;
  int* abort_flag;
  float* red;            // [33]
};

__host__ __device__ inline size_t fwd_stage_bytes(int N) { return 16384u + static_cast<size_t>(N) * 128u; }

__host__ __device__ inline size_t fwd_smem_bytes(int N, int n_stages, int d, int K, int E, bool gauss) {
  size_t b = static_cast<size_t>(n_stages) * fwd_stage_bytes(N);
  if (gauss) b += 2u * sizeof(float) * static_cast<size_t>(round_up(d, kFwdBK));
  b += sizeof(float) * (static_cast<size_t>(K) * 128u + 256u);
  b += sizeof(int) * static_cast<size_t>(round_up(E, 4));
  b += sizeof(uint64_t) * (2u * n_stages + 9u);
  b += 16u + 33u * sizeof(float);
  return b + 1024u;   // alignment slack
}

template <bool kGauss>
__global__ void __launch_bounds__(kGauss ? 320 : 192, 1)
k_router_fwd_tc(const __grid_constant__ CUtensorMap tmX, const __grid_constant__ CUtensorMap tmW,
                const FwdParams p, const int N, const int n_stages) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const Dims& dm = p.dm;
  const int dpad = round_up(dm.d, kFwdBK);
  const int n_kb = dpad / kFwdBK;
  const size_t sbytes = fwd_stage_bytes(N);

  FwdSmem sm;
  uint8_t* q = base;
  sm.stage = q;                 q += n_stages * sbytes;
  sm.ga = reinterpret_cast<float*>(q);  q += kGauss ? sizeof(float) * dpad : 0;
  sm.gb = reinterpret_cast<float*>(q);  q += kGauss ? sizeof(float) * dpad : 0;
  sm.p_s = reinterpret_cast<float*>(q); q += sizeof(float) * dm.K * 128;
  sm.dll = reinterpret_cast<float*>(q); q += sizeof(float) * 256;
  sm.s_bin = reinterpret_cast<int*>(q); q += sizeof(int) * round_up(dm.E, 4);
  q = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(q) + 7) & ~uintptr_t(7));
  sm.full = reinterpret_cast<uint64_t*>(q);   q += 8 * n_stages;
  sm.empty = reinterpret_cast<uint64_t*>(q);  q += 8 * n_stages;
  sm.acc_full = reinterpret_cast<uint64_t*>(q);  q += 16;
  sm.acc_empty = reinterpret_cast<uint64_t*>(q); q += 16;
  sm.g_full = reinterpret_cast<uint64_t*>(q);    q += 16;
  sm.g_empty = reinterpret_cast<uint64_t*>(q);   q += 16;
  sm.drain = reinterpret_cast<uint64_t*>(q);     q += 8;
  sm.tmem_slot = reinterpret_cast<uint32_t*>(q); q += 4;
  sm.abort_flag = reinterpret_cast<int*>(q);     q += 4;
  sm.red = reinterpret_cast<float*>(q);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  WaitCtx wc{sm.abort_flag, p.ws.status, p.limit_ns};

  if (threadIdx.x == 0) {
    *sm.abort_flag = 0;
    for (int i = 0; i < n_stages; ++i) {
      mbar_init(sm.full + i, 1);
      mbar_init(sm.empty + i, 1 + (kGauss ? 4 : 0));
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(sm.acc_full + i, 1);
      mbar_init(sm.acc_empty + i, 128);
      mbar_init(sm.g_full + i, 128);
      mbar_init(sm.g_empty + i, 128);
    }
    mbar_init(sm.drain, 1);
    fence_mbar_init();
    tma_prefetch_desc(&tmX);
    tma_prefetch_desc(&tmW);
  }
  for (int e = threadIdx.x; e < dm.E; e += blockDim.x) sm.s_bin[e] = p.ws.expert_bin[e];
  float gc = 0.f;
  if (kGauss) gc = gauss_coefficients(p.mu, p.var, dm.d, dpad, sm.ga, sm.gb, sm.red, p.ws.status);
  const uint32_t tmem_cols = (2 * N <= 32) ? 32u : (2 * N <= 64) ? 64u : (2 * N <= 128) ? 128u
                                                 : (2 * N <= 256) ? 256u : 512u;
  if (warp == 1) tmem_alloc(sm.tmem_slot, tmem_cols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *sm.tmem_slot;

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
          if (!mbar_wait(sm.empty + st, ph ^ 1u, wc)) { ok = false; break; }
          uint8_t* xs = sm.stage + st * sbytes;
          mbar_arrive_expect_tx(sm.full + st, tx);
          tma_load_2d(xs, &tmX, sm.full + st, kb * kFwdBK, tile * kFwdBM);
          tma_load_2d(xs + 16384, &tmW, sm.full + st, kb * kFwdBK, 0);
          ++issued;
          if (++st == n_stages) { st = 0; ph ^= 1u; }
        }
      }
      if (!ok) {
        // drain: every issued copy must land before the CTA may exit
        WaitCtx wd{sm.abort_flag, p.ws.status, p.limit_ns};
        int dummy = 0;
        wd.abort_flag = &dummy;
        for (long qn = (issued > n_stages ? issued - n_stages : 0); qn < issued; ++qn)
          mbar_wait(sm.full + (qn % n_stages), static_cast<uint32_t>((qn / n_stages) & 1), wd);
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
        if (!mbar_wait(sm.acc_empty + buf, (use & 1u) ^ 1u, wc)) { ok = false; break; }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(buf * N);
        for (int kb = 0; kb < n_kb; ++kb) {
          if (!mbar_wait(sm.full + st, ph, wc)) { ok = false; break; }
          tc_fence_after();
          const uint8_t* xs = sm.stage + st * sbytes;
          const uint64_t da = sdesc_sw128(smem_u32(xs), 16, 1024);
          const uint64_t db = sdesc_sw128(smem_u32(xs + 16384), 16, 1024);
#pragma unroll
          for (int kk = 0; kk < kFwdBK / 16; ++kk)   // K = 16 per instruction: +32 bytes
            umma_bf16(d_tmem, da + 2u * kk, db + 2u * kk, idesc, (kb | kk) != 0 ? 1u : 0u);
          umma_commit(sm.empty + st);
          if (++st == n_stages) { st = 0; ph ^= 1u; }
        }
        if (ok) umma_commit(sm.acc_full + buf);
      }
      // make sure every issued MMA has completed before TMEM is released
      umma_commit(sm.drain);
      WaitCtx wd = wc;
      int dummy = 0;
      wd.abort_flag = &dummy;
      mbar_wait(sm.drain, 0, wd);
    }
  } else if (warp < 6) {
    // ---------------------------------------------------------------- epilogue (4 warps)
    const int lg = warp & 3;                 // TMEM lane group accessible to this warp
    const int row = lg * 32 + lane;          // tile row == TMEM lane == token offset
    int lt = 0;
    for (int tile = blockIdx.x; tile < p.n_tiles; tile += gridDim.x, ++lt) {
      const int buf = lt & 1;
      const uint32_t use = static_cast<uint32_t>(lt >> 1);
      if (!mbar_wait(sm.acc_full + buf, use & 1u, wc)) break;
      tc_fence_after();
      float dll = 0.f;
      struct Prov {
        uint32_t base;
        __device__ void load16(int c, float (&v)[16]) const { tmem_ld16(base + 16u * c, v); }
      } prov{tmem_base + (static_cast<uint32_t>(lg * 32) << 16) + static_cast<uint32_t>(buf * N)};
      struct Rel {                  // hand the accumulator buffer back to the MMA warp
        uint64_t* bar;
        __device__ void operator()() const { tc_fence_before(); mbar_arrive(bar); }
      } rel{sm.acc_empty + buf};
      if (kGauss) {
        if (!mbar_wait(sm.g_full + buf, use & 1u, wc)) break;
        dll = sm.dll[buf * 128 + row];
        mbar_arrive(sm.g_empty + buf);
      }
      const int j = tile * kFwdBM + row;
      const int wg = tile * (kFwdBM / 32) + lg;
      router_epilogue(p, prov, rel, N / 16, row, j, wg, dll + gc, sm.p_s, 128, sm.s_bin);
    }
  } else {
    // ---------------------------------------------------------------- Gaussian warps (4)
    if (kGauss) {
      const int row = (warp - 6) * 32 + lane;
      int st = 0;
      uint32_t ph = 0;
      int lt = 0;
      bool ok = true;
      for (int tile = blockIdx.x; tile < p.n_tiles && ok; tile += gridDim.x, ++lt) {
        const int buf = lt & 1;
        const uint32_t use = static_cast<uint32_t>(lt >> 1);
        if (!mbar_wait(sm.g_empty + buf, (use & 1u) ^ 1u, wc)) break;
        float acc = 0.f;
        for (int kb = 0; kb < n_kb; ++kb) {
          if (!mbar_wait(sm.full + st, ph, wc)) { ok = false; break; }
          const uint8_t* xr = sm.stage + st * sbytes + row * 128;
          const float* a = sm.ga + kb * kFwdBK;
          const float* b = sm.gb + kb * kFwdBK;
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
          if (lane == 0) mbar_arrive(sm.empty + st);
          if (++st == n_stages) { st = 0; ph ^= 1u; }
        }
        if (!ok) break;
        sm.dll[buf * 128 + row] = acc;
        mbar_arrive(sm.g_full + buf);
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem_base, tmem_cols);
}

// ------------------------------------------------------------------ FFMA forward (fp32)
// 32 tokens per block; thread (row r = t/4, quarter q = t%4) accumulates the logits of experts
// e = q + 4i over d, and a quarter of the Gaussian sum. Warp 0 then runs the epilogue.
constexpr int kF32MaxE = 64;

template <bool kGauss>
__global__ void __launch_bounds__(128)
k_router_fwd_f32(const FwdParams p) {
  extern __shared__ float fs[];
  const Dims& dm = p.dm;
  const int E = dm.E, d = dm.d;
  const int E16 = round_up(E, 16);
  const int dpad = round_up(d, 32);
  float* xs = fs;                          // [32][33]
  float* wsm = xs + 32 * 33;               // [E][33]
  float* zs = wsm + E * 33;                // [32][E16 + 1]
  float* ga = zs + 32 * (E16 + 1);         // [dpad]
  float* gb = ga + dpad;                   // [dpad]
  float* p_s = gb + dpad;                  // [K][32]
  float* red = p_s + dm.K * 32;            // [8]
  int* s_bin = reinterpret_cast<int*>(red + 8);

  const int t = threadIdx.x, r = t >> 2, qd = t & 3;
  const int j0 = blockIdx.x * 32;
  for (int e = t; e < E; e += 128) s_bin[e] = p.ws.expert_bin[e];
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
    for (int i = t; i < 32 * 32; i += 128) {
      const int rr = i >> 5, cc = i & 31;
      xs[rr * 33 + cc] =
          (j0 + rr < dm.T && d0 + cc < d) ? X[static_cast<size_t>(j0 + rr) * d + d0 + cc] : 0.f;
    }
    for (int i = t; i < E * 32; i += 128) {
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
  float* dll_s = reinterpret_cast<float*>(s_bin + round_up(E, 4));   // [32]
  if (qd == 0) dll_s[r] = gacc + gc;
  __syncthreads();
  if (t < 32) {
    struct Prov {
      const float* z;
      __device__ void load16(int c, float (&v)[16]) const {
#pragma unroll
        for (int i = 0; i < 16; ++i) v[i] = z[16 * c + i];
      }
    } prov{zs + t * (E16 + 1)};
    struct Rel {
      __device__ void operator()() const {}
    } rel;
    router_epilogue(p, prov, rel, E16 / 16, t, j0 + t, blockIdx.x, kGauss ? dll_s[t] : 0.f, p_s, 32,
                    s_bin);
  }
}

size_t f32_smem_bytes(const Dims& dm) {
  const int E16 = round_up(dm.E, 16);
  const int dpad = round_up(dm.d, 32);
  return sizeof(float) * (32 * 33 + dm.E * 33 + 32 * (E16 + 1) + 2 * dpad + dm.K * 32 + 8) +
         sizeof(int) * round_up(dm.E, 4) + sizeof(float) * 32;
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
  if (gauss) {
    auto k = k_router_fwd_tc<true>;
    cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    k<<<grid, 320, smem, s>>>(tmX, tmW, p, N, n_stages);
  } else {
    auto k = k_router_fwd_tc<false>;
    cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    k<<<grid, 192, smem, s>>>(tmX, tmW, p, N, n_stages);
  }
  return cudaGetLastError();
}

cudaError_t launch_router_fwd_f32(const FwdParams& p, cudaStream_t s) {
  if (p.dm.E > kF32MaxE) return cudaErrorInvalidValue;
  const size_t smem = f32_smem_bytes(p.dm);
  const int grid = p.dm.n_groups;
  if (p.M_in == nullptr) {
    auto k = k_router_fwd_f32<true>;
    cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    k<<<grid, 128, smem, s>>>(p);
  } else {
    auto k = k_router_fwd_f32<false>;
    cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    k<<<grid, 128, smem, s>>>(p);
  }
  return cudaGetLastError();
}

}  // namespace smoes
