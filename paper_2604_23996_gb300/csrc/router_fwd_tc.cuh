// router_fwd_tc.cuh -- SMoES router forward on sm_103a: the device code shared by the forward's
// translation units (router_fwd.cu, router_fwd_var.cu) and the tensor-core kernel.
//
// One pass over X computes, per token: the gate logits z = W x (Sec. 3.1) on tcgen05 tensor
// cores (TMA-fed, accumulators in TMEM), the Gaussian modality score of eqs. (8)-(9) from the
// same shared-memory X tiles, softmax, top-k, bin sums p_k = sum_{e in B_k} g_e, and the
// per-(128-token tile, sample) partial sums of the joint table of eq. (12). The epilogue group
// that completes the last partial of a sample reduces that sample's joint to P (eq. 13),
// I (eq. 14) and the backward coefficient table; the one that completes the last sample writes
// the loss of eq. (15). All reductions run in a fixed order: results are bitwise reproducible.
//
// Code that runs once per tile is kept in compact loops: a kernel that streams one or two tiles
// per SM spends most of its epilogue fetching instructions and waiting on dependent latency,
// not issuing arithmetic.
#pragma once
#include <cuda_bf16.h>
#include <math_constants.h>

#include <cfloat>

#include <type_traits>

#include "device_common.cuh"
#include "ptx.cuh"
#include "smoes_internal.cuh"

namespace smoes {
namespace {

constexpr float kLog2e = 1.4426950408889634f;
constexpr int kTileRows = kPieceTokens;      // 128 tokens per tile and per partial-sum piece
constexpr int kPsStride = kTileRows + 1;     // padded row of the per-bin / per-modality tables
constexpr int kMaxNV = piece_values(kMaxBins);
constexpr int kCoefBars = 8;                 // Gaussian coefficient chunks with their own barrier

// Top-k selection key: the logit with its low `ib` mantissa bits replaced by the expert index,
// (2^ib - 1 - e) for a non-negative logit and e for a negative one, so that as floats the keys
// order by logit (to 23 - ib mantissa bits, at least 15) and, among equal logits, by ascending
// expert index. Keys compare with float min/max.
__device__ __forceinline__ float topk_key(float z, int e, uint32_t imask) {
  const uint32_t u = __float_as_uint(z);
  const uint32_t low = (u & 0x80000000u) ? static_cast<uint32_t>(e) : imask - static_cast<uint32_t>(e);
  return __uint_as_float((u & ~imask) | low);
}

// Expert index and logit (low bits set to the middle of their range, relative error below
// 2^(ib - 24)) of a key.
__device__ __forceinline__ int topk_index(float key, uint32_t imask) {
  const uint32_t u = __float_as_uint(key);
  return static_cast<int>((u & 0x80000000u) ? (u & imask) : imask - (u & imask));
}
__device__ __forceinline__ float topk_logit(float key, uint32_t imask) {
  return __uint_as_float((__float_as_uint(key) & ~imask) | ((imask + 1u) >> 1));
}

// Sorted (descending) insertion of key q into tk[0..KM): new[i] = max(tk[i], min(tk[i-1], q)).
template <int KM>
__device__ __forceinline__ void topk_push(float (&tk)[KM], float q) {
#pragma unroll
  for (int i = KM - 1; i > 0; --i) tk[i] = fmaxf(tk[i], fminf(tk[i - 1], q));
  tk[0] = fmaxf(tk[0], q);
}

// Coefficients of the feature pair (2i, 2i+1) (eqs. 8-9) into shared memory as
// {ga[2i], ga[2i+1], gb[2i], gb[2i+1]}; returns the pair's terms of -2 gc, NaN for invalid
// statistics. Not inlined: a CTA evaluates it a few times, so one copy of the code is fetched.
__device__ __noinline__ float gauss_coef_pair(float2 mv, float2 mt, float2 vv, float2 vt, float4* dst) {
  float a0, b0, c0, a1, b1, c1;
  const bool g0 = gauss_coef_feature(mv.x, mt.x, vv.x, vt.x, a0, b0, c0);
  const bool g1 = gauss_coef_feature(mv.y, mt.y, vv.y, vt.y, a1, b1, c1);
  *dst = make_float4(a0, a1, b0, b1);
  return (g0 && g1) ? c0 + c1 : CUDART_NAN_F;
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
// differences directly as well (see below). `red` is kMaxNV floats of shared scratch; the
// sample's pieces [pb, pe) and token count n are passed in when already loaded (pb < 0: load).
//
// dry: the same instruction path with every global access and fence skipped. The first epilogue
// warp runs it once while it waits for its first accumulator, so that this code, which a CTA
// otherwise runs once at the very end, is in the instruction cache when the last piece of a
// sample arrives (a dry run must not touch memory: its loads would queue behind the X stream).
__device__ __noinline__ void sample_reduce(const FwdParams& p, int s, float* red, int pb, int pe,
                                           int nt, bool dry) {
  const Dims& dm = p.dm;
  const int K = dm.K;
  const int NV = piece_values(K);
  const int lane = threadIdx.x & 31;
  if (pb < 0) {
    pb = p.ws.sample_pieces[s];
    pe = p.ws.sample_pieces[s + 1];
    nt = p.ws.offsets[s + 1] - p.ws.offsets[s];
  }
  // lane l sums value 32c + l over the sample's pieces in piece order, 32 loads in flight (one
  // round of memory latency per 32 pieces: the reduction sits on the forward's tail)
#pragma unroll 1
  for (int c = 0; c * 32 < NV; ++c) {
    const int v = 32 * c + lane;
    const bool in = v < NV;
    float acc = 0.f;
#pragma unroll 1
    for (int q0 = pb; q0 < pe; q0 += 32) {
      const float* src = p.ws.pieces + static_cast<size_t>(q0) * dm.pstride + (in ? v : 0);
      float t[32];
#pragma unroll
      for (int i = 0; i < 32; ++i)
        t[i] = (in && !dry && q0 + i < pe) ? __ldcg(src + static_cast<size_t>(i) * dm.pstride) : 0.f;
#pragma unroll
      for (int i = 0; i < 32; ++i) acc += t[i];
    }
    if (in) red[v] = acc;
  }
  __syncwarp();
  const bool act = lane < K;
  const int kk = act ? lane : 0;
  const float Q = act ? red[kk] : 0.f;
  const float Rv = red[K + kk], Rt = red[2 * K + kk];
  const float Nv = red[3 * K + kk], Nt = red[4 * K + kk];
  const float Dv = red[5 * K], Dt = red[5 * K + 1], Avd = red[5 * K + 2], Atd = red[5 * K + 3];
  const float n = static_cast<float>(nt);
  const float sumQ = warp_sum(Q);
  const float q = act ? Q / sumQ : 0.f;
  // per-modality mass and deviation of rho from 1
  const bool cv = Avd >= 0.25f * n, ct = Atd >= 0.25f * n;
  const float Av = cv ? 0.5f * n + Dv : Avd;
  const float At = ct ? 0.5f * n + Dt : Atd;
  const bool has_v = Av > 1e-12f, has_t = At > 1e-12f;   // absent modality: Sbar row = 0
  const float yv = 2.f * Dv / n, yt = 2.f * Dt / n;
  float ev = 0.f, et = 0.f;
  if (act && has_v) ev = cv ? (2.f * Rv / Q - yv) / (1.f + yv) : Nv * n / (Q * Av) - 1.f;
  if (act && has_t) et = ct ? (2.f * Rt / Q - yt) / (1.f + yt) : Nt * n / (Q * At) - 1.f;
  const float sv = warp_sum(q * ev), st = warp_sum(q * et);
  const float NB = static_cast<float>(dm.N_B);
  float Pv = 0.f, Pt = 0.f, a = 0.f, b = 0.f, h = 0.f, I = 0.f;
  if (K == 1) {                      // one bin carries no information: I = 0, P = 1/2 or 1
    Pv = has_v ? (has_t ? 0.5f : 1.f) : 0.f;
    Pt = has_t ? (has_v ? 0.5f : 1.f) : 0.f;
  } else if (has_v && has_t) {
    const float nbz = 2.f + sv + st;                               // N_B * Z
    Pv = q * (1.f + ev) / nbz;                                     // eq. (13)
    Pt = q * (1.f + et) / nbz;
    const float lk = log1pf(0.5f * (ev + et)), lz = log1pf(0.5f * (sv + st));
    const float Lv = act ? log1pf(ev) - lk + lz - log1pf(sv) : 0.f;
    const float Lt = act ? log1pf(et) - lk + lz - log1pf(st) : 0.f;
    I = warp_sum(Pv * Lv + Pt * Lt);                               // eq. (14)
    const float Z = nbz / NB;
    a = act ? (Lv - I) / (Z * NB * Av) : 0.f;
    b = act ? (Lt - I) / (Z * NB * At) : 0.f;
    if (cv && ct && act) {
      // h = (a + b) / 2 is second order (a ~ -b): form L_v + L_t and 1/A_v - 1/A_t directly,
      //   L_v + L_t = log1p(-(d/(1+m))^2) - log1p(-(d_s/(1+m_s))^2),
      // with m, d the half-sum and half-difference of (eps_v, eps_t) and m_s, d_s those of (s_v, s_t).
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
  if (act && !dry) {
    float* tb = p.ws.tabs + static_cast<size_t>(s) * 3 * K;
    tb[lane] = a;
    tb[K + lane] = b;
    tb[2 * K + lane] = h;
    if (p.joint) {
      p.joint[(static_cast<size_t>(s) * 2 + 0) * K + lane] = Pv;
      p.joint[(static_cast<size_t>(s) * 2 + 1) * K + lane] = Pt;
    }
  }
  if (lane == 0 && !dry) {
    p.mi[s] = I;
    p.ws.mi32[s] = I;
    const uint32_t absent = (has_v ? 0u : 1u) + (has_t ? 0u : 1u);
    if (absent) atomicAdd(p.ws.status + 1, absent);
    if (!isfinite(I) || !(sumQ > 0.f)) atomicOr(p.ws.status, kStatusData);
    p.ws.sample_ticket[s] = 0u;                       // ready for the next call
  }
  if (!dry) __threadfence();
  __syncwarp();
  uint32_t last = 0;
  if (lane == 0) last = dry || (atomicAdd(p.ws.loss_ticket, 1u) + 1u == static_cast<uint32_t>(dm.B));
  last = __shfl_sync(0xffffffffu, last, 0);
  if (last) {                                         // eq. (15) for one layer
    if (!dry) __threadfence();
    float t = 0.f;
    for (int i = lane; i < dm.B; i += 32) t += dry ? 0.f : __ldcg(p.ws.mi32 + i);
    t = warp_sum(t);
    if (lane == 0 && !dry) {
      *p.loss = -t / static_cast<float>(dm.B);
      *p.ws.loss_ticket = 0u;
    }
  }
}

// Metadata of one tile, loaded while its accumulator is still being computed: each item is a
// dependent global load that would otherwise sit on the tile's critical path.
struct TileMeta {
  int s0, s1;            // samples of the tile's first and last rows
  int pbase;             // first partial-sum piece of the tile
  int row_sample;        // sample of this thread's row, -1 past T
  int pb0, pe0, n0;      // pieces [pb, pe) and token count of sample s0
  int pb1, pe1, n1;      // the same for sample s1
};

__device__ __forceinline__ TileMeta load_tile_meta(const FwdParams& p, int tile, int row) {
  const Dims& dm = p.dm;
  const int t0 = tile * kTileRows;
  TileMeta m;
  m.row_sample = t0 + row < dm.T ? __ldg(p.ws.token_sample + t0 + row) : -1;
  m.s0 = __ldg(p.ws.token_sample + t0);
  m.s1 = __ldg(p.ws.token_sample + min(t0 + kTileRows - 1, dm.T - 1));
  m.pbase = __ldg(p.ws.piece_base + tile);
  m.pb0 = __ldg(p.ws.sample_pieces + m.s0);
  m.pe0 = __ldg(p.ws.sample_pieces + m.s0 + 1);
  m.n0 = __ldg(p.ws.offsets + m.s0 + 1) - __ldg(p.ws.offsets + m.s0);
  m.pb1 = __ldg(p.ws.sample_pieces + m.s1);
  m.pe1 = __ldg(p.ws.sample_pieces + m.s1 + 1);
  m.n1 = __ldg(p.ws.offsets + m.s1 + 1) - __ldg(p.ws.offsets + m.s1);
  return m;
}

// Shared memory of the per-tile epilogue: two groups of 128 threads, one token row per thread in
// each group (thread `row` of both groups owns tile row `row`); the groups split the logit
// columns. Each warp reads and writes only its own 32 rows of the row tables.
struct EpiSmem {
  float* p_s;            // [K][kPsStride] bin probabilities of the tile's rows
  float* m_s;            // [5][kPsStride] (M_v - 1/2, M_t - 1/2, M_v, M_t, 1) of the tile's rows
  float* wpart;          // [2][4][kMaxNV] per-lane-quarter partial piece sums (double buffer)
  float* red;            // [kMaxNV] sample-reduce scratch of the first warp
  int* ctot;             // [kMaxBins] (token, bin) pairs of the CTA's tiles (fused permutation)
  float* xmax;           // [2][128] per-group row maxima of the logits
  float* xsum;           // [2][128] per-group row sums of exp(z - max)
  float* xtk;            // [kMaxTopK][128] group 1's top-k keys of each row
  uint64_t* bar_in;      // count 256: the partials of one (tile, sample) are written
  uint64_t* bar_out;     // count 256: the tile's pieces are written
  uint64_t* xbar;        // [3] count 256: row maxima and keys / row sums / row tables exchanged
  uint64_t* perm_go;     // count 1: the CTA's top-k and pair counts are complete
  // optional staging of the tile's scores for coalesced TMA stores: 32-column blocks of
  // [128 rows][128 bytes], 16-byte chunks swizzled by row (the 128-byte TMA swizzle); each
  // group stages and stores its own blocks
  uint8_t* stg;          // null: scores are stored row by row
  uint64_t* stg_full;    // [2] count 128: a group's rows are staged
  uint64_t* stg_free;    // [2] count 1: a group's previous store has read the staging
  const CUtensorMap* tmG;
};

__host__ __device__ inline size_t epi_smem_floats(int K) {
  return static_cast<size_t>(K) * kPsStride + 5u * kPsStride + 2u * 4u * kMaxNV + kMaxNV + kMaxBins +
         4u * 128u + static_cast<size_t>(kMaxTopK) * 128u;
}

__device__ inline EpiSmem epi_smem(float* base, int K, uint64_t* bars) {
  EpiSmem es;
  es.p_s = base;
  es.m_s = es.p_s + K * kPsStride;
  es.wpart = es.m_s + 5 * kPsStride;
  es.red = es.wpart + 2 * 4 * kMaxNV;
  es.ctot = reinterpret_cast<int*>(es.red + kMaxNV);
  es.xmax = es.red + kMaxNV + kMaxBins;
  es.xsum = es.xmax + 256;
  es.xtk = es.xsum + 256;
  es.bar_in = bars;
  es.bar_out = bars + 1;
  es.xbar = bars + 2;
  es.perm_go = nullptr;
  es.stg = nullptr;
  es.stg_full = es.stg_free = nullptr;
  es.tmG = nullptr;
  return es;
}
constexpr int kEpiBars = 5;   // bar_in, bar_out, xbar[3]

__device__ inline void init_epi_bars(uint64_t* bars) {
  for (int i = 0; i < kEpiBars; ++i) mbar_init(bars + i, 256);
}

// Column split of the logits between the two epilogue groups: group 0 takes the 16-column chunks
// [0, nc0), group 1 [nc0, nch). nc0 is even (32-column staging blocks stay in one group) and,
// with consecutive bins, a multiple of N_B columns (no bin straddles the groups); otherwise
// group 0 takes every column.
__device__ __forceinline__ int epi_split(const Dims& dm) {
  const int nch = (dm.E + 15) >> 4;
  const int nc0 = 2 * ((nch + 3) >> 2);
  if (nc0 >= nch || !dm.contig_bins || (16 * nc0) % dm.N_B != 0) return nch;
  return nc0;
}

// Per-tile epilogue, run by both groups (grp 0, 1) for every tile. Src::load16(c, v) returns
// logits [16c, 16c+16) of this thread's row, -FLT_MAX past E (finite, so that its top-k key is
// not a NaN; warp-collective); release() is called after the last logit read. row: token row in
// the tile (0..127); lt: index of the tile among those this CTA processes; dll: the row's
// Gaussian log-likelihood difference (read by group 1); meta: the tile's metadata
// (load_tile_meta); n_in: completed phases of bar_in (identical in all 256 threads).
//
// Softmax in two passes over each group's columns: pass A finds the row maximum and top-k keys
// (merged across the groups through shared memory); pass B forms e = exp(z - max), its row sum,
// the bin sums of e and the saved scores (e is saved with 1/sum kept per row, so that nothing
// waits for the sum before storing). Group 0 then writes the top-k outputs and the permutation's
// pair counts, group 1 the modality score; both write the per-(tile, sample) partial sums of the
// joint table (eq. 12), each a half of the values. With the fused permutation, after the CTA's
// last tile the first warp arrives on es.perm_go once all rows are counted.
template <int KM, bool kVar, class Src, class Release>
__device__ void epilogue_tile(const FwdParams& p, const Src& src, const Release& release, int tile,
                              int grp, int row, int lt, float dll, const TileMeta& meta,
                              const EpiSmem& es, const WaitCtx& wc, uint32_t& n_in, bool last_tile) {
  const Dims& dm = p.dm;
  // router variants (sigmoid gate, top-k-masked bins): compiled in only where kVar is set
  const bool v_gate = kVar && dm.gate != 0, v_mask = kVar && dm.mask != 0;
  const int E = dm.E, K = dm.K, k = dm.k;
  const int wg = row >> 5, lane = row & 31;
  const int j = tile * kTileRows + row;
  const bool valid = j < dm.T;
  const int nch = (E + 15) >> 4;
  const int nc0 = epi_split(dm);
  const bool split = nc0 < nch;
  const int cb = grp ? nc0 : 0, ce = grp ? nch : nc0;
  const uint32_t imask = (1u << (32 - __clz(max(nch * 16 - 1, 1)))) - 1u;
  const uint32_t xph = static_cast<uint32_t>(lt & 1);

  // pass A: row maximum and top-k keys of this group's columns, even and odd columns in two
  // independent lists (two dependency chains), merged at the end
  float tk[KM], tk2[KM];
#pragma unroll
  for (int i = 0; i < KM; ++i) tk[i] = tk2[i] = -CUDART_INF_F;
  float mx = -CUDART_INF_F, mx2 = -CUDART_INF_F;
  if (!v_gate) {
#pragma unroll 1
    for (int c = cb; c < ce; ++c) {
      float v[16];
      src.load16(c, v);
#pragma unroll
      for (int t = 0; t < 16; t += 2) {
        mx = fmaxf(mx, v[t]);
        mx2 = fmaxf(mx2, v[t + 1]);
        topk_push<KM>(tk, topk_key(v[t], c * 16 + t, imask));
        topk_push<KM>(tk2, topk_key(v[t + 1], c * 16 + t + 1, imask));
      }
    }
  } else {                           // sigmoid gate: the choice ranks s + bias (padding stays last)
#pragma unroll 1
    for (int c = cb; c < ce; ++c) {
      float v[16];
      src.load16(c, v);
#pragma unroll
      for (int t = 0; t < 16; ++t) {
        const int e = c * 16 + t;
        mx = fmaxf(mx, v[t]);
        v[t] = e < E ? sigmoid_acc(v[t]) + (p.score_bias ? __ldg(p.score_bias + e) : 0.f) : -FLT_MAX;
      }
#pragma unroll
      for (int t = 0; t < 16; t += 2) {
        topk_push<KM>(tk, topk_key(v[t], c * 16 + t, imask));
        topk_push<KM>(tk2, topk_key(v[t + 1], c * 16 + t + 1, imask));
      }
    }
  }
  mx = fmaxf(mx, mx2);
#pragma unroll
  for (int i = 0; i < KM; ++i) topk_push<KM>(tk, tk2[i]);
  es.xmax[grp * 128 + row] = mx;
  if (grp == 1 && split) {
#pragma unroll
    for (int i = 0; i < KM; ++i) es.xtk[i * 128 + row] = tk[i];
  }
  mbar_arrive(es.xbar + 0);
  if (!mbar_wait(es.xbar + 0, xph, wc)) return;
  mx = fmaxf(es.xmax[row], es.xmax[128 + row]);
  if (grp == 0 && split) {
#pragma unroll
    for (int i = 0; i < KM; ++i) topk_push<KM>(tk, es.xtk[i * 128 + row]);
  }

  // pass B: e = exp(z - max), its sum, the bin sums of e and the saved scores
  const float mxl = mx * kLog2e;
  float* grow = p.ws.gsave + static_cast<size_t>(valid ? j : 0) * E;
  float* prow = es.p_s + row;                       // p_s[b][row] at prow[b * kPsStride]
  const bool vec = (E & 3) == 0;
  const bool stg = es.stg != nullptr;
  float sum = 0.f, run = 0.f;
  int cnt = 0, bin = split && grp ? 16 * nc0 / dm.N_B : 0;
  if (!dm.contig_bins && grp == 0)
    for (int b = 0; b < K; ++b) prow[b * kPsStride] = 0.f;
  if (stg && lt > 0 && !mbar_wait(es.stg_free + grp, static_cast<uint32_t>((lt - 1) & 1), wc)) return;
#pragma unroll 1
  for (int c = cb; c < ce; ++c) {
    float v[16];
    src.load16(c, v);
    float ps[4] = {0.f, 0.f, 0.f, 0.f};
    if (!v_gate) {
#pragma unroll
      for (int t = 0; t < 16; ++t) {
        v[t] = exp2f(fmaf(v[t], kLog2e, -mxl));                 // saved e = exp(z - max)
        ps[t & 3] += v[t];
      }
    } else {
#pragma unroll
      for (int t = 0; t < 16; ++t) {
        v[t] = sigmoid_acc(v[t]);                               // saved s = sigmoid(z)
        ps[t & 3] += v[t];
      }
    }
    sum += (ps[0] + ps[1]) + (ps[2] + ps[3]);
    if (stg) {
      uint8_t* rb = es.stg + (c >> 1) * 16384 + row * 128;
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const uint32_t qd = static_cast<uint32_t>((c & 1) * 4 + i);
        *reinterpret_cast<float4*>(rb + ((qd ^ static_cast<uint32_t>(row & 7)) << 4)) =
            make_float4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
      }
    } else if (valid) {
      if (vec && c * 16 + 16 <= E) {
#pragma unroll
        for (int t = 0; t < 16; t += 4)
          *reinterpret_cast<float4*>(grow + c * 16 + t) = make_float4(v[t], v[t + 1], v[t + 2], v[t + 3]);
      } else {
#pragma unroll
        for (int t = 0; t < 16; ++t)
          if (c * 16 + t < E) grow[c * 16 + t] = v[t];
      }
    }
    if (dm.contig_bins) {              // bins are runs of N_B experts, N_B a multiple of 4
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        if (c * 16 + 4 * q >= E) break;   // padding columns (e = 0 past E) end the last bin
        run += (v[4 * q] + v[4 * q + 1]) + (v[4 * q + 2] + v[4 * q + 3]);
        cnt += 4;
        if (cnt == dm.N_B) {
          if (bin < K) prow[bin * kPsStride] = run;
          run = 0.f;
          cnt = 0;
          ++bin;
        }
      }
    } else {                           // any expert -> bin map (group 0 holds every column)
#pragma unroll
      for (int t = 0; t < 16; ++t)
        if (c * 16 + t < E) prow[__ldg(p.ws.expert_bin + c * 16 + t) * kPsStride] += v[t];
    }
  }
  release();
  if (stg) {                      // the group's first thread stores its staged blocks (rows >= T clipped)
    fence_proxy_async_smem();
    mbar_arrive(es.stg_full + grp);
    if (row == 0 && mbar_wait(es.stg_full + grp, static_cast<uint32_t>(lt & 1), wc)) {
      for (int b = cb >> 1; cb < ce && b < (ce + 1) >> 1; ++b)
        tma_store_2d(es.tmG, es.stg + b * 16384, 32 * b, tile * kTileRows);
      tma_store_commit();
    }
  }
  es.xsum[grp * 128 + row] = sum;
  mbar_arrive(es.xbar + 1);
  if (!mbar_wait(es.xbar + 1, xph, wc)) return;
  const float tot = es.xsum[row] + es.xsum[128 + row];
  const float inv = 1.f / tot;
  // this group's bins (all of them for group 0 without a split): e sums -> probabilities
  const int kb0 = split && grp ? 16 * nc0 / dm.N_B : 0;
  const int kb1 = split && !grp ? 16 * nc0 / dm.N_B : (grp && !split ? 0 : K);
  if (!v_mask)                   // (the top-k-masked bins are written by group 0 below)
    for (int b = kb0; b < kb1; ++b) prow[b * kPsStride] = valid ? prow[b * kPsStride] * inv : 0.f;

  float Mv = 0.f, Mt = 0.f, dv = 0.f, dt = 0.f;
  if (grp == 0) {
    if (valid && !(isfinite(mx) && isfinite(tot) && tot > 0.f)) atomicOr(p.ws.status, kStatusData);
    // top-k outputs: indices from the keys; weights = the staged e, or e recomputed from the
    // keys' logits when the scores are not staged, times 1/sum
    if (valid) {
      float w[KM];
      float wsum = 0.f;
#pragma unroll
      for (int i = 0; i < KM; ++i) {
        w[i] = 0.f;
        if (i < k) {
          if (stg) {
            const uint32_t e = static_cast<uint32_t>(topk_index(tk[i], imask));
            const uint32_t qd = ((e & 31u) >> 2) ^ static_cast<uint32_t>(row & 7);
            w[i] = *reinterpret_cast<const float*>(es.stg + (e >> 5) * 16384u + row * 128 + (qd << 4) + (e & 3u) * 4u) * inv;
          } else if (v_gate) {      // s from the key s + bias (renormalised below)
            const int e = topk_index(tk[i], imask);
            w[i] = topk_logit(tk[i], imask) - (p.score_bias ? __ldg(p.score_bias + e) : 0.f);
          } else {
            w[i] = exp2f(fmaf(topk_logit(tk[i], imask), kLog2e, -mxl)) * inv;
          }
        }
        wsum += w[i];
      }
      const float wsc = dm.renorm ? 1.f / wsum : 1.f;
      int32_t* ti = p.topk_idx + static_cast<size_t>(j) * k;
      float* tw = p.topk_w + static_cast<size_t>(j) * k;
#pragma unroll
      for (int i = 0; i < KM; ++i) {
        if (i < k) {
          ti[i] = topk_index(tk[i], imask);
          tw[i] = w[i] * wsc;
        }
      }
      if (v_mask) {                 // eq. (12) on the gate restricted to the top-k, renormalised
        for (int b = 0; b < K; ++b) prow[b * kPsStride] = 0.f;
        const float iw = 1.f / wsum;
#pragma unroll
        for (int i = 0; i < KM; ++i) {
          if (i < k) {
            const int e = topk_index(tk[i], imask);
            const int b = dm.contig_bins ? e / dm.N_B : __ldg(p.ws.expert_bin + e);
            prow[b * kPsStride] += w[i] * iw;
          }
        }
      }
    } else if (v_mask) {
      for (int b = 0; b < K; ++b) prow[b * kPsStride] = 0.f;
    }
    if (p.perm.perm_token) {         // (token, bin) pairs of this warp's rows, per bin
      uint32_t bins = 0u;
      if (valid) {
#pragma unroll
        for (int i = 0; i < KM; ++i) {
          if (i < k) {
            const int e = topk_index(tk[i], imask);
            bins |= 1u << (dm.contig_bins ? e / dm.N_B : __ldg(p.ws.expert_bin + e));
          }
        }
      }
      for (int kb = 0; kb < K; ++kb) {
        const int c = __popc(__ballot_sync(0xffffffffu, (bins >> kb) & 1u));
        if (lane == kb && c) atomicAdd(es.ctot + kb, c);
      }
    }
  } else {
    // modality score of this token (eq. 9 for two modalities, or the provided scores)
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
      p.ws.ginv[j] = inv;
    }
    float* mrow = es.m_s + row;
    mrow[0] = dv;
    mrow[kPsStride] = dt;
    mrow[2 * kPsStride] = Mv;
    mrow[3 * kPsStride] = Mt;
    mrow[4 * kPsStride] = 1.f;
  }
  mbar_arrive(es.xbar + 2);
  if (!mbar_wait(es.xbar + 2, xph, wc)) return;
  if (valid && p.bin_prob)
    for (int b = grp; b < K; b += 2) p.bin_prob[static_cast<size_t>(j) * K + b] = prow[b * kPsStride];

  // partial sums of the joint table: one piece per (tile, sample); group g sums the values of
  // its half over the rows of each lane quarter (lane = value), the four quarters' partials are
  // then added in quarter order. The rows of a sample are contiguous: a ballot over the rows'
  // sample ids gives the warp's range.
  const int NV = piece_values(K);
  const int NVh = (NV + 1) >> 1;
  const int vb = grp ? NVh : 0, ve = grp ? NV : NVh;
  const int tid = grp * 128 + row;
  const int s0 = meta.s0, s1 = meta.s1;
  for (int s = s0; s <= s1; ++s) {
    const uint32_t mine = __ballot_sync(0xffffffffu, meta.row_sample == s);
    const int r0 = 32 * wg + (mine ? __ffs(mine) - 1 : 0);
    const int r1 = 32 * wg + (mine ? 32 - __clz(mine) : 0);
    float* wp = es.wpart + ((n_in & 1) * 4 + wg) * kMaxNV;
    for (int v = vb + lane; v < ve; v += 32) {
      // value v: kind v / K over bin v % K (kind 0: Q, 1..4: weighted by m_s rows 0..3),
      // or, past 5K, the plain sum of m_s row v - 5K
      const int kind = v < 5 * K ? v / K : 0;
      const float* a = v < 5 * K ? es.p_s + (v - kind * K) * kPsStride : es.m_s + (v - 5 * K) * kPsStride;
      const float* w = es.m_s + (v < 5 * K ? (kind + 4) % 5 : 4) * kPsStride;
      float acc = 0.f;
#pragma unroll 4
      for (int r = r0; r < r1; ++r) acc = fmaf(w[r], a[r], acc);
      wp[v] = acc;
    }
    mbar_arrive(es.bar_in);
    if (!mbar_wait(es.bar_in, n_in & 1u, wc)) return;
    const float* w0 = es.wpart + (n_in & 1) * 4 * kMaxNV;
    ++n_in;
    float* piece = p.ws.pieces + static_cast<size_t>(meta.pbase + (s - s0)) * dm.pstride;
    for (int v = tid; v < NV; v += 256)
      piece[v] = ((w0[v] + w0[kMaxNV + v]) + w0[2 * kMaxNV + v]) + w0[3 * kMaxNV + v];
  }
  if (stg && row == 0) {            // the staging may be rewritten once the store has read it
    tma_store_wait_read<0>();
    mbar_arrive(es.stg_free + grp);
  }
  __threadfence();
  mbar_arrive(es.bar_out);
  if (grp == 0 && wg == 0) {            // the first warp announces the pieces, reduces samples
    bool ok = true;
    if (lane == 0) ok = mbar_wait(es.bar_out, static_cast<uint32_t>(lt & 1), wc);
    ok = __shfl_sync(0xffffffffu, ok, 0);
    if (!ok) return;
    // every row of the CTA's last tile is done: its top-k and pair counts may be read
    if (p.perm.perm_token && last_tile && lane == 0) mbar_arrive(es.perm_go);
    for (int s = s0; s <= s1; ++s) {
      // a sample strictly inside the tile has this tile's piece only
      const int pb = s == s0 ? meta.pb0 : s == s1 ? meta.pb1 : meta.pbase + (s - s0);
      const int pe = s == s0 ? meta.pe0 : s == s1 ? meta.pe1 : pb + 1;
      const int nt = s == s0 ? meta.n0 : s == s1 ? meta.n1 : 0;
      uint32_t last = 0;
      if (lane == 0) last = (atomicAdd(p.ws.sample_ticket + s, 1u) + 1u == static_cast<uint32_t>(pe - pb));
      last = __shfl_sync(0xffffffffu, last, 0);
      if (last) {
        __threadfence();
        const bool known = s == s0 || s == s1;
        sample_reduce(p, s, es.red, known ? pb : -1, pe, nt, false);
      }
    }
  }
}

// ------------------------------------------------------------------ fused bin permutation
// The de-duplicated bin dispatch of Sec. 4.5 for the forward's own top-k, run at the end of the
// forward by a group of warps per CTA (warps that are idle once the CTA's gate GEMM is done),
// while the CTA's first epilogue warp reduces samples. Every CTA owns a contiguous run of tiles;
// its epilogue warps add their rows' (token, bin) pairs into a shared total. The group publishes
// the total; after a grid barrier (the launch is cooperative, so every CTA is resident) a CTA's
// base in bin b is the pairs of all bins before b plus those of the CTAs before it in bin b, and
// its tokens are placed in order with ballot ranks. Entries, offsets and counts equal those of
// the standalone permutation kernel: pairs grouped by bin, by token inside a bin; dispatch and
// expert counts are integer sums.
__host__ __device__ inline size_t perm_scratch_ints(int E) {
  return 7u * kMaxBins + static_cast<size_t>(kMaxBins) * kMaxBins + 2u * static_cast<size_t>(E) + 4u;
}

// One token's selection for the permutation: its experts with their bins and slot bits, its set
// of bins, modality (0 vision, 1 text) and dispatch home (-1: invalid).
template <int KM>
struct PermSel {
  int e[KM], b[KM];
  uint32_t sbit[KM];
  uint32_t bins;
  int m, home;
};

template <int KM>
__device__ __forceinline__ void perm_load_sel(const FwdParams& p, int j, PermSel<KM>& t) {
  const Dims& dm = p.dm;
  const FusedPerm& f = p.perm;
  const bool valid = j < dm.T;
  t.bins = 0u;
  t.m = 0;
  t.home = 0;
#pragma unroll
  for (int i = 0; i < KM; ++i) {
    t.e[i] = -1;
    t.b[i] = -1;
    t.sbit[i] = 0u;
    if (valid && i < dm.k) {
      const int e = __ldcg(p.topk_idx + static_cast<size_t>(j) * dm.k + i);   // this CTA's rows
      t.e[i] = e;
      t.b[i] = dm.contig_bins ? e / dm.N_B : __ldg(p.ws.expert_bin + e);
      t.sbit[i] = 1u << __ldg(p.ws.expert_slot + e);
      t.bins |= 1u << t.b[i];
    }
  }
  if (valid) {
    t.m = (f.is_vision && !f.is_vision[j]) ? 1 : 0;
    t.home = f.home ? f.home[j] : static_cast<int>((static_cast<long long>(j) * dm.K) / dm.T);
    if (t.home < 0 || t.home >= dm.K) {
      atomicOr(p.ws.status, kStatusData);
      t.home = -1;
    }
  }
}

// gtid: the thread's index in the group (0 .. 32 nw - 1); bar_id: a named barrier for the group;
// ctot: the CTA's pair counts per bin (complete at perm_go); scratch: perm_scratch_ints(E) ints of
// shared memory that nothing else uses after perm_go.
template <int KM>
__device__ void perm_tail(const FwdParams& p, int t_beg, int t_end, int gtid, int nw, int bar_id,
                          const int* ctot, int* scratch, uint64_t* perm_go, const WaitCtx& wc) {
  const Dims& dm = p.dm;
  const FusedPerm& f = p.perm;
  const int K = dm.K, E = dm.E;
  const int gs = nw * 32, gw = gtid >> 5, lane = gtid & 31;
  int* wcnt = scratch;                          // [4][kMaxBins] per-warp counts, then their bases
  int* base = wcnt + 4 * kMaxBins;              // [kMaxBins] next position of this CTA in bin b
  int* pre_s = base + kMaxBins;                 // [kMaxBins]
  int* tot_s = pre_s + kMaxBins;                // [kMaxBins]
  int* disp = tot_s + kMaxBins;                 // [K][K] dispatch of this CTA's tokens
  int* ecnt = disp + kMaxBins * kMaxBins;       // [2][E] expert counts of this CTA's tokens
  int* flag = ecnt + 2 * E;
  if (gtid == 0) *flag = mbar_wait(perm_go, 0, wc) ? 1 : 0;
  named_bar(bar_id, gs);
  if (!*flag) return;
  // the first round's selections (they land while the other CTAs finish), then the CTA's counts
  const int G = gridDim.x;
  PermSel<KM> sel;
  perm_load_sel<KM>(p, t_beg * kTileRows + gtid, sel);
  if (gtid < K) f.cta_counts[gtid * G + blockIdx.x] = ctot[gtid];
  for (int i = gtid; i < K * K; i += gs) disp[i] = 0;
  for (int i = gtid; i < 2 * E; i += gs) ecnt[i] = 0;
  if (blockIdx.x == 0) {                        // zeroed before any CTA passes the barrier
    for (int i = gtid; i < K * K; i += gs) f.dispatch[i] = 0;
    if (f.expert_counts)
      for (int i = gtid; i < 2 * E; i += gs) f.expert_counts[i] = 0;
  }
  if (gtid < K || blockIdx.x == 0) __threadfence();
  named_bar(bar_id, gs);
  if (gtid == 0) *flag = grid_barrier(f.sync, G, p.limit_ns, p.ws.status) ? 1 : 0;
  named_bar(bar_id, gs);
  if (!*flag) return;

  // this CTA's base in every bin
  for (int kb = gw; kb < K; kb += nw) {
    int pre = 0, tot = 0;
    const int* row = f.cta_counts + kb * G;
#pragma unroll 4
    for (int c = lane; c < G; c += 32) {
      const int v = __ldcg(row + c);
      tot += v;
      if (c < static_cast<int>(blockIdx.x)) pre += v;
    }
    pre = __reduce_add_sync(0xffffffffu, pre);
    tot = __reduce_add_sync(0xffffffffu, tot);
    if (lane == 0) {
      pre_s[kb] = pre;
      tot_s[kb] = tot;
    }
  }
  named_bar(bar_id, gs);
  if (gtid == 0) {
    int run = 0;
    for (int kb = 0; kb < K; ++kb) {
      base[kb] = run + pre_s[kb];
      if (blockIdx.x == 0) f.bin_offsets[kb] = run;
      run += tot_s[kb];
    }
    if (blockIdx.x == 0) f.bin_offsets[K] = run;
  }
  named_bar(bar_id, gs);

  // the CTA's tokens in order: per round, warp counts per bin -> bases over the group's warps ->
  // ballot ranks inside the warp
  const unsigned lt_mask = (1u << lane) - 1u;
  bool first = true;
  for (int tile = t_beg; tile < t_end; ++tile) {
    for (int r0 = 0; r0 < kTileRows; r0 += gs) {
      const int j = tile * kTileRows + r0 + gtid;
      if (!first) perm_load_sel<KM>(p, j, sel);
      first = false;
      for (int kb = 0; kb < K; ++kb) {
        const unsigned bal = __ballot_sync(0xffffffffu, (sel.bins >> kb) & 1u);
        if (lane == 0) wcnt[gw * kMaxBins + kb] = __popc(bal);
      }
      named_bar(bar_id, gs);
      if (gtid < K) {
        int run = base[gtid];
        for (int w = 0; w < nw; ++w) {
          const int t = wcnt[w * kMaxBins + gtid];
          wcnt[w * kMaxBins + gtid] = run;
          run += t;
        }
        base[gtid] = run;
      }
      named_bar(bar_id, gs);
      const unsigned same_home = __match_any_sync(0xffffffffu, sel.home);
      for (int kb = 0; kb < K; ++kb) {
        const unsigned bal = __ballot_sync(0xffffffffu, (sel.bins >> kb) & 1u);
        if ((sel.bins >> kb) & 1u) {
          const int pos = wcnt[gw * kMaxBins + kb] + __popc(bal & lt_mask);
          uint32_t mask = 0u;
#pragma unroll
          for (int i = 0; i < KM; ++i) mask |= (sel.b[i] == kb) ? sel.sbit[i] : 0u;
          f.perm_token[pos] = j;
          f.perm_mask[pos] = mask;
          const unsigned grp = bal & same_home;
          if (sel.home >= 0 && lane == __ffs(grp) - 1) atomicAdd(&disp[sel.home * K + kb], __popc(grp));
        }
      }
      if (f.expert_counts) {
#pragma unroll
        for (int i = 0; i < KM; ++i)
          if (sel.e[i] >= 0) atomicAdd(&ecnt[sel.m * E + sel.e[i]], 1);
      }
      named_bar(bar_id, gs);                    // wcnt is rewritten by the next round
    }
  }
  for (int i = gtid; i < K * K; i += gs)
    if (disp[i]) atomicAdd(f.dispatch + i, disp[i]);
  if (f.expert_counts)
    for (int i = gtid; i < 2 * E; i += gs)
      if (ecnt[i]) atomicAdd(f.expert_counts + i, ecnt[i]);
}

// ------------------------------------------------------------------ tcgen05 forward (bf16)

__host__ __device__ inline size_t fwd_stage_bytes(int N) { return 16384u + static_cast<size_t>(N) * 128u; }

// Staged softmax scores: 32-column blocks of [128 rows][32 floats].
__host__ __device__ inline size_t fwd_stg_bytes(int E) { return static_cast<size_t>(round_up(E, 32)) * 512u; }

__host__ __device__ inline size_t fwd_smem_bytes(int N, int n_stages, int d, int K, int E, bool gauss,
                                                 bool stg) {
  size_t b = static_cast<size_t>(n_stages) * fwd_stage_bytes(N);
  if (stg) b += fwd_stg_bytes(E);
  if (gauss) b += 2u * sizeof(float) * static_cast<size_t>(round_up(d, kFwdBK));
  b += sizeof(float) * (epi_smem_floats(K) + 256u + 8u);
  b += sizeof(uint64_t) * (2u * n_stages + 19u + kEpiBars + kCoefBars);
  b += 16u;
  return b + 1024u;   // alignment slack
}

// Roles: warp 0 TMA producer, warp 1 MMA issuer, warps 2-5 epilogue group 0, then (Gaussian
// score) warps 6-9 Gaussian and 10-13 epilogue group 1, or (provided scores) warps 6-9 epilogue
// group 1. With 14 warps four share a sub-partition's 16K registers: 128 per thread.
constexpr int fwd_threads(bool gauss) { return gauss ? 448 : 320; }

template <bool kGauss, int KM, bool kVar>
__global__ void __launch_bounds__(fwd_threads(kGauss), 1)
k_router_fwd_tc(const __grid_constant__ CUtensorMap tmX, const __grid_constant__ CUtensorMap tmW,
                const __grid_constant__ CUtensorMap tmG, const FwdParams p, const int N,
                const int n_stages, const int use_stg) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const Dims& dm = p.dm;
  const int dpad = round_up(dm.d, kFwdBK);
  const int n_kb = dpad / kFwdBK;
  // CTAs walk the K-blocks from different starting points, so that they do not all request the
  // same W tile from L2 at the same moment
  const int kb0 = blockIdx.x % n_kb;
  auto kb_at = [&](int i) { return (kb0 + i) % n_kb; };
  // a contiguous run of tiles per CTA (the fused permutation orders its entries by CTA)
  const int t_beg = static_cast<int>(static_cast<long long>(blockIdx.x) * p.n_tiles / gridDim.x);
  const int t_end = static_cast<int>(static_cast<long long>(blockIdx.x + 1) * p.n_tiles / gridDim.x);
  const size_t sbytes = fwd_stage_bytes(N);

  uint8_t* q = base;
  uint8_t* stage = q;                             q += n_stages * sbytes;
  uint8_t* stg = q;                               q += use_stg ? fwd_stg_bytes(dm.E) : 0;
  float4* cq = reinterpret_cast<float4*>(q);      q += kGauss ? 2 * sizeof(float) * dpad : 0;
  float* epi = reinterpret_cast<float*>(q);       q += sizeof(float) * epi_smem_floats(dm.K);
  float* dll_s = reinterpret_cast<float*>(q);     q += sizeof(float) * 256;
  float* gred = reinterpret_cast<float*>(q);      q += sizeof(float) * 8;
  q = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(q) + 7) & ~uintptr_t(7));
  uint64_t* full = reinterpret_cast<uint64_t*>(q);      q += 8 * n_stages;
  uint64_t* empty = reinterpret_cast<uint64_t*>(q);     q += 8 * n_stages;
  uint64_t* acc_full = reinterpret_cast<uint64_t*>(q);  q += 16;
  uint64_t* acc_empty = reinterpret_cast<uint64_t*>(q); q += 16;
  uint64_t* g_full = reinterpret_cast<uint64_t*>(q);    q += 16;
  uint64_t* g_empty = reinterpret_cast<uint64_t*>(q);   q += 16;
  uint64_t* drain = reinterpret_cast<uint64_t*>(q);     q += 8;
  uint64_t* ebars = reinterpret_cast<uint64_t*>(q);     q += 8 * kEpiBars;
  uint64_t* coef_bar = reinterpret_cast<uint64_t*>(q);  q += 8 * kCoefBars;
  uint64_t* coef_issued = reinterpret_cast<uint64_t*>(q);  q += 8;
  uint64_t* gc_bar = reinterpret_cast<uint64_t*>(q);    q += 8;
  uint64_t* perm_go = reinterpret_cast<uint64_t*>(q);   q += 8;
  uint64_t* stg_full = reinterpret_cast<uint64_t*>(q);  q += 16;
  uint64_t* stg_free = reinterpret_cast<uint64_t*>(q);  q += 16;
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
      mbar_init(acc_empty + i, 256);             // both epilogue groups read the accumulator
      mbar_init(g_full + i, 128);
      mbar_init(g_empty + i, 128);
      mbar_init(stg_full + i, 128);
      mbar_init(stg_free + i, 1);
    }
    mbar_init(drain, 1);
    init_epi_bars(ebars);
    mbar_init(coef_bar, 256);
    for (int i = 1; i < kCoefBars; ++i) mbar_init(coef_bar + i, 128);
    mbar_init(coef_issued, 256);
    mbar_init(gc_bar, 256);
    mbar_init(perm_go, 1);
    int* ctot = epi_smem(epi, dm.K, ebars).ctot;
    for (int i = 0; i < kMaxBins; ++i) ctot[i] = 0;
    fence_mbar_init();
    tma_prefetch_desc(&tmX);
    tma_prefetch_desc(&tmW);
  }
  const uint32_t tmem_cols = (2 * N <= 32) ? 32u : (2 * N <= 64) ? 64u : (2 * N <= 128) ? 128u
                                                 : (2 * N <= 256) ? 256u : 512u;
  if (warp == 1) tmem_alloc(tmem_slot, tmem_cols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  // X, W, the statistics and the outputs may be in use by the kernel before this one
  pdl_wait();
  pdl_trigger();
  if (blockIdx.x == 0 && threadIdx.x == 0) *p.ws.bal_flag = 0u;   // a new forward: no balance term yet

  if (kGauss && warp >= 2 && warp < 10) {
    // this CTA's Gaussian coefficients (eqs. 8-9), float4 {ga[2i], ga[2i+1], gb[2i], gb[2i+1]}
    // per feature pair i, computed in the order in which the CTA walks the K-blocks, in chunks
    // of eight blocks (256 pairs): chunk 0 by the epilogue and Gaussian warps together, one pair
    // per thread, so that the Gaussian warps consume the first stages early; the later chunks
    // by the four epilogue warps, two pairs per thread, while the stream runs. The loads of
    // chunks 0-3 are all issued before the producer starts the X stream.
    const int ct = threadIdx.x - 64;            // 0..255; 0..127 in the epilogue warps
    const bool epi_w = warp < 6;
    const float2* mu2 = reinterpret_cast<const float2*>(p.mu);
    const float2* var2 = reinterpret_cast<const float2*>(p.var);
    const int np = dm.d / 2;
    const int n_pos = n_kb * 32;
    const int n_chunks = (n_kb + 7) / 8;
    auto pair_at = [&](int pos) { return kb_at(pos >> 5) * 32 + (pos & 31); };
    auto load_pair = [&](int pos, float2 (&v)[4]) {
      const int i = pos < n_pos ? pair_at(pos) : np;
      const bool in = i < np;
      v[0] = in ? __ldg(mu2 + i) : make_float2(0.f, 0.f);
      v[1] = in ? __ldg(mu2 + np + i) : make_float2(0.f, 0.f);
      v[2] = in ? __ldg(var2 + i) : make_float2(1.f, 1.f);
      v[3] = in ? __ldg(var2 + np + i) : make_float2(1.f, 1.f);
    };
    float part = 0.f;
    auto store_pair = [&](int pos, const float2 (&v)[4]) {
      if (pos < n_pos) part += gauss_coef_pair(v[0], v[1], v[2], v[3], cq + pair_at(pos));
    };
    constexpr int kPre = 3;                     // chunks 1..3: loads issued up front
    float2 c0[4], pre[kPre][2][4];
    load_pair(ct, c0);
    if (epi_w) {
#pragma unroll
      for (int c = 1; c <= kPre; ++c) {
        load_pair(256 * c + ct, pre[c - 1][0]);
        load_pair(256 * c + 128 + ct, pre[c - 1][1]);
      }
    }
    mbar_arrive(coef_issued);
    store_pair(ct, c0);
    mbar_arrive(coef_bar);
    if (epi_w) {
      // chunk c completes barrier min(c, kCoefBars - 1); the last barrier covers every chunk
      // from kCoefBars - 1 on and completes after the last one
#pragma unroll
      for (int c = 1; c <= kPre; ++c) {
        if (c < n_chunks) {
          store_pair(256 * c + ct, pre[c - 1][0]);
          store_pair(256 * c + 128 + ct, pre[c - 1][1]);
          if (c < kCoefBars - 1 || c == n_chunks - 1) mbar_arrive(coef_bar + min(c, kCoefBars - 1));
        }
      }
      for (int c = kPre + 1; c < n_chunks; ++c) {
        float2 v0[4], v1[4];
        load_pair(256 * c + ct, v0);
        load_pair(256 * c + 128 + ct, v1);
        store_pair(256 * c + ct, v0);
        store_pair(256 * c + 128 + ct, v1);
        if (c < kCoefBars - 1 || c == n_chunks - 1) mbar_arrive(coef_bar + min(c, kCoefBars - 1));
      }
    }
    if (!isfinite(part)) atomicOr(p.ws.status, kStatusData);
    part = warp_sum(part);
    if (lane == 0) gred[warp - 2] = part;
    mbar_arrive(gc_bar);
  }

  if (warp == 0) {
    // ---------------------------------------------------------------- TMA producer
    if (lane == 0) {
      int st = 0;
      uint32_t ph = 0;
      long issued = 0;
      bool ok = true;
      const uint32_t tx = static_cast<uint32_t>(sbytes);
      // the Gaussian statistics are requested before the X stream floods the memory system
      if (kGauss) ok = mbar_wait(coef_issued, 0, wc);
      for (int tile = t_beg; tile < t_end && ok; ++tile) {
        for (int kb = 0; kb < n_kb; ++kb) {
          if (!mbar_wait(empty + st, ph ^ 1u, wc)) { ok = false; break; }
          uint8_t* xs = stage + st * sbytes;
          mbar_arrive_expect_tx(full + st, tx);
          const int kx = kb_at(kb);
          tma_load_2d(xs, &tmX, full + st, kx * kFwdBK, tile * kFwdBM);
          tma_load_2d(xs + 16384, &tmW, full + st, kx * kFwdBK, 0);
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
      for (int tile = t_beg; tile < t_end && ok; ++tile, ++lt) {
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
  } else if (warp < 6 || warp >= (kGauss ? 10 : 6)) {
    // ---------------------------------------------------------------- epilogue (2 x 4 warps)
    const int grp = warp < 6 ? 0 : 1;        // column half of the logits
    const int lg = warp & 3;                 // TMEM lane group accessible to this warp
    const int row = lg * 32 + lane;          // tile row == TMEM lane == token offset
    EpiSmem es = epi_smem(epi, dm.K, ebars);
    es.perm_go = perm_go;
    if (use_stg) {
      es.stg = stg;
      es.stg_full = stg_full;
      es.stg_free = stg_free;
      es.tmG = &tmG;
    }
    struct Src {                    // logits of this warp's rows from TMEM
      uint32_t base;
      int E;
      __device__ void load16(int c, float (&v)[16]) const {
        tmem_ld16(base + 16u * c, v);
        if (16 * c + 16 > E) {
#pragma unroll
          for (int t = 0; t < 16; ++t)
            if (16 * c + t >= E) v[t] = -FLT_MAX;
        }
      }
    };
    struct Rel {                    // hand the accumulator buffer back to the MMA warp
      uint64_t* bar;
      __device__ void operator()() const { tc_fence_before(); mbar_arrive(bar); }
    };
    const uint32_t tl = tmem_base + (static_cast<uint32_t>(lg * 32) << 16);
    float gc = 0.f;                          // constant term of eq. (8), -1/2 sum of the parts
    if (kGauss && grp == 1 && mbar_wait(gc_bar, 0, wc)) {
      for (int w = 0; w < 8; ++w) gc += gred[w];
      gc *= -0.5f;
    }
    // the sample reduction's code into the instruction cache while the first tile streams in
    if (grp == 0 && lg == 0) sample_reduce(p, 0, es.red, 0, 1, 1, true);
    uint32_t n_in = 0;
    int lt = 0;
    for (int tile = t_beg; tile < t_end; ++tile, ++lt) {
      const int buf = lt & 1;
      const uint32_t use = static_cast<uint32_t>(lt >> 1);
      const TileMeta meta = load_tile_meta(p, tile, row);    // lands while the tile streams in
      if (!mbar_wait(acc_full + buf, use & 1u, wc)) break;
      tc_fence_after();
      float dll = 0.f;
      if (kGauss && grp == 1) {
        if (!mbar_wait(g_full + buf, use & 1u, wc)) break;
        dll = dll_s[buf * 128 + row] + gc;
        mbar_arrive(g_empty + buf);
      }
      epilogue_tile<KM, kVar>(p, Src{tl + static_cast<uint32_t>(buf * N), dm.E}, Rel{acc_empty + buf},
                        tile, grp, row, lt, dll, meta, es, wc, n_in, tile == t_end - 1);
    }
    if (use_stg && row == 0) tma_store_wait_all<0>();   // the score stores complete before exit
  } else {
    // ---------------------------------------------------------------- Gaussian warps (4)
    // Warp w owns tile rows 32w..32w+31 and lane l the feature pair (2l, 2l+1) of every K-block:
    // per stage a lane reads one float4 of coefficients and one 4-byte word of each of its
    // warp's rows, and keeps a running pair of sums per row (even and odd features, two FMAs in
    // one instruction); a butterfly over the lanes gives the row totals at the end of the tile.
    // These warps hold every X stage until they have read it, so their instruction count per
    // stage sets how fast stages return to the producer.
    if (kGauss) {                            // (warps 6-9)
      const int gw = warp - 6;
      const int gt = gw * 32 + lane;
      bool ok = true;
      // byte offset of this lane's word inside a 128-byte swizzled row r: chunk (l/4) ^ (r & 7)
      const uint32_t wcol = static_cast<uint32_t>(lane & 3) * 4u;
      const uint32_t chk = static_cast<uint32_t>(lane >> 2);
      int st = 0;
      uint32_t ph = 0;
      int lt = 0;
      for (int tile = t_beg; tile < t_end && ok; ++tile, ++lt) {
        const int buf = lt & 1;
        const uint32_t use = static_cast<uint32_t>(lt >> 1);
        if (!mbar_wait(g_empty + buf, (use & 1u) ^ 1u, wc)) break;
        uint64_t acc2[32];                   // per row: {sum over even features, over odd}
#pragma unroll
        for (int r = 0; r < 32; ++r) acc2[r] = 0ull;
        for (int kb = 0; kb < n_kb; ++kb) {
          // the coefficients of this block's chunk (complete for every later tile)
          if (lt == 0 && (kb & 7) == 0 && kb < 8 * kCoefBars &&
              !mbar_wait(coef_bar + (kb >> 3), 0, wc)) { ok = false; break; }
          if (!mbar_wait(full + st, ph, wc)) { ok = false; break; }
          const uint8_t* xs = stage + st * sbytes + gw * 32 * 128;
          // {a_2l, a_2l+1} and {b_2l, b_2l+1} of the float4 {ga, ga, gb, gb}
          const ulonglong2 cf = reinterpret_cast<const ulonglong2*>(cq)[kb_at(kb) * 32 + lane];
#pragma unroll
          for (int r = 0; r < 32; ++r) {
            const uint32_t u = *reinterpret_cast<const uint32_t*>(xs + r * 128 + ((chk ^ (r & 7)) << 4) + wcol);
            // {x_2l, x_2l+1} widened from the bf16 pair
            const uint64_t x2 = (static_cast<uint64_t>(u & 0xffff0000u) << 32) | static_cast<uint32_t>(u << 16);
            acc2[r] = ffma2(x2, ffma2(x2, cf.x, cf.y), acc2[r]);    // x (a x + b) + acc, per half
          }
          __syncwarp();
          if (lane == 0) mbar_arrive(empty + st);
          if (++st == n_stages) { st = 0; ph ^= 1u; }
        }
        if (!ok) break;
        float acc[32];
#pragma unroll
        for (int r = 0; r < 32; ++r)
          acc[r] = __uint_as_float(static_cast<uint32_t>(acc2[r])) + __uint_as_float(static_cast<uint32_t>(acc2[r] >> 32));
        dll_s[buf * 128 + gt] = warp_transpose_sum(acc);
        mbar_arrive(g_full + buf);
      }
    }
  }
  // the fused permutation, by the Gaussian warps (without them, the producer and MMA warps)
  // once their part of the CTA's tiles is done; the stage buffers are free after perm_go
  if (p.perm.perm_token) {
    int* ps = reinterpret_cast<int*>(stage);
    const int* ctot = epi_smem(epi, dm.K, ebars).ctot;
    if (kGauss && warp >= 6 && warp < 10)
      perm_tail<KM>(p, t_beg, t_end, threadIdx.x - 192, 4, 1, ctot, ps, perm_go, wc);
    if (!kGauss && warp < 2) perm_tail<KM>(p, t_beg, t_end, threadIdx.x, 2, 1, ctot, ps, perm_go, wc);
  }

  // the role branches leave single lanes running on their own: the warp reconverges before
  // the block barrier, so that no thread passes it while another of its warp is still working
  __syncwarp();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem_base, tmem_cols);
}

// Top-k insertion width: k rounded up to 2, 4, 6, 8 or 16.
template <class F>
cudaError_t dispatch_km(int k, F&& f) {
  if (k <= 2) return f(std::integral_constant<int, 2>());
  if (k <= 4) return f(std::integral_constant<int, 4>());
  if (k <= 6) return f(std::integral_constant<int, 6>());
  if (k <= 8) return f(std::integral_constant<int, 8>());
  return f(std::integral_constant<int, 16>());
}


// The tensor-core forward with or without the router variants compiled in.
template <bool kVar>
cudaError_t launch_fwd_tc(const FwdParams& p, const CUtensorMap& tmX, const CUtensorMap& tmW,
                          const CUtensorMap* tmG, int n_sms, cudaStream_t s) {
  const int N = round_up(p.dm.E, 16);
  const bool gauss = p.M_in == nullptr;
  // as many pipeline stages as fit next to the epilogue's shared memory; the scores are staged
  // for a coalesced store when that still leaves five stages
  auto stages_for = [&](bool stg) {
    int n = 8;
    while (n > 2 && fwd_smem_bytes(N, n, p.dm.d, p.dm.K, p.dm.E, gauss, stg) > 227u * 1024u) --n;
    return n;
  };
  const bool use_stg = tmG != nullptr && stages_for(true) >= 5;
  const int n_stages = stages_for(use_stg);
  const size_t smem = fwd_smem_bytes(N, n_stages, p.dm.d, p.dm.K, p.dm.E, gauss, use_stg);
  if (smem > 227u * 1024u) return cudaErrorInvalidConfiguration;
  if (p.perm.perm_token && static_cast<size_t>(n_stages) * fwd_stage_bytes(N) < sizeof(int) * perm_scratch_ints(p.dm.E))
    return cudaErrorInvalidConfiguration;
  const int grid = p.n_tiles < n_sms ? p.n_tiles : n_sms;
  const CUtensorMap& tg = use_stg ? *tmG : tmX;           // unused without staging
  return dispatch_km(p.dm.k, [&](auto km) -> cudaError_t {
    constexpr int KM = decltype(km)::value;
    auto k = gauss ? k_router_fwd_tc<true, KM, kVar> : k_router_fwd_tc<false, KM, kVar>;
    cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    if (!p.perm.perm_token)
      return launch_pdl(k, dim3(grid), dim3(fwd_threads(gauss)), smem, s, tmX, tmW, tg, p, N, n_stages,
                        use_stg ? 1 : 0);
    // the fused permutation has a grid barrier: every CTA must be resident (cooperative launch)
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(fwd_threads(gauss));
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeCooperative;
    attr[0].val.cooperative = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    return cudaLaunchKernelEx(&cfg, k, tmX, tmW, tg, p, N, n_stages, use_stg ? 1 : 0);
  });
}

}  // namespace
}  // namespace smoes
