// router_bwd.cu -- backward of loss_scale * L_MI (eq. 15) on sm_103a.
//
// With the soft scores held constant, the gradient reaching the gate logits is
//   dz_je = scale * g_je * (u_j,b(e) - sum_e' g_je' u_j,b(e'))           (scale = -loss_scale/B)
//   u_jk  = h_k + (M_jv - 1/2) a_k + (M_jt - 1/2) b_k
// with the per-sample coefficients (a, b, h) written by the forward. Optionally an upstream
// gradient of the top-k weights is pushed through the (renormalised) softmax as well.
// Then dW = dz^T X and dX = dz W.
//
// tcgen05 path (bf16): k_dz_prep writes dz of every 64-token tile as a bf16 hi/lo pair
// (dz = hi + lo to ~2^-17 relative) directly in the 128-byte-swizzled shared-memory image the
// tensor cores read. The main kernel runs CTA (token group g, d-slice s): per tile it bulk-copies
// that image, and one thread issues, per 128-column d-block of the slice,
//   dW^T[d-block] += X^T(tile) . (hi + lo)  (M = 128 d, N = E_pad, K = 64 tokens)  -> TMEM, kept
//   dX^T[d-block]  = W^T(d-block) . hi^T    (M = 128 d, N = 64 tokens, K = E_pad)  -> TMEM, drained
// dW (fp32 output, sums over many tokens that cancel) takes both halves; dX, stored in bf16, is
// formed from the bf16-rounded dz alone (bf16 inputs, fp32 accumulation: each element within one
// bf16 ulp plus 2^-8 sum_e |dz_je W_ed| of the exact value). The tensor pipe, not memory, set the
// tile rate with the lo half in dX as well: its 64-token MMAs read 6 KB of operands for 128 x 64 x
// 16 products.
// X tiles arrive by TMA; the W slice stays resident in shared memory; dX leaves by TMA store.
// The per-group dW^T slice is written once at the end and summed over groups in fixed order.
#include <cuda_bf16.h>

#include <type_traits>

#include "device_common.cuh"
#include "ptx.cuh"
#include "smoes_internal.cuh"

namespace smoes {
namespace {

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  const __nv_bfloat16 a = __float2bfloat16_rn(lo), b = __float2bfloat16_rn(hi);
  return static_cast<uint32_t>(__bfloat16_as_ushort(a)) |
         (static_cast<uint32_t>(__bfloat16_as_ushort(b)) << 16);
}

// Upstream top-k weight gradient of one token, folded into per-expert terms:
//   dt[e] = sum over top-k slots i with idx_i == e of dtil_i, and gdt = sum_i g_{idx_i} dtil_i,
// where dtil_i = d_i (raw weights) or (d_i - sum_i' d_i' w_i') / G (renormalised, G = sum g_sel).
struct Upstream {
  int idx[kMaxTopK];
  float dtil[kMaxTopK];
  float gdt;
};

__device__ __forceinline__ void load_upstream(const BwdParams& p, int j, Upstream& u) {
  const int k = p.dm.k;
  float gsel[kMaxTopK], d[kMaxTopK];
  float G = 0.f, dw = 0.f;
  const float* g = p.ws.gsave + static_cast<size_t>(j) * p.dm.E;
  const float ginv = p.ws.ginv[j];
#pragma unroll
  for (int i = 0; i < kMaxTopK; ++i) {
    u.idx[i] = -1;
    u.dtil[i] = 0.f;
    gsel[i] = 0.f;
    d[i] = 0.f;
    if (i < k) {
      u.idx[i] = p.topk_idx[static_cast<size_t>(j) * k + i];
      d[i] = p.d_topk_w[static_cast<size_t>(j) * k + i];
      const int e = u.idx[i];
      gsel[i] = (e >= 0 && e < p.dm.E) ? g[e] * ginv : 0.f;
      G += gsel[i];
    }
  }
  if (p.dm.renorm) {
#pragma unroll
    for (int i = 0; i < kMaxTopK; ++i)
      if (i < k) dw += d[i] * gsel[i] / G;
  }
  float gdt = 0.f;
#pragma unroll
  for (int i = 0; i < kMaxTopK; ++i) {
    if (i < k) {
      u.dtil[i] = p.dm.renorm ? (d[i] - dw) / G : d[i];
      gdt += gsel[i] * u.dtil[i];
    }
  }
  u.gdt = gdt;
}

__device__ __forceinline__ float upstream_at(const Upstream& u, int k, int e) {
  float r = 0.f;
#pragma unroll
  for (int i = 0; i < kMaxTopK; ++i)
    if (i < k && u.idx[i] == e) r += u.dtil[i];
  return r;
}

// Gradient of the bin-level balance loss (eq. 16) at one token's logits, added to dz[N] of the
// thread's N experts (g: their gate values, be: their bins (-1: none), fe: their f_e, fac: the
// gate's own factor, 1 for the softmax and 1 - s for the sigmoid): for every bin k the token
// routes to, dz_e += a_k h_e (f_e - sum_{e' in B_k} f_e' h_e') fac_e with h = g / (bin sum). The bin sums run over the token's GS-lane thread group (xor shuffles); every lane takes
// the same k iterations, and a bin repeated among the token's selections adds nothing again.
template <int GS, int N>
__device__ __forceinline__ void add_balance_grad(const BwdParams& p, int j, bool valid, const float (&g)[N],
                                                 const int (&be)[N], const float (&fe)[N],
                                                 const float (&fac)[N], float (&dz)[N]) {
  const int k = p.dm.k;
  int seen[kMaxTopK];
#pragma unroll
  for (int s = 0; s < kMaxTopK; ++s) {
    if (s >= k) break;
    const int es = valid ? __ldg(p.topk_idx + static_cast<size_t>(j) * k + s) : -1;
    const int bs = (es >= 0 && es < p.dm.E) ? (p.dm.contig_bins ? es / p.dm.N_B : __ldg(p.ws.expert_bin + es)) : -1;
    seen[s] = bs;
    bool dup = bs < 0;
#pragma unroll
    for (int s2 = 0; s2 < kMaxTopK; ++s2)
      if (s2 < s) dup = dup || seen[s2] == bs;
    float v = 0.f, w = 0.f;
#pragma unroll
    for (int i = 0; i < N; ++i) {
      v += be[i] == bs ? g[i] : 0.f;
      w += be[i] == bs ? fe[i] * g[i] : 0.f;
    }
#pragma unroll
    for (int o = 1; o < GS; o <<= 1) {
      v += __shfl_xor_sync(0xffffffffu, v, o);
      w += __shfl_xor_sync(0xffffffffu, w, o);
    }
    if (!dup && v > 0.f) {
      const float a = __ldg(p.ws.bal_a + bs), iv = 1.f / v, phi = w * iv;
#pragma unroll
      for (int i = 0; i < N; ++i)
        if (be[i] == bs) dz[i] = fmaf(a * g[i] * iv * fac[i], fe[i] - phi, dz[i]);
    }
  }
}

// MI gradient at one token's logits for the thread's N experts (a GS-lane group holds the token):
//   dz_e = scale fac_e w_e (u_e - sum_e' w_e' u_e'),
// with w the gate values that enter eq. (12) (the dense gate g, or with the top-k mask g on the
// chosen experts renormalised over them) and fac_e = 1 (softmax) or 1 - s_e (sigmoid: through
// g = s / sum s, s = sigmoid(z)). raw: the saved exp(z - max) or s; g = raw / sum raw.
template <int GS, int N, bool kVar = true>
__device__ __forceinline__ void mi_grad(const BwdParams& p, int j, bool valid, const int (&eidx)[N],
                                        const float (&raw)[N], const float (&g)[N], const float (&u)[N],
                                        float (&fac)[N], float (&dz)[N]) {
  const Dims& dm = p.dm;
  const bool gate = kVar && dm.gate, mask = kVar && dm.mask;   // kVar false: the softmax router
  float w[N];
#pragma unroll
  for (int i = 0; i < N; ++i) w[i] = g[i];
  if (mask) {
    bool sel[N];
#pragma unroll
    for (int i = 0; i < N; ++i) sel[i] = false;
    for (int s = 0; s < dm.k; ++s) {
      const int es = valid ? __ldg(p.topk_idx + static_cast<size_t>(j) * dm.k + s) : -1;
#pragma unroll
      for (int i = 0; i < N; ++i) sel[i] = sel[i] || (eidx[i] == es);
    }
    float G = 0.f;
#pragma unroll
    for (int i = 0; i < N; ++i) G += sel[i] ? g[i] : 0.f;
#pragma unroll
    for (int o = 1; o < GS; o <<= 1) G += __shfl_xor_sync(0xffffffffu, G, o);
    const float iG = G > 0.f ? 1.f / G : 0.f;
#pragma unroll
    for (int i = 0; i < N; ++i) w[i] = sel[i] ? g[i] * iG : 0.f;
  }
  float part = 0.f;
#pragma unroll
  for (int i = 0; i < N; ++i) part = fmaf(w[i], u[i], part);
#pragma unroll
  for (int o = 1; o < GS; o <<= 1) part += __shfl_xor_sync(0xffffffffu, part, o);
#pragma unroll
  for (int i = 0; i < N; ++i) {
    fac[i] = gate ? 1.f - raw[i] : 1.f;
    dz[i] = p.scale * fac[i] * w[i] * (u[i] - part);
  }
}

// ------------------------------------------------------------------ dz preparation (bf16 path)
// TPT = E_pad/8 threads per token, 8 experts each; the token's sum over experts is a shuffle
// reduction inside its TPT-lane group. dz is written as the bf16 hi/lo pair (dz = hi + lo to
// ~2^-17 relative) in the 128-byte-swizzled operand image of its 64-token tile,
// [tile][hi | lo][E_pad/64][64 rows][128 B], which the main kernel bulk-copies. Rows beyond T and
// padded experts are zeros. With consecutive bins of a multiple of 4 experts, a thread's 8
// experts lie in at most two bins: their coefficients are read once per bin. Every thread group
// handles kDzRep tokens (a block's token sets kDzRep apart) with all their loads issued before
// any is used, so enough bytes are in flight to stream the saved scores at HBM speed. kUp: an
// upstream gradient of the top-k weights is present (its per-token tables stay out of the
// register budget otherwise).
constexpr int kDzRep = 2;

template <int TPT, bool kUp, bool kBal, bool kVar>
__global__ void __launch_bounds__(256) k_dz_prep(const BwdParams p) {
  pdl_wait();                                         // scores and tables of the forward
  pdl_trigger();
  const Dims& dm = p.dm;
  const int E = dm.E, K = dm.K, k = dm.k;
  constexpr int kEp = TPT * 8;
  constexpr int kGroups = 256 / TPT;                  // token groups per block and set
  const int c = threadIdx.x % TPT;
  const int e0 = c * 8;
  const int n_rows = p.n_tiles * kBwdBT;
  int j[kDzRep];
  bool valid[kDzRep];
#pragma unroll
  for (int q = 0; q < kDzRep; ++q) {
    j[q] = (blockIdx.x * kDzRep + q) * kGroups + threadIdx.x / TPT;
    valid[q] = j[q] < dm.T;
  }
  // every load of the block's tokens first
  float4 ga[kDzRep], gb[kDzRep];
  float ginv[kDzRep];
  float2 m[kDzRep];
  int smp[kDzRep];
  const bool vec = (E & 3) == 0 && e0 + 8 <= E;
  // the balance term (eq. 16) when smoes_bin_balance armed this backward
  const bool bal = kBal && p.topk_idx != nullptr && __ldcg(p.ws.bal_flag) != 0u;
  int be[8];
  float fe[8];
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const int e = e0 + i;
    be[i] = -1;
    fe[i] = 0.f;
    if (bal && e < E) {
      be[i] = dm.contig_bins ? e / dm.N_B : __ldg(p.ws.expert_bin + e);
      fe[i] = __ldg(p.ws.bal_f + e);
    }
  }
#pragma unroll
  for (int q = 0; q < kDzRep; ++q) {
    ga[q] = gb[q] = make_float4(0.f, 0.f, 0.f, 0.f);
    ginv[q] = 0.f;
    m[q] = make_float2(0.5f, 0.5f);
    smp[q] = 0;
    if (valid[q]) {
      const float* grow = p.ws.gsave + static_cast<size_t>(j[q]) * E;
      if (vec) {
        ga[q] = __ldcg(reinterpret_cast<const float4*>(grow + e0));
        gb[q] = __ldcg(reinterpret_cast<const float4*>(grow + e0 + 4));
      } else {
        float t[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) t[u] = (e0 + u < E) ? __ldcg(grow + e0 + u) : 0.f;
        ga[q] = make_float4(t[0], t[1], t[2], t[3]);
        gb[q] = make_float4(t[4], t[5], t[6], t[7]);
      }
      ginv[q] = __ldcg(p.ws.ginv + j[q]);
      m[q] = __ldg(reinterpret_cast<const float2*>(p.M) + j[q]);
      smp[q] = __ldg(p.ws.token_sample + j[q]);
    }
  }
#pragma unroll
  for (int q = 0; q < kDzRep; ++q) {
    if (j[q] >= n_rows) continue;                     // whole TPT groups skip together
    const float raw[8] = {ga[q].x, ga[q].y, ga[q].z, ga[q].w, gb[q].x, gb[q].y, gb[q].z, gb[q].w};
    float g[8], u[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) { g[i] = raw[i] * ginv[q]; u[i] = 0.f; }   // the gate value g_je
    if (valid[q]) {
      const float dv = m[q].x - 0.5f, dt = m[q].y - 0.5f;
      // the sample's coefficient table was written by the forward kernel and is read-only here
      const float* tb = p.ws.tabs + static_cast<size_t>(smp[q]) * 3 * K;
      if (dm.contig_bins && e0 + 8 <= E) {
        const int b0 = e0 / dm.N_B, b1 = (e0 + 7) / dm.N_B;
        const float u0 = __ldg(tb + 2 * K + b0) + dv * __ldg(tb + b0) + dt * __ldg(tb + K + b0);
        const float u1 = __ldg(tb + 2 * K + b1) + dv * __ldg(tb + b1) + dt * __ldg(tb + K + b1);
#pragma unroll
        for (int i = 0; i < 8; ++i) u[i] = (e0 + i) / dm.N_B == b0 ? u0 : u1;
      } else {
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          if (e0 + i < E) {
            const int b = __ldg(p.ws.expert_bin + e0 + i);
            u[i] = __ldg(tb + 2 * K + b) + dv * __ldg(tb + b) + dt * __ldg(tb + K + b);
          }
        }
      }
    }
    int eidx[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) eidx[i] = e0 + i < E ? e0 + i : -2;
    float dz[8], fac[8];
    mi_grad<TPT, 8, kVar>(p, j[q], valid[q], eidx, raw, g, u, fac, dz);
    if (kUp && valid[q]) {
      Upstream up;
      load_upstream(p, j[q], up);
#pragma unroll
      for (int i = 0; i < 8; ++i)
        if (e0 + i < E)
          dz[i] += (kVar && dm.gate) ? fac[i] * g[i] * upstream_at(up, k, e0 + i)   // diagonal
                                     : g[i] * (upstream_at(up, k, e0 + i) - up.gdt);
    }
    if (kBal && bal) add_balance_grad<TPT, 8>(p, j[q], valid[q], g, be, fe, fac, dz);
    if (valid[q] && p.dlogits) {
      float* dl = p.dlogits + static_cast<size_t>(j[q]) * E;
      if (vec) {
        *reinterpret_cast<float4*>(dl + e0) = make_float4(dz[0], dz[1], dz[2], dz[3]);
        *reinterpret_cast<float4*>(dl + e0 + 4) = make_float4(dz[4], dz[5], dz[6], dz[7]);
      } else {
#pragma unroll
        for (int i = 0; i < 8; ++i)
          if (e0 + i < E) dl[e0 + i] = dz[i];
      }
    }
    uint32_t hw[4], lw[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const __nv_bfloat16 h0 = __float2bfloat16_rn(dz[2 * i]), h1 = __float2bfloat16_rn(dz[2 * i + 1]);
      hw[i] = static_cast<uint32_t>(__bfloat16_as_ushort(h0)) | (static_cast<uint32_t>(__bfloat16_as_ushort(h1)) << 16);
      lw[i] = pack_bf16x2(dz[2 * i] - __bfloat162float(h0), dz[2 * i + 1] - __bfloat162float(h1));
    }
    const int tile = j[q] / kBwdBT, r = j[q] % kBwdBT;
    uint8_t* img = p.ws.dz_img + static_cast<size_t>(tile) * (2 * kEp * 128);
    const uint32_t off = (e0 >> 6) * 8192u + sw128_offset(static_cast<uint32_t>(r), static_cast<uint32_t>(e0 & 63));
    *reinterpret_cast<uint4*>(img + off) = make_uint4(hw[0], hw[1], hw[2], hw[3]);
    *reinterpret_cast<uint4*>(img + kEp * 128 + off) = make_uint4(lw[0], lw[1], lw[2], lw[3]);
  }
}

// ------------------------------------------------------------------ tcgen05 backward (bf16)

struct BwdLayout {
  uint32_t wsl, dz, xst, stg, bars, total;
};

// dX^T accumulators in TMEM: kDxBufs buffers of 64 columns after the dW^T blocks (which take at
// most 256 columns: slice width x E_pad = 32768), drained by two warp groups in turn.
constexpr int kDxBufs = 4;
constexpr int kDrainGroups = 2;
constexpr int kBwdThreads = 64 + kDrainGroups * 128;

__host__ __device__ inline BwdLayout bwd_layout(int E_pad, int n_xst) {
  BwdLayout L;
  uint32_t o = 0;
  L.wsl = o;  o += 65536u;                                         // W slice (ds * E_pad * 2 B)
  L.dz = o;   o += 2u * 2u * static_cast<uint32_t>(E_pad) * 128u;   // 2 buffers x (hi, lo)
  L.xst = o;  o += static_cast<uint32_t>(n_xst) * 16384u;          // X stages [2 atoms][64][128 B]
  L.stg = o;  o += kDrainGroups * 16384u;                          // dX staging [64][128] bf16 per group
  L.bars = o; o += 8u * (2u * n_xst + 32u) + 16u;
  L.total = o + 1024u;
  return L;
}

// Roles (320 threads): warp 0 TMA / bulk-copy producer, warp 1 MMA issuer, warps 2-5 and 6-9 two
// drain groups: d-block iteration `it` of the CTA uses dX^T buffer it % 4 and is drained by group
// it % 2 through the group's own staging buffer, so two drains run while the tensor cores fill
// the other buffers. An X stage is released as soon as the d-block's dW^T MMAs complete (the dX^T
// MMAs read W and dz only). After the last tile every CTA writes its dW^T partial (both groups,
// alternate d-blocks); k_dw_reduce sums them.
template <int E_pad>
__global__ void __launch_bounds__(kBwdThreads, 1)
k_router_bwd_tc(const __grid_constant__ CUtensorMap tmX, const __grid_constant__ CUtensorMap tmW,
                const __grid_constant__ CUtensorMap tmDX, const BwdParams p, const int n_xst) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const Dims& dm = p.dm;
  const BwdLayout L = bwd_layout(E_pad, n_xst);
  uint8_t* wsl = base + L.wsl;
  uint8_t* dzb = base + L.dz;               // buffer zb: hi at zb*2*E_pad*128, lo right after
  uint8_t* xst = base + L.xst;
  uint8_t* stg = base + L.stg;
  uint64_t* bars = reinterpret_cast<uint64_t*>(base + L.bars);
  uint64_t* xfull = bars;
  uint64_t* xempty = bars + n_xst;
  uint64_t* dz_full = bars + 2 * n_xst;       // [2] the tile's dz image has landed
  uint64_t* dz_empty = dz_full + 2;           // [2] the tile's MMAs have read it
  uint64_t* dx_full = dz_full + 4;            // [kDxBufs]
  uint64_t* dx_empty = dx_full + kDxBufs;     // [kDxBufs]
  uint64_t* wfull = dx_empty + kDxBufs;
  uint64_t* dw_full = wfull + 1;
  uint64_t* drain = wfull + 2;
  uint64_t* stg_free = wfull + 3;             // [kDrainGroups] a group's staging may be rewritten
  uint64_t* stg_full = stg_free + kDrainGroups;   // [kDrainGroups] a group's staging is written
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(stg_full + kDrainGroups);
  int* abort_flag = reinterpret_cast<int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int S = p.slices, G = p.groups;
  const int sl = blockIdx.x % S, grp = blockIdx.x / S;
  const int d0 = sl * p.slice_width;
  const int nb = min(p.slice_width, round_up(dm.d - d0, kBwdBD)) / kBwdBD;   // d-blocks here
  const bool want_dx = p.dX != nullptr;
  constexpr uint32_t dz_half = static_cast<uint32_t>(E_pad) * 128u;         // one of hi / lo
  constexpr uint32_t dz_buf_bytes = 2u * dz_half;                           // hi + lo
  WaitCtx wc{abort_flag, p.ws.status, p.limit_ns};

  if (threadIdx.x == 0) {
    *abort_flag = 0;
    for (int i = 0; i < n_xst; ++i) {
      mbar_init(xfull + i, 1);
      mbar_init(xempty + i, 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(dz_full + i, 1);
      mbar_init(dz_empty + i, 1);
    }
    for (int i = 0; i < kDxBufs; ++i) {
      mbar_init(dx_full + i, 1);
      mbar_init(dx_empty + i, 128);
    }
    for (int i = 0; i < kDrainGroups; ++i) {
      mbar_init(stg_free + i, 1);
      mbar_init(stg_full + i, 128);
    }
    mbar_init(wfull, 1);
    mbar_init(dw_full, 1);
    mbar_init(drain, 1);
    fence_mbar_init();
    tma_prefetch_desc(&tmX);
    tma_prefetch_desc(&tmW);
    tma_prefetch_desc(&tmDX);
  }
  if (warp == 1) tmem_alloc(tmem_slot, 512);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const uint32_t tm_dx = tmem + 256u;          // kDxBufs 64-column dX^T buffers after the dW^T blocks
  if (warp == 0 && lane == 0) {
    // W slice (atom a = columns d0 + 64a .. +64), requested before the dz prep kernel has
    // finished: that kernel does not write W, and it started only after all earlier work
    mbar_arrive_expect_tx(wfull, static_cast<uint32_t>(nb) * 2u * dz_half);
    for (int a = 0; a < 2 * nb; ++a) tma_load_2d(wsl + a * dz_half, &tmW, wfull, d0 + 64 * a, 0);
  }
  pdl_wait();                                  // the dz images, X and dX
  pdl_trigger();

  if (warp == 0) {
    // -------------------------------------------------------------- TMA producer
    if (lane == 0) {
      bool ok = true;
      int st = 0;
      uint32_t ph = 0;
      long issued = 0, dz_issued = 0;
      int lt = 0;
      for (int t = grp; t < p.n_tiles && ok; t += G, ++lt) {
        const int zb = lt & 1;
        const uint32_t zuse = static_cast<uint32_t>(lt >> 1);
        if (!mbar_wait(dz_empty + zb, (zuse & 1u) ^ 1u, wc)) { ok = false; break; }
        mbar_arrive_expect_tx(dz_full + zb, dz_buf_bytes);
        bulk_load(dzb + zb * dz_buf_bytes, p.ws.dz_img + static_cast<size_t>(t) * dz_buf_bytes,
                  dz_buf_bytes, dz_full + zb);
        ++dz_issued;
        for (int b = 0; b < nb; ++b) {
          if (!mbar_wait(xempty + st, ph ^ 1u, wc)) { ok = false; break; }
          uint8_t* xs = xst + st * 16384;
          mbar_arrive_expect_tx(xfull + st, 16384u);
          tma_load_2d(xs, &tmX, xfull + st, d0 + b * kBwdBD, t * kBwdBT);
          tma_load_2d(xs + 8192, &tmX, xfull + st, d0 + b * kBwdBD + 64, t * kBwdBT);
          ++issued;
          if (++st == n_xst) { st = 0; ph ^= 1u; }
        }
      }
      WaitCtx wd = wc;
      int dummy = 0;
      wd.abort_flag = &dummy;
      mbar_wait(wfull, 0, wd);                // the W slice copy must land before exit
      if (!ok) {                              // so must every issued X and dz copy
        for (long q = (issued > n_xst ? issued - n_xst : 0); q < issued; ++q)
          mbar_wait(xfull + (q % n_xst), static_cast<uint32_t>((q / n_xst) & 1), wd);
        for (long q = (dz_issued > 2 ? dz_issued - 2 : 0); q < dz_issued; ++q)
          mbar_wait(dz_full + (q & 1), static_cast<uint32_t>((q >> 1) & 1), wd);
      }
    }
  } else if (warp == 1) {
    // -------------------------------------------------------------- MMA issuer
    if (lane == 0) {
      const uint32_t id_dw = idesc_bf16(128, E_pad, true, true);
      const uint32_t id_dx = idesc_bf16(128, kBwdBT, true, false);
      bool ok = mbar_wait(wfull, 0, wc);
      tc_fence_after();
      int st = 0;
      uint32_t ph = 0;
      int it = 0;                              // d-block iterations of this CTA
      int lt = 0;
      for (int t = grp; t < p.n_tiles && ok; t += G, ++lt) {
        const int zb = lt & 1;
        const uint32_t zuse = static_cast<uint32_t>(lt >> 1);
        if (!mbar_wait(dz_full + zb, zuse & 1u, wc)) { ok = false; break; }
        tc_fence_after();
        const uint32_t hi = smem_u32(dzb + zb * dz_buf_bytes);
        const uint32_t lo = hi + dz_half;
        for (int b = 0; b < nb; ++b, ++it) {
          if (!mbar_wait(xfull + st, ph, wc)) { ok = false; break; }
          tc_fence_after();
          const uint32_t xs = smem_u32(xst + st * 16384);
          const uint32_t dwc = tmem + static_cast<uint32_t>(b * E_pad);
#pragma unroll
          for (int ks = 0; ks < kBwdBT / 16; ++ks) {     // K = 16 tokens per instruction
            const uint64_t da = sdesc_sw128(xs + ks * 2048, 8192, 1024);
            const uint64_t dh = sdesc_sw128(hi + ks * 2048, 8192, 1024);
            const uint64_t dl = sdesc_sw128(lo + ks * 2048, 8192, 1024);
            umma_bf16(dwc, da, dh, id_dw, (lt > 0 || ks > 0) ? 1u : 0u);
            umma_bf16(dwc, da, dl, id_dw, 1u);
          }
          umma_commit(xempty + st);             // the X stage is free once these MMAs complete
          if (++st == n_xst) { st = 0; ph ^= 1u; }
          if (want_dx) {
            const int xb = it % kDxBufs;
            const uint32_t xuse = static_cast<uint32_t>(it / kDxBufs);
            if (!mbar_wait(dx_empty + xb, (xuse & 1u) ^ 1u, wc)) { ok = false; break; }
            tc_fence_after();
            const uint32_t dxc = tm_dx + static_cast<uint32_t>(xb * kBwdBT);
            const uint32_t wa = smem_u32(wsl + 2 * b * dz_half);
#pragma unroll
            for (int ke = 0; ke < E_pad / 16; ++ke) {    // K = 16 experts per instruction
              const uint64_t da = sdesc_sw128(wa + ke * 2048, dz_half, 1024);
              const uint32_t boff = (ke >> 2) * 8192 + (ke & 3) * 32;
              const uint64_t dh = sdesc_sw128(hi + boff, 16, 1024);
              umma_bf16(dxc, da, dh, id_dx, ke > 0 ? 1u : 0u);
            }
            umma_commit(dx_full + xb);
          }
        }
        if (!ok) break;
        umma_commit(dz_empty + zb);
      }
      if (ok) umma_commit(dw_full);
      umma_commit(drain);
      WaitCtx wd = wc;
      int dummy = 0;
      wd.abort_flag = &dummy;
      mbar_wait(drain, 0, wd);
    }
  } else {
    // -------------------------------------------------------------- dX drain + dW drain (2 groups)
    const int lg = warp & 3;                           // TMEM lane quarter of this warp
    const int dg = (warp - 2) >> 2;                    // drain group
    const int gtid = (threadIdx.x - 64) & 127;         // 0..127 within the group
    const bool issuer = (gtid == 0);
    uint8_t* sgb = stg + dg * 16384;
    bool ok = true;
    if (want_dx) {
      int it = 0, n_mine = 0;
      for (int t = grp; t < p.n_tiles && ok; t += G) {
        for (int b = 0; b < nb; ++b, ++it) {
          if ((it & 1) != dg) continue;
          const int xb = it % kDxBufs;
          const uint32_t xuse = static_cast<uint32_t>(it / kDxBufs);
          if (!mbar_wait(dx_full + xb, xuse & 1u, wc)) { ok = false; break; }
          tc_fence_after();
          if (issuer) {                                // this group's staging free again
            tma_store_wait_read<0>();
            mbar_arrive(stg_free + dg);
          }
          if (!mbar_wait(stg_free + dg, static_cast<uint32_t>(n_mine & 1), wc)) { ok = false; break; }
          __nv_bfloat16* sg = reinterpret_cast<__nv_bfloat16*>(sgb);
          const uint32_t ta = tm_dx + (static_cast<uint32_t>(lg * 32) << 16) + static_cast<uint32_t>(xb * kBwdBT);
          const int drow = lg * 32 + lane;
#pragma unroll
          for (int c = 0; c < kBwdBT / 32; ++c) {
            float v[32];
            tmem_ld32(ta + 32u * c, v);
#pragma unroll
            for (int q = 0; q < 32; ++q) sg[(c * 32 + q) * kBwdBD + drow] = __float2bfloat16_rn(v[q]);
          }
          tc_fence_before();
          mbar_arrive(dx_empty + xb);
          fence_proxy_async_smem();
          mbar_arrive(stg_full + dg);
          if (issuer) {
            if (!mbar_wait(stg_full + dg, static_cast<uint32_t>(n_mine & 1), wc)) { ok = false; break; }
            tma_store_2d(&tmDX, sg, d0 + b * kBwdBD, t * kBwdBT);
            tma_store_commit();
          }
          ++n_mine;
        }
      }
      if (issuer) tma_store_wait_all<0>();
    }
    // partial dW^T of this group: lanes = d rows, columns = experts; the two drain groups take
    // alternate d-blocks
    if (ok && mbar_wait(dw_full, 0, wc)) {
      tc_fence_after();
      for (int b = dg; b < nb; b += kDrainGroups) {
        const int drow = d0 + b * kBwdBD + lg * 32 + lane;
        const uint32_t ta = tmem + (static_cast<uint32_t>(lg * 32) << 16) + static_cast<uint32_t>(b * E_pad);
#pragma unroll 1
        for (int c = 0; c < E_pad / 32; ++c) {
          float v[32];
          tmem_ld32(ta + 32u * c, v);
#pragma unroll
          for (int q = 0; q < 32; ++q) {
            const int e = c * 32 + q;
            if (e < dm.E && drow < dm.d)
              p.ws.dw_part[(static_cast<size_t>(grp) * dm.E + e) * dm.d + drow] = v[q];
          }
        }
      }
    }
  }

  // the role branches leave single lanes running on their own: the warp reconverges before
  // the block barrier, so that no thread passes it while another of its warp is still working
  __syncwarp();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem, 512);
}

// ------------------------------------------------------------------ FFMA backward (fp32)
// CTA (64-token tile, 128-feature chunk): dz of the tile's tokens into shared memory (4 threads
// per token; every chunk of the tile forms the same dz, the first one writes dlogits), then
// thread (feature c, half h) holds W[:, c] in registers and walks 32 of the tile's rows: dX[j, c]
// = dz_j . W[:, c] and the partial dW[:, c] += dz_j x_jc. The two halves' dW partials are added
// in shared memory and written once per tile; k_dw_reduce sums the tiles in order.
constexpr int kF32MaxE = 64;
constexpr int kF32Cols = 128;

// EB = E rounded up to 16: the expert loops run to EB over zero-padded dz and W columns.
template <int EB>
__global__ void __launch_bounds__(256)
k_router_bwd_f32(const BwdParams p) {
  extern __shared__ float bs[];
  pdl_wait();
  pdl_trigger();
  const Dims& dm = p.dm;
  const int E = dm.E, K = dm.K, k = dm.k;
  const int nck = (dm.d + kF32Cols - 1) / kF32Cols;
  const int tile = blockIdx.x / nck, ck = blockIdx.x % nck;
  constexpr int kZs = EB + 4;                        // dz row stride (16-byte aligned rows)
  float* dzs = bs;                                   // [64][kZs], experts past E zero
  float* dws = dzs + 64 * kZs;                       // [E][128] second half's dW partial
  const int t = threadIdx.x;
  {
    const int r = t >> 2, qd = t & 3;
    const int j = tile * 64 + r;
    const bool valid = j < dm.T;
    float dv = 0.f, dt = 0.f;
    const float* tb = nullptr;
    if (valid) {
      const int s = p.ws.token_sample[j];
      dv = p.M[2 * static_cast<size_t>(j)] - 0.5f;
      dt = p.M[2 * static_cast<size_t>(j) + 1] - 0.5f;
      tb = p.ws.tabs + static_cast<size_t>(s) * 3 * K;
    }
    Upstream up;
    const bool has_up = valid && p.d_topk_w != nullptr;
    if (has_up) load_upstream(p, j, up);
    const float* g = p.ws.gsave + static_cast<size_t>(valid ? j : 0) * E;
    const float ginv = valid ? p.ws.ginv[j] : 0.f;
    // the token's 4-thread group holds experts qd, qd + 4, ...
    constexpr int NQ = EB / 4;
    int eidx[NQ], bq[NQ];
    float raw[NQ], gq[NQ], uq[NQ], fq[NQ], fac[NQ], dzv[NQ];
#pragma unroll
    for (int i = 0; i < NQ; ++i) {
      const int e = qd + 4 * i;
      const bool in = valid && e < E;
      eidx[i] = e < E ? e : -2;
      bq[i] = in ? p.ws.expert_bin[e] : -1;
      raw[i] = in ? g[e] : 0.f;
      gq[i] = raw[i] * ginv;
      uq[i] = in ? tb[2 * K + bq[i]] + dv * tb[bq[i]] + dt * tb[K + bq[i]] : 0.f;
    }
    mi_grad<4, NQ>(p, j, valid, eidx, raw, gq, uq, fac, dzv);
    if (has_up) {
#pragma unroll
      for (int i = 0; i < NQ; ++i)
        if (eidx[i] >= 0)
          dzv[i] += dm.gate ? fac[i] * gq[i] * upstream_at(up, k, eidx[i])
                            : gq[i] * (upstream_at(up, k, eidx[i]) - up.gdt);
    }
    if (p.topk_idx && __ldcg(p.ws.bal_flag) != 0u) {   // the balance term (eq. 16); block-uniform
#pragma unroll
      for (int i = 0; i < NQ; ++i) fq[i] = bq[i] >= 0 ? p.ws.bal_f[eidx[i]] : 0.f;
      add_balance_grad<4, NQ>(p, j, valid, gq, bq, fq, fac, dzv);
    }
#pragma unroll
    for (int i = 0; i < EB / 4; ++i) {
      const int e = qd + 4 * i;
      if (valid && e < E && p.dlogits && ck == 0) p.dlogits[static_cast<size_t>(j) * E + e] = dzv[i];
      dzs[r * kZs + e] = dzv[i];
    }
  }
  const float* X = static_cast<const float*>(p.X);
  const float* W = static_cast<const float*>(p.W);
  float* dX = static_cast<float*>(p.dX);
  const int c = ck * kF32Cols + (t & 127), h = t >> 7;
  const bool cin = c < dm.d;
  float wc[EB], acc[EB];
#pragma unroll
  for (int e = 0; e < EB; ++e) {
    wc[e] = (e < E && cin) ? __ldg(W + static_cast<size_t>(e) * dm.d + c) : 0.f;
    acc[e] = 0.f;
  }
  __syncthreads();
  const int r0 = 32 * h;
  const int rows = min(32, dm.T - tile * 64 - r0);
  constexpr int kU = 8;                              // rows loaded ahead
  for (int rb = 0; rb < rows; rb += kU) {
    float x[kU];
#pragma unroll
    for (int u = 0; u < kU; ++u) {
      const size_t j = static_cast<size_t>(tile) * 64 + r0 + rb + u;
      x[u] = (cin && rb + u < rows) ? __ldg(X + j * dm.d + c) : 0.f;
    }
#pragma unroll
    for (int u = 0; u < kU; ++u) {
      if (rb + u >= rows) break;
      const float* zr = dzs + (r0 + rb + u) * kZs;
      float dx = 0.f;
#pragma unroll
      for (int e = 0; e < EB; e += 4) {
        const float4 z = *reinterpret_cast<const float4*>(zr + e);
        dx = fmaf(z.x, wc[e], fmaf(z.y, wc[e + 1], fmaf(z.z, wc[e + 2], fmaf(z.w, wc[e + 3], dx))));
        acc[e] = fmaf(z.x, x[u], acc[e]);
        acc[e + 1] = fmaf(z.y, x[u], acc[e + 1]);
        acc[e + 2] = fmaf(z.z, x[u], acc[e + 2]);
        acc[e + 3] = fmaf(z.w, x[u], acc[e + 3]);
      }
      const size_t j = static_cast<size_t>(tile) * 64 + r0 + rb + u;
      if (dX && cin) dX[j * dm.d + c] = dx;
    }
  }
  if (h == 1) {
#pragma unroll
    for (int e = 0; e < EB; ++e)
      if (e < E) dws[e * kF32Cols + (t & 127)] = acc[e];
  }
  __syncthreads();
  if (h == 0 && cin) {
#pragma unroll
    for (int e = 0; e < EB; ++e)
      if (e < E)
        p.ws.dw_part[(static_cast<size_t>(tile) * E + e) * dm.d + c] = acc[e] + dws[e * kF32Cols + t];
  }
}

// dW[e][c] = (accumulate ? dW[e][c] : 0) + S, S = sum_{g=0}^{G-1} part[g][e][c]; the group sum is
// formed first, so an existing dW adds one rounding, not G. A block covers 32 float4 columns of
// dW with 8 threads each: thread slice t sums groups [t G/8, (t+1) G/8) in order with all its
// loads in flight at once, then the 8 slice sums are added in slice order (a fixed tree).
constexpr int kDwSlices = 8;
constexpr int kDwCols = 32;

__global__ void __launch_bounds__(kDwSlices * kDwCols) k_dw_reduce(const BwdParams p) {
  __shared__ float4 part_s[kDwSlices][kDwCols];
  pdl_wait();                                              // the partials of the main kernel
  pdl_trigger();
  const size_t n = static_cast<size_t>(p.dm.E) * p.dm.d;
  const bool vec = (n & 3) == 0;
  const size_t nv = vec ? n / 4 : n;                       // float4 (or scalar) columns
  const int col = threadIdx.x % kDwCols, sl = threadIdx.x / kDwCols;
  const size_t i = static_cast<size_t>(blockIdx.x) * kDwCols + col;
  const int G = p.groups;
  const int g0 = sl * G / kDwSlices, g1 = (sl + 1) * G / kDwSlices;
  float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
  if (i < nv) {
    constexpr int kU = 8;
    for (int g = g0; g < g1; g += kU) {
      float4 v[kU];
#pragma unroll
      for (int u = 0; u < kU; ++u) {
        v[u] = make_float4(0.f, 0.f, 0.f, 0.f);
        if (g + u < g1) {
          if (vec) {
            v[u] = __ldcg(reinterpret_cast<const float4*>(p.ws.dw_part) + static_cast<size_t>(g + u) * nv + i);
          } else {
            v[u].x = __ldcg(p.ws.dw_part + static_cast<size_t>(g + u) * nv + i);
          }
        }
      }
#pragma unroll
      for (int u = 0; u < kU; ++u) {
        acc.x += v[u].x; acc.y += v[u].y; acc.z += v[u].z; acc.w += v[u].w;
      }
    }
  }
  part_s[sl][col] = acc;
  __syncthreads();
  if (sl == 0 && i < nv) {
    float4 t = part_s[0][col];
#pragma unroll
    for (int q = 1; q < kDwSlices; ++q) {
      const float4 u = part_s[q][col];
      t.x += u.x; t.y += u.y; t.z += u.z; t.w += u.w;
    }
    if (vec) {
      float4* dW = reinterpret_cast<float4*>(p.dW);
      if (p.accumulate) {
        const float4 o = dW[i];
        t.x += o.x; t.y += o.y; t.z += o.z; t.w += o.w;
      }
      dW[i] = t;
    } else {
      p.dW[i] = p.accumulate ? p.dW[i] + t.x : t.x;
    }
  }
}

}  // namespace

cudaError_t launch_dz_prep(const BwdParams& p, cudaStream_t s) {
  const int E_pad = round_up(p.dm.E, 64);
  const int tokens_per_block = kDzRep * 256 / (E_pad / 8);
  const long rows = static_cast<long>(p.n_tiles) * kBwdBT;
  const int blocks = static_cast<int>((rows + tokens_per_block - 1) / tokens_per_block);
  // the upstream-gradient and balance variants keep their tables out of the common kernel's
  // registers; the balance variant still checks the arming flag on the device
  const bool up = p.d_topk_w != nullptr, bal = p.balance_armed != 0;
  const bool var = p.dm.gate != 0 || p.dm.mask != 0;      // sigmoid gate or top-k-masked g
  auto pick = [&](auto tpt) {
    constexpr int TPT = decltype(tpt)::value;
    if (var)
      return up ? (bal ? k_dz_prep<TPT, true, true, true> : k_dz_prep<TPT, true, false, true>)
                : (bal ? k_dz_prep<TPT, false, true, true> : k_dz_prep<TPT, false, false, true>);
    return up ? (bal ? k_dz_prep<TPT, true, true, false> : k_dz_prep<TPT, true, false, false>)
              : (bal ? k_dz_prep<TPT, false, true, false> : k_dz_prep<TPT, false, false, false>);
  };
  if (E_pad == 64) return launch_pdl(pick(std::integral_constant<int, 8>()), dim3(blocks), dim3(256), 0, s, p);
  if (E_pad == 128) return launch_pdl(pick(std::integral_constant<int, 16>()), dim3(blocks), dim3(256), 0, s, p);
  return cudaErrorInvalidValue;
}

cudaError_t launch_router_bwd_bf16(const BwdParams& p, const CUtensorMap& tmX, const CUtensorMap& tmW,
                                   const CUtensorMap& tmDX, cudaStream_t s) {
  const int E_pad = round_up(p.dm.E, 64);
  if (E_pad > 128) return cudaErrorInvalidValue;
  int n_xst = 6;
  while (n_xst > 2 && bwd_layout(E_pad, n_xst).total > 227u * 1024u) --n_xst;
  const uint32_t smem = bwd_layout(E_pad, n_xst).total;
  if (smem > 227u * 1024u) return cudaErrorInvalidConfiguration;
  auto k = (E_pad == 64) ? k_router_bwd_tc<64> : k_router_bwd_tc<128>;
  cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  return launch_pdl(k, dim3(p.groups * p.slices), dim3(kBwdThreads), smem, s, tmX, tmW, tmDX, p, n_xst);
}


cudaError_t launch_router_bwd_f32(const BwdParams& p, cudaStream_t s) {
  if (p.dm.E > kF32MaxE) return cudaErrorInvalidValue;
  const int eb = round_up(p.dm.E, 16);
  const size_t smem = sizeof(float) * (64 * static_cast<size_t>(eb + 4) + static_cast<size_t>(p.dm.E) * kF32Cols);
  auto k = eb <= 16 ? k_router_bwd_f32<16> : eb <= 32 ? k_router_bwd_f32<32>
         : eb <= 48 ? k_router_bwd_f32<48> : k_router_bwd_f32<64>;
  cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  const int nck = (p.dm.d + kF32Cols - 1) / kF32Cols;
  return launch_pdl(k, dim3(p.n_tiles * nck), dim3(256), smem, s, p);
}

cudaError_t launch_dw_reduce(const BwdParams& p, cudaStream_t s) {
  size_t n = static_cast<size_t>(p.dm.E) * p.dm.d;
  if ((n & 3) == 0) n /= 4;
  const int blocks = static_cast<int>((n + kDwCols - 1) / kDwCols);
  return launch_pdl(k_dw_reduce, dim3(blocks), dim3(kDwSlices * kDwCols), 0, s, p);
}

}  // namespace smoes
