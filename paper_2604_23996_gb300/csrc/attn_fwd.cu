// attn_fwd.cu -- causal attention forward that also yields the attention-accumulated vision score
// (eqs. 2-4): the score is attention with the carried score m as one more value column, so one
// pass gives the layer's output O = softmax(s Q K^T + bias) V and, per query,
//   Mtilde_v = (1/H) sum_h sum_j' softmax_j'(s q.k_j' + beta_j') m_j'.
// Grouped-query attention: K and V have H_kv heads; query head h reads key/value head h / (H / H_kv).
//
// A work item is (sequence, head, 128-query tile); items run longest first on persistent CTAs.
// Per 128-key block the tensor cores form S = Q K^T into one of two TMEM buffers (tcgen05,
// TMA-fed). Two softmax warp groups (four warps each, one query row per thread) take the two
// halves of the block's keys and keep independent online states: the running maximum used for
// the exponentials, the normaliser l and the vision mass a = sum P m. Each half writes its P (bf16,
// as FlashAttention passes it to the tensor cores) to its half of a shared-memory tile and the
// tensor cores accumulate O_h += P_h V_h into the half's own TMEM accumulator. The maximum in use
// is only raised when a block's maximum exceeds it by more than 2^8 (then O_h, l and a are
// rescaled), so the exponentials stay below 2^8 and rescales are rare. At the end of an item the
// first group merges the halves (O = (2^(m0-m) O_0 + 2^(m1-m) O_1) / l), O leaves through a TMA
// store, a / l goes to the per-head partials, and the last head of each (sequence, query tile) to
// finish averages the heads in fixed order and writes M (optionally blended with the carried score
// by eq. 4).
#include <cuda_bf16.h>
#include <math_constants.h>

#include "device_common.cuh"
#include "ptx.cuh"
#include "smoes_internal.cuh"

namespace smoes {
namespace {

constexpr int kFT = 128;                       // queries per tile, keys per block
constexpr int kFHd = 128;                      // head dimension handled here
constexpr uint32_t kFTile = kFT * kFHd * 2;    // bytes of a Q tile, K or V block, P or O tile
constexpr int kFStages = 2;                    // K/V blocks in flight
constexpr int kFHalf = kFT / 2;                // keys of a block per softmax group
constexpr int kFThreads = 64 + 2 * 128;        // producer, MMA issuer, two softmax groups
constexpr float kRescale = 8.f;                // raise the maximum in use only past +2^8

struct FwdAttnLayout {
  uint32_t q, k, v, pbuf, stg, mrg, bars, total;
};

// Q tile, K/V stages, the P tile (also the staging of O at the end of an item), per-stage key
// terms (bias [128] fp32 and the carried score [128] fp32 or uint8).
__host__ __device__ inline FwdAttnLayout fwd_attn_layout() {
  FwdAttnLayout L;
  uint32_t o = 0;
  L.q = o;    o += kFTile;
  L.k = o;    o += kFStages * kFTile;
  L.v = o;    o += kFStages * kFTile;
  L.pbuf = o; o += kFTile;
  L.stg = o;  o += kFStages * 2u * kFT * 4u;
  L.mrg = o;  o += 2u * 3u * kFT * 4u;            // second half's (max, l, a) per row, by item parity
  L.bars = o; o += 8u * (4u * kFStages + 24u) + 32u;
  L.total = o + 1024u;
  return L;
}

__device__ __forceinline__ float ex2f(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ uint32_t pack2_bf16(float lo, float hi) {
  return static_cast<uint32_t>(__bfloat16_as_ushort(__float2bfloat16_rn(lo))) |
         (static_cast<uint32_t>(__bfloat16_as_ushort(__float2bfloat16_rn(hi))) << 16);
}

// Item -> (sequence b, query head h, query tile qt): query tiles from the last (longest under the
// causal mask) down; within one tile index the heads of all sequences follow each other.
struct FItem {
  int b, h, qt;
};

__device__ __forceinline__ FItem decode_fitem(const AttnParams& p, int item) {
  const int BH = p.B * p.H;
  FItem it;
  it.qt = p.n_qtiles - 1 - item / BH;
  const int bh = item - (item / BH) * BH;
  it.b = bh / p.H;
  it.h = bh - it.b * p.H;
  return it;
}

__device__ __forceinline__ int fblocks_of(const AttnParams& p, int qt) {
  const int nk = p.S / kFT;
  return p.causal ? min(qt + 1, nk) : nk;
}

template <bool kFloatM>
__global__ void __launch_bounds__(kFThreads, 1)
k_attn_fwd(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
           const __grid_constant__ CUtensorMap tmV, const __grid_constant__ CUtensorMap tmO,
           const AttnFwdParams fp) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const AttnParams& p = fp.a;
  const FwdAttnLayout L = fwd_attn_layout();
  uint8_t* qs = base + L.q;
  uint8_t* ks = base + L.k;
  uint8_t* vs = base + L.v;
  uint8_t* pb = base + L.pbuf;
  float* kt = reinterpret_cast<float*>(base + L.stg);   // [stage][bias 128 | m 128]
  uint64_t* bars = reinterpret_cast<uint64_t*>(base + L.bars);
  uint64_t* kvfull = bars;                    // [kFStages] K, V and the key terms have landed
  uint64_t* kvempty = bars + kFStages;        // [kFStages] the block's P V has completed
  float* mrg = reinterpret_cast<float*>(base + L.mrg);   // [item parity][max | l | a][128]
  uint64_t* q_full = bars + 2 * kFStages;
  uint64_t* q_empty = q_full + 1;             // the item's last S has read Q
  uint64_t* s_full = q_full + 2;              // [2]
  uint64_t* s_empty = q_full + 4;             // [2] count 256 (both groups)
  uint64_t* p_full = q_full + 6;              // [2 halves] count 128
  uint64_t* p_empty = q_full + 8;             // [2 halves] the half's P V has read its P
  uint64_t* o_full = q_full + 10;             // the item's last P V has completed
  uint64_t* o_empty = q_full + 11;            // count 128: O read by the epilogue
  uint64_t* stg_full = q_full + 12;           // count 128: O staged
  uint64_t* stg_free = q_full + 13;           // the O store has read the staging
  uint64_t* out_bar = q_full + 14;            // count 128: head partials written
  uint64_t* dec_bar = q_full + 15;            // the tile's last-head decision is known
  uint64_t* drain = q_full + 16;              // all of the MMA warp's work has completed
  uint64_t* mrg_bar = q_full + 17;            // [2] count 128: the second half's state is handed over
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(q_full + 19);
  int* abort_flag = reinterpret_cast<int*>(tmem_slot + 1);
  uint32_t* decision = reinterpret_cast<uint32_t*>(tmem_slot + 2);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int G = fp.Hkv > 0 ? p.H / fp.Hkv : 1;           // query heads per key/value head
  WaitCtx wc{abort_flag, p.status, p.limit_ns};
  if (threadIdx.x == 0) {
    *abort_flag = 0;
    for (int i = 0; i < kFStages; ++i) {
      mbar_init(kvfull + i, 1);
      mbar_init(kvempty + i, 1);
    }
    mbar_init(q_full, 1);
    mbar_init(q_empty, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(s_full + i, 1);
      mbar_init(s_empty + i, 256);
      mbar_init(p_full + i, 128);
      mbar_init(p_empty + i, 1);
      mbar_init(mrg_bar + i, 128);
    }
    mbar_init(o_full, 1);
    mbar_init(o_empty, 128);
    mbar_init(stg_full, 128);
    mbar_init(stg_free, 1);
    mbar_init(out_bar, 128);
    mbar_init(dec_bar, 1);
    mbar_init(drain, 1);
    fence_mbar_init();
    tma_prefetch_desc(&tmQ);
    tma_prefetch_desc(&tmK);
    tma_prefetch_desc(&tmV);
    tma_prefetch_desc(&tmO);
  }
  if (warp == 1) tmem_alloc(tmem_slot, 512);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;             // S buffers at columns 0 and 128, O_0 at 256, O_1 at 384
  pdl_wait();                                   // Q, K, V, the scores and M of earlier work
  pdl_trigger();
  const int n_items = p.n_items;

  if (warp == 0) {
    // -------------------------------------------------------------- TMA producer
    if (lane == 0) {
      bool ok = true;
      int st = 0;
      uint32_t ph = 0;
      long issued = 0;
      int n = 0;
      const uint32_t mbytes = kFloatM ? kFT * 4u : kFT * 1u;
      const uint32_t tx = 2u * kFTile + (p.key_bias ? kFT * 4u : 0u) + mbytes;
      for (int item = blockIdx.x; item < n_items && ok; item += gridDim.x, ++n) {
        const FItem it = decode_fitem(p, item);
        const int hk = it.h / G;
        if (!mbar_wait(q_empty, (static_cast<uint32_t>(n) & 1u) ^ 1u, wc)) { ok = false; break; }
        const int qrow = (it.b * p.H + it.h) * p.S + it.qt * kFT;
        mbar_arrive_expect_tx(q_full, kFTile);
        tma_load_2d(qs, &tmQ, q_full, 0, qrow);
        tma_load_2d(qs + kFTile / 2, &tmQ, q_full, 64, qrow);
        const int nb = fblocks_of(p, it.qt);
        for (int j = 0; j < nb; ++j) {
          if (!mbar_wait(kvempty + st, ph ^ 1u, wc)) { ok = false; break; }
          const int krow = (it.b * fp.Hkv + hk) * p.S + j * kFT;
          const size_t key0 = static_cast<size_t>(it.b) * p.S + j * kFT;
          mbar_arrive_expect_tx(kvfull + st, tx);
          uint8_t* kb = ks + st * kFTile;
          uint8_t* vb = vs + st * kFTile;
          tma_load_2d(kb, &tmK, kvfull + st, 0, krow);
          tma_load_2d(kb + kFTile / 2, &tmK, kvfull + st, 64, krow);
          tma_load_2d(vb, &tmV, kvfull + st, 0, krow);
          tma_load_2d(vb + kFTile / 2, &tmV, kvfull + st, 64, krow);
          float* kts = kt + st * 2 * kFT;
          if (p.key_bias) bulk_load(kts, p.key_bias + key0, kFT * 4u, kvfull + st);
          if (kFloatM) bulk_load(kts + kFT, p.m_prev + key0, mbytes, kvfull + st);
          else bulk_load(kts + kFT, p.is_vision + key0, mbytes, kvfull + st);
          ++issued;
          if (++st == kFStages) { st = 0; ph ^= 1u; }
        }
      }
      if (!ok) {                    // every issued copy lands before the CTA may exit
        WaitCtx wd = wc;
        int dummy = 0;
        wd.abort_flag = &dummy;
        for (long q = (issued > kFStages ? issued - kFStages : 0); q < issued; ++q)
          mbar_wait(kvfull + (q % kFStages), static_cast<uint32_t>((q / kFStages) & 1), wd);
      }
    }
  } else if (warp == 1) {
    // -------------------------------------------------------------- MMA issuer
    if (lane == 0) {
      const uint32_t id_s = idesc_bf16(kFT, kFT, false, false);      // S = Q K^T (both K-major)
      const uint32_t id_o = idesc_bf16(kFT, kFHd, false, true);      // O += P V (V MN-major)
      const uint32_t tm_o = tmem + 256u;
      bool ok = true;
      int st = 0, pst = 0;
      uint32_t ph = 0;
      long g = 0;                                                    // blocks of this CTA so far
      int n = 0;
      for (int item = blockIdx.x; item < n_items && ok; item += gridDim.x, ++n) {
        const FItem it = decode_fitem(p, item);
        const int nb = fblocks_of(p, it.qt);
        if (!mbar_wait(q_full, static_cast<uint32_t>(n) & 1u, wc)) { ok = false; break; }
        tc_fence_after();
        const uint32_t qa = smem_u32(qs);
        for (int j = 0; j <= nb && ok; ++j) {
          if (j < nb) {
            // S_j = Q K_j^T into buffer g % 2
            if (!mbar_wait(kvfull + st, ph, wc)) { ok = false; break; }
            const int sb = static_cast<int>(g & 1);
            if (!mbar_wait(s_empty + sb, (static_cast<uint32_t>(g >> 1) & 1u) ^ 1u, wc)) { ok = false; break; }
            tc_fence_after();
            const uint32_t kb = smem_u32(ks + st * kFTile);
#pragma unroll
            for (int kk = 0; kk < kFHd / 16; ++kk) {     // K = 16 of the head dimension per step
              const uint32_t off = (kk >> 2) * (kFTile / 2) + (kk & 3) * 32;
              umma_bf16(tmem + static_cast<uint32_t>(sb * kFT), sdesc_sw128(qa + off, 16, 1024),
                        sdesc_sw128(kb + off, 16, 1024), id_s, kk > 0 ? 1u : 0u);
            }
            umma_commit(s_full + sb);
            if (j == nb - 1) umma_commit(q_empty);
          }
          if (j > 0) {
            // O_h += P_h V_h of block j - 1, each half once its softmax group has written its P
            const long gp = g - 1;                              // global index of block j - 1
            const uint32_t pa = smem_u32(pb);
            const uint32_t vb = smem_u32(vs + pst * kFTile);
            for (int hf = 0; hf < 2 && ok; ++hf) {
              if (!mbar_wait(p_full + hf, static_cast<uint32_t>(gp) & 1u, wc)) { ok = false; break; }
              if (j == 1 && hf == 0 && !mbar_wait(o_empty, (static_cast<uint32_t>(n) & 1u) ^ 1u, wc)) { ok = false; break; }
              tc_fence_after();
#pragma unroll
              for (int kk = 0; kk < kFHalf / 16; ++kk) {   // K = 16 keys per step
                const uint64_t da = sdesc_sw128(pa + hf * (kFTile / 2) + kk * 32, 16, 1024);
                const uint64_t dv = sdesc_sw128(vb + (hf * (kFHalf / 16) + kk) * 2048, kFTile / 2, 1024);
                umma_bf16(tm_o + static_cast<uint32_t>(hf * kFHd), da, dv, id_o, (j > 1 || kk > 0) ? 1u : 0u);
              }
              umma_commit(p_empty + hf);
            }
            if (!ok) break;
            umma_commit(kvempty + pst);
            if (++pst == kFStages) pst = 0;
            if (j == nb) umma_commit(o_full);
          }
          if (j < nb) {
            ++g;
            if (++st == kFStages) { st = 0; ph ^= 1u; }
          }
        }
      }
      umma_commit(drain);                 // every issued MMA completes before TMEM is released
      WaitCtx wd = wc;
      int dummy = 0;
      wd.abort_flag = &dummy;
      mbar_wait(drain, 0, wd);
    }
  } else {
    // -------------------------------------------------------------- softmax groups (2 x 4 warps)
    const int hf = (warp - 2) >> 2;              // half of each block's keys
    const int lg = warp & 3;                     // TMEM lane quarter of this warp
    const int row = lg * 32 + lane;              // query row of the tile
    const int gtid = (threadIdx.x - 64) & 127;   // thread of the group
    const uint32_t lane_off = static_cast<uint32_t>(lg * 32) << 16;
    const uint32_t to = tmem + lane_off + 256u + static_cast<uint32_t>(hf * kFHd);   // O_hf
    bool ok = true;
    long g = 0;
    int st = 0;
    uint32_t ph = 0;
    int n = 0;
    for (int item = blockIdx.x; item < n_items && ok; item += gridDim.x, ++n) {
      const FItem it = decode_fitem(p, item);
      const int nb = fblocks_of(p, it.qt);
      const int qi = it.qt * kFT + row;          // query index in the sequence
      float m_used = -CUDART_INF_F, l = 0.f, a = 0.f;
      for (int j = 0; j < nb; ++j, ++g) {
        const int sb = static_cast<int>(g & 1);
        if (!mbar_wait(kvfull + st, ph, wc)) { ok = false; break; }
        if (!mbar_wait(s_full + sb, static_cast<uint32_t>(g >> 1) & 1u, wc)) { ok = false; break; }
        tc_fence_after();
        const float* kts = kt + st * 2 * kFT;
        const uint8_t* mkb = reinterpret_cast<const uint8_t*>(kts + kFT);
        const bool diag = p.causal && j == it.qt;
        const uint32_t ts = tmem + lane_off + static_cast<uint32_t>(sb * kFT + hf * kFHalf);
        // the half's 64 logits of this row, log2-scaled, masked above the diagonal
        float t[kFHalf];
        {
          float v[32];
          tmem_ld32(ts, v);
#pragma unroll
          for (int q = 0; q < 32; ++q) t[q] = v[q];
          tmem_ld32(ts + 32u, v);
#pragma unroll
          for (int q = 0; q < 32; ++q) t[32 + q] = v[q];
        }
        tc_fence_before();
        mbar_arrive(s_empty + sb);               // the S buffer may be rewritten
        float mx = -CUDART_INF_F;
#pragma unroll
        for (int q = 0; q < kFHalf; ++q) {
          const int key = hf * kFHalf + q;
          const float b = p.key_bias ? kts[key] * 1.4426950408889634f : 0.f;
          t[q] = (diag && key > row) ? -CUDART_INF_F : fmaf(t[q], p.scale_log2, b);
          mx = fmaxf(mx, t[q]);
        }
        const float m_new = fmaxf(m_used, mx);
        const bool raise = j == 0 || m_new > m_used + kRescale;
        // the half's previous P V has read its P and updated O_hf before either changes; at the
        // first block of an item the staging of the previous item's O must have been stored
        if (j > 0) {
          if (!mbar_wait(p_empty + hf, static_cast<uint32_t>(g - 1) & 1u, wc)) { ok = false; break; }
        } else if (n > 0) {
          if (!mbar_wait(stg_free, static_cast<uint32_t>(n - 1) & 1u, wc)) { ok = false; break; }
        }
        if (__any_sync(0xffffffffu, raise && j > 0)) {          // rescale O_hf, l and a (rare)
          tc_fence_after();
          const float alpha = (raise && j > 0) ? (m_used == -CUDART_INF_F ? 0.f : ex2f(m_used - m_new)) : 1.f;
#pragma unroll 1
          for (int c = 0; c < kFHd / 32; ++c) {
            float v[32];
            tmem_ld32(to + 32u * c, v);
#pragma unroll
            for (int q = 0; q < 32; ++q) v[q] *= alpha;
            tmem_st32(to + 32u * c, v);
          }
          l *= alpha;
          a *= alpha;
        }
        if (raise) m_used = m_new;
        // P = 2^(logit - max in use) in bf16 to the half's atom of the P tile; l and the mass. A
        // half whose keys are all above the diagonal so far (max -inf) has P = 0.
        const float msub = m_used == -CUDART_INF_F ? 0.f : m_used;
        uint32_t pk[kFHalf / 2];
#pragma unroll
        for (int q = 0; q < kFHalf; q += 2) {
          const int k0 = hf * kFHalf + q;
          const float p0 = ex2f(t[q] - msub), p1 = ex2f(t[q + 1] - msub);
          const float m0 = kFloatM ? kts[kFT + k0] : (mkb[k0] ? 1.f : 0.f);
          const float m1 = kFloatM ? kts[kFT + k0 + 1] : (mkb[k0 + 1] ? 1.f : 0.f);
          l += p0 + p1;
          a = fmaf(p0, m0, fmaf(p1, m1, a));
          pk[q >> 1] = pack2_bf16(p0, p1);
        }
        uint8_t* prow = pb + hf * (kFTile / 2) + row * 128;
#pragma unroll
        for (int u = 0; u < 8; ++u) {
          const uint32_t chunk = static_cast<uint32_t>(u) ^ static_cast<uint32_t>(row & 7);
          *reinterpret_cast<uint4*>(prow + (chunk << 4)) = make_uint4(pk[4 * u], pk[4 * u + 1], pk[4 * u + 2], pk[4 * u + 3]);
        }
        fence_proxy_async_smem();
        mbar_arrive(p_full + hf);
        if (++st == kFStages) { st = 0; ph ^= 1u; }
      }
      if (!ok) break;
      float* mb = mrg + (n & 1) * 3 * kFT;
      if (hf == 1) {                             // hand the half's state to the first group
        mb[row] = m_used;
        mb[kFT + row] = l;
        mb[2 * kFT + row] = a;
        mbar_arrive(mrg_bar + (n & 1));
        continue;
      }
      // epilogue (first group): merge the halves, O / l through the staging (the P tile, free
      // once the last P V completed)
      if (!mbar_wait(o_full, static_cast<uint32_t>(n) & 1u, wc)) { ok = false; break; }
      if (!mbar_wait(mrg_bar + (n & 1), static_cast<uint32_t>(n >> 1) & 1u, wc)) { ok = false; break; }
      tc_fence_after();
      const float m1 = mb[row], l1 = mb[kFT + row], a1 = mb[2 * kFT + row];
      const float mm = fmaxf(m_used, m1);                   // finite: the first half sees key 0
      const float c0 = ex2f(m_used - mm), c1 = m1 == -CUDART_INF_F ? 0.f : ex2f(m1 - mm);
      l = l * c0 + l1 * c1;
      a = a * c0 + a1 * c1;
      const float il = 1.f / l;
      const float s0 = c0 * il, s1 = c1 * il;
      const uint32_t o0 = tmem + lane_off + 256u;
#pragma unroll 1
      for (int c = 0; c < kFHd / 32; ++c) {
        float v[32], w[32];
        tmem_ld32(o0 + 32u * c, v);
        tmem_ld32(o0 + kFHd + 32u * c, w);
        uint32_t pk[16];
#pragma unroll
        for (int q = 0; q < 32; q += 2)
          pk[q >> 1] = pack2_bf16(fmaf(v[q], s0, w[q] * s1), fmaf(v[q + 1], s0, w[q + 1] * s1));
        uint8_t* orow = pb + (c >> 1) * (kFTile / 2) + row * 128;
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const uint32_t chunk = static_cast<uint32_t>((c & 1) * 4 + u) ^ static_cast<uint32_t>(row & 7);
          *reinterpret_cast<uint4*>(orow + (chunk << 4)) = make_uint4(pk[4 * u], pk[4 * u + 1], pk[4 * u + 2], pk[4 * u + 3]);
        }
      }
      tc_fence_before();
      mbar_arrive(o_empty);
      fence_proxy_async_smem();
      mbar_arrive(stg_full);
      const int orow0 = (it.b * p.H + it.h) * p.S + it.qt * kFT;
      if (gtid == 0) {
        if (mbar_wait(stg_full, static_cast<uint32_t>(n) & 1u, wc)) {
          tma_store_2d(&tmO, pb, 0, orow0);
          tma_store_2d(&tmO, pb + kFTile / 2, 64, orow0);
          tma_store_commit();
          tma_store_wait_read<0>();
        }
        mbar_arrive(stg_free);
      }
      if (!mbar_wait(stg_free, static_cast<uint32_t>(n) & 1u, wc)) { ok = false; break; }
      // this head's score, then the head average of the tile by the last head to finish
      const size_t tok = static_cast<size_t>(it.b) * p.S + qi;
      p.part[static_cast<size_t>(it.h) * p.T + tok] = a * il;
      __threadfence();
      mbar_arrive(out_bar);
      if (gtid == 0) {
        uint32_t last = 0u;
        if (mbar_wait(out_bar, static_cast<uint32_t>(n) & 1u, wc)) {
          const uint32_t cnt = atomicAdd(p.ticket + it.b * p.n_qtiles + it.qt, 1u) + 1u;
          last = (cnt == static_cast<uint32_t>(p.H)) ? 1u : 0u;
          if (last) p.ticket[it.b * p.n_qtiles + it.qt] = 0u;        // ready for the next call
        }
        *decision = last;
        mbar_arrive(dec_bar);
      }
      if (!mbar_wait(dec_bar, static_cast<uint32_t>(n) & 1u, wc)) { ok = false; break; }
      if (*decision) {
        __threadfence();
        float sum = 0.f;
        for (int hh = 0; hh < p.H; ++hh) sum += __ldcg(p.part + static_cast<size_t>(hh) * p.T + tok);
        float mv = sum / static_cast<float>(p.H);                       // eq. (3)
        if (p.xattn_norm) {                                              // eq. (4)
          const float an = __ldg(p.xattn_norm + tok), rn = __ldg(p.x_norm + tok);
          const float mprev = kFloatM ? __ldg(p.m_prev + tok) : static_cast<float>(__ldg(p.is_vision + tok) != 0);
          mv = (an * mv + rn * mprev) / (an + rn);
        }
        reinterpret_cast<float2*>(p.M)[tok] = make_float2(mv, 1.f - mv);
      }
    }
    if (hf == 0 && gtid == 0) tma_store_wait_all<0>();
  }

  // the role branches leave single lanes running on their own: the warp reconverges before
  // the block barrier, so that no thread passes it while another of its warp is still working
  __syncwarp();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem, 512);
}

}  // namespace

cudaError_t launch_attn_fwd(const AttnFwdParams& fp, const CUtensorMap& tmQ, const CUtensorMap& tmK,
                            const CUtensorMap& tmV, const CUtensorMap& tmO, int n_sms, cudaStream_t s) {
  const AttnParams& p = fp.a;
  if (p.hd != kFHd || p.S % kFT != 0 || fp.Hkv < 1 || p.H % fp.Hkv != 0) return cudaErrorNotSupported;
  const uint32_t smem = fwd_attn_layout().total;
  if (smem > 227u * 1024u) return cudaErrorInvalidConfiguration;
  const int grid = p.n_items < n_sms ? p.n_items : n_sms;
  auto k = p.m_prev ? k_attn_fwd<true> : k_attn_fwd<false>;
  cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  return launch_pdl(k, dim3(grid), dim3(kFThreads), smem, s, tmQ, tmK, tmV, tmO, fp);
}

}  // namespace smoes
