// attn_mass.cu -- attention-accumulated vision score, eqs. (2)-(4).
//
// For sequence b and query j:  Mtilde_v[b,j] = (1/H) sum_h sum_{j'} softmax_{j'}(s q_j.k_j' + beta_j') m_j',
// the head-averaged attention matrix applied to the keys' carried vision score m (eq. 3; the hard
// labels of eq. 2 at layer 0). As the paper notes, this equals attention with the score as the
// value vector, so it runs FlashAttention-style without materialising the attention matrix:
// per (sequence, head, 128-query tile) the scores S = Q K^T of each 128-key block are formed on
// tcgen05 tensor cores (TMA-fed, accumulator in TMEM); four softmax warps (one query row per
// thread) keep the online max, the normaliser l = sum e^(s - max) and the vision mass
// a = sum e^(s - max) m_j'. The head's score a / l goes to the workspace; the last head of each
// (sequence, query tile) to finish averages the heads in fixed order and writes M (optionally
// blended with the carried score by eq. 4).
#include <cuda_bf16.h>
#include <math_constants.h>

#include "device_common.cuh"
#include "ptx.cuh"
#include "smoes_internal.cuh"

namespace smoes {
namespace {

constexpr int kAT = 128;                      // queries per tile, keys per block
constexpr int kHd = 128;                      // head dimension handled here
constexpr uint32_t kTile = kAT * kHd * 2;     // bytes of one Q tile or K block (2 swizzle atoms)

struct AttnLayout {
  uint32_t q, k, mk, bars, total;
};

__host__ __device__ inline AttnLayout attn_layout(int n_ks) {
  AttnLayout L;
  uint32_t o = 0;
  L.q = o;    o += kTile;                                  // Q tile [2 atoms][128 rows][128 B]
  L.k = o;    o += static_cast<uint32_t>(n_ks) * kTile;    // K blocks
  L.mk = o;   o += 2u * kAT * 8u;                          // (bias*log2e, m) per key, 2 buffers
  L.bars = o; o += 8u * (2u * n_ks + 12u) + 16u;
  L.total = o + 1024u;
  return L;
}

// Work item -> (sequence b, head h, query tile qt). Items are ordered head-major so that the
// items running at the same time share keys in L2; a CTA's items cycle through tile sizes.
__device__ __forceinline__ void decode_item(const AttnParams& p, int item, int& b, int& h, int& qt) {
  const int bh = item / p.n_qtiles;
  qt = item - bh * p.n_qtiles;
  b = bh / p.H;
  h = bh - b * p.H;
}

__device__ __forceinline__ int kblocks_of(const AttnParams& p, int qt) {
  const int nk = (p.S + kAT - 1) / kAT;
  return p.causal ? min(qt + 1, nk) : nk;
}

template <bool kFloatM>
__global__ void __launch_bounds__(192, 1)
k_attn_mass(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
            const AttnParams p, const int n_ks) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const AttnLayout L = attn_layout(n_ks);
  uint8_t* qs = base + L.q;
  uint8_t* ks = base + L.k;
  float2* mk = reinterpret_cast<float2*>(base + L.mk);
  uint64_t* bars = reinterpret_cast<uint64_t*>(base + L.bars);
  uint64_t* kfull = bars;
  uint64_t* kempty = bars + n_ks;
  uint64_t* q_full = bars + 2 * n_ks;
  uint64_t* q_empty = q_full + 1;
  uint64_t* s_full = q_full + 2;      // [2]
  uint64_t* s_empty = q_full + 4;     // [2]
  uint64_t* mk_bar = q_full + 6;      // [2] keys' (bias, m) staged by the softmax group
  uint64_t* out_bar = q_full + 8;     // head results of the tile written
  uint64_t* drain = q_full + 9;
  uint64_t* dec_bar = q_full + 10;    // the ticket decision of the tile is published
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(q_full + 12);
  int* abort_flag = reinterpret_cast<int*>(tmem_slot + 1);
  volatile uint32_t* decision = reinterpret_cast<volatile uint32_t*>(tmem_slot + 2);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  WaitCtx wc{abort_flag, p.status, p.limit_ns};
  if (threadIdx.x == 0) {
    *abort_flag = 0;
    for (int i = 0; i < n_ks; ++i) {
      mbar_init(kfull + i, 1);
      mbar_init(kempty + i, 1);
    }
    mbar_init(q_full, 1);
    mbar_init(q_empty, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(s_full + i, 1);
      mbar_init(s_empty + i, 128);
      mbar_init(mk_bar + i, 128);
    }
    mbar_init(out_bar, 128);
    mbar_init(dec_bar, 1);
    mbar_init(drain, 1);
    fence_mbar_init();
    tma_prefetch_desc(&tmQ);
    tma_prefetch_desc(&tmK);
  }
  if (warp == 1) tmem_alloc(tmem_slot, 256);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    // ---------------------------------------------------------------- TMA producer
    if (lane == 0) {
      int st = 0;
      uint32_t ph = 0;
      int it = 0;
      long issued = 0;
      bool ok = true;
      for (int item = blockIdx.x; item < p.n_items && ok; item += gridDim.x, ++it) {
        int b, h, qt;
        decode_item(p, item, b, h, qt);
        const int row0 = (b * p.H + h) * p.S;
        if (!mbar_wait(q_empty, (static_cast<uint32_t>(it) & 1u) ^ 1u, wc)) { ok = false; break; }
        mbar_arrive_expect_tx(q_full, kTile);
        tma_load_2d(qs, &tmQ, q_full, 0, row0 + qt * kAT);
        tma_load_2d(qs + kTile / 2, &tmQ, q_full, 64, row0 + qt * kAT);
        const int nkb = kblocks_of(p, qt);
        for (int kb = 0; kb < nkb; ++kb) {
          if (!mbar_wait(kempty + st, ph ^ 1u, wc)) { ok = false; break; }
          uint8_t* kd = ks + st * kTile;
          mbar_arrive_expect_tx(kfull + st, kTile);
          tma_load_2d(kd, &tmK, kfull + st, 0, row0 + kb * kAT);
          tma_load_2d(kd + kTile / 2, &tmK, kfull + st, 64, row0 + kb * kAT);
          ++issued;
          if (++st == n_ks) { st = 0; ph ^= 1u; }
        }
      }
      if (!ok) {
        WaitCtx wd = wc;
        int dummy = 0;
        wd.abort_flag = &dummy;
        for (long q = (issued > n_ks ? issued - n_ks : 0); q < issued; ++q)
          mbar_wait(kfull + (q % n_ks), static_cast<uint32_t>((q / n_ks) & 1), wd);
        mbar_wait(q_full, static_cast<uint32_t>((it) & 1), wd);
      }
    }
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA issuer
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16(kAT, kAT, false, false);
      int st = 0;
      uint32_t ph = 0;
      int blk = 0;                      // running block count: selects the TMEM buffer
      int it = 0;
      bool ok = true;
      for (int item = blockIdx.x; item < p.n_items && ok; item += gridDim.x, ++it) {
        int b, h, qt;
        decode_item(p, item, b, h, qt);
        if (!mbar_wait(q_full, static_cast<uint32_t>(it) & 1u, wc)) { ok = false; break; }
        tc_fence_after();
        const uint32_t qa = smem_u32(qs);
        const int nkb = kblocks_of(p, qt);
        for (int kb = 0; kb < nkb; ++kb, ++blk) {
          const int buf = blk & 1;
          if (!mbar_wait(s_empty + buf, (static_cast<uint32_t>(blk >> 1) & 1u) ^ 1u, wc)) { ok = false; break; }
          if (!mbar_wait(kfull + st, ph, wc)) { ok = false; break; }
          tc_fence_after();
          const uint32_t kbase = smem_u32(ks + st * kTile);
          const uint32_t d_tmem = tmem + static_cast<uint32_t>(buf * kAT);
#pragma unroll
          for (int kk = 0; kk < kHd / 16; ++kk) {
            const uint32_t off = (kk >> 2) * (kTile / 2) + (kk & 3) * 32;
            umma_bf16(d_tmem, sdesc_sw128(qa + off, 16, 1024), sdesc_sw128(kbase + off, 16, 1024), idesc,
                      kk > 0 ? 1u : 0u);
          }
          umma_commit(kempty + st);
          umma_commit(s_full + buf);
          if (++st == n_ks) { st = 0; ph ^= 1u; }
        }
        if (!ok) break;
        umma_commit(q_empty);           // the Q tile may be replaced once its MMAs are done
      }
      umma_commit(drain);
      WaitCtx wd = wc;
      int dummy = 0;
      wd.abort_flag = &dummy;
      mbar_wait(drain, 0, wd);
    }
  } else {
    // ---------------------------------------------------------------- softmax group (4 warps)
    const int lg = warp & 3;
    const int row = lg * 32 + lane;            // query row in the tile == TMEM lane
    const int gt = threadIdx.x - 64;           // 0..127 inside the group
    int blk = 0;
    int it = 0;
    for (int item = blockIdx.x; item < p.n_items; item += gridDim.x, ++it) {
      int b, h, qt;
      decode_item(p, item, b, h, qt);
      const int q = qt * kAT + row;             // query position in the sequence
      const int nkb = kblocks_of(p, qt);
      float mrun = -CUDART_INF_F, l = 0.f, a = 0.f;
      bool ok = true;
      for (int kb = 0; kb < nkb; ++kb, ++blk) {
        const int buf = blk & 1;
        const uint32_t use = static_cast<uint32_t>(blk >> 1);
        // stage this block's keys: (bias * log2 e, carried score), masked keys get -inf
        {
          const int key = kb * kAT + gt;
          float bias = -CUDART_INF_F, m = 0.f;
          if (key < p.S) {
            const size_t t = static_cast<size_t>(b) * p.S + key;
            bias = p.key_bias ? __ldg(p.key_bias + t) * 1.4426950408889634f : 0.f;
            m = kFloatM ? __ldg(p.m_prev + t) : static_cast<float>(__ldg(p.is_vision + t) != 0);
          }
          mk[buf * kAT + gt] = make_float2(bias, m);
          mbar_arrive(mk_bar + buf);
        }
        if (!mbar_wait(mk_bar + buf, use & 1u, wc)) { ok = false; break; }
        if (!mbar_wait(s_full + buf, use & 1u, wc)) { ok = false; break; }
        tc_fence_after();
        const uint32_t ta = tmem + (static_cast<uint32_t>(lg * 32) << 16) + static_cast<uint32_t>(buf * kAT);
        const float2* mkb = mk + buf * kAT;
        const bool diag = p.causal && kb == qt;
#pragma unroll 1
        for (int c = 0; c < kAT / 32; ++c) {
          float v[32];
          tmem_ld32(ta + 32u * c, v);
          float cmax = -CUDART_INF_F;
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            const int kc = c * 32 + i;
            const float2 bm = mkb[kc];
            float s = fmaf(v[i], p.scale_log2, bm.x);
            if (diag && kc > row) s = -CUDART_INF_F;
            v[i] = s;
            cmax = fmaxf(cmax, s);
          }
          const float mnew = fmaxf(mrun, cmax);
          if (mnew != -CUDART_INF_F) {
            const float corr = exp2f(mrun - mnew);
            l *= corr;
            a *= corr;
            mrun = mnew;
#pragma unroll
            for (int i = 0; i < 32; ++i) {
              const float e = exp2f(v[i] - mnew);
              l += e;
              a = fmaf(e, mkb[c * 32 + i].y, a);
            }
          }
        }
        tc_fence_before();
        mbar_arrive(s_empty + buf);
      }
      if (!ok) break;
      // head result, then the head average of the tile by the last head to finish
      const bool valid = q < p.S;
      const size_t tok = static_cast<size_t>(b) * p.S + q;
      if (valid) p.part[static_cast<size_t>(h) * p.T + tok] = a / l;
      __threadfence();
      mbar_arrive(out_bar);
      if (gt == 0) {
        uint32_t last = 0u;
        if (mbar_wait(out_bar, static_cast<uint32_t>(it) & 1u, wc)) {
          const uint32_t n = atomicAdd(p.ticket + b * p.n_qtiles + qt, 1u) + 1u;
          last = (n == static_cast<uint32_t>(p.H)) ? 1u : 0u;
          if (last) p.ticket[b * p.n_qtiles + qt] = 0u;     // ready for the next call
        }
        *decision = last;
        mbar_arrive(dec_bar);
      }
      if (!mbar_wait(dec_bar, static_cast<uint32_t>(it) & 1u, wc)) break;
      if (*decision && valid) {
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
  }

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem, 256);
}

}  // namespace

cudaError_t launch_attn_mass(const AttnParams& p, const CUtensorMap& tmQ, const CUtensorMap& tmK,
                             int n_sms, cudaStream_t s) {
  if (p.hd != kHd) return cudaErrorNotSupported;
  const int n_ks = 4;
  const uint32_t smem = attn_layout(n_ks).total;
  const int grid = p.n_items < n_sms ? p.n_items : n_sms;
  auto k = p.m_prev ? k_attn_mass<true> : k_attn_mass<false>;
  cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  k<<<grid, 192, smem, s>>>(tmQ, tmK, p, n_ks);
  return cudaGetLastError();
}

}  // namespace smoes
