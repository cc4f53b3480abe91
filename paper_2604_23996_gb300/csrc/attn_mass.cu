// attn_mass.cu -- attention-accumulated vision score, eqs. (2)-(4).
//
// For sequence b and query j:  Mtilde_v[b,j] = (1/H) sum_h sum_{j'} softmax_{j'}(s q_j.k_j' + beta_j') m_j',
// the head-averaged attention matrix applied to the keys' carried vision score m (eq. 3; the hard
// labels of eq. 2 at layer 0). This equals attention with the score as the value vector, so it
// runs FlashAttention-style without materialising the attention matrix.
//
// A work item is (sequence, head, pair of adjacent 128-query tiles). The two tiles share one
// stream of 128-key blocks: for each block the tensor cores form S = Q K^T of both tiles
// (tcgen05, TMA-fed, accumulators in TMEM, two buffers per tile). Four softmax groups of four
// warps (one query row per thread; a group per tile and half of the 128 keys of a block) keep
// the online max, the normaliser l = sum e^(s - max) and the vision mass a = sum e^(s - max) m_j'
// of their keys; at the end of an item the second half's state is merged into the first's (fixed
// order). Sixteen softmax warps keep the special-function unit, which evaluates one
// exponential per score, busier than eight could. The head's score a / l goes to the workspace;
// the last head of each (sequence, query tile) to finish averages the heads in fixed order and
// writes M (optionally blended with the carried score by eq. 4). Items are ordered longest
// first and dealt to the CTAs in rounds of alternating direction, so that the CTAs finish
// together.
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

constexpr int kHalf = kAT / 2;                // keys of a block per softmax group
constexpr int kAttnThreads = 64 + 4 * 128;    // producer, MMA issuer, four softmax groups

struct AttnLayout {
  uint32_t q, k, mk, mrg, bars, total;
};

__host__ __device__ inline AttnLayout attn_layout(int n_ks) {
  AttnLayout L;
  uint32_t o = 0;
  L.q = o;    o += 2u * kTile;                             // two Q tiles [2 atoms][128 rows][128 B]
  L.k = o;    o += static_cast<uint32_t>(n_ks) * kTile;    // K blocks
  L.mk = o;   o += 4u * 2u * 2u * kHalf * 4u;              // bias*log2e [64] | m [64]: group x buffer
  L.mrg = o;  o += 2u * 2u * 3u * kAT * 4u;                // second half's (max, l, a): tile x buffer
  L.bars = o; o += 8u * (2u * n_ks + 36u) + 32u;
  L.total = o + 1024u;
  return L;
}

// 2^x on the special-function unit (flushes results below 2^-126 to zero).
__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Packed fp32 pair arithmetic (one instruction for two lanes' worth of work per thread):
// (d0, d1) = (a0, a1) * (b0, b1) + (c0, c1), and (d0, d1) = (a0, a1) + (b0, b1).
__device__ __forceinline__ void fma2(float& d0, float& d1, float a0, float a1, float b0, float b1,
                                     float c0, float c1) {
  asm("{\n\t.reg .b64 ra, rb, rc, rd;\n\t"
      "mov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %5};\n\tmov.b64 rc, {%6, %7};\n\t"
      "fma.rn.f32x2 rd, ra, rb, rc;\n\t"
      "mov.b64 {%0, %1}, rd;\n\t}"
      : "=f"(d0), "=f"(d1) : "f"(a0), "f"(a1), "f"(b0), "f"(b1), "f"(c0), "f"(c1));
}
__device__ __forceinline__ void add2(float& d0, float& d1, float a0, float a1, float b0, float b1) {
  asm("{\n\t.reg .b64 ra, rb, rd;\n\t"
      "mov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %5};\n\t"
      "add.rn.f32x2 rd, ra, rb;\n\t"
      "mov.b64 {%0, %1}, rd;\n\t}"
      : "=f"(d0), "=f"(d1) : "f"(a0), "f"(a1), "f"(b0), "f"(b1));
}

// Work items of a persistent kernel, dealt to the CTAs in rounds of gridDim.x that alternate in
// direction: in round r CTA c takes item r * G + c when r is even and r * G + (G - 1 - c) when it
// is odd. With the items ordered longest first, each CTA's total stays within about one item of
// the mean, where a plain stride gives the low-numbered CTAs the longest item of every round.
__device__ __forceinline__ int dealt_item(int round) {
  const int g = static_cast<int>(gridDim.x), c = static_cast<int>(blockIdx.x);
  return round * g + ((round & 1) ? g - 1 - c : c);
}

// Bounded wait with its slow path out of line: the softmax warps keep the wait context in
// memory instead of in registers, which their 96-register budget needs for the scores.
__device__ __noinline__ bool wait_slow(uint64_t* bar, uint32_t parity, const WaitCtx& w) {
  return mbar_wait(bar, parity, w);
}
__device__ __forceinline__ bool wait_bar(uint64_t* bar, uint32_t parity, const WaitCtx& w) {
  return mbar_try_wait(bar, parity) || wait_slow(bar, parity, w);
}

// Work item -> (sequence b, head h, query-tile pair pr). Pairs run longest (last) first; within
// a pair index the heads of all sequences follow each other, so concurrent items share L2 keys.
struct Item {
  int b, h, qt0, nq;          // first query tile, tiles in the pair (1 or 2)
};

__device__ __forceinline__ Item decode_item(const AttnParams& p, int item) {
  const int n_pairs = (p.n_qtiles + 1) / 2;
  const int BH = p.B * p.H;
  const int pr = n_pairs - 1 - item / BH;
  const int bh = item - (item / BH) * BH;
  Item it;
  it.b = bh / p.H;
  it.h = bh - it.b * p.H;
  it.qt0 = 2 * pr;
  it.nq = min(2, p.n_qtiles - it.qt0);
  return it;
}

// Key blocks query tile qt attends to.
__device__ __forceinline__ int kblocks_of(const AttnParams& p, int qt) {
  const int nk = (p.S + kAT - 1) / kAT;
  return p.causal ? min(qt + 1, nk) : nk;
}

template <bool kFloatM>
__global__ void __launch_bounds__(kAttnThreads, 1)
k_attn_mass(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
            const AttnParams p, const int n_ks) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const AttnLayout L = attn_layout(n_ks);
  uint8_t* qs = base + L.q;
  uint8_t* ks = base + L.k;
  float* mk = reinterpret_cast<float*>(base + L.mk);
  float* mrg = reinterpret_cast<float*>(base + L.mrg);
  uint64_t* bars = reinterpret_cast<uint64_t*>(base + L.bars);
  uint64_t* kfull = bars;
  uint64_t* kempty = bars + n_ks;
  uint64_t* q_full = bars + 2 * n_ks;   // [2] per tile of the pair
  uint64_t* q_empty = q_full + 2;       // [2]
  uint64_t* s_full = q_full + 4;        // [tile][buf]
  uint64_t* s_empty = q_full + 8;       // [tile][buf]
  uint64_t* mk_bar = q_full + 12;       // [group][buf] keys' (bias, m) staged by that group
  uint64_t* out_bar = q_full + 20;      // [tile] head results of the tile written
  uint64_t* dec_bar = q_full + 22;      // [tile] the ticket decision of the tile is published
  uint64_t* mrg_full = q_full + 24;     // [tile][merge buffer] the second half's state is written
  uint64_t* mrg_free = q_full + 28;     // [tile][merge buffer] the first half has read it
  uint64_t* drain = q_full + 32;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(q_full + 34);
  int* abort_flag = reinterpret_cast<int*>(tmem_slot + 1);
  volatile uint32_t* decision = reinterpret_cast<volatile uint32_t*>(tmem_slot + 2);   // [2]

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int BH = p.B * p.H;
  const int n_items = ((p.n_qtiles + 1) / 2) * BH;
  WaitCtx wc{abort_flag, p.status, p.limit_ns};
  if (threadIdx.x == 0) {
    *abort_flag = 0;
    for (int i = 0; i < n_ks; ++i) {
      mbar_init(kfull + i, 1);
      mbar_init(kempty + i, 1);
    }
    for (int t = 0; t < 2; ++t) {
      mbar_init(q_full + t, 1);
      mbar_init(q_empty + t, 1);
      mbar_init(out_bar + t, 128);
      mbar_init(dec_bar + t, 1);
      for (int i = 0; i < 2; ++i) {
        mbar_init(mrg_full + 2 * t + i, 128);
        mbar_init(mrg_free + 2 * t + i, 128);
      }
      for (int i = 0; i < 2; ++i) {
        mbar_init(s_full + 2 * t + i, 1);
        mbar_init(s_empty + 2 * t + i, 256);     // both key halves read the scores
      }
    }
    for (int i = 0; i < 8; ++i) mbar_init(mk_bar + i, 128);
    mbar_init(drain, 1);
    fence_mbar_init();
    tma_prefetch_desc(&tmQ);
    tma_prefetch_desc(&tmK);
  }
  if (warp == 1) tmem_alloc(tmem_slot, 512);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  pdl_wait();                                 // Q, K and the outputs may be in use before this
  pdl_trigger();

  if (warp == 0) {
    // ---------------------------------------------------------------- TMA producer
    if (lane == 0) {
      int st = 0;
      uint32_t ph = 0;
      int nqt[2] = {0, 0};              // items that used Q buffer t: its barrier phase
      long issued = 0;
      bool ok = true;
      for (int rd = 0; ok; ++rd) {
        const int item = dealt_item(rd);
        if (item >= n_items) break;
        const Item w = decode_item(p, item);
        const int row0 = (w.b * p.H + w.h) * p.S;
        for (int t = 0; t < w.nq && ok; ++t) {
          if (!mbar_wait(q_empty + t, (static_cast<uint32_t>(nqt[t]) & 1u) ^ 1u, wc)) { ok = false; break; }
          ++nqt[t];
          mbar_arrive_expect_tx(q_full + t, kTile);
          tma_load_2d(qs + t * kTile, &tmQ, q_full + t, 0, row0 + (w.qt0 + t) * kAT);
          tma_load_2d(qs + t * kTile + kTile / 2, &tmQ, q_full + t, 64, row0 + (w.qt0 + t) * kAT);
        }
        const int nkb = kblocks_of(p, w.qt0 + w.nq - 1);
        for (int kb = 0; kb < nkb && ok; ++kb) {
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
        for (int t = 0; t < 2; ++t)
          if (nqt[t] > 0) mbar_wait(q_full + t, static_cast<uint32_t>(nqt[t] - 1) & 1u, wd);
      }
    }
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA issuer
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16(kAT, kAT, false, false);
      int st = 0;
      uint32_t ph = 0;
      int blk[2] = {0, 0};              // running block count per tile: selects its TMEM buffer
      int nqt[2] = {0, 0};
      bool ok = true;
      for (int rd = 0; ok; ++rd) {
        const int item = dealt_item(rd);
        if (item >= n_items) break;
        const Item w = decode_item(p, item);
        for (int t = 0; t < w.nq && ok; ++t)
          if (!mbar_wait(q_full + t, static_cast<uint32_t>(nqt[t]++) & 1u, wc)) ok = false;
        if (!ok) break;
        tc_fence_after();
        const int nkb0 = kblocks_of(p, w.qt0), nkb = kblocks_of(p, w.qt0 + w.nq - 1);
        for (int kb = 0; kb < nkb; ++kb) {
          if (!mbar_wait(kfull + st, ph, wc)) { ok = false; break; }
          tc_fence_after();
          const uint32_t kbase = smem_u32(ks + st * kTile);
          for (int t = 0; t < w.nq; ++t) {
            if (t == 0 && kb >= nkb0) continue;       // past the first tile's diagonal
            const int buf = blk[t] & 1;
            if (!mbar_wait(s_empty + 2 * t + buf, (static_cast<uint32_t>(blk[t] >> 1) & 1u) ^ 1u, wc)) {
              ok = false;
              break;
            }
            tc_fence_after();
            const uint32_t qa = smem_u32(qs + t * kTile);
            const uint32_t d_tmem = tmem + static_cast<uint32_t>((2 * t + buf) * kAT);
#pragma unroll
            for (int kk = 0; kk < kHd / 16; ++kk) {
              const uint32_t off = (kk >> 2) * (kTile / 2) + (kk & 3) * 32;
              umma_bf16(d_tmem, sdesc_sw128(qa + off, 16, 1024), sdesc_sw128(kbase + off, 16, 1024), idesc,
                        kk > 0 ? 1u : 0u);
            }
            umma_commit(s_full + 2 * t + buf);
            ++blk[t];
          }
          if (!ok) break;
          umma_commit(kempty + st);
          if (++st == n_ks) { st = 0; ph ^= 1u; }
        }
        if (!ok) break;
        for (int t = 0; t < w.nq; ++t) umma_commit(q_empty + t);   // Q tiles may be replaced
      }
      umma_commit(drain);
      WaitCtx wd = wc;
      int dummy = 0;
      wd.abort_flag = &dummy;
      mbar_wait(drain, 0, wd);
    }
  } else {
    // ---------------------------------------------------------------- softmax groups (4 x 4 warps)
    const int grp = (warp - 2) >> 2;
    const int t = grp & 1;                     // query tile of the pair handled by this group
    const int hf = grp >> 1;                   // half of each key block: keys [64 hf, 64 hf + 64)
    const int lg = warp & 3;
    const int row = lg * 32 + lane;            // query row in the tile == TMEM lane
    const int gt = threadIdx.x - 64 - 128 * grp; // 0..127 inside the group
    float* mkg = mk + grp * 2 * kAT;           // this group's staging: [buf][bias 64 | m 64]
    float* mrt = mrg + t * 2 * 3 * kAT;        // the tile's merge buffers: [item parity][3][128]
    uint64_t* sfull = s_full + 2 * t;
    uint64_t* sempty = s_empty + 2 * t;
    uint64_t* mkbar = mk_bar + 2 * grp;
    int blk = 0;
    int ng = 0;                                // items this group has processed
    for (int rd = 0; ; ++rd) {
      const int item = dealt_item(rd);
      if (item >= n_items) break;
      const Item w = decode_item(p, item);
      if (t >= w.nq) continue;
      const int qt = w.qt0 + t;
      const int q = qt * kAT + row;             // query position in the sequence
      const int nkb = kblocks_of(p, qt);
      float mrun = -CUDART_INF_F;
      float l4[4] = {0.f, 0.f, 0.f, 0.f}, a4[4] = {0.f, 0.f, 0.f, 0.f};
      bool ok = true;
      // keys' (bias * log2 e, carried score) of this half of block kb for thread gt < 64, masked
      // keys get -inf; loaded one block ahead so that the global round trip overlaps the block
      auto key_vals = [&](int kb, float& bias, float& m) {
        const int key = kb * kAT + kHalf * hf + gt;
        bias = -CUDART_INF_F;
        m = 0.f;
        if (gt < kHalf && key < p.S) {
          const size_t tk = static_cast<size_t>(w.b) * p.S + key;
          bias = p.key_bias ? __ldg(p.key_bias + tk) * 1.4426950408889634f : 0.f;
          m = kFloatM ? __ldg(p.m_prev + tk) : static_cast<float>(__ldg(p.is_vision + tk) != 0);
        }
      };
      float nb_bias, nb_m;
      key_vals(0, nb_bias, nb_m);
      for (int kb = 0; kb < nkb; ++kb, ++blk) {
        const int buf = blk & 1;
        const uint32_t use = static_cast<uint32_t>(blk >> 1);
        if (gt < kHalf) {
          mkg[buf * kAT + gt] = nb_bias;
          mkg[buf * kAT + kHalf + gt] = nb_m;
        }
        mbar_arrive(mkbar + buf);
        if (kb + 1 < nkb) key_vals(kb + 1, nb_bias, nb_m);
        if (!wait_bar(mkbar + buf, use & 1u, wc)) { ok = false; break; }
        if (!wait_bar(sfull + buf, use & 1u, wc)) { ok = false; break; }
        tc_fence_after();
        const uint32_t ta = tmem + (static_cast<uint32_t>(lg * 32) << 16) + static_cast<uint32_t>((2 * t + buf) * kAT);
        const float4* bias4 = reinterpret_cast<const float4*>(mkg + buf * kAT);
        const float4* m4 = reinterpret_cast<const float4*>(mkg + buf * kAT + kHalf);
        const bool diag = p.causal && kb == qt;
#pragma unroll 1
        for (int cc = 0; cc < kHalf / 32; ++cc) {
          const int c = 2 * hf + cc;            // 32-key chunk of the block
          float v[32];
          tmem_ld32(ta + 32u * c, v);
          float cm[4] = {-CUDART_INF_F, -CUDART_INF_F, -CUDART_INF_F, -CUDART_INF_F};
#pragma unroll
          for (int i4 = 0; i4 < 8; ++i4) {
            const float4 bb = bias4[cc * 8 + i4];
            const float bv[4] = {bb.x, bb.y, bb.z, bb.w};
            const int i = 4 * i4;
            fma2(v[i], v[i + 1], v[i], v[i + 1], p.scale_log2, p.scale_log2, bv[0], bv[1]);
            fma2(v[i + 2], v[i + 3], v[i + 2], v[i + 3], p.scale_log2, p.scale_log2, bv[2], bv[3]);
          }
          if (diag) {                           // causal mask inside the diagonal block only
#pragma unroll
            for (int i = 0; i < 32; ++i)
              if (c * 32 + i > row) v[i] = -CUDART_INF_F;
          }
#pragma unroll
          for (int i = 0; i < 32; ++i) cm[i & 3] = fmaxf(cm[i & 3], v[i]);
          const float mnew = fmaxf(mrun, fmaxf(fmaxf(cm[0], cm[1]), fmaxf(cm[2], cm[3])));
          if (mnew != -CUDART_INF_F) {
            if (mnew != mrun) {                 // rescale the running sums to the new maximum
              const float corr = ex2(mrun - mnew);
#pragma unroll
              for (int u = 0; u < 4; ++u) {
                l4[u] *= corr;
                a4[u] *= corr;
              }
              mrun = mnew;
            }
#pragma unroll
            for (int i4 = 0; i4 < 8; ++i4) {
              const float4 mm = m4[cc * 8 + i4];
              const float mv[4] = {mm.x, mm.y, mm.z, mm.w};
              const int i = 4 * i4;
              float t0, t1, t2, t3;
              add2(t0, t1, v[i], v[i + 1], -mnew, -mnew);
              add2(t2, t3, v[i + 2], v[i + 3], -mnew, -mnew);
              const float e0 = ex2(t0), e1 = ex2(t1), e2 = ex2(t2), e3 = ex2(t3);
              add2(l4[0], l4[1], l4[0], l4[1], e0, e1);
              add2(l4[2], l4[3], l4[2], l4[3], e2, e3);
              fma2(a4[0], a4[1], e0, e1, mv[0], mv[1], a4[0], a4[1]);
              fma2(a4[2], a4[3], e2, e3, mv[2], mv[3], a4[2], a4[3]);
            }
          }
        }
        tc_fence_before();
        mbar_arrive(sempty + buf);
      }
      if (!ok) break;
      float l = (l4[0] + l4[1]) + (l4[2] + l4[3]);
      float a = (a4[0] + a4[1]) + (a4[2] + a4[3]);
      const uint32_t nt = static_cast<uint32_t>(ng++);   // this item's phase of the group's barriers
      // the second half hands its state to the first, which merges it (maxima in log2 units).
      // Two merge buffers alternate by item; the second half may run ahead of the first by up
      // to two S buffers of keys, which can span whole short items, so it refills a buffer only
      // once the first half has read the buffer's previous state (full / free pair per buffer).
      const uint32_t mbuf = nt & 1u, muse = nt >> 1;
      float* mb = mrt + mbuf * 3 * kAT;
      uint64_t* mfull = mrg_full + 2 * t + mbuf;
      uint64_t* mfree = mrg_free + 2 * t + mbuf;
      if (hf == 1) {
        if (!wait_bar(mfree, (muse & 1u) ^ 1u, wc)) break;
        mb[row] = mrun;
        mb[kAT + row] = l;
        mb[2 * kAT + row] = a;
        mbar_arrive(mfull);
        continue;
      }
      if (!wait_bar(mfull, muse & 1u, wc)) break;
      {
        const float m1 = mb[row], l1 = mb[kAT + row], a1 = mb[2 * kAT + row];
        mbar_arrive(mfree);
        const float mm = fmaxf(mrun, m1);
        if (mm == -CUDART_INF_F) {
          l = 0.f;
          a = 0.f;
        } else {
          const float c0 = ex2(mrun - mm), c1 = ex2(m1 - mm);
          l = l * c0 + l1 * c1;
          a = a * c0 + a1 * c1;
        }
      }
      // head result, then the head average of the tile by the last head to finish
      const bool valid = q < p.S;
      const size_t tok = static_cast<size_t>(w.b) * p.S + q;
      if (valid) p.part[static_cast<size_t>(w.h) * p.T + tok] = a / l;
      __threadfence();
      mbar_arrive(out_bar + t);
      if (gt == 0) {
        uint32_t last = 0u;
        if (wait_bar(out_bar + t, nt & 1u, wc)) {
          const uint32_t n = atomicAdd(p.ticket + w.b * p.n_qtiles + qt, 1u) + 1u;
          last = (n == static_cast<uint32_t>(p.H)) ? 1u : 0u;
          if (last) p.ticket[w.b * p.n_qtiles + qt] = 0u;     // ready for the next call
        }
        decision[t] = last;
        mbar_arrive(dec_bar + t);
      }
      if (!wait_bar(dec_bar + t, nt & 1u, wc)) break;
      if (decision[t] && valid) {
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

  // the role branches leave single lanes running on their own: the warp reconverges before
  // the block barrier, so that no thread passes it while another of its warp is still working
  __syncwarp();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem, 512);
}

}  // namespace

cudaError_t launch_attn_mass(const AttnParams& p, const CUtensorMap& tmQ, const CUtensorMap& tmK,
                             int n_sms, cudaStream_t s) {
  if (p.hd != kHd) return cudaErrorNotSupported;
  const int n_ks = 4;
  const uint32_t smem = attn_layout(n_ks).total;
  if (smem > 227u * 1024u) return cudaErrorInvalidConfiguration;
  const int n_items = ((p.n_qtiles + 1) / 2) * p.B * p.H;
  const int grid = n_items < n_sms ? n_items : n_sms;
  auto k = p.m_prev ? k_attn_mass<true> : k_attn_mass<false>;
  cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  return launch_pdl(k, dim3(grid), dim3(kAttnThreads), smem, s, tmQ, tmK, p, n_ks);
}

}  // namespace smoes
