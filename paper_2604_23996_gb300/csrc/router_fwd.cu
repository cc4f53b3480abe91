// router_fwd.cu -- SMoES router forward on sm_103a.
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
//
// The tensor-core kernel and the epilogue it shares with the fp32 kernel are in router_fwd_tc.cuh;
// this file holds the fp32 kernel and the launchers (router_fwd_var.cu instantiates the
// tensor-core kernel with the router variants).
#include "router_fwd_tc.cuh"

namespace smoes {
namespace {

// ------------------------------------------------------------------ FFMA forward (fp32)
// The fp32 layers of the workloads are small (d ~ 512, E <= 64): one 128-token tile per CTA
// would leave most SMs idle, so the hidden dimension is split as well. CTA (tile, chunk) stages
// its 128 x 128 block of X and the matching [E, 128] block of W in shared memory (16-byte
// asynchronous copies, all in flight at once), evaluates the chunk's Gaussian coefficients
// (eqs. 8-9) and forms the partial logits and the partial log-likelihood difference of the
// tile's rows over its 128 features. The last CTA of the tile to finish (a ticket) adds the
// chunks' partials in chunk order (bitwise reproducible) and runs the same two-group epilogue as
// the tensor-core path (logits read from shared memory).
constexpr int kF32MaxE = 64;
constexpr int kF32Cols = 128;                 // features per CTA
constexpr int kF32XStride = kF32Cols + 4;     // row stride of the staged X block (floats)

__host__ __device__ inline size_t f32_smem_floats(const Dims& dm) {
  const int E16 = round_up(dm.E, 16);
  const size_t xs = static_cast<size_t>(kF32Cols) * kF32XStride;
  const size_t zs = 128 * static_cast<size_t>(E16 + 1);
  return (xs > zs ? xs : zs) + static_cast<size_t>(round_up(dm.E, 16)) * kF32Cols + 3 * kF32Cols + 8 +
         epi_smem_floats(dm.K) + 3 * 128 + 8;
}

__device__ __forceinline__ void cp_async16(void* dst, const void* src, bool in) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;"
               ::"r"(smem_u32(dst)), "l"(src), "r"(in ? 16 : 0) : "memory");
}

// EB = E rounded up to 16 (16, 32, 48 or 64): the expert loops are unrolled to EB with the padding
// experts' W rows zero, so no expert is predicated off.
template <bool kGauss, int KM, int EB>
__global__ void __launch_bounds__(256)
k_router_fwd_f32(const FwdParams p) {
  extern __shared__ float fs[];
  const Dims& dm = p.dm;
  const int E = dm.E, d = dm.d;
  const int E16 = round_up(E, 16);
  const int nck = p.f32_chunks;
  const int tile = blockIdx.x / nck, ck = blockIdx.x % nck;
  const int j0 = tile * kTileRows, c0 = ck * kF32Cols;
  float* xs = fs;                                        // [128][kF32XStride]; later zs [128][E16 + 1]
  float* zs = fs;
  const size_t big = static_cast<size_t>(kF32Cols) * kF32XStride > 128 * static_cast<size_t>(E16 + 1)
                         ? static_cast<size_t>(kF32Cols) * kF32XStride : 128 * static_cast<size_t>(E16 + 1);
  float* wsm = fs + big;                                 // [EB][128], rows past E zero
  float* ga = wsm + EB * kF32Cols;                       // [128]
  float* gb = ga + kF32Cols;                             // [128]
  float* hsum = gb + kF32Cols;                           // [128] second half's Gaussian sums
  float* gcw = hsum + kF32Cols;                          // [8] per-warp constant terms
  float* epi = gcw + 8;
  float* dll_s = epi + epi_smem_floats(dm.K);            // [128]
  int* flag_s = reinterpret_cast<int*>(dll_s + 128);
  uint64_t* bars = reinterpret_cast<uint64_t*>(
      (reinterpret_cast<uintptr_t>(dll_s + 3 * 128) + 7) & ~uintptr_t(7));   // [kEpiBars]
  int* abort_flag = reinterpret_cast<int*>(bars + kEpiBars);

  const int t = threadIdx.x, r = t & 127, h = t >> 7;
  pdl_wait();
  pdl_trigger();
  if (blockIdx.x == 0 && t == 0) *p.ws.bal_flag = 0u;             // a new forward: no balance term yet
  const float* X = static_cast<const float*>(p.X);
  const float* W = static_cast<const float*>(p.W);
  // the tile's 128 x 128 block of X and the [E, 128] block of W, zero past T and d
  for (int i = t; i < 128 * (kF32Cols / 4); i += 256) {
    const int rr = i >> 5, q = (i & 31) * 4;
    const bool in = j0 + rr < dm.T && c0 + q < d;
    cp_async16(xs + rr * kF32XStride + q, in ? X + static_cast<size_t>(j0 + rr) * d + c0 + q : X, in);
  }
  for (int i = t; i < EB * (kF32Cols / 4); i += 256) {
    const int e = i >> 5, q = (i & 31) * 4;
    const bool in = e < E && c0 + q < d;
    cp_async16(wsm + e * kF32Cols + q, in ? W + static_cast<size_t>(e) * d + c0 + q : W, in);
  }
  asm volatile("cp.async.commit_group;" ::: "memory");
  if (t == 0) {
    *abort_flag = 0;
    init_epi_bars(bars);
    fence_mbar_init();
  }
  if (kGauss && t < kF32Cols) {                          // this chunk's coefficients (eqs. 8-9)
    const int c = c0 + t;
    float a = 0.f, b = 0.f, cc = 0.f;
    if (c < d && !gauss_coef_feature(p.mu[c], p.mu[d + c], p.var[c], p.var[d + c], a, b, cc))
      atomicOr(p.ws.status, kStatusData);
    ga[t] = a;
    gb[t] = b;
    cc = warp_sum(cc);
    if ((t & 31) == 0) gcw[t >> 5] = cc;
  }
  asm volatile("cp.async.wait_all;" ::: "memory");
  __syncthreads();

  // partial logits of row r, experts e = 2i + h, over the chunk's features
  float acc[EB / 2];
#pragma unroll
  for (int i = 0; i < EB / 2; ++i) acc[i] = 0.f;
  float gs = 0.f;
  const float* xr = xs + r * kF32XStride;
#pragma unroll 1
  for (int q = 0; q < kF32Cols; q += 4) {
    const float4 x = *reinterpret_cast<const float4*>(xr + q);
#pragma unroll
    for (int i = 0; i < EB / 2; ++i) {
      const float4 w = *reinterpret_cast<const float4*>(wsm + (2 * i + h) * kF32Cols + q);
      acc[i] = fmaf(x.x, w.x, fmaf(x.y, w.y, fmaf(x.z, w.z, fmaf(x.w, w.w, acc[i]))));
    }
    if (kGauss && (q >> 6) == h) {                        // half h of the features: sum x (ga x + gb)
      const float4 a = *reinterpret_cast<const float4*>(ga + q);
      const float4 b = *reinterpret_cast<const float4*>(gb + q);
      gs = fmaf(x.x, fmaf(a.x, x.x, b.x), gs);
      gs = fmaf(x.y, fmaf(a.y, x.y, b.y), gs);
      gs = fmaf(x.z, fmaf(a.z, x.z, b.z), gs);
      gs = fmaf(x.w, fmaf(a.w, x.w, b.w), gs);
    }
  }
  float* pz = p.f32_part + static_cast<size_t>(tile * nck + ck) * (E + 1) * 128;
#pragma unroll
  for (int i = 0; i < EB / 2; ++i) {
    const int e = 2 * i + h;
    if (e < E) pz[e * 128 + r] = acc[i];
  }
  if (kGauss) {
    if (h == 1) hsum[r] = gs;
    __syncthreads();
    if (h == 0) {
      const float gc = ((gcw[0] + gcw[1]) + (gcw[2] + gcw[3]));
      pz[E * 128 + r] = (gs + hsum[r]) - 0.5f * gc;
    }
  }
  // the last CTA of the tile sums the chunks in order and runs the epilogue
  __threadfence();
  __syncthreads();
  if (t == 0) *flag_s = atomicAdd(p.tile_ticket + tile, 1u) == static_cast<uint32_t>(nck - 1);
  __syncthreads();
  if (!*flag_s) return;
  __threadfence();
  if (t == 0) p.tile_ticket[tile] = 0u;                  // ready for the next call
  const float* pt = p.f32_part + static_cast<size_t>(tile * nck) * (E + 1) * 128;
  // thread (r, h) sums values e = 2i + h (the logits, then the log-likelihood difference at e = E)
  // over the chunks in chunk order; the loads of CB chunks of every e are issued together
  {
    constexpr int NI = EB / 2 + 1;
    constexpr int CB = EB <= 16 ? 4 : EB <= 32 ? 2 : 1;
    float zz[NI];
#pragma unroll
    for (int i = 0; i < NI; ++i) zz[i] = 0.f;
#pragma unroll 1
    for (int c0 = 0; c0 < nck; c0 += CB) {
      float t[NI][CB];
#pragma unroll
      for (int i = 0; i < NI; ++i) {
        const int e = 2 * i + h;
        const bool on = e < E || (kGauss && e == E);
#pragma unroll
        for (int u = 0; u < CB; ++u)
          t[i][u] = (on && c0 + u < nck)
                        ? __ldcg(pt + static_cast<size_t>(c0 + u) * (E + 1) * 128 + e * 128 + r) : 0.f;
      }
#pragma unroll
      for (int i = 0; i < NI; ++i) {
#pragma unroll
        for (int u = 0; u < CB; ++u)
          if (c0 + u < nck) zz[i] += t[i][u];
      }
    }
#pragma unroll
    for (int i = 0; i < NI; ++i) {
      const int e = 2 * i + h;
      if (e < E16) zs[r * (E16 + 1) + e] = zz[i];       // padding experts: logit 0, masked below
      if (kGauss && e == E) dll_s[r] = zz[i];
    }
  }
  __syncthreads();
  {
    const int grp = h, row = r;
    struct Src {
      const float* z;
      int E;
      __device__ void load16(int c, float (&v)[16]) const {
#pragma unroll
        for (int i = 0; i < 16; ++i) v[i] = (16 * c + i < E) ? z[16 * c + i] : -FLT_MAX;
      }
    } src{zs + row * (E16 + 1), E};
    struct Rel {
      __device__ void operator()() const {}
    } rel;
    WaitCtx wc{abort_flag, p.ws.status, p.limit_ns};
    const EpiSmem es = epi_smem(epi, dm.K, bars);
    uint32_t n_in = 0;
    const TileMeta meta = load_tile_meta(p, tile, row);   // (no fused permutation on this path)
    epilogue_tile<KM, true>(p, src, rel, tile, grp, row, 0, kGauss ? dll_s[row] : 0.f, meta, es, wc, n_in, true);
  }
}

}  // namespace

// Plans without router variants run kernels compiled without their code (the epilogue of a
// kernel that streams one or two tiles per SM is bound by instruction fetch and latency, and
// the variant branches lengthen it); plans with a variant run those of router_fwd_var.cu.
cudaError_t launch_router_fwd_bf16(const FwdParams& p, const CUtensorMap& tmX,
                                   const CUtensorMap& tmW, const CUtensorMap* tmG, int n_sms,
                                   cudaStream_t s) {
  if (p.dm.gate || p.dm.mask) return launch_router_fwd_bf16_var(p, tmX, tmW, tmG, n_sms, s);
  return launch_fwd_tc<false>(p, tmX, tmW, tmG, n_sms, s);
}

cudaError_t launch_router_fwd_f32(const FwdParams& p, cudaStream_t s) {
  if (p.dm.E > kF32MaxE) return cudaErrorInvalidValue;
  const size_t smem = sizeof(float) * f32_smem_floats(p.dm) + sizeof(uint64_t) * kEpiBars + 64;
  if (smem > 227u * 1024u) return cudaErrorInvalidConfiguration;
  const bool gauss = p.M_in == nullptr;
  const int eb = round_up(p.dm.E, 16);
  return dispatch_km(p.dm.k, [&](auto km) -> cudaError_t {
    constexpr int KM = decltype(km)::value;
    auto pick = [&](auto ebc) {
      constexpr int EB = decltype(ebc)::value;
      return gauss ? k_router_fwd_f32<true, KM, EB> : k_router_fwd_f32<false, KM, EB>;
    };
    auto k = eb <= 16 ? pick(std::integral_constant<int, 16>())
           : eb <= 32 ? pick(std::integral_constant<int, 32>())
           : eb <= 48 ? pick(std::integral_constant<int, 48>())
                      : pick(std::integral_constant<int, 64>());
    cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    return launch_pdl(k, dim3(p.n_tiles * p.f32_chunks), dim3(256), smem, s, p);
  });
}

int f32_chunks(int d) { return (d + kF32Cols - 1) / kF32Cols; }

}  // namespace smoes
