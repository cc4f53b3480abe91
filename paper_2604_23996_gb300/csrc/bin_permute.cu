// bin_permute.cu -- de-duplicated bin dispatch (Sec. 4.5, "DeDup").
//
// Every token is sent once to each bin that holds at least one of its top-k experts; the
// entry carries a bit mask of the chosen experts' slots inside the bin. Entries are grouped by
// bin (ascending) and ordered by token inside a bin. One cooperative launch, all integer work:
//   count    per-block pair counts per bin (warp ballots);
//   barrier  a bounded grid barrier (all blocks are resident: cooperative launch);
//   offsets  each block sums the count table: its prefix inside every bin and the bin bases;
//   scatter  stable positions from ballots, tokens and masks written, and the dispatch matrix
//            and per-modality expert counts added (integer atomics: order-independent).
#include <algorithm>
#include <mutex>

#include "device_common.cuh"
#include "ptx.cuh"
#include "smoes_internal.cuh"

namespace smoes {
namespace {

constexpr int kPermThreads = 256;                    // one token per thread and round
constexpr int kPermWarps = kPermThreads / 32;

// One token's selection: its chosen experts (-1 for none) with their bins and slot bits, the
// set of the bins and the token's modality (0 vision, 1 text). KM >= k, a compile-time bound
// that keeps the arrays in registers.
template <int KM>
struct TokenSel {
  int e[KM];
  int b[KM];
  uint32_t sbit[KM];
  uint32_t bins;
  int m;
};

template <int KM>
__device__ __forceinline__ void load_sel(const PermParams& p, const int* s_bin, const int* s_slot,
                                         int j, TokenSel<KM>& s) {
  s.bins = 0u;
  int e[KM];
#pragma unroll
  for (int i = 0; i < KM; ++i) e[i] = i < p.k ? p.topk_idx[static_cast<size_t>(j) * p.k + i] : -1;
  s.m = (p.is_vision && !p.is_vision[j]) ? 1 : 0;
#pragma unroll
  for (int i = 0; i < KM; ++i) {
    s.e[i] = -1;
    s.b[i] = -1;
    s.sbit[i] = 0u;
    if (i < p.k) {
      if (e[i] >= 0 && e[i] < p.E) {
        s.e[i] = e[i];
        s.b[i] = s_bin[e[i]];
        s.sbit[i] = 1u << s_slot[e[i]];
        s.bins |= 1u << s.b[i];
      } else {
        atomicOr(p.status, kStatusData);
      }
    }
  }
}

template <int KM>
__global__ void __launch_bounds__(kPermThreads) k_perm(const PermParams p) {
  __shared__ int s_bin[kMaxExperts];
  __shared__ int s_slot[kMaxExperts];
  __shared__ int wcnt[kPermWarps][kMaxBins];
  __shared__ int base[kMaxBins];
  __shared__ int pre_s[kMaxBins], tot_s[kMaxBins];
  __shared__ int disp[kMaxBins * kMaxBins];
  __shared__ int ecnt[2 * kMaxExperts];
  __shared__ int ok_s;
  // a cooperative grid launched with programmatic serialization: the top-k of the kernel before
  // it are read only after that kernel has completed
  pdl_wait();
  pdl_trigger();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int K = p.K;
  for (int e = threadIdx.x; e < p.E; e += kPermThreads) {
    s_bin[e] = p.expert_bin[e];
    s_slot[e] = p.expert_slot[e];
  }
  for (int i = threadIdx.x; i < K * K; i += kPermThreads) disp[i] = 0;
  for (int i = threadIdx.x; i < 2 * p.E; i += kPermThreads) ecnt[i] = 0;
  __syncthreads();

  // count: lane kb of each warp accumulates the warp's pairs in bin kb; the first round's
  // selections stay in registers for the scatter
  int cnt = 0;
  TokenSel<KM> s0;
  s0.bins = 0u;
  s0.m = 0;
  for (int r = 0; r < p.rounds; ++r) {
    const int j = (blockIdx.x * p.rounds + r) * kPermThreads + threadIdx.x;
    TokenSel<KM> s;
    s.bins = 0u;
    s.m = 0;
    if (j < p.T) load_sel<KM>(p, s_bin, s_slot, j, s);
    if (r == 0) s0 = s;
    for (int kb = 0; kb < K; ++kb) {
      const int c = __popc(__ballot_sync(0xffffffffu, (s.bins >> kb) & 1u));
      if (lane == kb) cnt += c;
    }
  }
  if (lane < kMaxBins) wcnt[warp][lane] = cnt;
  __syncthreads();
  if (threadIdx.x < K) {
    int t = 0;
    for (int w = 0; w < kPermWarps; ++w) t += wcnt[w][threadIdx.x];
    p.blk_counts[threadIdx.x * p.n_blocks + blockIdx.x] = t;     // bin-major
  }
  if (blockIdx.x == 0) {
    for (int i = threadIdx.x; i < K * K; i += kPermThreads) p.dispatch[i] = 0;
    if (p.expert_counts)
      for (int i = threadIdx.x; i < 2 * p.E; i += kPermThreads) p.expert_counts[i] = 0;
  }
  __syncthreads();
  if (threadIdx.x == 0) ok_s = grid_barrier(p.sync, gridDim.x, p.limit_ns, p.status) ? 1 : 0;
  __syncthreads();
  if (!ok_s) return;

  // offsets: warp w sums bins w, w + 8, ... over all blocks (lanes stride the blocks, eight
  // loads in flight per lane and round)
  for (int kb = warp; kb < K; kb += kPermWarps) {
    int pre = 0, tot = 0;
    const int* row = p.blk_counts + kb * p.n_blocks;
    for (int b0 = lane; b0 < p.n_blocks; b0 += 8 * 32) {
      int c[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) c[u] = b0 + 32 * u < p.n_blocks ? __ldcg(row + b0 + 32 * u) : 0;
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        tot += c[u];
        if (b0 + 32 * u < static_cast<int>(blockIdx.x)) pre += c[u];
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      pre += __shfl_xor_sync(0xffffffffu, pre, o);
      tot += __shfl_xor_sync(0xffffffffu, tot, o);
    }
    if (lane == 0) {
      pre_s[kb] = pre;
      tot_s[kb] = tot;
    }
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    int run = 0;
    for (int kb = 0; kb < K; ++kb) {
      base[kb] = run + pre_s[kb];
      if (blockIdx.x == 0) p.bin_offsets[kb] = run;
      run += tot_s[kb];
    }
    if (blockIdx.x == 0) p.bin_offsets[K] = run;
  }
  __syncthreads();

  // scatter: per round, warp counts per bin -> exclusive scan over warps -> ballot ranks
  const unsigned lt_mask = (1u << lane) - 1u;
  for (int r = 0; r < p.rounds; ++r) {
    const int j = (blockIdx.x * p.rounds + r) * kPermThreads + threadIdx.x;
    const bool valid = j < p.T;
    TokenSel<KM> s;
    s.bins = 0u;
    s.m = 0;
    if (r == 0) {
      s = s0;
    } else if (valid) {
      load_sel<KM>(p, s_bin, s_slot, j, s);
    }
    int home = 0;
    if (valid) {
      home = p.home ? p.home[j] : static_cast<int>((static_cast<long long>(j) * K) / p.T);
      if (home < 0 || home >= K) {
        atomicOr(p.status, kStatusData);
        home = -1;
      }
    }
    for (int kb = 0; kb < K; ++kb) {
      const unsigned bal = __ballot_sync(0xffffffffu, (s.bins >> kb) & 1u);
      if (lane == 0) wcnt[warp][kb] = __popc(bal);
    }
    __syncthreads();
    if (threadIdx.x < K) {                              // exclusive scan over warps, per bin
      int run = base[threadIdx.x];
      for (int w = 0; w < kPermWarps; ++w) {
        const int t = wcnt[w][threadIdx.x];
        wcnt[w][threadIdx.x] = run;
        run += t;
      }
      base[threadIdx.x] = run;                          // carried into the next round
    }
    __syncthreads();
    // lanes with the same dispatch home add their pairs with one atomic per (warp, bin, home)
    const unsigned same_home = __match_any_sync(0xffffffffu, home);
    for (int kb = 0; kb < K; ++kb) {
      const unsigned bal = __ballot_sync(0xffffffffu, (s.bins >> kb) & 1u);
      if ((s.bins >> kb) & 1u) {
        const int pos = wcnt[warp][kb] + __popc(bal & lt_mask);
        uint32_t mask = 0u;
#pragma unroll
        for (int i = 0; i < KM; ++i) mask |= (s.b[i] == kb) ? s.sbit[i] : 0u;
        p.perm_token[pos] = j;
        p.perm_mask[pos] = mask;
        const unsigned grp = bal & same_home;
        if (home >= 0 && lane == __ffs(grp) - 1) atomicAdd(&disp[home * K + kb], __popc(grp));
      }
    }
    if (valid && p.expert_counts) {
#pragma unroll
      for (int i = 0; i < KM; ++i)
        if (s.e[i] >= 0) atomicAdd(&ecnt[s.m * p.E + s.e[i]], 1);
    }
    __syncthreads();                                    // wcnt reused by the next round
  }
  for (int i = threadIdx.x; i < K * K; i += kPermThreads)
    if (disp[i]) atomicAdd(p.dispatch + i, disp[i]);
  if (p.expert_counts)
    for (int i = threadIdx.x; i < 2 * p.E; i += kPermThreads)
      if (ecnt[i]) atomicAdd(p.expert_counts + i, ecnt[i]);
}
}  // namespace

// Scratch of the no-allocation permutation entry point (see smoes_bin_permute_noalloc): one copy
// per device that loads this library, alive until the process exits, shared by every call.
static __device__ __align__(256) unsigned char g_perm_static[sizeof(StaticPermScratch)];

// The host cannot use g_perm_static's name as a device address; it asks the runtime once per
// device, with that device current, and caches the answer.
cudaError_t static_perm_scratch(StaticPermScratch** out) {
  constexpr int kMaxDevices = 64;
  static std::mutex mu;
  static void* addr[kMaxDevices] = {};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(mu);
  if (addr[dev] == nullptr) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_perm_static);
    if (e != cudaSuccess) return e;
    addr[dev] = p;
  }
  *out = static_cast<StaticPermScratch*>(addr[dev]);
  return cudaSuccess;
}

// The plan's bin map and slots travel to the device as kernel parameters (2 KB, by value, so no
// host buffer is referenced once the launch returns); one block writes them into the fixed
// scratch and clears its status and grid-barrier words.
struct StaticPermMaps {
  int32_t expert_bin[kMaxExperts];
  int32_t expert_slot[kMaxExperts];
  int E;
};

__global__ void __launch_bounds__(kPermThreads) k_static_perm_prep(const StaticPermMaps m,
                                                                    StaticPermScratch* sp) {
  for (int e = threadIdx.x; e < m.E; e += kPermThreads) {
    sp->expert_bin[e] = m.expert_bin[e];
    sp->expert_slot[e] = m.expert_slot[e];
  }
  if (threadIdx.x < 4) {
    sp->status[threadIdx.x] = 0u;
    sp->sync[threadIdx.x] = 0u;
  }
}

cudaError_t launch_static_perm_prep(StaticPermScratch* sp, const int32_t* expert_bin,
                                    const int32_t* expert_slot, int E, cudaStream_t s) {
  if (E < 1 || E > kMaxExperts) return cudaErrorInvalidValue;
  StaticPermMaps m;
  for (int e = 0; e < kMaxExperts; ++e) {
    m.expert_bin[e] = e < E ? expert_bin[e] : 0;
    m.expert_slot[e] = e < E ? expert_slot[e] : 0;
  }
  m.E = E;
  k_static_perm_prep<<<1, kPermThreads, 0, s>>>(m, sp);
  return cudaGetLastError();
}

template <class F>
cudaError_t with_kernel(int k, F&& f) {
  if (k <= 2) return f(k_perm<2>);
  if (k <= 4) return f(k_perm<4>);
  if (k <= 6) return f(k_perm<6>);
  if (k <= 8) return f(k_perm<8>);
  return f(k_perm<16>);
}

// Blocks of the permutation: all must be resident at once (the grid barrier), and at most
// kStaticPermBlocks. Rounds of 256 tokens per block grow once the batch needs more blocks.
int perm_max_blocks(int k) {
  static std::mutex mu;
  static int cached[64][5] = {};
  const int v = k <= 2 ? 0 : k <= 4 ? 1 : k <= 6 ? 2 : k <= 8 ? 3 : 4;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 1;
  std::lock_guard<std::mutex> lock(mu);
  if (cached[dev][v] == 0) {
    int sms = 0, per_sm = 0;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 1;
    const cudaError_t e = with_kernel(k, [&](auto kern) {
      return cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kPermThreads, 0);
    });
    if (e != cudaSuccess) return 1;
    cached[dev][v] = std::max(1, std::min(kStaticPermBlocks, sms * per_sm));
  }
  return cached[dev][v];
}
int perm_rounds(int T, int k) {
  const int units = (T + kPermThreads - 1) / kPermThreads;
  const int cap = perm_max_blocks(k);
  return units <= cap ? 1 : (units + cap - 1) / cap;
}
int perm_blocks(int T, int k) {
  const int per = kPermThreads * perm_rounds(T, k);
  return (T + per - 1) / per;
}

cudaError_t launch_bin_permute(const PermParams& p, cudaStream_t s) {
  if (p.n_blocks > perm_max_blocks(p.k)) return cudaErrorInvalidValue;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(p.n_blocks);
  cfg.blockDim = dim3(kPermThreads);
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeCooperative;    // every block resident: the barrier is safe
  attr[0].val.cooperative = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return with_kernel(p.k, [&](auto kern) { return cudaLaunchKernelEx(&cfg, kern, p); });
}

}  // namespace smoes
