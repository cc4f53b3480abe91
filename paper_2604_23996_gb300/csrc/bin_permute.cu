// bin_permute.cu -- de-duplicated bin dispatch (Sec. 4.5, "DeDup").
//
// Every token is sent once to each bin that holds at least one of its top-k experts; the
// entry carries a bit mask of the chosen experts' slots inside the bin. Entries are grouped by
// bin (ascending) and ordered by token inside a bin. Three launches, all integer work:
//   count   per-block pair counts per bin (warp ballots), zeroes the atomic outputs;
//   scan    block offsets per bin and the bin offsets (one block, warp-shuffle scans);
//   scatter stable positions from ballots + block offsets, writes tokens and masks, and adds the
//           dispatch matrix and per-modality expert counts (integer atomics: order-independent).
#include <mutex>

#include "device_common.cuh"
#include "smoes_internal.cuh"

namespace smoes {
namespace {

constexpr int kPermThreads = 256;                    // one token per thread and round

struct TokenSel {
  int e[kMaxTopK];
  int b[kMaxTopK];
  uint32_t bins;
};

__device__ __forceinline__ void load_sel(const PermParams& p, int j, TokenSel& s) {
  s.bins = 0u;
#pragma unroll
  for (int i = 0; i < kMaxTopK; ++i) {
    s.e[i] = -1;
    s.b[i] = -1;
    if (i < p.k) {
      const int e = p.topk_idx[static_cast<size_t>(j) * p.k + i];
      if (e >= 0 && e < p.E) {
        s.e[i] = e;
        s.b[i] = p.expert_bin[e];
        s.bins |= 1u << s.b[i];
      } else {
        atomicOr(p.status, kStatusData);
      }
    }
  }
}

__global__ void __launch_bounds__(kPermThreads) k_perm_count(const PermParams p) {
  __shared__ int wc[kPermThreads / 32][kMaxBins];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  int cnt = 0;                                          // lane kb of each warp counts bin kb
  for (int r = 0; r < p.rounds; ++r) {
    const int j = (blockIdx.x * p.rounds + r) * kPermThreads + threadIdx.x;
    TokenSel s;
    s.bins = 0u;
    if (j < p.T) load_sel(p, j, s);
    for (int kb = 0; kb < p.K; ++kb) {
      const int c = __popc(__ballot_sync(0xffffffffu, (s.bins >> kb) & 1u));
      if (lane == kb) cnt += c;
    }
  }
  if (lane < kMaxBins) wc[warp][lane] = cnt;
  __syncthreads();
  if (threadIdx.x < p.K) {
    int t = 0;
    for (int w = 0; w < kPermThreads / 32; ++w) t += wc[w][threadIdx.x];
    p.blk_counts[blockIdx.x * p.K + threadIdx.x] = t;
  }
  if (blockIdx.x == 0) {
    for (int i = threadIdx.x; i < p.K * p.K; i += kPermThreads) p.dispatch[i] = 0;
    if (p.expert_counts)
      for (int i = threadIdx.x; i < 2 * p.E; i += kPermThreads) p.expert_counts[i] = 0;
  }
}

// One block of 1024 threads; thread b owns block b (n_blocks <= 1024). For every bin, an
// exclusive scan over blocks gives the block's first position inside the bin; the bin offsets
// are the exclusive scan of the bin totals.
__global__ void __launch_bounds__(1024) k_perm_scan(const PermParams p) {
  __shared__ int wsum[32][kMaxBins];
  __shared__ int tot[kMaxBins + 1];
  const int b = threadIdx.x, warp = b >> 5, lane = b & 31;
  const bool own = b < p.n_blocks;
  for (int kb = 0; kb < p.K; ++kb) {
    const int v = own ? p.blk_counts[b * p.K + kb] : 0;
    int x = v;                                          // inclusive warp scan
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, x, o);
      if (lane >= o) x += y;
    }
    if (lane == 31) wsum[warp][kb] = x;
    if (own) p.blk_offsets[b * p.K + kb] = x - v;       // exclusive within the warp (for now)
  }
  __syncthreads();
  if (b < p.K) {                                        // scan warp totals for bin b
    int run = 0;
    for (int w = 0; w < 32; ++w) {
      const int t = wsum[w][b];
      wsum[w][b] = run;
      run += t;
    }
    tot[b] = run;
  }
  __syncthreads();
  if (b == 0) {
    int run = 0;
    for (int kb = 0; kb < p.K; ++kb) {
      const int t = tot[kb];
      tot[kb] = run;
      p.bin_offsets[kb] = run;
      run += t;
    }
    p.bin_offsets[p.K] = run;
  }
  __syncthreads();
  if (own)
    for (int kb = 0; kb < p.K; ++kb) p.blk_offsets[b * p.K + kb] += wsum[warp][kb] + tot[kb];
}

__global__ void __launch_bounds__(kPermThreads) k_perm_scatter(const PermParams p) {
  __shared__ int wcnt[kPermThreads / 32][kMaxBins];
  __shared__ int base[kMaxBins];
  __shared__ int disp[kMaxBins * kMaxBins];
  __shared__ int ecnt[2 * kMaxExperts];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int i = threadIdx.x; i < p.K * p.K; i += kPermThreads) disp[i] = 0;
  for (int i = threadIdx.x; i < 2 * p.E; i += kPermThreads) ecnt[i] = 0;
  if (threadIdx.x < p.K) base[threadIdx.x] = p.blk_offsets[blockIdx.x * p.K + threadIdx.x];
  __syncthreads();
  const unsigned lt_mask = (1u << lane) - 1u;
  for (int r = 0; r < p.rounds; ++r) {
    const int j = (blockIdx.x * p.rounds + r) * kPermThreads + threadIdx.x;
    const bool valid = j < p.T;
    TokenSel s;
    s.bins = 0u;
    if (valid) load_sel(p, j, s);
    int home = 0;
    if (valid) {
      home = p.home ? p.home[j] : static_cast<int>((static_cast<long long>(j) * p.K) / p.T);
      if (home < 0 || home >= p.K) {
        atomicOr(p.status, kStatusData);
        home = -1;
      }
    }
    // ballots: per bin, rank inside the warp and the warp's count
    for (int kb = 0; kb < p.K; ++kb) {
      const unsigned bal = __ballot_sync(0xffffffffu, (s.bins >> kb) & 1u);
      if (lane == 0) wcnt[warp][kb] = __popc(bal);
    }
    __syncthreads();
    if (threadIdx.x < p.K) {                            // exclusive scan over warps, per bin
      int run = base[threadIdx.x];
      for (int w = 0; w < kPermThreads / 32; ++w) {
        const int t = wcnt[w][threadIdx.x];
        wcnt[w][threadIdx.x] = run;
        run += t;
      }
      base[threadIdx.x] = run;                          // carried into the next round
    }
    __syncthreads();
    for (int kb = 0; kb < p.K; ++kb) {
      const unsigned bal = __ballot_sync(0xffffffffu, (s.bins >> kb) & 1u);
      if ((s.bins >> kb) & 1u) {
        const int pos = wcnt[warp][kb] + __popc(bal & lt_mask);
        uint32_t mask = 0u;
#pragma unroll
        for (int i = 0; i < kMaxTopK; ++i)
          if (i < p.k && s.b[i] == kb) mask |= 1u << p.expert_slot[s.e[i]];
        p.perm_token[pos] = j;
        p.perm_mask[pos] = mask;
        if (home >= 0) atomicAdd(&disp[home * p.K + kb], 1);
      }
    }
    if (valid && p.expert_counts) {
      const int m = p.is_vision[j] ? 0 : 1;
#pragma unroll
      for (int i = 0; i < kMaxTopK; ++i)
        if (i < p.k && s.e[i] >= 0) atomicAdd(&ecnt[m * p.E + s.e[i]], 1);
    }
    __syncthreads();                                    // wcnt reused by the next round
  }
  for (int i = threadIdx.x; i < p.K * p.K; i += kPermThreads)
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

// Rounds of 256 tokens per block: 1 while that keeps the block count <= 1024 (the scan runs in
// one block of 1024 threads), more for larger batches.
int perm_rounds(int T) {
  const int units = (T + kPermThreads - 1) / kPermThreads;
  return units <= 1024 ? 1 : (units + 1023) / 1024;
}
int perm_blocks(int T) {
  const int per = kPermThreads * perm_rounds(T);
  return (T + per - 1) / per;
}

cudaError_t launch_bin_permute(const PermParams& p, cudaStream_t s) {
  if (p.n_blocks > 1024) return cudaErrorInvalidValue;
  k_perm_count<<<p.n_blocks, kPermThreads, 0, s>>>(p);
  k_perm_scan<<<1, 1024, 0, s>>>(p);
  k_perm_scatter<<<p.n_blocks, kPermThreads, 0, s>>>(p);
  return cudaGetLastError();
}

}  // namespace smoes
