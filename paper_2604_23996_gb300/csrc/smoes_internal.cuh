// smoes_internal.cuh -- types shared by the host API (api.cu) and the kernels.
#pragma once

#include <cstddef>
#include <cstdint>
#include <cuda.h>
#include <cuda_runtime.h>

#include "smoes.h"

namespace smoes {

constexpr int kMaxTopK = 16;
constexpr int kMaxBins = 32;
constexpr int kMaxExperts = 256;           // bound of the permutation and metadata arrays
constexpr int kMaxExpertsBf16 = 128;       // experts a bf16 plan accepts
constexpr int kMaxExpertsF32 = 64;         // experts an fp32 plan accepts
constexpr int kPieceTokens = 128;          // tokens per partial-sum "piece" (one forward tile)
constexpr uint32_t kStatusData = 1u;       // status word bits
constexpr uint32_t kStatusTimeout = 2u;
constexpr uint64_t kWaitLimitNs = 2000000000ull;   // 2 s for any bounded device wait

// Values accumulated per piece (a warp's tokens of one sample), in this order:
//   Q[k] = sum p_jk, Rv[k] = sum dv_j p_jk, Rt[k] = sum dt_j p_jk, Nv[k] = sum Mv_j p_jk,
//   Nt[k] = sum Mt_j p_jk, then Dv = sum dv_j, Dt = sum dt_j, Av = sum Mv_j, At = sum Mt_j,
// where dm_j = M_jm - 1/2. The centred sums carry the modality/bin covariance without
// cancellation when M is close to 1/2 (the Gaussian score at tau = 0.5 d); the direct sums
// stay accurate when a modality's mass is small.
__host__ __device__ constexpr int piece_values(int K) { return 5 * K + 4; }
__host__ __device__ constexpr int piece_stride(int K) { return (piece_values(K) + 3) & ~3; }

// Device view of the caller-owned workspace (all pointers inside one allocation).
struct WsView {
  uint32_t* status;          // [4]: status bits, absent-modality count, spare, spare
  uint32_t* sample_ticket;   // [B] pieces completed per sample (self-resetting)
  uint32_t* loss_ticket;     // [1] samples completed (self-resetting)
  const int32_t* offsets;    // [B+1]
  const int32_t* token_sample;   // [T]
  const int32_t* expert_bin;     // [E]
  const int32_t* expert_slot;    // [E]
  const int32_t* piece_base;     // [n_groups+1] first piece of each 128-token tile
  const int32_t* sample_pieces;  // [B+1] pieces of sample i are [sp[i], sp[i+1])
  float* pieces;             // [n_pieces * piece_stride]
  float* mi32;               // [B] per-sample MI for the loss
  float* tabs;               // [B * 3 * K]: a_k, b_k, h_k per sample (backward coefficients)
  float* gsave;              // [T * E] exp(z_je - max_e z_je) saved by the forward
  float* ginv;               // [T] 1 / sum_e exp(z_je - max_e z_je): g_je = gsave * ginv
  float* dw_part;            // [G * E * d] per-token-group partial dW
  uint8_t* dz_img;           // [ceil(T/64)][hi|lo][E_pad/64][64 rows][128 B] dz in the MMA layout
  int32_t* perm_scratch;     // permutation block counts [n_blocks * K]
  uint32_t* attn_ticket;     // [B * ceil(S/128)] head tickets of the attention score
  float* attn_part;          // [H_max * T] per-head vision mass
  float* gcoef;              // Gaussian score coefficients: ga[dcoef], gb[dcoef], part[dcoef/256]
  int dcoef;                 // round_up(d, 256)
  // bin-level load balance (eq. 16): the backward adds its gradient while *bal_flag != 0 (set by
  // smoes_bin_balance, cleared by every forward); bal_f [E] = f_e, bal_a [K] = scale N_B / |U_k|
  uint32_t* bal_flag;
  float* bal_f;
  float* bal_a;
};

struct Dims {
  int T, d, E, k, K, B, N_B, renorm;
  int gate;                  // 0 softmax, 1 sigmoid (affinities s; g = s / sum s; renorm forced)
  int mask;                  // 1: the g of eq. (12) is restricted to the top-k and renormalised
  int pstride;               // piece_stride(K)
  int n_groups;              // ceil(T / 128): forward tiles = partial-sum groups
  int contig_bins;           // bin b holds experts [b N_B, (b+1) N_B) and N_B % 4 == 0
};

// The bin permutation of the forward's own top-k, done inside the forward launch (Sec. 4.5);
// perm_token == null: not requested.
struct FusedPerm {
  const int32_t* home;       // [T] or null (contiguous split)
  const uint8_t* is_vision;  // [T] (required with expert_counts)
  int32_t* bin_offsets;
  int32_t* perm_token;
  uint32_t* perm_mask;
  int32_t* dispatch;
  int32_t* expert_counts;
  int32_t* cta_counts;       // [K][G] pairs of each bin in each CTA's tiles (workspace)
  uint32_t* sync;            // [2] grid barrier words (workspace, zero between calls)
};

struct FwdParams {
  Dims dm;
  WsView ws;
  const void* X;
  const void* W;             // [E, d] (read directly by the fp32 path; bf16 goes through TMA)
  const float* M_in;         // provided scores, or null when the Gaussian score is fused
  const float* score_bias;   // [E] selection bias of the sigmoid gate, or null
  const float* mu;           // [2, d] (Gaussian mode)
  const float* var;          // [2, d]
  float inv_tau;
  float* M_out;
  int32_t* topk_idx;
  float* topk_w;
  float* bin_prob;
  float* joint;
  float* mi;
  float* loss;
  FusedPerm perm;
  int n_tiles;
  uint64_t limit_ns;
  // fp32 path: feature chunks per tile, per-(tile, chunk) partial logits and Gaussian sums
  // [n_tiles * f32_chunks][E + 1][128], per-tile tickets [n_tiles] (zero between calls)
  int f32_chunks;
  float* f32_part;
  uint32_t* tile_ticket;
};

struct BwdParams {
  Dims dm;
  WsView ws;
  const void* X;
  const void* W;
  const float* M;
  const int32_t* topk_idx;
  const float* d_topk_w;
  float scale;               // -loss_scale / B
  void* dX;
  float* dlogits;
  float* dW;
  int accumulate;
  int groups;                // G token groups (partial dW blocks)
  int slices;                // d-slices per token group (tcgen05 path)
  int slice_width;           // columns per d-slice
  int n_tiles;               // token tiles
  uint64_t limit_ns;
  int balance_armed;         // host's view: smoes_bin_balance was called since the last forward
};

struct PermParams {
  int T, k, E, K;
  const int32_t* topk_idx;
  const int32_t* home;
  const uint8_t* is_vision;
  const int32_t* expert_bin;
  const int32_t* expert_slot;
  int32_t* bin_offsets;
  int32_t* perm_token;
  uint32_t* perm_mask;
  int32_t* dispatch;
  int32_t* expert_counts;
  int32_t* blk_counts;       // [n_blocks * K] pair counts per block and bin
  uint32_t* sync;            // [2] grid barrier: arrivals, generation (zero between calls)
  uint32_t* status;
  int n_blocks;
  int rounds;                // 256-token rounds per block
  uint64_t limit_ns;
};

struct GaussParams {
  int T, d;
  const void* X;
  const float* gcoef;        // written by the coefficient kernel launched just before
  int dcoef;
  float inv_tau;
  float* M;
  uint32_t* status;
};

// Gaussian-mixture score: C components per modality, F = 2C - 1 forms relative to (text, 0).
constexpr int kGmmMaxComponents = 4;
constexpr int kGmmMaxForms = 2 * kGmmMaxComponents - 1;
struct GmmParams {
  int T, d, C, F, dcoef;
  const void* X;
  const float* log_pi;       // [2, C]
  const float* mu;           // [2, C, d]
  const float* var;          // [2, C, d]
  float inv_tau;
  float* coef;               // workspace: [F][2][dcoef] + [F][dcoef / 256]
  float* M;
  uint32_t* status;
};

struct AttnParams {
  int B, H, S, hd, T;
  const void* Q;
  const void* K;
  const uint8_t* is_vision;
  const float* m_prev;
  const float* key_bias;
  float scale_log2;          // sm_scale * log2(e)
  int causal;
  const float* xattn_norm;
  const float* x_norm;
  float* M;
  float* part;               // [H * T]
  uint32_t* ticket;          // [B * n_qtiles]
  uint32_t* status;
  int n_qtiles;
  int n_items;
  uint64_t limit_ns;
};

// Online Gaussian statistics (eqs. 5-7): state N [2], S_mu [2, d], S_var [2, d] (fp64, updated
// in place); per-block shifted sums part [G][4][d] and vision-row counts nvis [G] (workspace).
struct StatsParams {
  int T, d, G;
  const void* X;
  const uint8_t* is_vision;
  double beta;
  double* N;
  double* S_mu;
  double* S_var;
  float* mu_out;             // [2, d] S_mu / N or null
  float* var_out;            // [2, d] S_var / N or null
  float* part;
  int32_t* nvis;
  double* N0;                // [2] copy of N_{t-1}
};

// Bin-level load-balance loss (eq. 16) from the forward's saved scores: per-block partials
// part_h [G][E] (sums of the bin-renormalised gate over the bin's routed tokens), part_s [G][E]
// (selections), part_u [G][K] (routed tokens per bin), then f, P, the loss and the table.
struct BalParams {
  int T, E, k, K, N_B, G;
  const float* gsave;
  const int32_t* topk_idx;
  const int32_t* expert_bin;
  const int32_t* expert_bin_host;   // the plan's bin map on the host (kernel choice)
  double scale;
  float* part_h;
  int32_t* part_s;
  int32_t* part_u;
  float* tab_f;
  float* tab_a;
  uint32_t* flag;
  float* loss;
  float* f_out;              // [E] or null
  float* P_out;              // [E] or null
};

// Momentum-adaptive binning (eqs. 10-11).
struct BinsParams {
  int E, N_B;
  double beta;
  const int32_t* counts;     // [2, E] this step's selections by hard modality
  double* C_bar;             // [2, E] EMA loads, updated in place
  int32_t* expert_bin;       // [E] output
  double* f_spec;            // [E] output or null
};

// Fixed-size scratch of smoes_bin_permute_noalloc, kept in a file-scope __device__ array of
// bin_permute.cu (for callers that cannot allocate): room for 1024 permutation blocks x 32 bins
// and 256 experts, which covers every plan smoes_plan_create accepts.
constexpr int kStaticPermBlocks = 1024;
struct StaticPermScratch {
  int32_t blk_counts[kStaticPermBlocks * kMaxBins];
  int32_t expert_bin[kMaxExperts];
  int32_t expert_slot[kMaxExperts];
  uint32_t status[4];
  uint32_t sync[4];
};
// Device address of that array on the current device (resolved once per device).
cudaError_t static_perm_scratch(StaticPermScratch** out);
// Writes a plan's bin map and slots (host arrays of E entries, passed to the kernel by value)
// into that array and clears its status and barrier words, in stream order.
cudaError_t launch_static_perm_prep(StaticPermScratch* sp, const int32_t* expert_bin,
                                    const int32_t* expert_slot, int E, cudaStream_t s);

// ------------------------------------------------------------------ launchers (in .cu files)
// Every kernel of the library is launched with programmatic stream serialization: its CTAs may
// be scheduled while the kernel before it in the stream is finishing, which hides the launch
// latency between the calls of a step. The protocol that keeps this exact: a kernel calls
// pdl_wait() before it reads or writes memory that any earlier work in the stream may touch,
// and pdl_trigger() only after its own pdl_wait(), so that a kernel that starts early knows
// that every kernel before its immediate predecessor has completed; only data that the
// immediate predecessor does not write (a plan table, W in the backward) is read earlier.
template <class... KArgs, class... Args>
cudaError_t launch_pdl(void (*k)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                       Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, k, static_cast<Args&&>(args)...);
}

// tmG: TMA map of the saved softmax scores [T, E] fp32 (box 32 x 128, 128-byte swizzle), or
// null to store them row by row.
cudaError_t launch_router_fwd_bf16(const FwdParams& p, const CUtensorMap& tmX,
                                   const CUtensorMap& tmW, const CUtensorMap* tmG, int n_sms,
                                   cudaStream_t s);
cudaError_t launch_router_fwd_bf16_var(const FwdParams& p, const CUtensorMap& tmX,
                                       const CUtensorMap& tmW, const CUtensorMap* tmG, int n_sms,
                                       cudaStream_t s);   // router variants compiled in
cudaError_t launch_router_fwd_f32(const FwdParams& p, cudaStream_t s);
int f32_chunks(int d);     // feature chunks of the fp32 forward and backward (128 features each)
cudaError_t launch_router_bwd_bf16(const BwdParams& p, const CUtensorMap& tmX,
                                   const CUtensorMap& tmW, const CUtensorMap& tmDX,
                                   cudaStream_t s);
cudaError_t launch_router_bwd_f32(const BwdParams& p, cudaStream_t s);
cudaError_t launch_dz_prep(const BwdParams& p, cudaStream_t s);
cudaError_t launch_dw_reduce(const BwdParams& p, cudaStream_t s);
cudaError_t launch_bin_permute(const PermParams& p, cudaStream_t s);
cudaError_t launch_gauss_score(const GaussParams& p, smoes_dtype dt, int n_sms, cudaStream_t s);
// Coefficients of the Gaussian log-likelihood difference (eq. 8) into coef = ga | gb | part.
cudaError_t launch_gauss_coef(const float* mu, const float* var, int d, int dcoef, float* coef,
                              uint32_t* status, cudaStream_t s);
cudaError_t launch_stats_update(const StatsParams& p, bool bf16, cudaStream_t s);
cudaError_t launch_adaptive_bins(const BinsParams& p, cudaStream_t s);
cudaError_t launch_bin_balance(const BalParams& p, cudaStream_t s);
// Attention forward with the vision score as one more value column (eqs. 2-4), grouped-query
// heads: K and V have Hkv heads, query head h reads key/value head h / (H / Hkv). O [B, H, S, hd]
// bf16 (written through the TMA map), M as for the mass-only kernel.
struct AttnFwdParams {
  AttnParams a;
  int Hkv;
};
cudaError_t launch_attn_fwd(const AttnFwdParams& p, const CUtensorMap& tmQ, const CUtensorMap& tmK,
                            const CUtensorMap& tmV, const CUtensorMap& tmO, int n_sms, cudaStream_t s);
cudaError_t launch_gmm_score(const GmmParams& p, smoes_dtype dt, int n_sms, cudaStream_t s);
cudaError_t launch_attn_mass(const AttnParams& p, const CUtensorMap& tmQ, const CUtensorMap& tmK,
                             int n_sms, cudaStream_t s);

// Shape helpers shared by host and device code.
__host__ __device__ constexpr int round_up(int x, int m) { return (x + m - 1) / m * m; }

// Forward (tcgen05): 128-token tiles, K-blocks of 64 bf16 (128-byte rows).
constexpr int kFwdBM = 128;
constexpr int kFwdBK = 64;
// Backward (tcgen05): 64-token tiles, 128-column d-blocks.
constexpr int kBwdBT = 64;
constexpr int kBwdBD = 128;

}  // namespace smoes
