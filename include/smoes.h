/*
 * smoes.h -- C ABI of the GB300 (sm_103a) SMoES router hot path.
 *
 * SMoES ("Soft Modality-Guided Expert Specialization in MoE-VLMs") regularises an MoE router
 * so that groups of experts ("bins") specialise by modality. Per MoE layer the hot path is:
 *   soft modality score (Sec. 3.2: Gaussian statistics, eqs. (8)-(9), or attention mass,
 *   eqs. (2)-(4)) -> gate logits z = W x, softmax, top-k (Sec. 3.1) -> expert-to-bin sums
 *   -> per-sample inter-bin mutual information and the MI loss (Sec. 3.4, eqs. (12)-(15))
 *   -> gradient of the MI loss to W and x -> bin-grouped token permutation with
 *   de-duplicated expert-parallel dispatch counts (Sec. 4.5).
 *
 * Conventions shared by every call
 *   - Arrays are dense, row-major, device pointers, 16-byte aligned; the caller owns every
 *     buffer, including the workspace. The library never allocates device memory.
 *   - X is [T, d] (tokens x hidden), W is [E, d] (the torch Linear layout of W_gate).
 *   - Modality index 0 = vision, 1 = text. M is [T, 2] float32, rows sum to 1.
 *   - Sample i (the paper's index i) is the contiguous token range
 *     [sample_offsets[i], sample_offsets[i+1]).
 *   - All work is enqueued asynchronously on the given stream. Argument errors are found on the
 *     host before any launch and leave every output untouched. Errors found while kernels run
 *     (non-finite values, non-positive variances, invalid indices, a bounded device wait that
 *     ran out) set a status word inside the workspace; read it with smoes_read_device_status.
 *   - Calls that share one workspace must be ordered on the GPU (same stream, or synchronised).
 */
#ifndef SMOES_H
#define SMOES_H

#include <stddef.h>
#include <stdint.h>

#include <cuda_runtime_api.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  SMOES_OK = 0,
  SMOES_ERR_INVALID_ARG = -1,     /* bad size, pointer, map or offsets; nothing launched      */
  SMOES_ERR_UNSUPPORTED = -2,     /* valid but outside what the library supports            */
  SMOES_ERR_ALIGNMENT = -3,       /* a pointer is not 16-byte aligned                        */
  SMOES_ERR_WORKSPACE = -4,       /* workspace missing or smaller than smoes_workspace_bytes */
  SMOES_ERR_CUDA = -5,            /* a CUDA runtime/driver call or a launch failed           */
  SMOES_ERR_DEVICE_TIMEOUT = -6,  /* (device status) a bounded wait inside a kernel expired  */
  SMOES_ERR_DATA = -7             /* (device status) non-finite or out-of-range input data   */
} smoes_status;

typedef enum { SMOES_F32 = 0, SMOES_BF16 = 1 } smoes_dtype;

typedef enum {
  SMOES_SCORE_PROVIDED = 0,       /* M is given by the caller                       */
  SMOES_SCORE_GAUSS = 1,          /* Gaussian-statistics score, eqs. (8)-(9)        */
  SMOES_SCORE_ATTN = 2,           /* attention-accumulated score, eqs. (2)-(4)      */
  SMOES_SCORE_GMM = 3             /* Gaussian-mixture estimator (supplementary)     */
} smoes_score_mode;

typedef enum { SMOES_GATE_SOFTMAX = 0, SMOES_GATE_SIGMOID = 1 } smoes_gate;

typedef enum {
  SMOES_CALL_ROUTER_FWD = 0,          /* smoes_router_fwd                                 */
  SMOES_CALL_ROUTER_FWD_PERMUTE = 1,  /* smoes_router_fwd_permute                         */
  SMOES_CALL_ROUTER_BWD = 2,          /* smoes_router_bwd                                 */
  SMOES_CALL_BIN_PERMUTE = 3,         /* smoes_bin_permute                                */
  SMOES_CALL_ATTN_SCORE = 4           /* smoes_modality_score with SMOES_SCORE_ATTN       */
} smoes_call;

typedef struct smoes_plan_s* smoes_plan;

/* Shape and routing metadata of one router layer (Secs. 3.1, 3.3).
 *   T tokens (0..2^20); d hidden size (d % 8 == 0, d >= 8); E routed experts (1..128 for
 *   SMOES_BF16 plans, 1..64 for SMOES_F32 plans; larger E returns SMOES_ERR_UNSUPPORTED);
 *   k top-k (1..16, k <= E); n_bins bins (1..32, E % n_bins == 0, E / n_bins <= 32);
 *   n_samples >= 1 when T > 0 (0 when T == 0). Every plan this call accepts runs in every
 *   call below (the attention score adds its own limit on the head size).
 *   sample_offsets_host [n_samples+1]: 0 = o_0 < o_1 < ... < o_B = T (no empty sample).
 *   expert_bin_host [E]: bin of each expert, each bin holding exactly E / n_bins experts.
 *   renorm_topk: 0 -> top-k weights are the softmax scores; 1 -> renormalised over the top-k.
 *   attn_max_heads: largest head count passed to smoes_modality_score(SMOES_SCORE_ATTN)
 *   (sizes the per-head partial sums in the workspace); 0 if the attention score is not used.
 *   gate: SMOES_GATE_SOFTMAX (Sec. 3.1) or SMOES_GATE_SIGMOID (the sigmoid router with a
 *   selection bias of the paper's backbone table: affinities s = sigmoid(z), experts chosen by
 *   the top-k of s + score_bias, top-k weights s / sum of the chosen s (always renormalised), and
 *   the g of eq. (12) read as s / sum_e s).
 *   score_bias: device array [E] float32 read by every forward of a SMOES_GATE_SIGMOID plan (the
 *   caller may update it in place between steps), or NULL for no bias.
 *   mi_topk_mask: 0 -> the g summed into the bins of eq. (12) is the dense gate; 1 -> it is the
 *   gate restricted to the chosen experts and renormalised over them (a reading the paper leaves
 *   open). bin_prob then reports these masked bin sums.
 * Both host arrays are copied; the caller may free them after smoes_plan_create returns. */
typedef struct {
  int T, d, E, k, n_bins, n_samples;
  smoes_dtype dtype;                   /* element type of X, W and dX                          */
  const int32_t* sample_offsets_host;
  const int32_t* expert_bin_host;
  int renorm_topk;
  int attn_max_heads;
  int gate;                            /* smoes_gate                                           */
  const float* score_bias;
  int mi_topk_mask;
} smoes_router_desc;

/* Gaussian-statistics score inputs, eqs. (8)-(9).
 *   X [T, d] (plan dtype); mu, var [2, d] float32 (row 0 vision, row 1 text), var > 0;
 *   tau > 0 the temperature, or tau <= 0 for the paper's default 0.5 * d (Sec. 4.1). */
typedef struct {
  const void* X;
  const float* mu;
  const float* var;
  float tau;
} smoes_gauss_args;

/* Attention-accumulated score inputs, eqs. (2)-(4).
 *   Q, K [B, H, S, hd] bf16 with B * S == T (token b*S + j is query j of sequence b);
 *   hd == 128 (other head sizes return SMOES_ERR_UNSUPPORTED); 1 <= H <= attn_max_heads of
 *   the plan (else SMOES_ERR_WORKSPACE).
 *   Exactly one of is_vision ([T] uint8, the hard labels of eq. (2)) or m_prev ([T] float32,
 *   the previous layer's vision score) gives the score carried by every key.
 *   key_bias [T] float32 or NULL: added to the logit of key j of its sequence.
 *   sm_scale: logit scale (1/sqrt(hd) for standard attention). causal: 1 = keys j' <= j only.
 *   xattn_norm, x_norm [T] float32 or NULL: when both are given, eq. (4) blends the aggregated
 *   score with the carried one, weighted by |x_attn| and |x|.                               */
typedef struct {
  const void* Q;
  const void* K;
  int B, H, S, hd;
  const uint8_t* is_vision;
  const float* m_prev;
  const float* key_bias;
  float sm_scale;
  int causal;
  const float* xattn_norm;
  const float* x_norm;
} smoes_attn_args;

/* Gaussian-mixture score inputs (the estimator the paper explores beyond eq. (8)): each
 *   modality's features follow n_components (1..4) diagonal Gaussians with weights pi.
 *   X [T, d] (plan dtype); log_pi [2, C] float32 (log weights, each row summing to 1 in the
 *   linear domain); mu, var [2, C, d] float32, var > 0; tau as for smoes_gauss_args.
 *   M_v = sigmoid((LL_v - LL_t) / tau) with LL_m = log sum_c pi_mc N(x; mu_mc, var_mc);
 *   n_components = 1 gives the score of eqs. (8)-(9). */
typedef struct {
  const void* X;
  int n_components;
  const float* log_pi;
  const float* mu;
  const float* var;
  float tau;
} smoes_gmm_args;

typedef struct {
  smoes_gauss_args gauss;
  smoes_attn_args attn;
  smoes_gmm_args gmm;
} smoes_score_args;

/* Validates the descriptor and builds the host-side plan (no device memory is touched).
 * Returns SMOES_ERR_INVALID_ARG / SMOES_ERR_UNSUPPORTED on bad or unsupported shapes. */
smoes_status smoes_plan_create(const smoes_router_desc* desc, smoes_plan* out);
void smoes_plan_destroy(smoes_plan plan);

/* Bytes of device workspace the plan needs (metadata, forward-to-backward state, partial sums,
 * status word). The workspace is caller-owned and 256-byte aligned. */
size_t smoes_workspace_bytes(smoes_plan plan);

/* Writes the plan's metadata into the workspace and clears its counters and status word.
 * Call once after allocating the workspace (and again after any device-side error), on the
 * stream that later calls use. */
smoes_status smoes_workspace_init(smoes_plan plan, void* ws, size_t ws_bytes, cudaStream_t stream);

/* Kernel launches one call makes on this plan (a host query: no GPU work, no allocation). Nothing
 * else is enqueued besides these kernels, except a cudaMemsetAsync of the outputs of empty
 * (T == 0) calls, counted as 0. smoes_router_fwd_permute is one launch when the permutation
 * runs inside the forward kernel (SMOES_BF16 plans of at most two 128-token tiles per SM), two
 * otherwise. Returns -1 for a null plan or an unknown call. */
int smoes_call_launches(smoes_plan plan, smoes_call call);

const char* smoes_status_string(smoes_status status);

/* Limit, in nanoseconds, of every bounded wait inside the plan's kernels (pipeline barriers,
 * the grid barriers of the cooperative launches, tickets). A wait that exceeds it records
 * SMOES_ERR_DEVICE_TIMEOUT in the workspace status word and the kernel returns without
 * finishing its outputs. The default is 2 s; limit_ns == 0 restores it. Applies to calls made
 * after it returns. */
smoes_status smoes_plan_set_wait_limit(smoes_plan plan, uint64_t limit_ns);

/* Synchronises `stream`, reads the workspace status word and returns SMOES_OK,
 * SMOES_ERR_DATA or SMOES_ERR_DEVICE_TIMEOUT. *n_absent_modality (optional) receives how many
 * (sample, modality) pairs had zero soft mass in the last forward (eq. (12) read as 0). */
smoes_status smoes_read_device_status(smoes_plan plan, const void* ws, cudaStream_t stream,
                                      int32_t* n_absent_modality);

/* (1) Soft modality score (Sec. 3.2).
 *   mode SMOES_SCORE_GAUSS: M[j] = softmax_m(LL[j, m] / tau) with LL of eq. (8).
 *   mode SMOES_SCORE_ATTN:  M[j, 0] = (1/H) sum_h sum_j' softmax_j'(s q.k_j' + bias_j') m_j'
 *                           (eq. (3), optionally followed by eq. (4)); M[j, 1] = 1 - M[j, 0].
 *   mode SMOES_SCORE_GMM:   eq. (9) on the Gaussian-mixture log-likelihoods of args->gmm
 *                           (n_components > 4 returns SMOES_ERR_UNSUPPORTED).
 *   M: [T, 2] float32 output. ws is needed by SMOES_SCORE_ATTN (head partial sums). */
smoes_status smoes_modality_score(smoes_plan plan, smoes_score_mode mode,
                                  const smoes_score_args* args, float* M,
                                  void* ws, size_t ws_bytes, cudaStream_t stream);

/* (1b) Causal attention forward that also yields the attention-accumulated score (Sec. 3.2.1,
 *   eqs. (2)-(4); the form the paper's supplementary gives for FlashAttention-style kernels: the
 *   carried score is one more value column). args as for SMOES_SCORE_ATTN (Q [B, H, S, hd], K with
 *   n_kv_heads heads [B, n_kv_heads, S, hd], bf16); V [B, n_kv_heads, S, hd] bf16; grouped-query
 *   heads: query head h reads key/value head h / (H / n_kv_heads) (H % n_kv_heads == 0).
 *   Outputs: O [B, H, S, hd] bf16 = softmax(sm_scale Q K^T + key_bias) V per head (the softmax
 *   weights pass to the tensor cores in bf16, as in FlashAttention), and M [T, 2] as for
 *   smoes_modality_score(SMOES_SCORE_ATTN) (the head-averaged vision mass, optionally blended
 *   by eq. (4)). Requires hd == 128 and S % 128 == 0 (else SMOES_ERR_UNSUPPORTED); key_bias,
 *   is_vision and m_prev 16-byte aligned; H <= attn_max_heads of the plan. */
smoes_status smoes_attention_fwd(smoes_plan plan, const smoes_attn_args* args, const void* V,
                                 int n_kv_heads, void* O, float* M, void* ws, size_t ws_bytes,
                                 cudaStream_t stream);

/* (2) Router forward with the MI regulariser (Secs. 3.1, 3.3, 3.4).
 *   X [T, d], W [E, d] (plan dtype). Scores: M_in [T, 2] (SMOES_SCORE_PROVIDED, gauss == NULL),
 *   or gauss != NULL (fused Gaussian score; gauss->X is ignored, X is used) and the scores are
 *   written to M_out [T, 2] (required then).
 *   Outputs: topk_idx [T, k] int32 (descending logit, equal logits -> lower expert index),
 *   topk_w [T, k] float32, bin_prob [T, n_bins] float32 (optional, NULL to skip),
 *   joint [B, 2, n_bins] float32 P_i(m, B_k) of eq. (13) (optional), mi [B] float32 I_i of
 *   eq. (14), loss [1] float32 = -(1/B) sum_i I_i (eq. (15), one layer).
 *   ws keeps the softmax scores and per-sample tables that smoes_router_bwd reads. */
smoes_status smoes_router_fwd(smoes_plan plan, const void* X, const void* W, const float* M_in,
                              const smoes_gauss_args* gauss, float* M_out,
                              int32_t* topk_idx, float* topk_w, float* bin_prob,
                              float* joint, float* mi, float* loss,
                              void* ws, size_t ws_bytes, cudaStream_t stream);

/* (2b) The forward (2) and the bin permutation (4) of its own top-k in one launch.
 *   Arguments: those of smoes_router_fwd, then those of smoes_bin_permute (topk_idx is the
 *   forward's output); results are identical to smoes_router_fwd followed by smoes_bin_permute.
 *   On bf16 plans with at most two 128-token tiles per SM the forward kernel counts each CTA's
 *   (token, bin) pairs from the top-k it holds in registers; after a grid-wide barrier (a
 *   cooperative launch: every CTA resident) the warps that are idle once the CTA's gate GEMM is
 *   done place the CTA's entries, while the per-sample MI reduction of eqs. (12)-(15) runs.
 *   Larger batches and fp32 plans make the two calls (the fused scatter runs after a CTA's last
 *   tile, serially over its tokens, and loses to the standalone kernel there). The paper has no
 *   counterpart for this fusion; it removes the separate launch and counting pass. */
smoes_status smoes_router_fwd_permute(smoes_plan plan, const void* X, const void* W,
                                      const float* M_in, const smoes_gauss_args* gauss,
                                      float* M_out, int32_t* topk_idx, float* topk_w,
                                      float* bin_prob, float* joint, float* mi, float* loss,
                                      const int32_t* home, const uint8_t* is_vision,
                                      int32_t* bin_offsets, int32_t* perm_token,
                                      uint32_t* perm_mask, int32_t* dispatch,
                                      int32_t* expert_counts, void* ws, size_t ws_bytes,
                                      cudaStream_t stream);

/* (3) Backward of loss_scale * L_MI (plus, optionally, an upstream gradient of topk_w).
 *   The soft scores are constants (no gradient flows into M). X, W, M and topk_idx must be the
 *   tensors of the preceding smoes_router_fwd on the same ws.
 *   dW [E, d] float32: written, or accumulated into when accumulate_dW != 0.
 *   dX [T, d] (plan dtype) or NULL; dlogits [T, E] float32 or NULL.
 *   d_topk_w [T, k] float32 or NULL.
 *   Precision on SMOES_BF16 plans: dW is formed from dz split into two bf16 parts (fp32-level
 *   accuracy); dX from dz rounded to bf16 (bf16 inputs, fp32 accumulation), stored in bf16. */
smoes_status smoes_router_bwd(smoes_plan plan, const void* X, const void* W, const float* M,
                              const int32_t* topk_idx, const float* d_topk_w, float loss_scale,
                              float* dW, int accumulate_dW, void* dX, float* dlogits,
                              void* ws, size_t ws_bytes, cudaStream_t stream);

/* (7) Bin-level load-balance loss (Sec. 3.5, eq. (16)) of the last forward on ws:
 *     L_bal = sum_k N_B sum_{e in B_k} f_e P_e,
 *   with U_k = the tokens that have at least one top-k expert in bin B_k, f_e = selections of e /
 *   selections of all of B_k's experts, P_e = mean over U_k of g_je / sum_{e' in B_k} g_je' (the
 *   gate renormalised inside the bin). A bin no token selects contributes 0. topk_idx [T, k]: the
 *   forward's top-k. loss_bal [1] float32 receives L_bal (one layer); f_e, P_e [E] float32 or NULL.
 *   The call also arms the backward: every smoes_router_bwd of this plan on the same ws until the
 *   next forward adds the gradient of loss_scale * L_bal, taken with the counts f_e constant, to
 *   the MI gradient (dlogits, dW and dX; topk_idx must then be passed to smoes_router_bwd). The
 *   arming is tracked both on the host (the plan) and in ws (the forward kernels clear it).
 *   Sums are fp32, in a fixed order (bitwise reproducible). */
smoes_status smoes_bin_balance(smoes_plan plan, const int32_t* topk_idx, float loss_scale,
                               float* loss_bal, float* f_e, float* P_e, void* ws, size_t ws_bytes,
                               cudaStream_t stream);

/* (4) Bin-grouped permutation with de-duplicated dispatch (Sec. 4.5, "DeDup").
 *   One entry per unique (token, bin) pair, ordered by bin ascending then token ascending.
 *   topk_idx [T, k] int32 in [0, E). home [T] int32 in [0, n_bins) or NULL for the contiguous
 *   split home(j) = floor(j * n_bins / T). is_vision [T] uint8 (required if expert_counts).
 *   Outputs: bin_offsets [n_bins+1] int32; perm_token and perm_mask with capacity
 *   T * min(k, n_bins) (bit s of perm_mask = the expert in slot s of the bin, slots ordering a
 *   bin's experts by index); dispatch [n_bins, n_bins] int32, dispatch[h][b] = pairs whose
 *   token lives on device h and goes to bin b; expert_counts [2, E] int32 (optional) = tokens
 *   of each hard modality that chose each expert (the count C_{m,e} of eq. (10)). */
smoes_status smoes_bin_permute(smoes_plan plan, const int32_t* topk_idx, const int32_t* home,
                               const uint8_t* is_vision, int32_t* bin_offsets,
                               int32_t* perm_token, uint32_t* perm_mask, int32_t* dispatch,
                               int32_t* expert_counts, void* ws, size_t ws_bytes,
                               cudaStream_t stream);

/* (5) Online statistics of the Gaussian modality score (Sec. 3.2, eqs. (5)-(7)): one step of the
 *   EMA variant of Welford's algorithm for both modalities, in place.
 *   X [T, d] (plan dtype); is_vision [T] uint8 (the hard labels: T_m is the batch's modality-m
 *   tokens); beta in [0, 1] the EMA decay (the paper uses 0.99).
 *   State (device, fp64, updated in place): N [2], S_mu [2, d], S_var [2, d] (row 0 vision,
 *   row 1 text); all zeros is the empty state. Per modality m with n = |T_m|:
 *     N = beta N + n;  S_mu = beta S_mu + n mu_T;
 *     S_var = beta S_var + sum_{x in T_m} (x - mu_T)^2 + (mu_T - S_mu_old / N_old)^2 beta N_old n / (beta N_old + n),
 *   the last term taken as 0 when N_old = 0 or n = 0 (mu_T the batch mean; see the paper for the
 *   symbols). mu, var [2, d] float32 or NULL: S_mu / N and S_var / N after the update (the
 *   statistics the next score uses; NaN for a modality never seen).
 *   The batch sums are shifted by the previous mean (exact algebra, no cancellation); partial
 *   sums are fp32 per block of rows and fp64 across blocks, in a fixed order (reproducible).
 *   ws: the plan's workspace (per-block partial sums). */
smoes_status smoes_gaussian_stats_update(smoes_plan plan, const void* X, const uint8_t* is_vision,
                                         double beta, double* N, double* S_mu, double* S_var,
                                         float* mu, float* var, void* ws, size_t ws_bytes,
                                         cudaStream_t stream);

/* (6) Momentum-adaptive binning (Sec. 3.3, eqs. (10)-(11)).
 *   expert_counts [2, E] int32: this step's selections of each expert by the tokens of each hard
 *   modality (the expert_counts output of (4)); C_bar [2, E] fp64, updated in place:
 *   C_bar = beta C_bar + (1 - beta) C (eq. (10)). f_spec(e) = C_bar[text, e] / (C_bar[text, e] +
 *   C_bar[vision, e]) (eq. (11); 1/2 for an expert with no load), written to f_spec [E] fp64
 *   when not NULL. expert_bin [E] int32 receives the new map: experts sorted by ascending f_spec
 *   (equal values in expert-index order) and cut into n_bins runs of E / n_bins, so bin 0 holds
 *   the most vision-biased experts. All arithmetic is fp64 with separately rounded operations:
 *   the map is reproducible bit for bit. The plan keeps its own map; a caller that adopts the
 *   new one creates a plan from it (expert groupings change rarely: the loads are EMAs). */
smoes_status smoes_adaptive_bins(smoes_plan plan, const int32_t* expert_counts, double beta,
                                 double* C_bar, int32_t* expert_bin, double* f_spec,
                                 cudaStream_t stream);

/* (4b) The bin permutation of (4) without a workspace, for callers that cannot allocate device
 *   memory. The paper has no counterpart; this is a deployment convenience. Some callers cannot
 *   call cudaMalloc: serving runtimes whose device memory is planned up front by an arena that
 *   hands out no further blocks, plug-ins that receive only their input and output buffers from a
 *   host framework, and latency-critical loops that must not risk the implicit device-wide
 *   synchronisation an allocation can cause.
 *   Same arguments and results as smoes_bin_permute, minus the workspace. The scratch it needs
 *   (about 130 KB: block counts for up to 1024 permutation blocks x 32 bins, the bin
 *   map of up to 256 experts, a status word) is a fixed array inside the library, one per device
 *   that loads it, held until the process exits; this covers every plan smoes_plan_create
 *   accepts, and larger shapes return SMOES_ERR_UNSUPPORTED. Each call first writes the plan's
 *   bin map (passed to a small kernel by value) into that array and clears its status and
 *   barrier words, on the given stream.
 *   The first call on a device looks up that array's device address (once per device); make that
 *   first call before any stream capture. Every call shares the one array (each call rewrites
 *   what it reads), so calls that overlap on the GPU, on any stream, race: order them. Device-side
 *   data errors are recorded in the array's status word only, not reported. */
smoes_status smoes_bin_permute_noalloc(smoes_plan plan, const int32_t* topk_idx, const int32_t* home,
                                       const uint8_t* is_vision, int32_t* bin_offsets,
                                       int32_t* perm_token, uint32_t* perm_mask, int32_t* dispatch,
                                       int32_t* expert_counts, cudaStream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* SMOES_H */
