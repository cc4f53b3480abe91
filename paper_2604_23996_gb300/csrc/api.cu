// api.cu -- host side of the C ABI in include/smoes.h: plans, workspace layout, argument
// validation, TMA descriptors and launch sequencing. No device memory is allocated here.
#include <algorithm>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <new>
#include <vector>

#include "smoes_internal.cuh"

namespace smoes {
int perm_blocks(int T, int k);
int perm_rounds(int T, int k);
}

using namespace smoes;

namespace {

constexpr size_t kAlign = 256;
inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

struct Layout {
  size_t status, sample_ticket, loss_ticket, offsets, token_sample, expert_bin, expert_slot,
      piece_base, sample_pieces, pieces, mi32, tabs, gsave, ginv, dw_part, dz_img, perm, attn_ticket, attn_part,
      gcoef, perm_sync, fperm, stat_part, stat_nvis, stat_n0, f32_part, tile_ticket, bal_flag,
      bal_f, bal_a, bal_h, bal_s, bal_u, gmmcoef;
  size_t header_bytes;   // [0, header_bytes) is cleared by smoes_workspace_init
  size_t total;
};

}  // namespace

struct smoes_plan_s {
  smoes_router_desc desc{};
  int N_B = 1;
  int n_groups = 0;      // ceil(T / 128): forward tiles, one partial-sum piece per (tile, sample)
  int n_pieces = 0;
  int n_sms = 148;
  // backward decomposition
  int bwd_tiles = 0;     // 64-token tiles
  int bwd_groups = 1, bwd_slices = 1, bwd_slice_width = 0;
  int perm_nblocks = 0;
  int dcoef = 256;       // Gaussian coefficient vectors padded to 256 features
  int stat_blocks = 1;   // blocks of the statistics pass (one partial each)
  bool contig_bins = false;
  uint64_t limit_ns = kWaitLimitNs;   // bounded device waits
  bool balance_armed = false;         // smoes_bin_balance enqueued since the last forward
  std::vector<int32_t> offsets, expert_bin, expert_slot, token_sample, piece_base, sample_pieces;
  Layout L{};
};

namespace {

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

WsView make_view(const smoes_plan_s* P, void* ws) {
  uint8_t* b = static_cast<uint8_t*>(ws);
  const Layout& L = P->L;
  WsView v;
  v.status = reinterpret_cast<uint32_t*>(b + L.status);
  v.sample_ticket = reinterpret_cast<uint32_t*>(b + L.sample_ticket);
  v.loss_ticket = reinterpret_cast<uint32_t*>(b + L.loss_ticket);
  v.offsets = reinterpret_cast<const int32_t*>(b + L.offsets);
  v.token_sample = reinterpret_cast<const int32_t*>(b + L.token_sample);
  v.expert_bin = reinterpret_cast<const int32_t*>(b + L.expert_bin);
  v.expert_slot = reinterpret_cast<const int32_t*>(b + L.expert_slot);
  v.piece_base = reinterpret_cast<const int32_t*>(b + L.piece_base);
  v.sample_pieces = reinterpret_cast<const int32_t*>(b + L.sample_pieces);
  v.pieces = reinterpret_cast<float*>(b + L.pieces);
  v.mi32 = reinterpret_cast<float*>(b + L.mi32);
  v.tabs = reinterpret_cast<float*>(b + L.tabs);
  v.gsave = reinterpret_cast<float*>(b + L.gsave);
  v.ginv = reinterpret_cast<float*>(b + L.ginv);
  v.dw_part = reinterpret_cast<float*>(b + L.dw_part);
  v.dz_img = b + L.dz_img;
  v.perm_scratch = reinterpret_cast<int32_t*>(b + L.perm);
  v.attn_ticket = reinterpret_cast<uint32_t*>(b + L.attn_ticket);
  v.attn_part = reinterpret_cast<float*>(b + L.attn_part);
  v.gcoef = reinterpret_cast<float*>(b + L.gcoef);
  v.dcoef = P->dcoef;
  v.bal_flag = reinterpret_cast<uint32_t*>(b + L.bal_flag);
  v.bal_f = reinterpret_cast<float*>(b + L.bal_f);
  v.bal_a = reinterpret_cast<float*>(b + L.bal_a);
  return v;
}

Dims make_dims(const smoes_plan_s* P) {
  const smoes_router_desc& d = P->desc;
  Dims m;
  m.T = d.T;
  m.d = d.d;
  m.E = d.E;
  m.k = d.k;
  m.K = d.n_bins;
  m.B = d.n_samples;
  m.N_B = P->N_B;
  m.renorm = (d.renorm_topk || d.gate == SMOES_GATE_SIGMOID) ? 1 : 0;
  m.gate = d.gate == SMOES_GATE_SIGMOID ? 1 : 0;
  m.mask = d.mi_topk_mask ? 1 : 0;
  m.pstride = piece_stride(d.n_bins);
  m.n_groups = P->n_groups;
  m.contig_bins = P->contig_bins ? 1 : 0;
  return m;
}

// ---------------------------------------------------------------- TMA descriptor encoding
using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                   const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                   const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                   CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn get_encode() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(ptr);
  });
  return fn;
}

// 2-D row-major bf16 tensor [rows, cols]; box [box_rows, box_cols]; OOB reads return zeros.
bool encode_bf16_2d(CUtensorMap* m, const void* ptr, uint64_t rows, uint64_t cols, uint32_t box_rows,
                    uint32_t box_cols, bool swizzle128) {
  EncodeTiledFn enc = get_encode();
  if (!enc) return false;
  const cuuint64_t dims[2] = {cols, rows};
  const cuuint64_t strides[1] = {cols * 2};
  const cuuint32_t box[2] = {box_cols, box_rows};
  const cuuint32_t estr[2] = {1, 1};
  return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides, box, estr,
             CU_TENSOR_MAP_INTERLEAVE_NONE,
             swizzle128 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_NONE,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// 2-D row-major fp32 tensor [rows, cols] (cols * 4 a multiple of 16); box [box_rows, box_cols].
bool encode_f32_2d(CUtensorMap* m, const void* ptr, uint64_t rows, uint64_t cols, uint32_t box_rows,
                   uint32_t box_cols, bool swizzle128) {
  EncodeTiledFn enc = get_encode();
  if (!enc) return false;
  const cuuint64_t dims[2] = {cols, rows};
  const cuuint64_t strides[1] = {cols * 4};
  const cuuint32_t box[2] = {box_cols, box_rows};
  const cuuint32_t estr[2] = {1, 1};
  return enc(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<void*>(ptr), dims, strides, box, estr,
             CU_TENSOR_MAP_INTERLEAVE_NONE,
             swizzle128 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_NONE,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

int device_sms() {
  int dev = 0, n = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 148;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) return 148;
  return n;
}

smoes_status check_ws(const smoes_plan_s* P, const void* ws, size_t ws_bytes) {
  if (!ws || ws_bytes < P->L.total) return SMOES_ERR_WORKSPACE;
  if ((reinterpret_cast<uintptr_t>(ws) & (kAlign - 1)) != 0) return SMOES_ERR_ALIGNMENT;
  return SMOES_OK;
}

smoes_status cuda_status(cudaError_t e) { return e == cudaSuccess ? SMOES_OK : SMOES_ERR_CUDA; }

// The permutation runs inside the forward launch on the tensor-core path when every CTA holds at
// most two tiles (the fused scatter runs after a CTA's last tile, serially over its tokens: with
// many tiles per CTA the standalone permutation, spread over the whole GPU, is faster).
bool fuse_permute(const smoes_plan_s* P) {
  const smoes_router_desc& d = P->desc;
  const int fwd_tiles = (d.T + kFwdBM - 1) / kFwdBM;
  return d.dtype == SMOES_BF16 && d.T > 0 && d.n_bins <= kMaxBins && d.E <= kMaxExperts &&
         fwd_tiles <= 2 * P->n_sms;
}

// The forward of smoes_router_fwd; perm: the fused permutation's outputs (tensor-core path), or null.
smoes_status router_fwd(smoes_plan P, const void* X, const void* W, const float* M_in,
                        const smoes_gauss_args* gauss, float* M_out, int32_t* topk_idx,
                        float* topk_w, float* bin_prob, float* joint, float* mi, float* loss,
                        const FusedPerm* perm, void* ws, size_t ws_bytes, cudaStream_t stream) {
  if (!P) return SMOES_ERR_INVALID_ARG;
  smoes_status st = check_ws(P, ws, ws_bytes);
  if (st != SMOES_OK) return st;
  const smoes_router_desc& d = P->desc;
  if (!loss) return SMOES_ERR_INVALID_ARG;
  if (d.T == 0) return cuda_status(cudaMemsetAsync(loss, 0, sizeof(float), stream));
  if (!X || !W || !topk_idx || !topk_w || !mi) return SMOES_ERR_INVALID_ARG;
  if ((M_in == nullptr) == (gauss == nullptr)) return SMOES_ERR_INVALID_ARG;
  if (gauss && (!gauss->mu || !gauss->var || !M_out)) return SMOES_ERR_INVALID_ARG;
  if (!aligned16(X) || !aligned16(W) || (M_in && !aligned16(M_in)) || (M_out && !aligned16(M_out)) ||
      (gauss && (!aligned16(gauss->mu) || !aligned16(gauss->var))))
    return SMOES_ERR_ALIGNMENT;
  if (d.dtype == SMOES_F32 && d.E > 64) return SMOES_ERR_UNSUPPORTED;

  P->balance_armed = false;           // the forward kernel clears the device flag too
  FwdParams p{};
  p.dm = make_dims(P);
  p.ws = make_view(P, ws);
  p.X = X;
  p.W = W;
  p.M_in = M_in;
  p.score_bias = d.score_bias;
  p.mu = gauss ? gauss->mu : nullptr;
  p.var = gauss ? gauss->var : nullptr;
  p.inv_tau = gauss ? 1.f / (gauss->tau > 0.f ? gauss->tau : 0.5f * d.d) : 1.f;
  p.M_out = gauss ? M_out : nullptr;
  p.topk_idx = topk_idx;
  p.topk_w = topk_w;
  p.bin_prob = bin_prob;
  p.joint = joint;
  p.mi = mi;
  p.loss = loss;
  p.limit_ns = P->limit_ns;
  if (perm) {
    p.perm = *perm;
    p.perm.cta_counts = reinterpret_cast<int32_t*>(static_cast<uint8_t*>(ws) + P->L.fperm);
    p.perm.sync = reinterpret_cast<uint32_t*>(static_cast<uint8_t*>(ws) + P->L.perm_sync);
  }
  if (d.dtype == SMOES_BF16) {
    p.n_tiles = (d.T + kFwdBM - 1) / kFwdBM;
    CUtensorMap tx, tw;
    if (!encode_bf16_2d(&tx, X, d.T, d.d, kFwdBM, kFwdBK, true) ||
        !encode_bf16_2d(&tw, W, d.E, d.d, round_up(d.E, 16), kFwdBK, true))
      return SMOES_ERR_CUDA;
    // saved scores leave through TMA when their rows are 16-byte multiples
    CUtensorMap tg;
    const bool tma_g = d.E % 4 == 0 && d.E <= 128 && encode_f32_2d(&tg, p.ws.gsave, d.T, d.E, 128, 32, true);
    return cuda_status(launch_router_fwd_bf16(p, tx, tw, tma_g ? &tg : nullptr, P->n_sms, stream));
  }
  p.n_tiles = P->n_groups;
  p.f32_chunks = f32_chunks(d.d);
  p.f32_part = reinterpret_cast<float*>(static_cast<uint8_t*>(ws) + P->L.f32_part);
  p.tile_ticket = reinterpret_cast<uint32_t*>(static_cast<uint8_t*>(ws) + P->L.tile_ticket);
  return cuda_status(launch_router_fwd_f32(p, stream));
}

}  // namespace

extern "C" {

const char* smoes_status_string(smoes_status s) {
  switch (s) {
    case SMOES_OK: return "ok";
    case SMOES_ERR_INVALID_ARG: return "invalid argument";
    case SMOES_ERR_UNSUPPORTED: return "unsupported shape or mode";
    case SMOES_ERR_ALIGNMENT: return "pointer not aligned";
    case SMOES_ERR_WORKSPACE: return "workspace missing or too small";
    case SMOES_ERR_CUDA: return "CUDA error";
    case SMOES_ERR_DEVICE_TIMEOUT: return "bounded device wait expired";
    case SMOES_ERR_DATA: return "invalid input data found on the device";
  }
  return "unknown status";
}

smoes_status smoes_plan_create(const smoes_router_desc* desc, smoes_plan* out) {
  if (!desc || !out) return SMOES_ERR_INVALID_ARG;
  *out = nullptr;
  const smoes_router_desc& d = *desc;
  if (d.T < 0 || d.d < 8 || d.d % 8 != 0 || d.E < 1 || d.k < 1 || d.n_bins < 1)
    return SMOES_ERR_INVALID_ARG;
  if (d.dtype != SMOES_F32 && d.dtype != SMOES_BF16) return SMOES_ERR_INVALID_ARG;
  if (d.gate != SMOES_GATE_SOFTMAX && d.gate != SMOES_GATE_SIGMOID) return SMOES_ERR_INVALID_ARG;
  if (d.mi_topk_mask != 0 && d.mi_topk_mask != 1) return SMOES_ERR_INVALID_ARG;
  if (d.score_bias && (d.gate != SMOES_GATE_SIGMOID || !aligned16(d.score_bias))) return SMOES_ERR_INVALID_ARG;
  if (d.k > d.E || d.E % d.n_bins != 0) return SMOES_ERR_INVALID_ARG;
  if (d.E > kMaxExperts || d.k > kMaxTopK || d.n_bins > kMaxBins || d.E / d.n_bins > 32)
    return SMOES_ERR_UNSUPPORTED;
  if (d.T == 0 ? d.n_samples != 0 : d.n_samples < 1) return SMOES_ERR_INVALID_ARG;
  if (d.T > 0 && (!d.sample_offsets_host || !d.expert_bin_host)) return SMOES_ERR_INVALID_ARG;
  // what every later call can run: the backward's accumulators (bf16: E_pad <= 128 TMEM columns
  // per d-block; fp32: 64 logits per thread)
  if (d.E > (d.dtype == SMOES_BF16 ? kMaxExpertsBf16 : kMaxExpertsF32)) return SMOES_ERR_UNSUPPORTED;
  if (d.T > (1 << 20)) return SMOES_ERR_UNSUPPORTED;          // permutation: <= 1024 blocks
  if (static_cast<long long>(d.T) * d.d > (1ll << 40)) return SMOES_ERR_UNSUPPORTED;

  smoes_plan_s* P = new (std::nothrow) smoes_plan_s();
  if (!P) return SMOES_ERR_INVALID_ARG;
  P->desc = d;
  P->desc.sample_offsets_host = nullptr;
  P->desc.expert_bin_host = nullptr;
  P->N_B = d.E / d.n_bins;
  const int B = d.n_samples, T = d.T, E = d.E, K = d.n_bins;

  // sample offsets: 0 = o_0 < o_1 < ... < o_B = T
  P->offsets.assign(B + 1, 0);
  if (T > 0) {
    for (int i = 0; i <= B; ++i) P->offsets[i] = d.sample_offsets_host[i];
    bool ok = P->offsets[0] == 0 && P->offsets[B] == T;
    for (int i = 0; i < B && ok; ++i) ok = P->offsets[i + 1] > P->offsets[i];
    if (!ok) { delete P; return SMOES_ERR_INVALID_ARG; }
  }
  // expert -> bin map with exactly N_B experts per bin; slot = rank of the expert in its bin
  P->expert_bin.assign(E, 0);
  P->expert_slot.assign(E, 0);
  std::vector<int> fill(K, 0);
  for (int e = 0; e < E; ++e) {
    const int b = (T > 0 || d.expert_bin_host) ? d.expert_bin_host[e] : e / P->N_B;
    if (b < 0 || b >= K) { delete P; return SMOES_ERR_INVALID_ARG; }
    P->expert_bin[e] = b;
    P->expert_slot[e] = fill[b]++;
  }
  for (int b = 0; b < K; ++b)
    if (fill[b] != P->N_B) { delete P; return SMOES_ERR_INVALID_ARG; }
  // consecutive bins of a multiple of 4 experts: the forward sums bins in 4-expert groups
  P->contig_bins = P->N_B % 4 == 0;
  for (int e = 0; e < E && P->contig_bins; ++e) P->contig_bins = P->expert_bin[e] == e / P->N_B;
  P->dcoef = round_up(d.d, 256);

  // token -> sample, 128-token groups -> pieces (one piece per (group, sample) pair)
  P->n_groups = (T + kPieceTokens - 1) / kPieceTokens;
  P->token_sample.assign(std::max(T, 1), 0);
  for (int i = 0; i < B; ++i)
    for (int j = P->offsets[i]; j < P->offsets[i + 1]; ++j) P->token_sample[j] = i;
  P->piece_base.assign(P->n_groups + 1, 0);
  for (int w = 0; w < P->n_groups; ++w) {
    const int s0 = P->token_sample[w * kPieceTokens];
    const int s1 = P->token_sample[std::min(w * kPieceTokens + kPieceTokens - 1, T - 1)];
    P->piece_base[w + 1] = P->piece_base[w] + (s1 - s0 + 1);
  }
  P->n_pieces = P->piece_base[P->n_groups];
  // pieces of sample i are contiguous: groups are visited in order and each group's pieces are
  // ordered by sample, so sample i's first piece is in the group holding its first token
  P->sample_pieces.assign(B + 1, P->n_pieces);
  for (int i = 0; i < B; ++i) {
    const int w = P->offsets[i] / kPieceTokens;
    P->sample_pieces[i] = P->piece_base[w] + (i - P->token_sample[w * kPieceTokens]);
  }

  // backward decomposition
  P->n_sms = device_sms();
  P->bwd_tiles = (T + kBwdBT - 1) / kBwdBT;
  if (d.dtype == SMOES_BF16) {
    const int E_pad = round_up(E, 64);
    const int ds_full = 32768 / std::min(E_pad, 128);
    const int dround = round_up(d.d, kBwdBD);
    P->bwd_slice_width = std::min(ds_full, dround);
    P->bwd_slices = (dround + P->bwd_slice_width - 1) / P->bwd_slice_width;
    P->bwd_groups = std::max(1, std::min(P->bwd_tiles, P->n_sms / P->bwd_slices));
  } else {
    P->bwd_slice_width = d.d;
    P->bwd_slices = 1;
    P->bwd_groups = std::max(1, P->bwd_tiles);
  }
  P->perm_nblocks = std::max(1, perm_blocks(T, d.k));

  // workspace layout
  Layout& L = P->L;
  size_t o = 0;
  auto take = [&](size_t bytes) { const size_t at = o; o = align_up(o + std::max<size_t>(bytes, 1), kAlign); return at; };
  L.status = take(16);
  L.sample_ticket = take(sizeof(uint32_t) * std::max(B, 1));
  L.loss_ticket = take(sizeof(uint32_t) * 4);
  L.attn_ticket = take(sizeof(uint32_t) * (static_cast<size_t>(T) + 1));
  L.perm_sync = take(sizeof(uint32_t) * 4);
  L.tile_ticket = take(sizeof(uint32_t) * static_cast<size_t>(std::max(P->n_groups, 1)));
  L.bal_flag = take(sizeof(uint32_t) * 4);
  L.header_bytes = o;
  L.offsets = take(sizeof(int32_t) * (B + 1));
  L.token_sample = take(sizeof(int32_t) * std::max(T, 1));
  L.expert_bin = take(sizeof(int32_t) * E);
  L.expert_slot = take(sizeof(int32_t) * E);
  L.piece_base = take(sizeof(int32_t) * (P->n_groups + 1));
  L.sample_pieces = take(sizeof(int32_t) * (B + 1));
  L.pieces = take(sizeof(float) * static_cast<size_t>(std::max(P->n_pieces, 1)) * piece_stride(K));
  L.mi32 = take(sizeof(float) * std::max(B, 1));
  L.tabs = take(sizeof(float) * 3 * K * static_cast<size_t>(std::max(B, 1)));
  L.gsave = take(sizeof(float) * static_cast<size_t>(T) * E);
  L.ginv = take(sizeof(float) * static_cast<size_t>(std::max(T, 1)));
  L.dw_part = take(sizeof(float) * static_cast<size_t>(P->bwd_groups) * E * d.d);
  L.dz_img = take(d.dtype == SMOES_BF16 && E <= 128
                      ? static_cast<size_t>(P->bwd_tiles) * 2 * round_up(E, 64) * 128 : 0);
  L.perm = take(sizeof(int32_t) * static_cast<size_t>(P->perm_nblocks) * K);
  L.fperm = take(sizeof(int32_t) * static_cast<size_t>(std::max(P->n_sms, 1)) * K);   // per-CTA counts
  L.attn_part = take(sizeof(float) * static_cast<size_t>(T) * std::max(0, d.attn_max_heads));
  L.gcoef = take(sizeof(float) * (2 * static_cast<size_t>(P->dcoef) + P->dcoef / 256));
  P->stat_blocks = std::max(1, std::min(2 * P->n_sms, (T + 63) / 64));
  L.stat_part = take(sizeof(float) * 4 * static_cast<size_t>(P->stat_blocks) * d.d);
  L.stat_nvis = take(sizeof(int32_t) * static_cast<size_t>(P->stat_blocks));
  L.stat_n0 = take(sizeof(double) * 2);
  L.gmmcoef = take(sizeof(float) * kGmmMaxForms * (2 * static_cast<size_t>(P->dcoef) + P->dcoef / 256));
  L.bal_f = take(sizeof(float) * E);
  L.bal_a = take(sizeof(float) * K);
  L.bal_h = take(sizeof(float) * static_cast<size_t>(P->stat_blocks) * E);
  L.bal_s = take(sizeof(int32_t) * static_cast<size_t>(P->stat_blocks) * E);
  L.bal_u = take(sizeof(int32_t) * static_cast<size_t>(P->stat_blocks) * K);
  L.f32_part = take(d.dtype == SMOES_F32 ? sizeof(float) * static_cast<size_t>(P->n_groups) *
                                               f32_chunks(d.d) * (E + 1) * 128 : 0);
  L.total = o;
  *out = P;
  return SMOES_OK;
}

void smoes_plan_destroy(smoes_plan plan) { delete plan; }

smoes_status smoes_plan_set_wait_limit(smoes_plan plan, uint64_t limit_ns) {
  if (!plan) return SMOES_ERR_INVALID_ARG;
  plan->limit_ns = limit_ns ? limit_ns : kWaitLimitNs;
  return SMOES_OK;
}

size_t smoes_workspace_bytes(smoes_plan plan) { return plan ? plan->L.total : 0; }

smoes_status smoes_workspace_init(smoes_plan P, void* ws, size_t ws_bytes, cudaStream_t stream) {
  if (!P) return SMOES_ERR_INVALID_ARG;
  smoes_status st = check_ws(P, ws, ws_bytes);
  if (st != SMOES_OK) return st;
  uint8_t* b = static_cast<uint8_t*>(ws);
  const Layout& L = P->L;
  const int B = P->desc.n_samples, E = P->desc.E, T = P->desc.T;
  cudaError_t e = cudaMemsetAsync(b, 0, L.header_bytes, stream);
  auto up = [&](size_t off, const std::vector<int32_t>& v, size_t n) {
    if (e == cudaSuccess && n > 0)
      e = cudaMemcpyAsync(b + off, v.data(), n * sizeof(int32_t), cudaMemcpyHostToDevice, stream);
  };
  up(L.offsets, P->offsets, B + 1);
  up(L.token_sample, P->token_sample, T);
  up(L.expert_bin, P->expert_bin, E);
  up(L.expert_slot, P->expert_slot, E);
  up(L.piece_base, P->piece_base, P->n_groups + 1);
  up(L.sample_pieces, P->sample_pieces, B + 1);
  if (e == cudaSuccess) e = cudaStreamSynchronize(stream);   // host vectors must outlive the copies
  return cuda_status(e);
}

int smoes_call_launches(smoes_plan P, smoes_call call) {
  if (!P) return -1;
  const smoes_router_desc& d = P->desc;
  const int any = d.T > 0 ? 1 : 0;
  switch (call) {
    case SMOES_CALL_ROUTER_FWD: return any;
    case SMOES_CALL_ROUTER_FWD_PERMUTE: return any ? (fuse_permute(P) ? 1 : 2) : 0;
    case SMOES_CALL_ROUTER_BWD: return any ? (d.dtype == SMOES_BF16 ? 3 : 2) : 0;  // (dz prep,) main, dW sum
    case SMOES_CALL_BIN_PERMUTE: return any;
    case SMOES_CALL_ATTN_SCORE: return any;
  }
  return -1;
}

smoes_status smoes_read_device_status(smoes_plan P, const void* ws, cudaStream_t stream,
                                      int32_t* n_absent) {
  if (!P || !ws) return SMOES_ERR_INVALID_ARG;
  uint32_t h[4] = {0, 0, 0, 0};
  cudaError_t e = cudaStreamSynchronize(stream);
  if (e == cudaSuccess)
    e = cudaMemcpy(h, static_cast<const uint8_t*>(ws) + P->L.status, sizeof(h), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return SMOES_ERR_CUDA;
  if (n_absent) *n_absent = static_cast<int32_t>(h[1]);
  if (h[0] & kStatusTimeout) return SMOES_ERR_DEVICE_TIMEOUT;
  if (h[0] & kStatusData) return SMOES_ERR_DATA;
  return SMOES_OK;
}

smoes_status smoes_modality_score(smoes_plan P, smoes_score_mode mode, const smoes_score_args* args,
                                  float* M, void* ws, size_t ws_bytes, cudaStream_t stream) {
  if (!P || !args || !M) return SMOES_ERR_INVALID_ARG;
  smoes_status st = check_ws(P, ws, ws_bytes);
  if (st != SMOES_OK) return st;
  if (!aligned16(M)) return SMOES_ERR_ALIGNMENT;
  const smoes_router_desc& d = P->desc;
  WsView v = make_view(P, ws);
  if (mode == SMOES_SCORE_GAUSS) {
    const smoes_gauss_args& g = args->gauss;
    if (!g.X || !g.mu || !g.var) return SMOES_ERR_INVALID_ARG;
    if (!aligned16(g.X)) return SMOES_ERR_ALIGNMENT;
    if (d.T == 0) return SMOES_OK;
    GaussParams p{};
    p.T = d.T;
    p.d = d.d;
    p.X = g.X;
    p.gcoef = v.gcoef;
    p.dcoef = v.dcoef;
    p.inv_tau = 1.f / (g.tau > 0.f ? g.tau : 0.5f * d.d);
    p.M = M;
    p.status = v.status;
    cudaError_t e = launch_gauss_coef(g.mu, g.var, d.d, v.dcoef, v.gcoef, v.status, stream);
    if (e == cudaSuccess) e = launch_gauss_score(p, d.dtype, P->n_sms, stream);
    return cuda_status(e);
  }
  if (mode == SMOES_SCORE_GMM) {
    const smoes_gmm_args& g = args->gmm;
    if (!g.X || !g.log_pi || !g.mu || !g.var) return SMOES_ERR_INVALID_ARG;
    if (g.n_components < 1) return SMOES_ERR_INVALID_ARG;
    if (g.n_components > kGmmMaxComponents) return SMOES_ERR_UNSUPPORTED;
    // the forms' coefficients stay in shared memory: 2 (2C - 1) round_up(d, 256) floats + padding
    if (sizeof(float) * 2 * (2 * g.n_components - 1) * static_cast<size_t>(round_up(d.d, 256) / 8 * 9) > 227u * 1024u)
      return SMOES_ERR_UNSUPPORTED;
    if (!aligned16(g.X)) return SMOES_ERR_ALIGNMENT;
    if (d.T == 0) return SMOES_OK;
    GmmParams p{};
    p.T = d.T;
    p.d = d.d;
    p.C = g.n_components;
    p.F = 2 * g.n_components - 1;
    p.dcoef = v.dcoef;
    p.X = g.X;
    p.log_pi = g.log_pi;
    p.mu = g.mu;
    p.var = g.var;
    p.inv_tau = 1.f / (g.tau > 0.f ? g.tau : 0.5f * d.d);
    p.coef = reinterpret_cast<float*>(static_cast<uint8_t*>(ws) + P->L.gmmcoef);
    p.M = M;
    p.status = v.status;
    return cuda_status(launch_gmm_score(p, d.dtype, P->n_sms, stream));
  }
  if (mode == SMOES_SCORE_ATTN) {
    const smoes_attn_args& a = args->attn;
    if (!a.Q || !a.K || a.B < 1 || a.H < 1 || a.S < 1) return SMOES_ERR_INVALID_ARG;
    if (static_cast<long long>(a.B) * a.S != d.T) return SMOES_ERR_INVALID_ARG;
    if ((a.is_vision == nullptr) == (a.m_prev == nullptr)) return SMOES_ERR_INVALID_ARG;
    if ((a.xattn_norm == nullptr) != (a.x_norm == nullptr)) return SMOES_ERR_INVALID_ARG;
    if (a.hd != 128) return SMOES_ERR_UNSUPPORTED;
    if (a.H > d.attn_max_heads) return SMOES_ERR_WORKSPACE;
    if (!aligned16(a.Q) || !aligned16(a.K)) return SMOES_ERR_ALIGNMENT;
    AttnParams p{};
    p.B = a.B;
    p.H = a.H;
    p.S = a.S;
    p.hd = a.hd;
    p.T = d.T;
    p.Q = a.Q;
    p.K = a.K;
    p.is_vision = a.is_vision;
    p.m_prev = a.m_prev;
    p.key_bias = a.key_bias;
    p.scale_log2 = a.sm_scale * 1.4426950408889634f;
    p.causal = a.causal ? 1 : 0;
    p.xattn_norm = a.xattn_norm;
    p.x_norm = a.x_norm;
    p.M = M;
    p.part = v.attn_part;
    p.ticket = v.attn_ticket;
    p.status = v.status;
    p.n_qtiles = (a.S + 127) / 128;
    p.n_items = a.B * p.n_qtiles * a.H;
    p.limit_ns = P->limit_ns;
    CUtensorMap tq, tk;
    const uint64_t rows = static_cast<uint64_t>(a.B) * a.H * a.S;
    if (!encode_bf16_2d(&tq, a.Q, rows, a.hd, 128, 64, true) ||
        !encode_bf16_2d(&tk, a.K, rows, a.hd, 128, 64, true))
      return SMOES_ERR_CUDA;
    const cudaError_t e = launch_attn_mass(p, tq, tk, P->n_sms, stream);
    if (e == cudaErrorNotSupported) return SMOES_ERR_UNSUPPORTED;
    return cuda_status(e);
  }
  return SMOES_ERR_INVALID_ARG;
}

smoes_status smoes_attention_fwd(smoes_plan P, const smoes_attn_args* args, const void* V,
                                 int n_kv_heads, void* O, float* M, void* ws, size_t ws_bytes,
                                 cudaStream_t stream) {
  if (!P || !args || !M || !O || !V) return SMOES_ERR_INVALID_ARG;
  smoes_status st = check_ws(P, ws, ws_bytes);
  if (st != SMOES_OK) return st;
  const smoes_router_desc& d = P->desc;
  const smoes_attn_args& a = *args;
  if (!a.Q || !a.K || a.B < 1 || a.H < 1 || a.S < 1 || n_kv_heads < 1) return SMOES_ERR_INVALID_ARG;
  if (static_cast<long long>(a.B) * a.S != d.T) return SMOES_ERR_INVALID_ARG;
  if ((a.is_vision == nullptr) == (a.m_prev == nullptr)) return SMOES_ERR_INVALID_ARG;
  if ((a.xattn_norm == nullptr) != (a.x_norm == nullptr)) return SMOES_ERR_INVALID_ARG;
  if (a.H % n_kv_heads != 0) return SMOES_ERR_INVALID_ARG;
  if (a.hd != 128 || a.S % 128 != 0) return SMOES_ERR_UNSUPPORTED;
  if (a.H > d.attn_max_heads) return SMOES_ERR_WORKSPACE;
  if (!aligned16(a.Q) || !aligned16(a.K) || !aligned16(V) || !aligned16(O) || !aligned16(M) ||
      (a.key_bias && !aligned16(a.key_bias)) || (a.is_vision && !aligned16(a.is_vision)) ||
      (a.m_prev && !aligned16(a.m_prev)))
    return SMOES_ERR_ALIGNMENT;
  WsView v = make_view(P, ws);
  AttnFwdParams fp{};
  AttnParams& p = fp.a;
  p.B = a.B;
  p.H = a.H;
  p.S = a.S;
  p.hd = a.hd;
  p.T = d.T;
  p.Q = a.Q;
  p.K = a.K;
  p.is_vision = a.is_vision;
  p.m_prev = a.m_prev;
  p.key_bias = a.key_bias;
  p.scale_log2 = a.sm_scale * 1.4426950408889634f;
  p.causal = a.causal ? 1 : 0;
  p.xattn_norm = a.xattn_norm;
  p.x_norm = a.x_norm;
  p.M = M;
  p.part = v.attn_part;
  p.ticket = v.attn_ticket;
  p.status = v.status;
  p.n_qtiles = a.S / 128;
  p.n_items = a.B * a.H * p.n_qtiles;
  p.limit_ns = P->limit_ns;
  fp.Hkv = n_kv_heads;
  CUtensorMap tq, tk, tv, to;
  const uint64_t rq = static_cast<uint64_t>(a.B) * a.H * a.S, rk = static_cast<uint64_t>(a.B) * n_kv_heads * a.S;
  if (!encode_bf16_2d(&tq, a.Q, rq, a.hd, 128, 64, true) || !encode_bf16_2d(&tk, a.K, rk, a.hd, 128, 64, true) ||
      !encode_bf16_2d(&tv, V, rk, a.hd, 128, 64, true) || !encode_bf16_2d(&to, O, rq, a.hd, 128, 64, true))
    return SMOES_ERR_CUDA;
  const cudaError_t e = launch_attn_fwd(fp, tq, tk, tv, to, P->n_sms, stream);
  if (e == cudaErrorNotSupported) return SMOES_ERR_UNSUPPORTED;
  return cuda_status(e);
}

smoes_status smoes_router_fwd(smoes_plan P, const void* X, const void* W, const float* M_in,
                              const smoes_gauss_args* gauss, float* M_out, int32_t* topk_idx,
                              float* topk_w, float* bin_prob, float* joint, float* mi, float* loss,
                              void* ws, size_t ws_bytes, cudaStream_t stream) {
  return router_fwd(P, X, W, M_in, gauss, M_out, topk_idx, topk_w, bin_prob, joint, mi, loss,
                    nullptr, ws, ws_bytes, stream);
}

smoes_status smoes_router_fwd_permute(smoes_plan P, const void* X, const void* W, const float* M_in,
                                      const smoes_gauss_args* gauss, float* M_out,
                                      int32_t* topk_idx, float* topk_w, float* bin_prob,
                                      float* joint, float* mi, float* loss, const int32_t* home,
                                      const uint8_t* is_vision, int32_t* bin_offsets,
                                      int32_t* perm_token, uint32_t* perm_mask, int32_t* dispatch,
                                      int32_t* expert_counts, void* ws, size_t ws_bytes,
                                      cudaStream_t stream) {
  if (!P) return SMOES_ERR_INVALID_ARG;
  const smoes_router_desc& d = P->desc;
  if (!bin_offsets || !dispatch) return SMOES_ERR_INVALID_ARG;
  if (expert_counts && !is_vision) return SMOES_ERR_INVALID_ARG;
  if (d.T > 0 && (!perm_token || !perm_mask)) return SMOES_ERR_INVALID_ARG;
  // inside the forward launch when fuse_permute(P); otherwise the two calls in order
  if (fuse_permute(P)) {
    FusedPerm f{};
    f.home = home;
    f.is_vision = is_vision;
    f.bin_offsets = bin_offsets;
    f.perm_token = perm_token;
    f.perm_mask = perm_mask;
    f.dispatch = dispatch;
    f.expert_counts = expert_counts;
    return router_fwd(P, X, W, M_in, gauss, M_out, topk_idx, topk_w, bin_prob, joint, mi, loss,
                      &f, ws, ws_bytes, stream);
  }
  smoes_status st = router_fwd(P, X, W, M_in, gauss, M_out, topk_idx, topk_w, bin_prob, joint, mi,
                               loss, nullptr, ws, ws_bytes, stream);
  if (st != SMOES_OK) return st;
  return smoes_bin_permute(P, topk_idx, home, is_vision, bin_offsets, perm_token, perm_mask,
                           dispatch, expert_counts, ws, ws_bytes, stream);
}

smoes_status smoes_router_bwd(smoes_plan P, const void* X, const void* W, const float* M,
                              const int32_t* topk_idx, const float* d_topk_w, float loss_scale,
                              float* dW, int accumulate_dW, void* dX, float* dlogits, void* ws,
                              size_t ws_bytes, cudaStream_t stream) {
  if (!P) return SMOES_ERR_INVALID_ARG;
  smoes_status st = check_ws(P, ws, ws_bytes);
  if (st != SMOES_OK) return st;
  const smoes_router_desc& d = P->desc;
  if (!dW) return SMOES_ERR_INVALID_ARG;
  if (d.T == 0) {
    if (accumulate_dW) return SMOES_OK;
    return cuda_status(cudaMemsetAsync(dW, 0, sizeof(float) * static_cast<size_t>(d.E) * d.d, stream));
  }
  if (!X || !W || !M) return SMOES_ERR_INVALID_ARG;
  if ((d_topk_w || d.mi_topk_mask) && !topk_idx) return SMOES_ERR_INVALID_ARG;
  if (!aligned16(X) || !aligned16(W) || !aligned16(M) || !aligned16(dW) || (dX && !aligned16(dX)))
    return SMOES_ERR_ALIGNMENT;
  if (d.dtype == SMOES_BF16 && d.E > 128) return SMOES_ERR_UNSUPPORTED;
  if (d.dtype == SMOES_F32 && d.E > 64) return SMOES_ERR_UNSUPPORTED;

  BwdParams p{};
  p.dm = make_dims(P);
  p.ws = make_view(P, ws);
  p.X = X;
  p.W = W;
  p.M = M;
  p.topk_idx = topk_idx;
  p.d_topk_w = d_topk_w;
  p.scale = -loss_scale / static_cast<float>(d.n_samples);
  p.dX = dX;
  p.dlogits = dlogits;
  p.dW = dW;
  p.accumulate = accumulate_dW ? 1 : 0;
  p.groups = P->bwd_groups;
  p.slices = P->bwd_slices;
  p.slice_width = P->bwd_slice_width;
  p.n_tiles = P->bwd_tiles;
  p.limit_ns = P->limit_ns;
  p.balance_armed = P->balance_armed ? 1 : 0;
  cudaError_t e;
  if (d.dtype == SMOES_BF16) {
    const int E_pad = round_up(d.E, 64);
    CUtensorMap tx, tw, tdx;
    if (!encode_bf16_2d(&tx, X, d.T, d.d, kBwdBT, 64, true) ||
        !encode_bf16_2d(&tw, W, d.E, d.d, E_pad, 64, true))
      return SMOES_ERR_CUDA;
    if (dX) {
      if (!encode_bf16_2d(&tdx, dX, d.T, d.d, kBwdBT, kBwdBD, false)) return SMOES_ERR_CUDA;
    } else {
      tdx = tx;   // unused
    }
    e = launch_dz_prep(p, stream);
    if (e == cudaSuccess) e = launch_router_bwd_bf16(p, tx, tw, tdx, stream);
  } else {
    e = launch_router_bwd_f32(p, stream);
  }
  if (e == cudaSuccess) e = launch_dw_reduce(p, stream);
  return cuda_status(e);
}

smoes_status smoes_bin_permute(smoes_plan P, const int32_t* topk_idx, const int32_t* home,
                               const uint8_t* is_vision, int32_t* bin_offsets, int32_t* perm_token,
                               uint32_t* perm_mask, int32_t* dispatch, int32_t* expert_counts,
                               void* ws, size_t ws_bytes, cudaStream_t stream) {
  if (!P) return SMOES_ERR_INVALID_ARG;
  smoes_status st = check_ws(P, ws, ws_bytes);
  if (st != SMOES_OK) return st;
  const smoes_router_desc& d = P->desc;
  if (!bin_offsets || !dispatch) return SMOES_ERR_INVALID_ARG;
  if (expert_counts && !is_vision) return SMOES_ERR_INVALID_ARG;
  if (d.T == 0) {
    cudaError_t e = cudaMemsetAsync(bin_offsets, 0, sizeof(int32_t) * (d.n_bins + 1), stream);
    if (e == cudaSuccess) e = cudaMemsetAsync(dispatch, 0, sizeof(int32_t) * d.n_bins * d.n_bins, stream);
    if (e == cudaSuccess && expert_counts) e = cudaMemsetAsync(expert_counts, 0, sizeof(int32_t) * 2 * d.E, stream);
    return cuda_status(e);
  }
  if (!topk_idx || !perm_token || !perm_mask) return SMOES_ERR_INVALID_ARG;
  WsView v = make_view(P, ws);
  PermParams p{};
  p.T = d.T;
  p.k = d.k;
  p.E = d.E;
  p.K = d.n_bins;
  p.topk_idx = topk_idx;
  p.home = home;
  p.is_vision = is_vision;
  p.expert_bin = v.expert_bin;
  p.expert_slot = v.expert_slot;
  p.bin_offsets = bin_offsets;
  p.perm_token = perm_token;
  p.perm_mask = perm_mask;
  p.dispatch = dispatch;
  p.expert_counts = expert_counts;
  p.blk_counts = v.perm_scratch;
  p.sync = reinterpret_cast<uint32_t*>(static_cast<uint8_t*>(ws) + P->L.perm_sync);
  p.status = v.status;
  p.n_blocks = P->perm_nblocks;
  p.rounds = perm_rounds(d.T, d.k);
  p.limit_ns = P->limit_ns;
  return cuda_status(launch_bin_permute(p, stream));
}

smoes_status smoes_gaussian_stats_update(smoes_plan P, const void* X, const uint8_t* is_vision,
                                         double beta, double* N, double* S_mu, double* S_var,
                                         float* mu, float* var, void* ws, size_t ws_bytes,
                                         cudaStream_t stream) {
  if (!P) return SMOES_ERR_INVALID_ARG;
  smoes_status st = check_ws(P, ws, ws_bytes);
  if (st != SMOES_OK) return st;
  const smoes_router_desc& d = P->desc;
  if (!N || !S_mu || !S_var) return SMOES_ERR_INVALID_ARG;
  if (d.T > 0 && (!X || !is_vision)) return SMOES_ERR_INVALID_ARG;
  if (!(beta >= 0.0 && beta <= 1.0)) return SMOES_ERR_INVALID_ARG;
  if ((X && !aligned16(X)) || !aligned16(N) || !aligned16(S_mu) || !aligned16(S_var) ||
      (mu && !aligned16(mu)) || (var && !aligned16(var)))
    return SMOES_ERR_ALIGNMENT;
  uint8_t* b = static_cast<uint8_t*>(ws);
  StatsParams p{};
  p.T = d.T;
  p.d = d.d;
  p.G = P->stat_blocks;
  p.X = X;
  p.is_vision = is_vision;
  p.beta = beta;
  p.N = N;
  p.S_mu = S_mu;
  p.S_var = S_var;
  p.mu_out = mu;
  p.var_out = var;
  p.part = reinterpret_cast<float*>(b + P->L.stat_part);
  p.nvis = reinterpret_cast<int32_t*>(b + P->L.stat_nvis);
  p.N0 = reinterpret_cast<double*>(b + P->L.stat_n0);
  return cuda_status(launch_stats_update(p, d.dtype == SMOES_BF16, stream));
}

smoes_status smoes_bin_balance(smoes_plan P, const int32_t* topk_idx, float loss_scale,
                               float* loss_bal, float* f_e, float* P_e, void* ws, size_t ws_bytes,
                               cudaStream_t stream) {
  if (!P || !loss_bal) return SMOES_ERR_INVALID_ARG;
  smoes_status st = check_ws(P, ws, ws_bytes);
  if (st != SMOES_OK) return st;
  const smoes_router_desc& d = P->desc;
  if (d.T == 0) return cuda_status(cudaMemsetAsync(loss_bal, 0, sizeof(float), stream));
  if (!topk_idx) return SMOES_ERR_INVALID_ARG;
  if (!aligned16(topk_idx) || (f_e && !aligned16(f_e)) || (P_e && !aligned16(P_e)))
    return SMOES_ERR_ALIGNMENT;
  uint8_t* b = static_cast<uint8_t*>(ws);
  WsView v = make_view(P, ws);
  BalParams p{};
  p.T = d.T;
  p.E = d.E;
  p.k = d.k;
  p.K = d.n_bins;
  p.N_B = P->N_B;
  p.G = P->stat_blocks;
  p.gsave = v.gsave;
  p.topk_idx = topk_idx;
  p.expert_bin = v.expert_bin;
  p.expert_bin_host = P->expert_bin.data();
  p.scale = loss_scale;
  p.part_h = reinterpret_cast<float*>(b + P->L.bal_h);
  p.part_s = reinterpret_cast<int32_t*>(b + P->L.bal_s);
  p.part_u = reinterpret_cast<int32_t*>(b + P->L.bal_u);
  p.tab_f = v.bal_f;
  p.tab_a = v.bal_a;
  p.flag = v.bal_flag;
  p.loss = loss_bal;
  p.f_out = f_e;
  p.P_out = P_e;
  const smoes_status r = cuda_status(launch_bin_balance(p, stream));
  if (r == SMOES_OK) P->balance_armed = true;
  return r;
}

smoes_status smoes_adaptive_bins(smoes_plan P, const int32_t* expert_counts, double beta,
                                 double* C_bar, int32_t* expert_bin, double* f_spec,
                                 cudaStream_t stream) {
  if (!P || !expert_counts || !C_bar || !expert_bin) return SMOES_ERR_INVALID_ARG;
  if (!(beta >= 0.0 && beta <= 1.0)) return SMOES_ERR_INVALID_ARG;
  if (!aligned16(expert_counts) || !aligned16(C_bar) || !aligned16(expert_bin) ||
      (f_spec && !aligned16(f_spec)))
    return SMOES_ERR_ALIGNMENT;
  BinsParams p{};
  p.E = P->desc.E;
  p.N_B = P->N_B;
  p.beta = beta;
  p.counts = expert_counts;
  p.C_bar = C_bar;
  p.expert_bin = expert_bin;
  p.f_spec = f_spec;
  return cuda_status(launch_adaptive_bins(p, stream));
}

}  // extern "C"

extern "C" smoes_status smoes_bin_permute_noalloc(smoes_plan P, const int32_t* topk_idx,
                                                  const int32_t* home, const uint8_t* is_vision,
                                                  int32_t* bin_offsets, int32_t* perm_token,
                                                  uint32_t* perm_mask, int32_t* dispatch,
                                                  int32_t* expert_counts, cudaStream_t stream) {
  if (!P) return SMOES_ERR_INVALID_ARG;
  const smoes_router_desc& d = P->desc;
  if (!bin_offsets || !dispatch) return SMOES_ERR_INVALID_ARG;
  if (expert_counts && !is_vision) return SMOES_ERR_INVALID_ARG;
  if (P->perm_nblocks > kStaticPermBlocks || d.n_bins > kMaxBins || d.E > kMaxExperts)
    return SMOES_ERR_UNSUPPORTED;                  // beyond the fixed scratch
  if (d.T == 0) {
    cudaError_t e = cudaMemsetAsync(bin_offsets, 0, sizeof(int32_t) * (d.n_bins + 1), stream);
    if (e == cudaSuccess) e = cudaMemsetAsync(dispatch, 0, sizeof(int32_t) * d.n_bins * d.n_bins, stream);
    if (e == cudaSuccess && expert_counts) e = cudaMemsetAsync(expert_counts, 0, sizeof(int32_t) * 2 * d.E, stream);
    return cuda_status(e);
  }
  if (!topk_idx || !perm_token || !perm_mask) return SMOES_ERR_INVALID_ARG;
  StaticPermScratch* sp = nullptr;
  cudaError_t e = static_perm_scratch(&sp);
  if (e != cudaSuccess) return SMOES_ERR_CUDA;
  // the plan's bin map and slots into the scratch (kernel parameters, by value: nothing on the
  // host is read after this call returns); the status and barrier words start at zero
  e = launch_static_perm_prep(sp, P->expert_bin.data(), P->expert_slot.data(), d.E, stream);
  if (e != cudaSuccess) return SMOES_ERR_CUDA;
  PermParams p{};
  p.T = d.T;
  p.k = d.k;
  p.E = d.E;
  p.K = d.n_bins;
  p.topk_idx = topk_idx;
  p.home = home;
  p.is_vision = is_vision;
  p.expert_bin = sp->expert_bin;
  p.expert_slot = sp->expert_slot;
  p.bin_offsets = bin_offsets;
  p.perm_token = perm_token;
  p.perm_mask = perm_mask;
  p.dispatch = dispatch;
  p.expert_counts = expert_counts;
  p.blk_counts = sp->blk_counts;
  p.sync = sp->sync;
  p.status = sp->status;
  p.n_blocks = P->perm_nblocks;
  p.rounds = perm_rounds(d.T, d.k);
  p.limit_ns = P->limit_ns;
  return cuda_status(launch_bin_permute(p, stream));
}
