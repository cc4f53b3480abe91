"""Seeded synthetic inputs shaped like the paper's MoE-VLM router layers.

This module only draws random numbers and lays out tokens; it holds none of the router's
arithmetic. Both the CUDA path and the fp64 oracle receive exactly the arrays made here (the
oracle widens them to float64).

Recipe (the paper's datasets and checkpoints are not used; these stand in for them):
  * tokens: each sample is one image block followed by its text tokens (576 image tokens per
    image follows CLIP ViT-L/14 at 336 px, Sec. A.1); samples are contiguous.
  * features: x = alpha * mu_v + (1 - alpha) * mu_t + N(0, I), with mu_v, mu_t random unit
    vectors scaled to norm 3; alpha is drawn per token from the workload's Beta law.
  * gate weight W ~ N(0, 0.02^2) (std 0.02), shape [E, d].
  * Gaussian statistics mu[m], var[m]: the plain mean and biased variance of this batch's
    tokens of hard modality m (the paper's EMA statistics after one step from an empty state).
  * bins: consecutive experts, expert_bin[e] = e // N_B.
  * attention workload: q, k ~ N(0, 1) stored in bf16, logit scale 1/sqrt(head_dim), and a
    +0.5 logit bias on vision keys.
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import Optional

import numpy as np
import torch


@dataclass
class RouterWorkload:
    name: str
    T: int
    d: int
    E: int
    k: int
    n_bins: int
    dtype: torch.dtype
    sample_offsets: np.ndarray          # int32 [B+1]
    expert_bin: np.ndarray              # int32 [E]
    is_vision: np.ndarray               # uint8 [T]
    X: torch.Tensor                     # [T, d] in dtype (CPU)
    W: torch.Tensor                     # [E, d] in dtype (CPU)
    mu: torch.Tensor                    # float32 [2, d] (row 0 vision, row 1 text)
    var: torch.Tensor                   # float32 [2, d]
    tau: float
    renorm_topk: int = 0
    seed: int = 0
    extra: dict = field(default_factory=dict)

    @property
    def B(self) -> int:
        return len(self.sample_offsets) - 1


@dataclass
class AttnWorkload:
    B: int
    H: int
    S: int
    hd: int
    Q: torch.Tensor                     # bf16 [B, H, S, hd] (CPU)
    K: torch.Tensor                     # bf16 [B, H, S, hd]
    is_vision: np.ndarray               # uint8 [B*S]
    key_bias: np.ndarray                # float32 [B*S]
    sm_scale: float


def layout(n_image: int, n_text: int, n_samples: int):
    """Token layout: n_samples samples of [n_image image tokens, then n_text text tokens]."""
    per = n_image + n_text
    offs = np.arange(n_samples + 1, dtype=np.int32) * per
    is_vis = np.zeros(per * n_samples, dtype=np.uint8)
    for i in range(n_samples):
        is_vis[i * per:i * per + n_image] = 1
    return offs, is_vis


def _unit(rng, d):
    v = rng.standard_normal(d)
    return v / np.linalg.norm(v)


def _alphas(rng, is_vis, law):
    T = len(is_vis)
    if law == 'beta51':          # vision ~ Beta(5,1), text ~ Beta(1,5)
        a = np.where(is_vis == 1, rng.beta(5.0, 1.0, T), rng.beta(1.0, 5.0, T))
    elif law == 'beta22':        # both modalities ~ Beta(2,2) (mid-layer fusion)
        a = rng.beta(2.0, 2.0, T)
    elif law == 'mix3':          # 0.3 near-pure vision, 0.3 near-pure text, 0.4 cross-modal
        c = rng.choice(3, size=T, p=[0.3, 0.3, 0.4])
        a = np.where(c == 0, rng.beta(20.0, 1.0, T),
                     np.where(c == 1, rng.beta(1.0, 20.0, T), rng.beta(2.0, 2.0, T)))
    else:
        raise ValueError(law)
    return a.astype(np.float32)


def make_features(rng, is_vis, d, law, chunk=8192):
    """x = alpha * mu_v + (1 - alpha) * mu_t + N(0, I) in float32, plus the two means."""
    mu_v = (3.0 * _unit(rng, d)).astype(np.float32)
    mu_t = (3.0 * _unit(rng, d)).astype(np.float32)
    a = _alphas(rng, is_vis, law)
    T = len(is_vis)
    X = np.empty((T, d), dtype=np.float32)
    for s in range(0, T, chunk):
        e = min(T, s + chunk)
        X[s:e] = rng.standard_normal((e - s, d), dtype=np.float32)
        X[s:e] += a[s:e, None] * mu_v[None, :] + (1.0 - a[s:e, None]) * mu_t[None, :]
    return X, mu_v, mu_t


def batch_moments(Xq: torch.Tensor, is_vis: np.ndarray):
    """Per-modality mean and biased variance of the (already quantised) features, float32."""
    mu = np.zeros((2, Xq.shape[1]), dtype=np.float64)
    var = np.zeros((2, Xq.shape[1]), dtype=np.float64)
    sel = [is_vis == 1, is_vis == 0]
    for m in range(2):
        rows = np.nonzero(sel[m])[0]
        acc = np.zeros(Xq.shape[1])
        acc2 = np.zeros(Xq.shape[1])
        for s in range(0, len(rows), 8192):
            blk = Xq[torch.from_numpy(rows[s:s + 8192])].double().numpy()
            acc += blk.sum(axis=0)
            acc2 += (blk * blk).sum(axis=0)
        n = max(len(rows), 1)
        mu[m] = acc / n
        var[m] = np.maximum(acc2 / n - mu[m] ** 2, 1e-6)
    return torch.from_numpy(mu.astype(np.float32)), torch.from_numpy(var.astype(np.float32))


def router_workload(name, T_img, T_txt, n_samples, d, E, k, n_bins, dtype, law, seed,
                    aligned=False, renorm_topk=0, T_override=None):
    """Build one router workload. ``aligned`` is the parity-only variant (tau = 1 and the gate
    weights of the first half of the bins tilted toward mu_v - mu_t) that makes the MI large."""
    rng = np.random.default_rng(seed)
    offs, is_vis = layout(T_img, T_txt, n_samples)
    X32, mu_v, mu_t = make_features(rng, is_vis, d, law)
    W32 = (0.02 * rng.standard_normal((E, d))).astype(np.float32)
    N_B = E // n_bins
    expert_bin = (np.arange(E) // N_B).astype(np.int32)
    tau = 0.5 * d
    if aligned:
        tilt = 0.5 * (mu_v - mu_t) / 3.0
        sign = np.where(expert_bin < n_bins // 2, 1.0, -1.0).astype(np.float32)
        W32 = W32 + sign[:, None] * tilt[None, :]
        tau = 1.0
    X = torch.from_numpy(X32).to(dtype)
    W = torch.from_numpy(W32).to(dtype)
    mu, var = batch_moments(X, is_vis)
    T = len(is_vis)
    return RouterWorkload(name=name, T=T, d=d, E=E, k=k, n_bins=n_bins, dtype=dtype,
                          sample_offsets=offs, expert_bin=expert_bin, is_vision=is_vis, X=X, W=W,
                          mu=mu, var=var, tau=tau, renorm_topk=renorm_topk, seed=seed)


# The five workload shapes (token layout, hidden size, experts, top-k, bins, dtype, alpha law).
CONFIGS = {
    'tiny_fp32':      dict(T_img=2458, T_txt=1638, n_samples=1, d=512, E=16, k=2, n_bins=4,
                           dtype=torch.float32, law='beta51', seed=0),
    'dsmoe_vlm':      dict(T_img=576, T_txt=1472, n_samples=8, d=2048, E=64, k=6, n_bins=8,
                           dtype=torch.bfloat16, law='beta22', seed=1),
    'small_hidden':   dict(T_img=729, T_txt=1319, n_samples=16, d=1280, E=64, k=6, n_bins=8,
                           dtype=torch.bfloat16, law='mix3', seed=2),
    'attn_router':    dict(T_img=1024, T_txt=3072, n_samples=8, d=2048, E=64, k=6, n_bins=8,
                           dtype=torch.bfloat16, law='beta22', seed=3),
    'large_fine':     dict(T_img=1024, T_txt=3072, n_samples=32, d=2048, E=128, k=8, n_bins=16,
                           dtype=torch.bfloat16, law='beta22', seed=4),
}


def config_workload(key: str, aligned: bool = False, n_samples: Optional[int] = None):
    c = dict(CONFIGS[key])
    if n_samples is not None:
        c['n_samples'] = n_samples
    return router_workload(key, aligned=aligned, **c)


def attn_workload(B=8, H=16, S=4096, hd=128, n_image=1024, seed=3, bias=0.5):
    """Attention-score workload: q, k ~ N(0,1) in bf16, image tokens first in each sequence."""
    rng = np.random.default_rng(seed + 1000)
    Q = torch.from_numpy(rng.standard_normal((B, H, S, hd), dtype=np.float32)).to(torch.bfloat16)
    K = torch.from_numpy(rng.standard_normal((B, H, S, hd), dtype=np.float32)).to(torch.bfloat16)
    is_vis = np.zeros(B * S, dtype=np.uint8)
    for b in range(B):
        is_vis[b * S:b * S + n_image] = 1
    key_bias = (bias * is_vis).astype(np.float32)
    return AttnWorkload(B=B, H=H, S=S, hd=hd, Q=Q, K=K, is_vision=is_vis, key_bias=key_bias,
                        sm_scale=1.0 / float(np.sqrt(hd)))


def random_router_case(seed, T, d, E, k, n_bins, sample_lengths, dtype=torch.bfloat16,
                       tau=None, aligned=False, vision_frac=0.3):
    """Small awkward cases for parity tests: arbitrary sample lengths (ragged), T not a multiple
    of the tile size, any E/k/n_bins. Each sample starts with round(vision_frac*len) image tokens."""
    rng = np.random.default_rng(seed)
    offs = np.zeros(len(sample_lengths) + 1, dtype=np.int32)
    offs[1:] = np.cumsum(sample_lengths)
    assert offs[-1] == T
    is_vis = np.zeros(T, dtype=np.uint8)
    for i, L in enumerate(sample_lengths):
        is_vis[offs[i]:offs[i] + int(round(vision_frac * L))] = 1
    X32, mu_v, mu_t = make_features(rng, is_vis, d, 'beta51')
    W32 = (0.02 * rng.standard_normal((E, d))).astype(np.float32)
    expert_bin = (np.arange(E) // (E // n_bins)).astype(np.int32)
    if aligned:
        tilt = 0.5 * (mu_v - mu_t) / 3.0
        sign = np.where(expert_bin < max(n_bins // 2, 1), 1.0, -1.0).astype(np.float32)
        W32 = W32 + sign[:, None] * tilt[None, :]
    X = torch.from_numpy(X32).to(dtype)
    W = torch.from_numpy(W32).to(dtype)
    mu, var = batch_moments(X, is_vis)
    return RouterWorkload(name=f'case{seed}', T=T, d=d, E=E, k=k, n_bins=n_bins, dtype=dtype,
                          sample_offsets=offs, expert_bin=expert_bin, is_vision=is_vis, X=X, W=W,
                          mu=mu, var=var, tau=(1.0 if tau is None and aligned else
                                               (0.5 * d if tau is None else tau)), seed=seed)
