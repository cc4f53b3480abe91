"""Parity at the full workload sizes, through the same plan and calls bench.py times.

The GPU runs each workload once at full size; the fp64 oracle is evaluated sample by sample
(samples are independent in eqs. 12-15; dW is the sum of the per-sample contributions), so host
memory stays small. Every workload also runs in its aligned variant (tau = 1, bins tilted by
modality), where the MI is far above the absolute floor of the scalar check. For the attention
workload the score is compared on every query and head of the first and the last sequence
(2 of 8 whole sequences; the full fp64 attention of all eight is ~5e11 flops), and its router
stage runs at full size twice: with the hard labels (the layer-0 score of eq. 2) and with the
GPU's own attention score as the provided scores (the score-to-router chain end to end).
"""
import numpy as np
import pytest
import torch

from oracle import smoes_oracle as O
from paper_2604_23996_gb300.workloads import attn_workload, config_workload

from .parity import (REL, assert_bf16_close, assert_scalar_close, assert_tensor_close,
                     assert_valid_topk, dx_operand_bound, tie_free_tokens)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def bd():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2604_23996_gb300 import binding
    return binding


class _Acc:
    """Running ||gpu - ref||^2, ||ref||^2 and max|.| over chunks."""

    def __init__(self):
        self.d2 = self.r2 = self.dmax = self.rmax = 0.0

    def add(self, gpu, ref):
        gpu = np.asarray(gpu, np.float64)
        ref = np.asarray(ref, np.float64)
        self.d2 += float(np.sum((gpu - ref) ** 2))
        self.r2 += float(np.sum(ref ** 2))
        self.dmax = max(self.dmax, float(np.abs(gpu - ref).max()))
        self.rmax = max(self.rmax, float(np.abs(ref).max()))

    def check(self, what, rel=REL):
        r = np.sqrt(self.d2 / self.r2) if self.r2 > 0 else np.sqrt(self.d2)
        assert r <= rel, f"{what}: rel L2 error {r:.3e}"
        assert self.dmax <= rel * self.rmax, f"{what}: max abs error {self.dmax:.3e}"
        return r


def _run_full(bd, wl, M_in=None, fused=True):
    """fused: the permutation comes from the forward call, as bench.py runs the step."""
    dev = "cuda"
    dt = bd.SMOES_BF16 if wl.dtype == torch.bfloat16 else bd.SMOES_F32
    r = bd.Router(wl.T, wl.d, wl.E, wl.k, wl.n_bins, wl.sample_offsets, wl.expert_bin, dt)
    X, W = wl.X.to(dev), wl.W.to(dev)
    isv = torch.from_numpy(wl.is_vision).to(dev)
    fwd = (lambda **kw: r.forward_permute(is_vision=isv, **kw)) if fused else r.forward
    if M_in is None:
        fwd(X=X, W=W, mu=wl.mu.to(dev), var=wl.var.to(dev), tau=wl.tau)
        M = r.M
    else:
        M = torch.from_numpy(M_in).to(dev)
        fwd(X=X, W=W, M_in=M)
    dW = torch.empty((wl.E, wl.d), dtype=torch.float32, device=dev)
    dX = torch.empty_like(X)
    dl = torch.empty((wl.T, wl.E), dtype=torch.float32, device=dev)
    r.backward(X, W, M, dW, dX=dX, dlogits=dl, loss_scale=1.0)
    if not fused:
        r.permute(is_vision=isv)
    assert r.device_status()[0] == 0
    torch.cuda.synchronize()
    n = int(r.bin_offsets[-1].item())
    return dict(M=M.cpu().numpy(), topk_idx=r.topk_idx.cpu().numpy(), topk_w=r.topk_w.cpu().numpy(),
                bin_prob=r.bin_prob.cpu().numpy(), mi=r.mi.cpu().numpy(), loss=float(r.loss.item()),
                dW=dW.cpu().numpy(), dX=dX.float().cpu().numpy(), dl=dl.cpu().numpy(),
                offsets=r.bin_offsets.cpu().numpy(), perm=r.perm_token[:n].cpu().numpy(),
                mask=r.perm_mask[:n].cpu().numpy().view(np.uint32), dispatch=r.dispatch.cpu().numpy(),
                expert_counts=r.expert_counts.cpu().numpy())


def _check_per_sample(wl, g, M_provided=None):
    """Oracle sample by sample; every GPU output compared."""
    offs = wl.sample_offsets
    B = wl.B
    mu, var = wl.mu.double().numpy(), wl.var.double().numpy()
    Wd = wl.W.double().numpy()
    acc = {k: _Acc() for k in ("M", "topk_w", "bin_prob", "dl")}
    dW_ref = np.zeros((wl.E, wl.d))
    dx_acc = _Acc()
    mis = np.zeros(B)
    excluded = 0
    for i in range(B):
        s, e = int(offs[i]), int(offs[i + 1])
        Xd = wl.X[s:e].double().numpy()
        M = (O.gaussian_score(Xd, mu, var, wl.tau) if M_provided is None
             else M_provided[s:e].astype(np.float64))
        one = np.array([0, e - s])
        fwd = O.router_forward(Xd, Wd, M, wl.expert_bin, wl.n_bins, one, wl.k)
        # loss = -(1/B) sum_i I_i: a one-sample oracle call divides by 1, so scale by 1/B
        dz, dW_i, dX_i = O.router_backward(Xd, Wd, M, fwd, wl.expert_bin, one, 1.0 / B)
        mis[i] = fwd["mi"][0]
        acc["M"].add(g["M"][s:e], M)
        ok = tie_free_tokens(fwd["z"], wl.k)
        excluded += int((~ok).sum())
        np.testing.assert_array_equal(g["topk_idx"][s:e][ok], fwd["topk_idx"][ok], err_msg=f"topk s{i}")
        assert_valid_topk(g["topk_idx"][s:e][~ok], fwd["z"][~ok], wl.k)
        acc["topk_w"].add(g["topk_w"][s:e][ok], fwd["topk_w"][ok])
        acc["bin_prob"].add(g["bin_prob"][s:e], fwd["p"])
        acc["dl"].add(g["dl"][s:e], dz)
        dW_ref += dW_i
        if wl.dtype == torch.bfloat16:
            assert_bf16_close(g["dX"][s:e], dX_i, f"dX sample {i}", operand_bound=dx_operand_bound(dz, Wd))
        dx_acc.add(g["dX"][s:e], dX_i)
    for k, a in acc.items():
        a.check(k)
    assert_tensor_close(g["dW"], dW_ref, "dW")
    if wl.dtype != torch.bfloat16:
        dx_acc.check("dX")
    assert_scalar_close(g["mi"][:B], mis, "mi")
    assert_scalar_close(g["loss"], -mis.mean(), "loss")
    pr = O.bin_permute(g["topk_idx"], wl.expert_bin, wl.n_bins, is_vision=wl.is_vision)
    for key in ("offsets", "perm", "dispatch", "expert_counts"):
        np.testing.assert_array_equal(g[key], pr[key], err_msg=key)
    np.testing.assert_array_equal(g["mask"].astype(np.uint64), pr["mask"])
    return excluded


@pytest.mark.parametrize("key", ["tiny_fp32", "dsmoe_vlm", "small_hidden", "large_fine"])
def test_fullsize_router(bd, key):
    wl = config_workload(key)
    g = _run_full(bd, wl)
    excl = _check_per_sample(wl, g)
    print(f"{key}: T={wl.T} tie-excluded tokens {excl}")


def test_fullsize_fused_equals_separate(bd):
    # 256 tiles on at most 152 CTAs: CTAs with two tiles; every output bit for bit
    wl = config_workload("small_hidden")
    a = _run_full(bd, wl, fused=True)
    b = _run_full(bd, wl, fused=False)
    for key in a:
        np.testing.assert_array_equal(np.asarray(a[key]), np.asarray(b[key]), err_msg=key)


@pytest.mark.parametrize("key", ["tiny_fp32", "dsmoe_vlm", "small_hidden", "large_fine"])
def test_fullsize_aligned_variant(bd, key):
    # same shapes, tau = 1 and bins tilted by modality: the MI is far from zero
    wl = config_workload(key, aligned=True)
    g = _run_full(bd, wl)
    _check_per_sample(wl, g)
    assert g["mi"].min() > 1e-7          # 100x above the 1e-9 absolute floor of the MI check


def test_fullsize_attention_workload(bd):
    aw = attn_workload()
    T = aw.B * aw.S
    r = bd.Router(T, 64, 16, 2, 4, [0, T], np.arange(16) // 4, attn_max_heads=aw.H)
    M = torch.empty((T, 2), dtype=torch.float32, device="cuda")
    attn = dict(Q=aw.Q.cuda(), K=aw.K.cuda(), B=aw.B, H=aw.H, S=aw.S, hd=aw.hd, sm_scale=aw.sm_scale,
                causal=1, key_bias=torch.from_numpy(aw.key_bias).cuda(),
                is_vision=torch.from_numpy(aw.is_vision).cuda())
    r.modality_score(bd.SMOES_SCORE_ATTN, M, attn=attn)
    assert r.device_status()[0] == 0
    Mg = M.cpu().numpy()
    got = Mg[:, 0].reshape(aw.B, aw.S)
    np.testing.assert_array_equal(Mg[:, 1], (1.0 - Mg[:, 0]).astype(np.float32))
    m = aw.is_vision.reshape(aw.B, aw.S).astype(np.float64)
    bias = aw.key_bias.reshape(aw.B, aw.S)
    Qd, Kd = aw.Q, aw.K
    for b in (0, aw.B - 1):                  # every query of every head of two whole sequences
        ref = O.attention_vision_mass(Qd[b:b + 1].double().numpy(), Kd[b:b + 1].double().numpy(),
                                      m[b:b + 1], aw.sm_scale, True, bias[b:b + 1])[0]
        assert_tensor_close(got[b], ref, f"attention vision mass, sequence {b} (all queries)")
    # the router stage of this workload at full size, fed the layer-0 hard labels
    wl = config_workload("attn_router")
    Mh = np.stack([wl.is_vision, 1 - wl.is_vision], 1).astype(np.float32)
    g = _run_full(bd, wl, M_in=Mh)
    _check_per_sample(wl, g, M_provided=Mh)
    # and fed the GPU's own attention score: the chain score -> router -> MI -> gradients
    g = _run_full(bd, wl, M_in=np.ascontiguousarray(Mg))
    _check_per_sample(wl, g, M_provided=Mg)
