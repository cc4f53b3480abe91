"""GPU parity of the router variants against the fp64 oracle: the sigmoid gate with a selection
bias (the Moonlight-MoE router of the paper's backbone table) and the top-k-masked reading of g in
eq. (12), alone and together, on bf16 and fp32 plans, with the fused permutation, an upstream
top-k weight gradient and the bin-level balance term.

The choice is compared bit for bit on tokens whose top-(k+1) selection keys (s + bias for the
sigmoid gate) are at least 1e-3 apart; everything after it is compared stage-wise on the GPU's
own choice (the masked bin sums, the MI and the gradients depend on it).
"""
import numpy as np
import pytest
import torch

from oracle import smoes_oracle as O
from paper_2604_23996_gb300.workloads import random_router_case

from .parity import (TIE_GAP, assert_bf16_close, assert_scalar_close, assert_tensor_close,
                     dx_operand_bound, tie_free_tokens)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def bd():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2604_23996_gb300 import binding
    return binding


CASES = {
    # name: (seed, T, d, E, k, K, lengths, dtype, gate, bias, mask, permuted bins, upstream, balance)
    "sigmoid_bias": (101, 1300, 256, 64, 6, 8, [600, 700], torch.bfloat16, 1, True, 0, False, False, False),
    "sigmoid_masked_e128": (102, 900, 192, 128, 8, 16, [400, 500], torch.bfloat16, 1, False, 1, False, False, False),
    "softmax_masked_perm": (103, 1000, 128, 48, 5, 6, [300, 700], torch.bfloat16, 0, False, 1, True, False, False),
    "sigmoid_bias_masked_fp32": (104, 700, 136, 32, 4, 4, [350, 350], torch.float32, 1, True, 1, False, False, False),
    "sigmoid_upstream": (105, 800, 128, 64, 6, 8, [800], torch.bfloat16, 1, True, 0, False, True, False),
    "sigmoid_balance": (106, 900, 128, 64, 6, 8, [450, 450], torch.bfloat16, 1, True, 0, False, False, True),
    "masked_upstream_fp32": (107, 500, 96, 16, 3, 4, [500], torch.float32, 0, False, 1, False, True, False),
}


@pytest.mark.parametrize("name", list(CASES))
def test_variant_parity(bd, name):
    seed, T, d, E, k, K, lens, dt, gate, use_bias, mask, perm, upstream, balance = CASES[name]
    wl = random_router_case(seed, T, d, E, k, K, lens, dtype=dt, aligned=True)
    rng = np.random.default_rng(seed)
    if perm:
        wl.expert_bin = rng.permutation(wl.expert_bin).astype(np.int32)
    bias = (0.05 * rng.standard_normal(E)).astype(np.float32) if use_bias else None
    dev = "cuda"
    bias_t = None if bias is None else torch.from_numpy(bias).to(dev)
    code = bd.SMOES_BF16 if dt == torch.bfloat16 else bd.SMOES_F32
    r = bd.Router(wl.T, wl.d, wl.E, wl.k, wl.n_bins, wl.sample_offsets, wl.expert_bin, code,
                  gate=gate, score_bias=bias_t, mi_topk_mask=mask)
    X, W = wl.X.to(dev), wl.W.to(dev)
    isv = torch.from_numpy(wl.is_vision).to(dev)
    r.forward_permute(X, W, mu=wl.mu.to(dev), var=wl.var.to(dev), tau=wl.tau, is_vision=isv)
    s_mi, s_bal = 0.9, 1.1
    if balance:
        lb = torch.empty(1, device=dev)
        assert bd.smoes_bin_balance(r.plan, r.topk_idx, s_bal, lb, r.ws) == 0
    dtw = (1e-3 * rng.standard_normal((T, k))).astype(np.float32) if upstream else None
    dW = torch.empty((E, d), device=dev)
    dX = torch.empty_like(X)
    dl = torch.empty((T, E), device=dev)
    r.backward(X, W, r.M, dW, dX=dX, dlogits=dl, loss_scale=s_mi,
               d_topk_w=None if dtw is None else torch.from_numpy(dtw).to(dev))
    assert r.device_status()[0] == 0
    torch.cuda.synchronize()
    g_idx = r.topk_idx.cpu().numpy()

    Xd, Wd = wl.X.double().numpy(), wl.W.double().numpy()
    M = O.gaussian_score(Xd, wl.mu.double().numpy(), wl.var.double().numpy(), wl.tau)
    gname = "sigmoid" if gate else "softmax"
    own = O.router_forward_variant(Xd, Wd, M, wl.expert_bin, K, wl.sample_offsets, k, gate=gname,
                                   score_bias=bias, mask=bool(mask))
    key = own["s"] + (0.0 if bias is None else bias[None, :]) if gate else own["z"]
    ok = tie_free_tokens(key, k)
    np.testing.assert_array_equal(g_idx[ok], own["topk_idx"][ok], err_msg="top-k")
    # stage-wise from here: the oracle on the GPU's own choice
    f = O.router_forward_variant(Xd, Wd, M, wl.expert_bin, K, wl.sample_offsets, k, gate=gname,
                                 score_bias=bias, mask=bool(mask), topk_idx=g_idx)
    assert_tensor_close(r.topk_w.cpu().numpy(), f["topk_w"], "topk_w")
    assert_tensor_close(r.bin_prob.cpu().numpy(), f["p"], "bin_prob")
    assert_scalar_close(r.mi.cpu().numpy()[:wl.B], f["mi"], "mi")
    assert_scalar_close(r.loss.item(), f["loss"], "loss")
    dz, _, _ = O.router_backward_variant(Xd, Wd, M, f, wl.expert_bin, wl.sample_offsets, s_mi)
    if upstream:
        dz = dz + (O.sigmoid_topk_weight_grad_logits(f["s"], g_idx, dtw) if gate
                   else O.topk_weight_grad_logits(f["g"], g_idx, dtw, False))
    if balance:
        dg = O.bin_balance_grad_gate(f["g"], g_idx, wl.expert_bin, K, s_bal)
        dz = dz + (O.sigmoid_grad_logits(f["s"], dg) if gate else O.softmax_grad_logits(f["g"], dg))
    assert_tensor_close(dl.cpu().numpy(), dz, "dlogits")
    assert_tensor_close(dW.cpu().numpy(), dz.T @ Xd, "dW")
    if dt == torch.bfloat16:
        assert_bf16_close(dX.float().cpu().numpy(), dz @ Wd, "dX", operand_bound=dx_operand_bound(dz, Wd))
    else:
        assert_tensor_close(dX.cpu().numpy(), dz @ Wd, "dX")
    pr = O.bin_permute(g_idx, wl.expert_bin, K, is_vision=wl.is_vision)
    n = int(r.bin_offsets[-1].item())
    np.testing.assert_array_equal(r.bin_offsets.cpu().numpy(), pr["offsets"])
    np.testing.assert_array_equal(r.perm_token[:n].cpu().numpy(), pr["perm"])
    print(f"{name}: {int((~ok).sum())} near-tie tokens of {T}; loss {r.loss.item():.4e}")


def test_variant_plan_arguments(bd):
    eb = np.arange(16) // 4
    b = torch.zeros(16, device="cuda")
    assert bd.smoes_plan_create(100, 64, 16, 2, 4, [0, 100], eb, bd.SMOES_BF16, gate=2)[0] == -1
    assert bd.smoes_plan_create(100, 64, 16, 2, 4, [0, 100], eb, bd.SMOES_BF16, score_bias=b)[0] == -1
    code, plan = bd.smoes_plan_create(100, 64, 16, 2, 4, [0, 100], eb, bd.SMOES_BF16, gate=1, score_bias=b,
                                      mi_topk_mask=1)
    assert code == 0
    bd.smoes_plan_destroy(plan)
