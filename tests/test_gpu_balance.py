"""GPU parity of the bin-level load-balance loss (Sec. 3.5, eq. 16) and of its gradient, added to
the MI gradient by the backward, against the fp64 oracle.

Stage-wise like the permutation: the oracle evaluates L_bal, f_e, P_e and the gradient on the
GPU's own top-k (the sets U_k and the counts f_e are integer decisions of the forward), with its
own fp64 softmax. Covered: bf16 and fp32 plans, consecutive and permuted bin maps, one bin (the
standard load-balance loss of the preliminaries), a ragged batch, and the arming rule (a new
forward disarms the balance term; a backward after it carries the MI gradient only).
"""
import numpy as np
import pytest
import torch

from oracle import smoes_oracle as O
from paper_2604_23996_gb300.workloads import random_router_case

from .parity import assert_bf16_close, assert_scalar_close, assert_tensor_close, dx_operand_bound

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def bd():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2604_23996_gb300 import binding
    return binding


CASES = {
    # name: (seed, T, d, E, k, n_bins, lengths, dtype, permute bins)
    "bf16_e64": (71, 1300, 256, 64, 6, 8, [600, 700], torch.bfloat16, False),
    "bf16_e128_ragged": (72, 777, 192, 128, 8, 16, [300, 477], torch.bfloat16, False),
    "bf16_permuted_bins": (73, 900, 128, 48, 5, 6, [450, 450], torch.bfloat16, True),
    "bf16_one_bin": (74, 500, 128, 16, 2, 1, [500], torch.bfloat16, False),
    "fp32_e16": (75, 640, 136, 16, 3, 4, [640], torch.float32, False),
    "fp32_permuted_e40": (76, 700, 96, 40, 4, 5, [300, 400], torch.float32, True),
}


def _setup(bd, name):
    seed, T, d, E, k, K, lens, dt, perm = CASES[name]
    wl = random_router_case(seed, T, d, E, k, K, lens, dtype=dt, aligned=True)
    if perm:
        wl.expert_bin = np.random.default_rng(seed).permutation(wl.expert_bin).astype(np.int32)
    code = bd.SMOES_BF16 if dt == torch.bfloat16 else bd.SMOES_F32
    r = bd.Router(wl.T, wl.d, wl.E, wl.k, wl.n_bins, wl.sample_offsets, wl.expert_bin, code)
    return wl, r


@pytest.mark.parametrize("name", list(CASES))
def test_balance_loss_and_gradient(bd, name):
    wl, r = _setup(bd, name)
    dev = "cuda"
    X, W = wl.X.to(dev), wl.W.to(dev)
    r.forward(X, W, mu=wl.mu.to(dev), var=wl.var.to(dev), tau=wl.tau)
    s_mi, s_bal = 0.7, 1.3
    lb = torch.full((1,), float("nan"), device=dev)
    f = torch.empty(wl.E, device=dev)
    P = torch.empty(wl.E, device=dev)
    assert bd.smoes_bin_balance(r.plan, r.topk_idx, s_bal, lb, r.ws, f_e=f, P_e=P) == 0
    dW = torch.empty((wl.E, wl.d), device=dev)
    dX = torch.empty_like(X)
    dl = torch.empty((wl.T, wl.E), device=dev)
    r.backward(X, W, r.M, dW, dX=dX, dlogits=dl, loss_scale=s_mi)
    assert r.device_status()[0] == 0
    torch.cuda.synchronize()
    topk = r.topk_idx.cpu().numpy()

    Xd, Wd = wl.X.double().numpy(), wl.W.double().numpy()
    M = O.gaussian_score(Xd, wl.mu.double().numpy(), wl.var.double().numpy(), wl.tau)
    z = O.gate_logits(Xd, Wd)
    g = O.softmax_gate(z)
    L_ref, parts = O.bin_balance_loss(g, topk, wl.expert_bin, wl.n_bins)
    assert_scalar_close(lb.item(), L_ref, "L_bal")
    np.testing.assert_allclose(f.cpu().numpy(), parts["f"], rtol=1e-6, atol=0)
    assert_tensor_close(P.cpu().numpy(), parts["P"], "P_e")
    fwd = O.router_forward(Xd, Wd, M, wl.expert_bin, wl.n_bins, wl.sample_offsets, wl.k)
    N_B = wl.E // wl.n_bins
    dz = (O.mi_grad_logits(M, fwd["g"], wl.expert_bin, wl.sample_offsets, fwd["tabs"], s_mi, N_B)
          + O.bin_balance_grad_logits(z, topk, wl.expert_bin, wl.n_bins, s_bal))
    assert_tensor_close(dl.cpu().numpy(), dz, "dlogits (MI + balance)")
    assert_tensor_close(dW.cpu().numpy(), dz.T @ Xd, "dW (MI + balance)")
    if wl.dtype == torch.bfloat16:
        assert_bf16_close(dX.float().cpu().numpy(), dz @ Wd, "dX (MI + balance)",
                          operand_bound=dx_operand_bound(dz, Wd))
    else:
        assert_tensor_close(dX.cpu().numpy(), dz @ Wd, "dX (MI + balance)")
    print(f"{name}: L_bal {lb.item():.6f} (oracle {L_ref:.6f})")


def test_a_new_forward_disarms_the_balance_term(bd):
    wl, r = _setup(bd, "bf16_e64")
    dev = "cuda"
    X, W = wl.X.to(dev), wl.W.to(dev)
    mu, var = wl.mu.to(dev), wl.var.to(dev)
    r.forward(X, W, mu=mu, var=var, tau=wl.tau)
    lb = torch.empty(1, device=dev)
    assert bd.smoes_bin_balance(r.plan, r.topk_idx, 5.0, lb, r.ws) == 0
    r.forward(X, W, mu=mu, var=var, tau=wl.tau)           # disarms
    dl = torch.empty((wl.T, wl.E), device=dev)
    dW = torch.empty((wl.E, wl.d), device=dev)
    r.backward(X, W, r.M, dW, dlogits=dl, loss_scale=1.0)
    torch.cuda.synchronize()
    Xd, Wd = wl.X.double().numpy(), wl.W.double().numpy()
    M = O.gaussian_score(Xd, wl.mu.double().numpy(), wl.var.double().numpy(), wl.tau)
    fwd = O.router_forward(Xd, Wd, M, wl.expert_bin, wl.n_bins, wl.sample_offsets, wl.k)
    dz = O.mi_grad_logits(M, fwd["g"], wl.expert_bin, wl.sample_offsets, fwd["tabs"], 1.0,
                          wl.E // wl.n_bins)
    assert_tensor_close(dl.cpu().numpy(), dz, "dlogits (MI only)")


def test_balance_of_an_evenly_loaded_bin_is_one(bd):
    # every token selects all experts of every bin with equal gates (W = 0): f = P = 1/N_B per
    # expert, so each bin contributes N_B * N_B * (1/N_B)^2 = 1 and L_bal = n_bins
    T, d, E, K = 256, 64, 16, 4
    r = bd.Router(T, d, E, E, K, [0, T], np.arange(E) // (E // K))
    X = torch.randn((T, d), device="cuda").to(torch.bfloat16)
    W = torch.zeros((E, d), device="cuda", dtype=torch.bfloat16)
    M = torch.full((T, 2), 0.5, device="cuda")
    r.forward(X, W, M_in=M)
    lb = torch.empty(1, device="cuda")
    assert bd.smoes_bin_balance(r.plan, r.topk_idx, 1.0, lb, r.ws) == 0
    torch.cuda.synchronize()
    assert abs(lb.item() - K) < 1e-5
