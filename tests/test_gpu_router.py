"""GPU parity of the router forward, backward and permutation (C ABI) against the fp64 oracle.

Small awkward cases cover several tiles with a ragged tail: T not a multiple of the 128/64-token
tiles, d not a multiple of the 64/128-column blocks, E not a multiple of 16, one-token samples,
non-consecutive bin maps, K = 1 and K = E, hard labels with an absent modality, renormalised
top-k with an upstream weight gradient, the fp32 path, and the column splits of the two
epilogue groups.
"""
import numpy as np
import pytest
import torch

from paper_2604_23996_gb300.workloads import random_router_case

from .parity import compare, run_gpu, run_oracle

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def bd():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2604_23996_gb300 import binding
    return binding


CASES = {
    # name: (seed, T, d, E, k, n_bins, sample lengths, dtype, tau/aligned)
    "ragged_aligned": (1, 1000, 256, 64, 6, 8, [300, 450, 250], torch.bfloat16, True),
    "default_tau": (2, 700, 512, 128, 8, 16, [128, 300, 272], torch.bfloat16, False),
    "odd_shapes": (3, 777, 136, 24, 3, 4, [1, 31, 33, 200, 512], torch.bfloat16, True),
    "one_bin": (4, 300, 64, 16, 2, 1, [300], torch.bfloat16, True),
    "bin_per_expert": (5, 260, 128, 16, 4, 16, [100, 160], torch.bfloat16, True),
    "single_token": (6, 1, 64, 16, 2, 4, [1], torch.bfloat16, True),
    "fp32": (7, 600, 128, 16, 2, 4, [600], torch.float32, True),
    "fp32_multi": (8, 333, 72, 32, 5, 8, [10, 200, 123], torch.float32, True),
    # the two epilogue groups: a second group with one 16-column chunk and a partial 32-column
    # staging block; consecutive bins that do not split at the half (group 0 takes all columns);
    # the fp32 kernel with both groups holding columns
    "split_odd_chunks": (9, 650, 256, 80, 5, 5, [330, 320], torch.bfloat16, True),
    "contig_no_split": (10, 500, 192, 96, 6, 8, [250, 250], torch.bfloat16, False),
    "fp32_split": (11, 300, 96, 64, 4, 8, [150, 150], torch.float32, True),
    # the fp32 path splits d into 128-feature chunks: three chunks, the last one partial
    "fp32_chunks": (12, 900, 328, 48, 5, 6, [400, 500], torch.float32, True),
}


@pytest.mark.parametrize("name", list(CASES))
def test_router_gauss_parity(bd, name):
    seed, T, d, E, k, K, lens, dt, aligned = CASES[name]
    wl = random_router_case(seed, T, d, E, k, K, lens, dtype=dt, aligned=aligned)
    g = run_gpu(wl, bd, mode="gauss", loss_scale=0.7)
    ref = run_oracle(wl, mode="gauss", loss_scale=0.7)
    res = compare(wl, g, ref)
    print(f"{name}: tie-excluded tokens {res['tie_excluded']} of {T}; errors "
          + ", ".join(f"{k} {v:.2e}" for k, v in res.items() if k != "tie_excluded"))


def test_provided_soft_scores_upstream_renorm_nonconsecutive_bins(bd):
    wl = random_router_case(21, 513, 192, 48, 5, 6, [200, 113, 200], aligned=True)
    rng = np.random.default_rng(0)
    wl.expert_bin = rng.permutation(wl.expert_bin).astype(np.int32)
    wl.renorm_topk = 1
    Mv = rng.uniform(0.02, 0.98, wl.T)
    M = np.stack([Mv, 1 - Mv], 1).astype(np.float32)
    dtw = rng.standard_normal((wl.T, wl.k)).astype(np.float32) * 1e-3
    g = run_gpu(wl, bd, mode="provided", M_in=M, d_topk_w=dtw, loss_scale=2.0)
    ref = run_oracle(wl, mode="provided", M_in=M.astype(np.float64), loss_scale=2.0,
                     d_topk_w=dtw.astype(np.float64), topk_idx_for_up=g["topk_idx"])
    compare(wl, g, ref)


def test_hard_labels_with_text_only_sample(bd):
    wl = random_router_case(22, 400, 128, 32, 4, 4, [150, 100, 150], aligned=True)
    wl.is_vision[150:250] = 0                      # sample 1 has no vision token
    M = np.stack([wl.is_vision, 1 - wl.is_vision], 1).astype(np.float32)
    g = run_gpu(wl, bd, mode="provided", M_in=M)
    ref = run_oracle(wl, mode="provided", M_in=M.astype(np.float64))
    compare(wl, g, ref)
    assert g["n_absent"] == 1
    assert g["mi"][1] == 0.0


@pytest.mark.parametrize("name", list(CASES))
def test_fused_permute_parity(bd, name):
    # smoes_router_fwd_permute: forward outputs and the permutation of its own top-k (one launch
    # on bf16 plans, two calls on fp32) against the oracle
    seed, T, d, E, k, K, lens, dt, aligned = CASES[name]
    wl = random_router_case(seed, T, d, E, k, K, lens, dtype=dt, aligned=aligned)
    g = run_gpu(wl, bd, mode="gauss", loss_scale=0.7, fused=True)
    ref = run_oracle(wl, mode="gauss", loss_scale=0.7)
    compare(wl, g, ref)


def test_fused_permute_provided_scores_custom_home(bd):
    # without the Gaussian warps the producer and MMA warps run the permutation; non-consecutive
    # bins and a custom dispatch home
    wl = random_router_case(27, 1500, 192, 48, 5, 6, [200, 1100, 200], aligned=True)
    rng = np.random.default_rng(1)
    wl.expert_bin = rng.permutation(wl.expert_bin).astype(np.int32)
    Mv = rng.uniform(0.02, 0.98, wl.T)
    M = np.stack([Mv, 1 - Mv], 1).astype(np.float32)
    home = (np.arange(wl.T) * 5) % wl.n_bins
    g = run_gpu(wl, bd, mode="provided", M_in=M, home=home, fused=True)
    ref = run_oracle(wl, mode="provided", M_in=M.astype(np.float64))
    compare(wl, g, ref, home=home)


def test_fused_permute_equals_separate_calls(bd):
    wl = random_router_case(26, 2000, 256, 64, 6, 8, [700, 1300], aligned=True)
    a = run_gpu(wl, bd, mode="gauss")
    b = run_gpu(wl, bd, mode="gauss", fused=True)
    for key in a:
        if a[key] is None:
            continue
        np.testing.assert_array_equal(np.asarray(a[key]), np.asarray(b[key]), err_msg=key)


def test_custom_home_dispatch(bd):
    wl = random_router_case(23, 640, 128, 32, 4, 4, [320, 320], aligned=True)
    home = (np.arange(wl.T) * 7) % wl.n_bins
    g = run_gpu(wl, bd, mode="gauss", home=home)
    from oracle import smoes_oracle as O
    pr = O.bin_permute(g["topk_idx"], wl.expert_bin, wl.n_bins, home=home, is_vision=wl.is_vision)
    np.testing.assert_array_equal(g["dispatch"], pr["dispatch"])


def test_determinism_bitwise(bd):
    wl = random_router_case(24, 900, 256, 64, 6, 8, [450, 450], aligned=True)
    a = run_gpu(wl, bd, mode="gauss")
    b = run_gpu(wl, bd, mode="gauss")
    for key in ("M", "topk_idx", "topk_w", "mi", "dW", "dX", "dlogits", "perm", "mask"):
        np.testing.assert_array_equal(a[key], b[key], err_msg=key)
    assert a["loss"] == b["loss"]


def test_accumulate_dw_and_no_dx(bd):
    wl = random_router_case(25, 300, 128, 64, 6, 8, [300], aligned=True)
    dev = "cuda"
    r = bd.Router(wl.T, wl.d, wl.E, wl.k, wl.n_bins, wl.sample_offsets, wl.expert_bin)
    X, W = wl.X.to(dev), wl.W.to(dev)
    r.forward(X, W, mu=wl.mu.to(dev), var=wl.var.to(dev), tau=wl.tau)
    dW1 = torch.zeros((wl.E, wl.d), device=dev)
    r.backward(X, W, r.M, dW1)
    dW2 = torch.ones((wl.E, wl.d), device=dev)
    r.backward(X, W, r.M, dW2, accumulate=True)
    torch.cuda.synchronize()
    # (1 + x) - 1 in fp32 carries up to 6e-8 absolute rounding
    np.testing.assert_allclose((dW2 - 1).cpu().numpy(), dW1.cpu().numpy(), rtol=1e-5, atol=2e-7)


def test_empty_batch(bd):
    r = bd.Router(0, 64, 16, 2, 4, [0], np.arange(16) // 4)
    X = torch.empty((0, 64), dtype=torch.bfloat16, device="cuda")
    W = torch.zeros((16, 64), dtype=torch.bfloat16, device="cuda")
    r.loss.fill_(7.0)
    r.forward(X, W, M_in=torch.empty((0, 2), device="cuda"))
    dW = torch.full((16, 64), 3.0, device="cuda")
    r.backward(X, W, torch.empty((0, 2), device="cuda"), dW)
    r.permute()
    torch.cuda.synchronize()
    assert r.loss.item() == 0.0
    assert float(dW.abs().max()) == 0.0
    assert int(r.bin_offsets.abs().max()) == 0


def test_invalid_input_sets_device_status(bd):
    wl = random_router_case(26, 200, 64, 16, 2, 4, [200], aligned=True)
    wl.var[0, 3] = -1.0                            # non-positive variance
    r = bd.Router(wl.T, wl.d, wl.E, wl.k, wl.n_bins, wl.sample_offsets, wl.expert_bin)
    X, W = wl.X.cuda(), wl.W.cuda()
    r.forward(X, W, mu=wl.mu.cuda(), var=wl.var.cuda(), tau=wl.tau)
    code, _ = r.device_status()
    assert code == -7
    # the workspace recovers after re-initialisation
    wl.var[0, 3] = 1.0
    assert bd.smoes_workspace_init(r.plan, r.ws) == 0
    r.forward(X, W, mu=wl.mu.cuda(), var=wl.var.cuda(), tau=wl.tau)
    assert r.device_status()[0] == 0


def test_host_validation_leaves_outputs_untouched(bd):
    wl = random_router_case(27, 100, 64, 16, 2, 4, [100], aligned=True)
    r = bd.Router(wl.T, wl.d, wl.E, wl.k, wl.n_bins, wl.sample_offsets, wl.expert_bin)
    X = wl.X.cuda()
    W = wl.W.cuda()
    r.loss.fill_(5.0)
    small_ws = torch.empty(256, dtype=torch.uint8, device="cuda")
    code = bd.smoes_router_fwd(r.plan, X, W, None, dict(mu=wl.mu.cuda(), var=wl.var.cuda()), r.M,
                               r.topk_idx, r.topk_w, None, None, r.mi, r.loss, small_ws)
    assert code == -4
    misaligned = X.view(-1)[1:].view(-1)               # 2-byte offset
    code = bd.smoes_router_fwd(r.plan, misaligned, W, None, dict(mu=wl.mu.cuda(), var=wl.var.cuda()),
                               r.M, r.topk_idx, r.topk_w, None, None, r.mi, r.loss, r.ws)
    assert code == -3
    code = bd.smoes_router_fwd(r.plan, X, W, r.M, dict(mu=wl.mu.cuda(), var=wl.var.cuda()), r.M,
                               r.topk_idx, r.topk_w, None, None, r.mi, r.loss, r.ws)
    assert code == -1                                  # both M_in and gauss given
    torch.cuda.synchronize()
    assert r.loss.item() == 5.0
