"""GPU parity of the online Gaussian statistics (Sec. 3.2, eqs. 5-7) and of momentum-adaptive
binning (Sec. 3.3, eqs. 10-11) against the fp64 oracle, over several consecutive steps.

Statistics: the state (N, S_mu, S_var) is carried on the device from the empty state through
batches with both modalities, a batch with no vision token (|T_m| = 0: the state only decays)
and a batch of another size; bf16 and fp32 features, d above one block's 2048-feature pass and
d not a multiple of 64. Tensors meet the 2e-3 bar of every other floating-point output (the
fp32 block sums give ~1e-6 in practice; the measured error is printed).

Binning: the EMA loads, f_spec and the new bin map are compared bit for bit (both sides take
the sort's decisions in fp64 with the same rounding), with counts from the router's own fused
permutation and synthetic counts full of ties (unused experts, equal columns).
"""
import numpy as np
import pytest
import torch

from oracle import smoes_oracle as O
from paper_2604_23996_gb300.workloads import make_features, random_router_case

from .parity import assert_tensor_close

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def bd():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2604_23996_gb300 import binding
    return binding


def _batch(seed, T, d, dtype, vision_frac):
    rng = np.random.default_rng(seed)
    is_vis = (rng.random(T) < vision_frac).astype(np.uint8)
    X32, _, _ = make_features(rng, is_vis, d, "beta51")
    return torch.from_numpy(X32).to(dtype), is_vis


def _plan(bd, T, d, dtype):
    dt = bd.SMOES_BF16 if dtype == torch.bfloat16 else bd.SMOES_F32
    return bd.Router(T, d, 16, 2, 4, [0, T], np.arange(16) // 4, dt)


@pytest.mark.parametrize("d,dtype,beta", [(2056, torch.bfloat16, 0.99), (1280, torch.bfloat16, 0.5),
                                          (72, torch.float32, 0.99)])
def test_gaussian_stats_update_several_steps(bd, d, dtype, beta):
    dev = "cuda"
    N = torch.zeros(2, dtype=torch.float64, device=dev)
    S_mu = torch.zeros((2, d), dtype=torch.float64, device=dev)
    S_var = torch.zeros((2, d), dtype=torch.float64, device=dev)
    mu = torch.empty((2, d), dtype=torch.float32, device=dev)
    var = torch.empty((2, d), dtype=torch.float32, device=dev)
    state = O.gaussian_stats_empty(d)
    # (seed, T, vision fraction): both modalities; again; no vision token; another batch size
    steps = [(1, 1500, 0.3), (2, 1500, 0.6), (3, 1500, 0.0), (4, 777, 0.45)]
    routers = {}
    for seed, T, vf in steps:
        X, is_vis = _batch(seed, T, d, dtype, vf)
        if T not in routers:
            routers[T] = _plan(bd, T, d, dtype)
        r = routers[T]
        code = bd.smoes_gaussian_stats_update(r.plan, X.to(dev), torch.from_numpy(is_vis).to(dev),
                                              beta, N, S_mu, S_var, mu, var, r.ws)
        assert code == 0, bd.smoes_status_string(code)
        torch.cuda.synchronize()
        state = O.gaussian_stats_update(state, X.double().numpy(), is_vis, beta)
        np.testing.assert_allclose(N.cpu().numpy(), state[0], rtol=1e-12, atol=0)
        e_mu = assert_tensor_close(S_mu.cpu().numpy(), state[1], f"S_mu step {seed}")
        e_var = assert_tensor_close(S_var.cpu().numpy(), state[2], f"S_var step {seed}")
        mu_ref, var_ref = O.gaussian_stats(state)
        assert_tensor_close(mu.cpu().numpy(), mu_ref, f"mu step {seed}")
        assert_tensor_close(var.cpu().numpy(), var_ref, f"var step {seed}")
        print(f"d={d} step {seed}: rel err S_mu {e_mu:.2e} S_var {e_var:.2e}")


def test_first_update_gives_the_batch_moments(bd):
    # from the empty state one update leaves mu = batch mean and var = biased batch variance per
    # hard modality (the statistics the timed workloads feed the score)
    wl = random_router_case(61, 2000, 256, 16, 2, 4, [2000])
    r = _plan(bd, wl.T, wl.d, wl.dtype)
    dev = "cuda"
    N = torch.zeros(2, dtype=torch.float64, device=dev)
    S_mu = torch.zeros((2, wl.d), dtype=torch.float64, device=dev)
    S_var = torch.zeros((2, wl.d), dtype=torch.float64, device=dev)
    mu = torch.empty((2, wl.d), dtype=torch.float32, device=dev)
    var = torch.empty((2, wl.d), dtype=torch.float32, device=dev)
    assert bd.smoes_gaussian_stats_update(r.plan, wl.X.to(dev), torch.from_numpy(wl.is_vision).to(dev),
                                          0.99, N, S_mu, S_var, mu, var, r.ws) == 0
    torch.cuda.synchronize()
    Xd = wl.X.double().numpy()
    for m, rows in enumerate((wl.is_vision == 1, wl.is_vision == 0)):
        assert_tensor_close(mu[m].cpu().numpy(), Xd[rows].mean(0), f"mu[{m}]")
        assert_tensor_close(var[m].cpu().numpy(), Xd[rows].var(0), f"var[{m}]")
    assert N.cpu().numpy().tolist() == [float((wl.is_vision == 1).sum()), float((wl.is_vision == 0).sum())]


def _bins_steps(bd, E, n_bins, counts_seq, beta):
    dev = "cuda"
    r = bd.Router(128, 64, E, 2, n_bins, [0, 128], np.arange(E) // (E // n_bins))
    C_bar = torch.zeros((2, E), dtype=torch.float64, device=dev)
    eb = torch.empty(E, dtype=torch.int32, device=dev)
    fs = torch.empty(E, dtype=torch.float64, device=dev)
    C_ref = np.zeros((2, E))
    for C in counts_seq:
        Ct = torch.as_tensor(np.ascontiguousarray(C), dtype=torch.int32).to(dev)
        assert bd.smoes_adaptive_bins(r.plan, Ct, beta, C_bar, eb, fs) == 0
        torch.cuda.synchronize()
        C_ref = O.expert_load_ema(C_ref, C, beta)
        f_ref = O.text_bias(C_ref)
        np.testing.assert_array_equal(C_bar.cpu().numpy(), C_ref)
        np.testing.assert_array_equal(fs.cpu().numpy(), f_ref)
        np.testing.assert_array_equal(eb.cpu().numpy(), O.adaptive_bins(f_ref, n_bins))


@pytest.mark.parametrize("E,n_bins", [(128, 16), (64, 8), (16, 1), (96, 3)])
def test_adaptive_bins_bit_exact_with_ties(bd, E, n_bins):
    rng = np.random.default_rng(E + n_bins)
    seq = []
    for t in range(5):
        C = rng.integers(0, 50, size=(2, E))
        C[:, rng.integers(0, E, 3)] = 0                    # unused experts: f = 1/2
        C[:, 1] = C[:, 0]                                  # equal columns: equal f_spec
        C[:, E - 1] = C[:, E // 2]
        seq.append(C)
    _bins_steps(bd, E, n_bins, seq, 0.99)


def test_adaptive_bins_from_the_routers_own_counts(bd):
    # C[m, e] from the fused forward + permutation of a real router step, several steps
    wl = random_router_case(62, 3000, 256, 64, 6, 8, [1500, 1500], aligned=True)
    dev = "cuda"
    r = bd.Router(wl.T, wl.d, wl.E, wl.k, wl.n_bins, wl.sample_offsets, wl.expert_bin)
    isv = torch.from_numpy(wl.is_vision).to(dev)
    seq = []
    for s in range(3):
        X = (wl.X.float() * (1.0 + 0.1 * s)).to(torch.bfloat16).to(dev)
        r.forward_permute(X, wl.W.to(dev), mu=wl.mu.to(dev), var=wl.var.to(dev), tau=wl.tau,
                          is_vision=isv)
        torch.cuda.synchronize()
        seq.append(r.expert_counts.cpu().numpy().copy())
    assert seq[0].sum() == wl.T * wl.k
    _bins_steps(bd, wl.E, wl.n_bins, seq, 0.99)


def test_stats_and_bins_reject_bad_arguments(bd):
    r = _plan(bd, 100, 64, torch.bfloat16)
    N = torch.zeros(2, dtype=torch.float64, device="cuda")
    S = torch.zeros((2, 64), dtype=torch.float64, device="cuda")
    X = torch.zeros((100, 64), dtype=torch.bfloat16, device="cuda")
    v = torch.zeros(100, dtype=torch.uint8, device="cuda")
    assert bd.smoes_gaussian_stats_update(r.plan, X, v, 1.5, N, S, S.clone(), None, None, r.ws) == -1
    assert bd.smoes_gaussian_stats_update(r.plan, X, None, 0.9, N, S, S.clone(), None, None, r.ws) == -1
    C = torch.zeros((2, 16), dtype=torch.int32, device="cuda")
    eb = torch.empty(16, dtype=torch.int32, device="cuda")
    assert bd.smoes_adaptive_bins(r.plan, C, -0.1, torch.zeros((2, 16), dtype=torch.float64,
                                                               device="cuda"), eb) == -1
