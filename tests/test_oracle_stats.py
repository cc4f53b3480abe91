"""Pins of the oracle's online Gaussian statistics (eqs. 5-7) and momentum-adaptive binning
(eqs. 10-11): against the exponentially weighted moments they must equal (the update is Chan's
merge of weighted samples), special cases with a closed form, and invariants of the binning."""
import numpy as np
import pytest
import torch

from oracle import smoes_oracle as O
from paper_2604_23996_gb300.workloads import batch_moments


def _batches(seed, d=6, sizes=(40, 25, 0, 33), vis_frac=(0.5, 0.0, 0.5, 0.7)):
    rng = np.random.default_rng(seed)
    out = []
    for n, fv in zip(sizes, vis_frac):
        X = rng.standard_normal((n, d)) * rng.uniform(0.5, 2.0, d) + rng.uniform(-1, 1, d)
        lab = (rng.uniform(size=n) < fv).astype(np.int32)
        out.append((X, lab))
    return out


@pytest.mark.parametrize("beta", [0.0, 0.5, 0.99])
def test_first_step_from_empty_is_the_batch_moments(beta):
    X, lab = _batches(0)[0]
    st = O.gaussian_stats_update(O.gaussian_stats_empty(X.shape[1]), X, lab, beta)
    mu, var = O.gaussian_stats(st)
    for m, rows in enumerate((lab == 1, lab == 0)):
        assert st[0][m] == rows.sum()
        np.testing.assert_allclose(mu[m], X[rows].mean(axis=0), rtol=1e-12)
        np.testing.assert_allclose(var[m], X[rows].var(axis=0), rtol=1e-12)   # biased


def test_workload_statistics_are_the_first_update():
    # the benchmarks' mu, var (input generator, fp32) are eqs. (5)-(7) after one step
    rng = np.random.default_rng(1)
    X = torch.from_numpy(rng.standard_normal((300, 16)).astype(np.float32)).to(torch.bfloat16)
    lab = (rng.uniform(size=300) < 0.4).astype(np.int64)
    mu_w, var_w = batch_moments(X, lab)
    st = O.gaussian_stats_update(O.gaussian_stats_empty(16), X.double().numpy(), lab, 0.99)
    mu, var = O.gaussian_stats(st)
    np.testing.assert_allclose(mu_w.double().numpy(), mu, rtol=1e-5, atol=1e-6)
    np.testing.assert_allclose(var_w.double().numpy(), var, rtol=1e-5, atol=1e-6)


@pytest.mark.parametrize("beta", [0.3, 0.9, 0.99])
def test_ema_welford_equals_exponentially_weighted_moments(beta):
    # after steps 1..t, N = sum w, mu = sum w x / N, var = sum w (x - mu)^2 / N with weight
    # w = beta^(t - t_x) for a token of step t_x (computed here from that definition)
    batches = _batches(2)
    d = batches[0][0].shape[1]
    st = O.gaussian_stats_empty(d)
    for t, (X, lab) in enumerate(batches):
        st = O.gaussian_stats_update(st, X, lab, beta)
        mu, var = O.gaussian_stats(st)
        for m, want in enumerate((1, 0)):
            xs, ws = [], []
            for t2, (X2, lab2) in enumerate(batches[:t + 1]):
                sel = X2[lab2 == want]
                xs.append(sel)
                ws.append(np.full(len(sel), beta ** (t - t2)))
            xs, ws = np.concatenate(xs), np.concatenate(ws)
            if ws.sum() == 0:
                continue
            mu_w = (ws[:, None] * xs).sum(axis=0) / ws.sum()
            var_w = (ws[:, None] * (xs - mu_w) ** 2).sum(axis=0) / ws.sum()
            assert st[0][m] == pytest.approx(ws.sum(), rel=1e-12)
            np.testing.assert_allclose(mu[m], mu_w, rtol=1e-10, atol=1e-12)
            np.testing.assert_allclose(var[m], var_w, rtol=1e-10, atol=1e-12)


def test_a_batch_without_a_modality_keeps_its_parameters():
    X, lab = _batches(3)[0]
    st = O.gaussian_stats_update(O.gaussian_stats_empty(X.shape[1]), X, lab, 0.9)
    mu0, var0 = O.gaussian_stats(st)
    X2 = np.random.default_rng(4).standard_normal((20, X.shape[1]))
    st2 = O.gaussian_stats_update(st, X2, np.ones(20, dtype=np.int32), 0.9)   # vision only
    mu1, var1 = O.gaussian_stats(st2)
    np.testing.assert_allclose(mu1[1], mu0[1], rtol=1e-12)       # text: decayed, not moved
    np.testing.assert_allclose(var1[1], var0[1], rtol=1e-12)
    assert st2[0][1] == pytest.approx(0.9 * st[0][1])


def test_expert_load_ema_closed_form():
    rng = np.random.default_rng(5)
    C0, C = rng.uniform(0, 9, (2, 8)), rng.integers(0, 50, (2, 8)).astype(float)
    beta, n = 0.99, 37
    Cb = C0
    for _ in range(n):
        Cb = O.expert_load_ema(Cb, C, beta)
    np.testing.assert_allclose(Cb, beta ** n * C0 + (1 - beta ** n) * C, rtol=1e-12)


def test_text_bias_values():
    C_bar = np.array([[4.0, 0.0, 3.0, 0.0],      # vision load
                      [0.0, 5.0, 3.0, 0.0]])     # text load
    np.testing.assert_array_equal(O.text_bias(C_bar), [0.0, 1.0, 0.5, 0.5])


def test_adaptive_bins_partition():
    f = np.array([0.9, 0.1, 0.5, 0.1, 0.7, 0.3, 0.5, 0.0])
    eb = O.adaptive_bins(f, 4)
    # ascending f: e7 (0.0), e1 (0.1), e3 (0.1), e5 (0.3), e2 (0.5), e6 (0.5), e4 (0.7), e0 (0.9)
    np.testing.assert_array_equal(eb, [3, 0, 2, 1, 3, 1, 2, 0])
    rng = np.random.default_rng(6)
    for E, K in ((16, 4), (64, 8), (128, 16)):
        f = rng.uniform(size=E).round(2)                 # ties included
        eb = O.adaptive_bins(f, K)
        assert np.all(np.bincount(eb, minlength=K) == E // K)
        for b in range(K - 1):
            assert f[eb == b].max() <= f[eb == b + 1].min()
        # equal scores keep expert order inside the sorted sequence
        order = np.lexsort((np.arange(E), f))
        np.testing.assert_array_equal(eb[order], np.arange(E) // (E // K))


def test_binning_from_the_routers_own_counts():
    # C[m, e] of the permutation -> eq. (10) -> eq. (11) -> a valid bin map with equal bins
    rng = np.random.default_rng(7)
    T, E, k, K = 200, 16, 2, 4
    z = rng.standard_normal((T, E))
    topk = np.argsort(-z, axis=1)[:, :k].astype(np.int32)
    is_vis = (rng.uniform(size=T) < 0.5).astype(np.uint8)
    res = O.bin_permute(topk, np.arange(E) // (E // K), K, is_vision=is_vis)
    C = res["expert_counts"]
    np.testing.assert_array_equal(C.sum(axis=0), np.bincount(topk.ravel(), minlength=E))
    eb = O.adaptive_bins(O.text_bias(O.expert_load_ema(np.zeros((2, E)), C, 0.99)), K)
    assert np.all(np.bincount(eb, minlength=K) == E // K)
