"""Pins of the fp64 oracle against what the paper and the mathematics fix (CPU only).

Each test fixes one part of the oracle with something other than the oracle itself: a closed
form derived by hand (tests/golden/closed_forms.json), an independent library routine, an
invariant the equations imply, brute force on tiny inputs, or central finite differences.
"""
import math

import numpy as np
import pytest
import torch

from oracle import smoes_oracle as O

RNG = np.random.default_rng(1234)


# ----------------------------------------------------------------------------- Gaussian score

def test_gauss_closed_form_equal_variance(golden):
    c = golden["gauss_equal_var_x_at_mu_v"]
    M = O.gaussian_score(c["X"], c["mu"], c["var"], c["tau"])
    assert M[0, 0] == pytest.approx(c["M_v"], rel=1e-14)
    assert M[0, 1] == pytest.approx(1.0 - c["M_v"], rel=1e-13)


def test_gauss_closed_form_variance_term(golden):
    # catches a dropped log-variance term or a wrong variance division
    c = golden["gauss_variance_only"]
    M = O.gaussian_score(c["X"], c["mu"], c["var"], c["tau"])
    np.testing.assert_allclose(M[:, 0], c["M_v"], rtol=1e-13)


def test_gauss_loglik_matches_scipy_logpdf():
    stats = pytest.importorskip("scipy.stats")
    d = 7
    X = RNG.standard_normal((5, d))
    mu = RNG.standard_normal((2, d))
    var = RNG.uniform(0.3, 3.0, (2, d))
    LL = O.gaussian_log_likelihood(X, mu, var)
    for m in range(2):
        ref = stats.norm.logpdf(X, loc=mu[m], scale=np.sqrt(var[m])).sum(axis=1)
        # eq. (8) omits the constant -d/2 log(2 pi), which cancels in eq. (9)
        np.testing.assert_allclose(LL[:, m] - 0.5 * d * math.log(2 * math.pi), ref, rtol=1e-13)


def test_gauss_equal_stats_give_half_and_rows_sum_to_one():
    d = 9
    X = RNG.standard_normal((11, d))
    mu = np.tile(RNG.standard_normal(d), (2, 1))
    var = np.tile(RNG.uniform(0.5, 2.0, d), (2, 1))
    np.testing.assert_allclose(O.gaussian_score(X, mu, var, 0.5 * d), 0.5, rtol=0, atol=1e-15)
    var2 = RNG.uniform(0.5, 2.0, (2, d))
    M = O.gaussian_score(X, RNG.standard_normal((2, d)), var2, 0.3)
    assert np.all((M >= 0) & (M <= 1))
    np.testing.assert_allclose(M.sum(axis=1), 1.0, atol=1e-15)


def test_gauss_temperature_is_a_sigmoid_of_the_difference():
    d = 6
    X = RNG.standard_normal((4, d))
    mu = RNG.standard_normal((2, d))
    var = RNG.uniform(0.5, 2.0, (2, d))
    LL = O.gaussian_log_likelihood(X, mu, var)
    for tau in (0.25, 1.0, 3.0):
        M = O.gaussian_score(X, mu, var, tau)
        np.testing.assert_allclose(M[:, 0], 1 / (1 + np.exp(-(LL[:, 0] - LL[:, 1]) / tau)), rtol=1e-13)


# ----------------------------------------------------------------------------- gate / top-k / bins

def test_softmax_and_topk_match_torch():
    z = RNG.standard_normal((13, 24))
    g = O.softmax_gate(z)
    np.testing.assert_allclose(g, torch.softmax(torch.from_numpy(z), dim=1).numpy(), rtol=1e-13)
    idx, w = O.topk_route(z, g, 5)
    tv, ti = torch.topk(torch.from_numpy(z), 5, dim=1, sorted=True)
    np.testing.assert_array_equal(idx, ti.numpy())
    np.testing.assert_allclose(w, np.take_along_axis(g, ti.numpy(), axis=1), rtol=1e-14)


def test_topk_tie_rule_and_renorm():
    z = np.array([[1.0, 3.0, 3.0, 2.0, 3.0]])
    g = O.softmax_gate(z)
    idx, w = O.topk_route(z, g, 4)
    np.testing.assert_array_equal(idx, [[1, 2, 4, 3]])          # equal logits -> lower index first
    _, wr = O.topk_route(z, g, 4, renorm=True)
    np.testing.assert_allclose(wr.sum(), 1.0, rtol=1e-15)
    np.testing.assert_allclose(wr, w / w.sum(), rtol=1e-15)


def test_gate_is_x_times_w_transposed():
    X = RNG.standard_normal((3, 4))
    W = RNG.standard_normal((5, 4))
    z = O.gate_logits(X, W)
    for j in range(3):
        for e in range(5):
            assert z[j, e] == pytest.approx(sum(X[j, t] * W[e, t] for t in range(4)), rel=1e-13)


def test_bin_probs_brute_force_and_sum_to_one():
    g = O.softmax_gate(RNG.standard_normal((7, 12)))
    eb = np.array([2, 0, 1, 2, 0, 1, 1, 0, 2, 1, 0, 2])       # a non-consecutive map, 4 per bin
    p = O.bin_probs(g, eb, 3)
    for j in range(7):
        for k in range(3):
            assert p[j, k] == pytest.approx(sum(g[j, e] for e in range(12) if eb[e] == k), rel=1e-14)
    np.testing.assert_allclose(p.sum(axis=1), 1.0, atol=1e-15)


# ----------------------------------------------------------------------------- mutual information

def test_mi_hand_example(golden):
    c = golden["mi_two_by_two"]
    p = O.bin_probs(np.array(c["g"]), c["expert_bin"], 2)
    tab = O.sample_joint(np.array(c["M"]), p, N_B=1)
    np.testing.assert_allclose(tab["P"], c["P"], rtol=1e-15)
    assert tab["I"] == pytest.approx(c["I"], rel=1e-14)


def test_mi_matches_sklearn_on_the_joint():
    metrics = pytest.importorskip("sklearn.metrics")
    M = RNG.uniform(0, 1, (40, 1))
    M = np.hstack([M, 1 - M])
    g = O.softmax_gate(3 * RNG.standard_normal((40, 8)))
    p = O.bin_probs(g, np.arange(8) // 2, 4)
    tab = O.sample_joint(M, p, N_B=2)
    # sklearn takes integer counts (and multiplies marginals in int64): scale the joint to 1e8
    counts = np.rint(tab["P"] * 1e8).astype(np.int64)
    ref = metrics.mutual_info_score(None, None, contingency=counts)
    assert tab["I"] == pytest.approx(ref, rel=1e-6)


def test_mi_hard_router_equals_modality_entropy(golden):
    # vision tokens -> bin 0, text tokens -> bin 1, logits scaled so p is one-hot to 1e-300
    T, E = 10, 4
    is_vis = np.array([1] * 4 + [0] * 6)
    M = np.stack([is_vis, 1 - is_vis], axis=1).astype(float)
    z = np.where(is_vis[:, None] == 1, [1.0, 0, 0, 0], [0, 0, 1.0, 0]) * 1e3
    p = O.bin_probs(O.softmax_gate(z), [0, 0, 1, 1], 2)
    tab = O.sample_joint(M, p, N_B=2)
    assert tab["I"] == pytest.approx(golden["mi_hard_router"]["I"], rel=1e-14)


def test_mi_bounds_and_uniform_modality_marginal():
    for trial in range(20):
        n, K, NB = 30, 4, 3
        Mv = RNG.uniform(0, 1, n)
        M = np.stack([Mv, 1 - Mv], axis=1)
        g = O.softmax_gate(2 * RNG.standard_normal((n, K * NB)))
        p = O.bin_probs(g, np.arange(K * NB) // NB, K)
        tab = O.sample_joint(M, p, NB)
        Hk = -np.sum(tab["Pk"] * np.log(tab["Pk"]))
        assert -1e-15 <= tab["I"] <= min(Hk, math.log(2)) + 1e-15
        # dense gate => sum_k Sbar[m,k] = 1/N_B for both modalities => P(m) = 1/2
        np.testing.assert_allclose(tab["Pm"], [0.5, 0.5], rtol=1e-13)


def test_mi_zero_when_scores_or_routing_constant():
    n, K, NB = 25, 4, 2
    g = O.softmax_gate(RNG.standard_normal((n, K * NB)))
    p = O.bin_probs(g, np.arange(K * NB) // NB, K)
    M_const = np.tile([0.3, 0.7], (n, 1))
    assert abs(O.sample_joint(M_const, p, NB)["I"]) < 1e-15
    Mv = RNG.uniform(0, 1, n)
    p_const = np.tile(p[0], (n, 1))
    assert abs(O.sample_joint(np.stack([Mv, 1 - Mv], 1), p_const, NB)["I"]) < 1e-15


def test_mi_absent_modality_gives_zero():
    n = 6
    M = np.tile([0.0, 1.0], (n, 1))                      # text-only sample
    p = O.bin_probs(O.softmax_gate(RNG.standard_normal((n, 4))), [0, 0, 1, 1], 2)
    tab = O.sample_joint(M, p, 2)
    assert tab["I"] == 0.0
    np.testing.assert_allclose(tab["Pm"], [0.0, 1.0])


def test_loss_is_minus_mean_mi():
    offs = np.array([0, 5, 12, 20])
    Mv = RNG.uniform(0, 1, 20)
    M = np.stack([Mv, 1 - Mv], 1)
    p = O.bin_probs(O.softmax_gate(RNG.standard_normal((20, 6))), [0, 0, 1, 1, 2, 2], 3)
    mis, joint, loss, _ = O.mi_loss(M, p, offs, 2)
    for i in range(3):
        assert mis[i] == pytest.approx(O.sample_joint(M[offs[i]:offs[i + 1]], p[offs[i]:offs[i + 1]], 2)["I"])
    assert loss == pytest.approx(-mis.mean(), rel=1e-15)


# ----------------------------------------------------------------------------- gradients

def _tiny_case(seed, T=14, d=5, E=6, n_bins=3, offs=(0, 6, 14)):
    rng = np.random.default_rng(seed)
    X = rng.standard_normal((T, d))
    W = 0.7 * rng.standard_normal((E, d))
    Mv = rng.uniform(0.05, 0.95, T)
    M = np.stack([Mv, 1 - Mv], 1)
    eb = np.arange(E) // (E // n_bins)
    return X, W, M, eb, n_bins, np.array(offs)


def _loss(X, W, M, eb, n_bins, offs, k=2):
    return O.router_forward(X, W, M, eb, n_bins, offs, k)["loss"]


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_mi_gradient_central_differences(seed):
    X, W, M, eb, K, offs = _tiny_case(seed)
    s = 0.37
    fwd = O.router_forward(X, W, M, eb, K, offs, 2)
    dz, dW, dX = O.router_backward(X, W, M, fwd, eb, offs, s)
    h = 1e-6
    for (A, G) in ((W, dW), (X, dX)):
        num = np.zeros_like(A)
        for idx in np.ndindex(A.shape):
            old = A[idx]
            A[idx] = old + h
            lp = _loss(X, W, M, eb, K, offs)
            A[idx] = old - h
            lm = _loss(X, W, M, eb, K, offs)
            A[idx] = old
            num[idx] = s * (lp - lm) / (2 * h)
        # central differences carry ~eps*|L|/h round-off (1e-12 here) plus O(h^2) truncation
        np.testing.assert_allclose(G, num, rtol=1e-5, atol=1e-7 * np.abs(num).max())


def test_mi_gradient_torch_autograd_second_opinion():
    X, W, M, eb, K, offs = _tiny_case(7, T=20, d=6, E=8, n_bins=4, offs=(0, 9, 20))
    s = 1.0
    fwd = O.router_forward(X, W, M, eb, K, offs, 3)
    _, dW, dX = O.router_backward(X, W, M, fwd, eb, offs, s)
    Xt = torch.tensor(X, requires_grad=True)
    Wt = torch.tensor(W, requires_grad=True)
    Mt = torch.tensor(M)
    g = torch.softmax(Xt @ Wt.T, dim=1)
    onehot = torch.nn.functional.one_hot(torch.tensor(eb), K).double()
    p = g @ onehot
    NB = len(eb) // K
    total = 0
    for i in range(len(offs) - 1):
        a, b = offs[i], offs[i + 1]
        Sb = (Mt[a:b].T @ p[a:b]) / (NB * Mt[a:b].sum(0)[:, None])
        P = Sb / Sb.sum()
        total = total + (P * torch.log(P / (P.sum(1, keepdim=True) * P.sum(0, keepdim=True)))).sum()
    loss = -total / (len(offs) - 1)
    loss.backward()
    np.testing.assert_allclose(dW, Wt.grad.numpy(), rtol=1e-9, atol=1e-14)
    np.testing.assert_allclose(dX, Xt.grad.numpy(), rtol=1e-9, atol=1e-14)


def test_mi_gradient_invariants():
    X, W, M, eb, K, offs = _tiny_case(3)
    fwd = O.router_forward(X, W, M, eb, K, offs, 2)
    dz, _, _ = O.router_backward(X, W, M, fwd, eb, offs, 1.0)
    np.testing.assert_allclose(dz.sum(axis=1), 0.0, atol=1e-15)       # softmax shift invariance
    Mc = np.tile([0.4, 0.6], (X.shape[0], 1))                           # constant scores: I = 0
    fwd = O.router_forward(X, W, Mc, eb, K, offs, 2)
    dz, dW, dX = O.router_backward(X, W, Mc, fwd, eb, offs, 1.0)
    assert np.abs(dW).max() < 1e-14 and np.abs(dX).max() < 1e-14


@pytest.mark.parametrize("renorm", [False, True])
def test_topk_weight_gradient_central_differences(renorm):
    rng = np.random.default_rng(5)
    z = rng.standard_normal((4, 7))
    k = 3
    idx, _ = O.topk_route(z, O.softmax_gate(z), k)
    d = rng.standard_normal((4, k))

    def f(zz):
        gg = O.softmax_gate(zz)
        w = np.take_along_axis(gg, idx, axis=1)
        if renorm:
            w = w / w.sum(axis=1, keepdims=True)
        return float(np.sum(d * w))

    G = O.topk_weight_grad_logits(O.softmax_gate(z), idx, d, renorm)
    h = 1e-6
    num = np.zeros_like(z)
    for ix in np.ndindex(z.shape):
        zp = z.copy(); zp[ix] += h
        zm = z.copy(); zm[ix] -= h
        num[ix] = (f(zp) - f(zm)) / (2 * h)
    np.testing.assert_allclose(G, num, rtol=1e-6, atol=1e-10)


# ----------------------------------------------------------------------------- permutation

def _perm_brute(topk_idx, eb, K, home, is_vis):
    T, k = topk_idx.shape
    E = len(eb)
    slot = [sum(1 for e2 in range(e) if eb[e2] == eb[e]) for e in range(E)]
    pairs = {}
    for j in range(T):
        for c in range(k):
            e = int(topk_idx[j, c])
            key = (int(eb[e]), j)
            pairs[key] = pairs.get(key, 0) | (1 << slot[e])
    keys = sorted(pairs)                                   # bin ascending, then token ascending
    offsets = [0] * (K + 1)
    for (kb, j) in keys:
        offsets[kb + 1] += 1
    for kb in range(K):
        offsets[kb + 1] += offsets[kb]
    dispatch = np.zeros((K, K), dtype=np.int64)
    for (kb, j) in keys:
        dispatch[home[j], kb] += 1
    ec = np.zeros((2, E), dtype=np.int64)
    for j in range(T):
        for c in range(k):
            ec[0 if is_vis[j] else 1, topk_idx[j, c]] += 1
    return (np.array(offsets), np.array([j for (_, j) in keys]),
            np.array([pairs[kk] for kk in keys], dtype=np.uint64), dispatch, ec)


@pytest.mark.parametrize("seed", [0, 1])
def test_bin_permute_brute_force_and_invariants(seed):
    rng = np.random.default_rng(seed)
    T, E, k, K = 37, 12, 4, 3
    z = rng.standard_normal((T, E))
    idx, _ = O.topk_route(z, O.softmax_gate(z), k)
    eb = rng.permutation(np.arange(E) // (E // K))           # non-consecutive bins
    is_vis = (rng.uniform(size=T) < 0.4).astype(np.uint8)
    home = O.default_home(T, K)
    r = O.bin_permute(idx, eb, K, home=None, is_vision=is_vis)
    offs, perm, mask, disp, ec = _perm_brute(idx, eb, K, home, is_vis)
    np.testing.assert_array_equal(r["offsets"], offs)
    np.testing.assert_array_equal(r["perm"], perm)
    np.testing.assert_array_equal(r["mask"], mask)
    np.testing.assert_array_equal(r["dispatch"], disp)
    np.testing.assert_array_equal(r["expert_counts"], ec)
    # invariants: monotone offsets, >=1 bit per entry, popcounts sum to T*k, dispatch sums to |U|
    assert np.all(np.diff(r["offsets"]) >= 0)
    assert np.all(r["mask"] != 0)
    assert sum(bin(int(m)).count("1") for m in r["mask"]) == T * k
    assert r["dispatch"].sum() == r["offsets"][-1]
    np.testing.assert_array_equal(r["expert_counts"].sum(0), np.bincount(idx.reshape(-1), minlength=E))


def test_default_home_is_contiguous_split():
    h = O.default_home(10, 4)
    np.testing.assert_array_equal(h, [0, 0, 0, 1, 1, 2, 2, 2, 3, 3])


# ----------------------------------------------------------------------------- attention score

def test_attn_zero_query_closed_form(golden):
    c = golden["attn_zero_query"]
    S, H, hd = c["S"], 3, 4
    Q = np.zeros((1, H, S, hd))
    K = RNG.standard_normal((1, H, S, hd))
    m = np.zeros((1, S)); m[0, :c["n_image"]] = 1
    bias = c["beta"] * m
    out = O.attention_vision_mass(Q, K, m, 0.5, True, bias)
    np.testing.assert_allclose(out[0], c["Mv"], rtol=1e-14)


def test_attn_image_first_causal_is_one_for_image_queries():
    B, H, S, hd, nimg = 2, 4, 12, 8, 5
    Q = RNG.standard_normal((B, H, S, hd))
    K = RNG.standard_normal((B, H, S, hd))
    m = np.zeros((B, S)); m[:, :nimg] = 1
    out = O.attention_vision_mass(Q, K, m, 1 / math.sqrt(hd), True)
    np.testing.assert_allclose(out[:, :nimg], 1.0, rtol=0, atol=1e-15)
    assert np.all(out[:, nimg:] < 1.0)


def test_attn_matches_torch_sdpa_with_scores_as_values():
    # the paper's FlashAttention equivalence: attention with V = m returns the aggregated score
    B, H, S, hd = 2, 3, 16, 8
    Q = RNG.standard_normal((B, H, S, hd))
    K = RNG.standard_normal((B, H, S, hd))
    m = RNG.uniform(0, 1, (B, S))
    bias = RNG.standard_normal((B, S))
    scale = 0.3
    out = O.attention_vision_mass(Q, K, m, scale, True, bias)
    mask = torch.full((S, S), float("-inf"), dtype=torch.float64).triu(1)
    attn_bias = mask[None, None] + torch.from_numpy(bias)[:, None, None, :]
    V = torch.from_numpy(m)[:, None, :, None].expand(B, H, S, 1)
    ref = torch.nn.functional.scaled_dot_product_attention(
        torch.from_numpy(Q), torch.from_numpy(K), V, attn_mask=attn_bias, scale=scale)
    np.testing.assert_allclose(out, ref[..., 0].mean(dim=1).numpy(), rtol=1e-12)
    # single-row path equals the blocked path
    rows = np.array([[0, 0], [1, 7], [0, 15]])
    np.testing.assert_allclose(O.attention_vision_mass(Q, K, m, scale, True, bias, queries=rows),
                               out[rows[:, 0], rows[:, 1]], rtol=1e-13)


def test_residual_update_is_norm_weighted_mean():
    r = O.residual_score_update(np.array([1.0, 0.0]), np.array([0.0, 1.0]), np.array([3.0, 1.0]),
                                np.array([1.0, 1.0]))
    np.testing.assert_allclose(r, [0.75, 0.5])


def test_msi_extremes():
    assert O.msi([[5, 0, 7], [0, 3, 0]]) == pytest.approx(1.0)
    assert O.msi([[2, 4], [1, 2]]) == pytest.approx(0.0, abs=1e-15)
