"""Pins of the oracle's router variants (no GPU): the GMM estimator of the supplementary material,
the sigmoid router with a selection bias (Moonlight-MoE in the backbone table) and the
top-k-masked reading of g in eq. (12). Each is fixed by a library routine, a reduction to a case
already pinned, or central differences."""
import numpy as np
import pytest
import torch

from oracle import smoes_oracle as O

scipy_stats = pytest.importorskip("scipy.stats")
scipy_special = pytest.importorskip("scipy.special")


def _gmm_case(seed, T=9, d=6, C=3):
    rng = np.random.default_rng(seed)
    X = rng.standard_normal((T, d))
    mu = rng.standard_normal((2, C, d))
    var = rng.uniform(0.3, 2.0, (2, C, d))
    w = rng.uniform(0.2, 1.0, (2, C))
    log_pi = np.log(w / w.sum(axis=1, keepdims=True))
    return X, log_pi, mu, var


def test_gmm_loglik_matches_scipy_mixture_density():
    X, log_pi, mu, var = _gmm_case(1)
    LL = O.gmm_log_likelihood(X, log_pi, mu, var)
    for m in range(2):
        comp = np.stack([log_pi[m, c] + scipy_stats.multivariate_normal(mu[m, c], np.diag(var[m, c])).logpdf(X)
                         for c in range(mu.shape[1])], axis=1)
        np.testing.assert_allclose(LL[:, m], scipy_special.logsumexp(comp, axis=1), rtol=1e-12)


def test_gmm_with_one_component_is_the_gaussian_score():
    X, _, mu, var = _gmm_case(2, C=1)
    tau = 1.7
    got = O.gmm_score(X, np.zeros((2, 1)), mu, var, tau)
    want = O.gaussian_score(X, mu[:, 0], var[:, 0], tau)
    np.testing.assert_allclose(got, want, rtol=1e-12, atol=1e-15)


def test_gmm_with_duplicate_components_is_one_gaussian():
    X, _, mu, var = _gmm_case(3, C=1)
    mu2 = np.concatenate([mu, mu], axis=1)
    var2 = np.concatenate([var, var], axis=1)
    lp = np.log(np.array([[0.3, 0.7], [0.5, 0.5]]))
    np.testing.assert_allclose(O.gmm_score(X, lp, mu2, var2, 2.0),
                               O.gaussian_score(X, mu[:, 0], var[:, 0], 2.0), rtol=1e-12)


def test_gmm_score_rows_sum_to_one_and_symmetric_stats_give_half():
    X, log_pi, mu, var = _gmm_case(4)
    M = O.gmm_score(X, log_pi, mu, var, 3.0)
    np.testing.assert_allclose(M.sum(axis=1), 1.0, rtol=1e-14)
    mu_s = np.stack([mu[0], mu[0]])
    var_s = np.stack([var[0], var[0]])
    lp_s = np.stack([log_pi[0], log_pi[0]])
    np.testing.assert_allclose(O.gmm_score(X, lp_s, mu_s, var_s, 3.0), 0.5, rtol=1e-14)


def test_sigmoid_gate_matches_torch_and_bias_only_steers_the_choice():
    rng = np.random.default_rng(5)
    z = rng.standard_normal((40, 12))
    out = O.sigmoid_gate(z, None, k=3)
    s = torch.sigmoid(torch.from_numpy(z)).numpy()
    np.testing.assert_allclose(out["s"], s, rtol=1e-14)
    np.testing.assert_allclose(out["g"].sum(axis=1), 1.0, rtol=1e-14)
    ref = torch.topk(torch.from_numpy(s), 3, dim=1).indices.numpy()
    np.testing.assert_array_equal(out["topk_idx"], ref)
    np.testing.assert_allclose(out["topk_w"].sum(axis=1), 1.0, rtol=1e-14)
    # a large bias on expert 7 puts it in every token's choice; the weights still come from s
    b = np.zeros(12)
    b[7] = 10.0
    ob = O.sigmoid_gate(z, b, k=3)
    assert np.all((ob["topk_idx"] == 7).any(axis=1))
    sel = np.take_along_axis(s, ob["topk_idx"].astype(np.int64), axis=1)
    np.testing.assert_allclose(ob["topk_w"], sel / sel.sum(axis=1, keepdims=True), rtol=1e-14)
    np.testing.assert_array_equal(ob["g"], out["g"])


def test_sigmoid_gradient_central_differences():
    rng = np.random.default_rng(6)
    z = rng.standard_normal((5, 7))
    c = rng.standard_normal((5, 7))               # a loss linear in g: L = sum c * g
    grad = O.sigmoid_grad_logits(O.sigmoid_gate(z)["s"], c)
    h = 1e-6
    num = np.zeros_like(z)
    for idx in np.ndindex(*z.shape):
        zp, zm = z.copy(), z.copy()
        zp[idx] += h
        zm[idx] -= h
        num[idx] = (np.sum(c * O.sigmoid_gate(zp)["g"]) - np.sum(c * O.sigmoid_gate(zm)["g"])) / (2 * h)
    np.testing.assert_allclose(grad, num, rtol=1e-6, atol=1e-9)


def test_topk_masked_gate_is_the_renormalised_topk_weight():
    rng = np.random.default_rng(7)
    z = rng.standard_normal((30, 10))
    g = O.softmax_gate(z)
    idx, w = O.topk_route(z, g, 4, renorm=True)
    gm = O.topk_masked_gate(g, idx)
    np.testing.assert_allclose(gm.sum(axis=1), 1.0, rtol=1e-14)
    np.testing.assert_allclose(np.take_along_axis(gm, idx.astype(np.int64), axis=1), w, rtol=1e-14)
    mask = np.zeros_like(g, dtype=bool)
    np.put_along_axis(mask, idx.astype(np.int64), True, axis=1)
    assert np.all(gm[~mask] == 0.0)


def _variant_case(seed, T=16, d=6, E=8, n_bins=4, offs=(0, 7, 16)):
    rng = np.random.default_rng(seed)
    X = rng.standard_normal((T, d))
    W = 0.5 * rng.standard_normal((E, d))
    Mv = rng.uniform(0.05, 0.95, T)
    M = np.stack([Mv, 1 - Mv], axis=1)
    eb = np.arange(E) // (E // n_bins)
    return X, W, M, eb, n_bins, np.array(offs)


def test_default_variant_is_the_pinned_router():
    X, W, M, eb, K, offs = _variant_case(10)
    a = O.router_forward(X, W, M, eb, K, offs, 3)
    b = O.router_forward_variant(X, W, M, eb, K, offs, 3)
    np.testing.assert_array_equal(a["topk_idx"], b["topk_idx"])
    np.testing.assert_allclose(b["mi"], a["mi"], rtol=1e-14, atol=1e-16)
    dz_a, dW_a, _ = O.router_backward(X, W, M, a, eb, offs, 0.8)
    dz_b, dW_b, _ = O.router_backward_variant(X, W, M, b, eb, offs, 0.8)
    np.testing.assert_allclose(dz_b, dz_a, rtol=1e-12, atol=1e-16)
    np.testing.assert_allclose(dW_b, dW_a, rtol=1e-12, atol=1e-16)


@pytest.mark.parametrize("gate,mask", [("softmax", True), ("sigmoid", False), ("sigmoid", True)])
def test_variant_gradient_central_differences(gate, mask):
    X, W, M, eb, K, offs = _variant_case(11)
    bias = np.linspace(-0.3, 0.3, W.shape[0]) if gate == "sigmoid" else None
    k = 3
    f0 = O.router_forward_variant(X, W, M, eb, K, offs, k, gate=gate, score_bias=bias, mask=mask)
    _, dW, dX = O.router_backward_variant(X, W, M, f0, eb, offs, 1.0)

    def loss(Xv, Wv):
        f = O.router_forward_variant(Xv, Wv, M, eb, K, offs, k, gate=gate, score_bias=bias, mask=mask)
        assert np.array_equal(f["topk_idx"], f0["topk_idx"])     # the choice is locally constant
        return f["loss"]

    h = 1e-6
    for A, grad, name in ((W, dW, "W"), (X, dX, "X")):
        num = np.zeros_like(A)
        for idx in np.ndindex(*A.shape):
            Ap, Am = A.copy(), A.copy()
            Ap[idx] += h
            Am[idx] -= h
            num[idx] = ((loss(Xv=X, Wv=Ap) - loss(Xv=X, Wv=Am)) if name == "W"
                        else (loss(Xv=Ap, Wv=W) - loss(Xv=Am, Wv=W))) / (2 * h)
        np.testing.assert_allclose(grad, num, rtol=2e-5, atol=5e-10, err_msg=f"{gate} mask={mask} d{name}")


def test_masked_bins_hold_only_chosen_experts():
    X, W, M, eb, K, offs = _variant_case(12)
    f = O.router_forward_variant(X, W, M, eb, K, offs, 2, mask=True)
    np.testing.assert_allclose(f["p"].sum(axis=1), 1.0, rtol=1e-14)
    chosen_bins = eb[f["topk_idx"]]
    for j in range(X.shape[0]):
        assert set(np.nonzero(f["p"][j] > 0)[0]) == set(chosen_bins[j])


def test_sigmoid_topk_weight_gradient_central_differences():
    rng = np.random.default_rng(13)
    z = rng.standard_normal((6, 9))
    d = rng.standard_normal((6, 3))
    idx = O.sigmoid_gate(z, None, k=3)["topk_idx"]

    def L(zv):
        s = O.sigmoid_gate(zv)["s"]
        w = np.take_along_axis(s, idx.astype(np.int64), axis=1)
        return float(np.sum(d * w / w.sum(axis=1, keepdims=True)))

    grad = O.sigmoid_topk_weight_grad_logits(O.sigmoid_gate(z)["s"], idx, d)
    h = 1e-6
    num = np.zeros_like(z)
    for i in np.ndindex(*z.shape):
        zp, zm = z.copy(), z.copy()
        zp[i] += h
        zm[i] -= h
        num[i] = (L(zp) - L(zm)) / (2 * h)
    np.testing.assert_allclose(grad, num, rtol=1e-6, atol=1e-9)


def test_balance_gradient_at_the_gate_central_differences():
    # dL/dg from bin_balance_grad_gate against differences of eq. (16) in g itself (f held at the
    # counts of the fixed choice), and the logits form through the softmax Jacobian
    rng = np.random.default_rng(14)
    z = rng.standard_normal((12, 8))
    g = O.softmax_gate(z)
    idx, _ = O.topk_route(z, g, 3)
    eb = np.arange(8) // 2
    dg = O.bin_balance_grad_gate(g, idx, eb, 4, 1.0)
    h = 1e-7
    num = np.zeros_like(g)
    for i in np.ndindex(*g.shape):
        gp, gm = g.copy(), g.copy()
        gp[i] += h
        gm[i] -= h
        num[i] = (O.bin_balance_loss(gp, idx, eb, 4)[0] - O.bin_balance_loss(gm, idx, eb, 4)[0]) / (2 * h)
    np.testing.assert_allclose(dg, num, rtol=1e-5, atol=1e-8)
    np.testing.assert_allclose(O.softmax_grad_logits(g, dg), O.bin_balance_grad_logits(z, idx, eb, 4, 1.0),
                               rtol=1e-12, atol=1e-15)
