"""Pins of the oracle's bin-level load-balance loss (eq. 16) and its gradient: the one-bin case
reduces to the standard load-balance loss of the preliminaries (eq. 1), even load gives one per
bin and no gradient, and the gradient matches central differences with the routing fixed."""
import numpy as np
import pytest

from oracle import smoes_oracle as O


def _case(seed, T=60, E=16, k=3, K=4, scale=1.0):
    rng = np.random.default_rng(seed)
    z = rng.standard_normal((T, E)) * scale
    g = O.softmax_gate(z)
    topk = np.argsort(-z, axis=1, kind="stable")[:, :k]
    return z, g, topk, np.arange(E) // (E // K)


def test_one_bin_is_the_standard_load_balance_loss():
    z, g, topk, _ = _case(0)
    T, E = g.shape
    k = topk.shape[1]
    L, _ = O.bin_balance_loss(g, topk, np.zeros(E, dtype=int), 1)
    f = np.bincount(topk.ravel(), minlength=E) / (T * k)      # fraction of the routed selections
    P = g.mean(axis=0)                                          # average gating score
    assert L == pytest.approx(E * np.sum(f * P), rel=1e-12)     # eq. (1), one layer


def test_even_load_gives_one_per_bin_and_no_gradient():
    # each token picks one expert per bin, cycling through the bin's slots: even f in every bin
    T, E, K = 64, 16, 4
    N_B = E // K
    eb = np.arange(E) // N_B
    topk = np.stack([k * N_B + (np.arange(T) % N_B) for k in range(K)], axis=1)
    z = np.random.default_rng(1).standard_normal((T, E))
    L, parts = O.bin_balance_loss(O.softmax_gate(z), topk, eb, K)
    np.testing.assert_allclose(parts["f"], 1.0 / N_B)
    assert L == pytest.approx(K, rel=1e-12)                     # sum_e P_e = 1 inside a bin
    dz = O.bin_balance_grad_logits(z, topk, eb, K, 1.0)
    np.testing.assert_allclose(dz, 0.0, atol=1e-15)


def test_unused_bin_contributes_nothing():
    z, g, topk, eb = _case(2)
    topk = np.where(eb[topk] == 3, 0, topk)                     # nobody selects bin 3
    L, parts = O.bin_balance_loss(g, topk, eb, 4)
    assert not parts["used"][3] and parts["used"][:3].all()
    L3 = sum(4 * np.sum(parts["f"][eb == b] * parts["P"][eb == b]) for b in range(3))
    assert L == pytest.approx(L3, rel=1e-12)


@pytest.mark.parametrize("seed", [3, 4])
def test_gradient_central_differences_with_fixed_routing(seed):
    z, g, topk, eb = _case(seed, T=12, E=8, k=2, K=2)
    scale = 0.37
    dz = O.bin_balance_grad_logits(z, topk, eb, 2, scale)
    h = 1e-6
    num = np.zeros_like(z)
    for j in range(z.shape[0]):
        for e in range(z.shape[1]):
            zp, zm = z.copy(), z.copy()
            zp[j, e] += h
            zm[j, e] -= h
            lp, _ = O.bin_balance_loss(O.softmax_gate(zp), topk, eb, 2)   # routing held fixed
            lm, _ = O.bin_balance_loss(O.softmax_gate(zm), topk, eb, 2)
            num[j, e] = scale * (lp - lm) / (2 * h)
    np.testing.assert_allclose(dz, num, rtol=1e-6, atol=1e-9)
    np.testing.assert_allclose(dz.sum(axis=1), 0.0, atol=1e-14)   # softmax invariance
