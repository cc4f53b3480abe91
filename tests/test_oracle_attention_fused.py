"""Pins of the oracle's fused attention forward with the vision score (the value column form of
eqs. 2-3) and its grouped-query variant: against the library routine for attention and against
the oracle's separate score."""
import numpy as np
import torch

from oracle import smoes_oracle as O

RNG = np.random.default_rng(11)


def _sdpa(Q, K, V, mask, scale, G):
    try:                                     # the library's grouped-query form
        return torch.nn.functional.scaled_dot_product_attention(Q, K, V, attn_mask=mask, scale=scale,
                                                                enable_gqa=G > 1)
    except TypeError:                        # older torch: expand the key/value heads by hand
        K = K.repeat_interleave(G, dim=1)
        V = V.repeat_interleave(G, dim=1)
        return torch.nn.functional.scaled_dot_product_attention(Q, K, V, attn_mask=mask, scale=scale)


def test_fused_output_and_score_match_library_attention():
    B, H, Hkv, S, hd, dv = 2, 4, 2, 12, 8, 5
    Q = RNG.standard_normal((B, H, S, hd))
    K = RNG.standard_normal((B, Hkv, S, hd))
    V = RNG.standard_normal((B, Hkv, S, dv))
    m = RNG.uniform(0, 1, (B, S))
    bias = RNG.standard_normal((B, S))
    scale = 0.35
    Ofused, mass = O.attention_forward_with_mass(Q, K, V, m, scale, True, bias)
    mask = torch.full((S, S), float("-inf"), dtype=torch.float64).triu(1)[None, None]
    mask = mask + torch.from_numpy(bias)[:, None, None, :]
    ref = _sdpa(torch.from_numpy(Q), torch.from_numpy(K), torch.from_numpy(V), mask, scale, H // Hkv)
    np.testing.assert_allclose(Ofused, ref.numpy(), rtol=1e-12, atol=1e-13)
    # the score column equals the separate score with the key heads expanded
    Kx = np.repeat(K, H // Hkv, axis=1)
    np.testing.assert_allclose(mass, O.attention_vision_mass(Q, Kx, m, scale, True, bias), rtol=1e-12)


def test_hard_labels_image_first_give_one_for_image_queries():
    # causal, image tokens first, hard labels: an image query attends to image keys only
    B, H, S, hd, n_img = 1, 2, 10, 4, 4
    Q = RNG.standard_normal((B, H, S, hd))
    K = RNG.standard_normal((B, 1, S, hd))
    V = RNG.standard_normal((B, 1, S, 3))
    m = np.zeros((B, S))
    m[:, :n_img] = 1.0
    _, mass = O.attention_forward_with_mass(Q, K, V, m, 0.5, True)
    np.testing.assert_allclose(mass[0, :n_img], 1.0, rtol=0, atol=1e-15)
    assert np.all(mass[0, n_img:] < 1.0) and np.all(mass[0, n_img:] > 0.0)
