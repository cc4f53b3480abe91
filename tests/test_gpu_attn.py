"""GPU parity of the attention-accumulated vision score (eqs. 2-4) against the fp64 oracle.

Cases: sequence lengths that are not multiples of the 128-query tile, causal and non-causal
attention, a vision-key logit bias, hard labels (eq. 2) and a carried soft score, the eq. (4)
residual blend, short sequences (S < 128), and many short work items per CTA (320 (sequence,
head) items of one or two key blocks on 152 CTAs: the second key half of a CTA can run a whole
item ahead of the first, which the merge hand-off between the halves has to absorb).
"""
import numpy as np
import pytest
import torch

from oracle import smoes_oracle as O

from .parity import assert_tensor_close

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def bd():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2604_23996_gb300 import binding
    return binding


def _case(seed, B, H, S, hd=128, n_img=None, soft=False, bias=0.5):
    rng = np.random.default_rng(seed)
    Q = torch.from_numpy(rng.standard_normal((B, H, S, hd), dtype=np.float32)).to(torch.bfloat16)
    K = torch.from_numpy(rng.standard_normal((B, H, S, hd), dtype=np.float32)).to(torch.bfloat16)
    n_img = S // 4 if n_img is None else n_img
    is_vis = np.zeros((B, S), dtype=np.uint8)
    is_vis[:, :n_img] = 1
    m = rng.uniform(0, 1, (B, S)).astype(np.float32) if soft else is_vis.astype(np.float32)
    key_bias = (bias * is_vis).astype(np.float32)
    return Q, K, is_vis, m, key_bias


def _run(bd, Q, K, is_vis, m, key_bias, causal, soft, norms=None):
    B, H, S, hd = Q.shape
    T = B * S
    r = bd.Router(T, 64, 16, 2, 4, [0, T], np.arange(16) // 4, attn_max_heads=H)
    M = torch.empty((T, 2), dtype=torch.float32, device="cuda")
    attn = dict(Q=Q.cuda(), K=K.cuda(), B=B, H=H, S=S, hd=hd, sm_scale=1.0 / np.sqrt(hd),
                causal=int(causal), key_bias=torch.from_numpy(key_bias.reshape(-1)).cuda())
    if soft:
        attn["m_prev"] = torch.from_numpy(m.reshape(-1)).cuda()
    else:
        attn["is_vision"] = torch.from_numpy(is_vis.reshape(-1)).cuda()
    if norms is not None:
        attn["xattn_norm"] = torch.from_numpy(norms[0]).cuda()
        attn["x_norm"] = torch.from_numpy(norms[1]).cuda()
    r.modality_score(bd.SMOES_SCORE_ATTN, M, attn=attn)
    code, _ = r.device_status()
    assert code == 0
    out = M.cpu().numpy()
    np.testing.assert_allclose(out.sum(axis=1), 1.0, rtol=0, atol=1e-6)
    return out[:, 0].reshape(B, S)


@pytest.mark.parametrize("B,H,S,causal,soft", [
    (2, 3, 300, True, False),
    (1, 2, 513, True, True),
    (2, 2, 200, False, False),
    (3, 4, 77, True, False),
    (1, 16, 1024, True, False),
    (20, 16, 256, True, False),
])
def test_attention_mass_parity(bd, B, H, S, causal, soft):
    Q, K, is_vis, m, key_bias = _case(B * 100 + S, B, H, S, soft=soft)
    got = _run(bd, Q, K, is_vis, m, key_bias, causal, soft)
    ref = O.attention_vision_mass(Q.double().numpy(), K.double().numpy(), m, 1.0 / np.sqrt(128),
                                  causal, key_bias)
    assert_tensor_close(got, ref, "attention vision mass")
    if causal and not soft:
        # image tokens come first: every image query attends to image keys only
        np.testing.assert_allclose(got[:, :S // 4], 1.0, rtol=0, atol=1e-6)


def test_attention_mass_residual_update(bd):
    B, H, S = 2, 2, 260
    Q, K, is_vis, m, key_bias = _case(5, B, H, S, soft=True)
    rng = np.random.default_rng(9)
    an = rng.uniform(0.5, 2.0, B * S).astype(np.float32)
    xn = rng.uniform(0.5, 2.0, B * S).astype(np.float32)
    got = _run(bd, Q, K, is_vis, m, key_bias, True, True, norms=(an, xn))
    mt = O.attention_vision_mass(Q.double().numpy(), K.double().numpy(), m, 1.0 / np.sqrt(128), True,
                                 key_bias)
    ref = O.residual_score_update(mt.reshape(-1), m.reshape(-1), an, xn).reshape(B, S)
    assert_tensor_close(got, ref, "eq. (4) blend")
