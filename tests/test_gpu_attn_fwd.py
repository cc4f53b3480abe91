"""GPU parity of the attention forward with the vision score as one more value column (Sec. 3.2.1,
eqs. 2-4) against the fp64 oracle: O = softmax(s Q K^T + bias) V per head and the head-averaged
vision mass, causal and not, grouped-query heads (H / H_kv = 1, 2, 4), hard labels and a carried
float score with the eq. (4) blend.

Tolerance of O (stored in bf16): the softmax weights reach the tensor cores in bf16 (relative
error 2^-9 each), which moves an output by at most 2^-9 max|V|, and the output's own rounding adds
half a bf16 ulp; the bar is one ulp of the exact value + 2^-8 max|V| per element, and 2e-3 + 2^-8
in norm. The score M (fp32 softmax weights) meets the 2e-3 bar of every floating-point output.
"""
import numpy as np
import pytest
import torch

from oracle import smoes_oracle as O
from paper_2604_23996_gb300.workloads import attn_workload

from .parity import assert_tensor_close, bf16_ulp

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def bd():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2604_23996_gb300 import binding
    return binding


def _case(B, H, Hkv, S, seed, n_image):
    aw = attn_workload(B=B, H=H, S=S, hd=128, n_image=n_image, seed=seed)
    rng = np.random.default_rng(seed + 7)
    # keys and values with H_kv heads (the query heads of a group share them)
    K = torch.from_numpy(rng.standard_normal((B, Hkv, S, 128), dtype=np.float32)).to(torch.bfloat16)
    V = torch.from_numpy(rng.standard_normal((B, Hkv, S, 128), dtype=np.float32)).to(torch.bfloat16)
    return aw, K, V


def _run(bd, aw, K, V, Hkv, causal=1, m_prev=None, norms=None):
    T = aw.B * aw.S
    r = bd.Router(T, 64, 16, 2, 4, [0, T], np.arange(16) // 4, attn_max_heads=aw.H)
    M = torch.empty((T, 2), device="cuda")
    Ot = torch.empty((aw.B, aw.H, aw.S, 128), dtype=torch.bfloat16, device="cuda")
    attn = dict(Q=aw.Q.cuda(), K=K.cuda(), B=aw.B, H=aw.H, S=aw.S, hd=128, sm_scale=aw.sm_scale,
                causal=causal, key_bias=torch.from_numpy(aw.key_bias).cuda())
    if m_prev is None:
        attn["is_vision"] = torch.from_numpy(aw.is_vision).cuda()
    else:
        attn["m_prev"] = torch.from_numpy(m_prev).cuda()
    if norms is not None:
        attn["xattn_norm"] = torch.from_numpy(norms[0]).cuda()
        attn["x_norm"] = torch.from_numpy(norms[1]).cuda()
    code = bd.smoes_attention_fwd(r.plan, attn, V.cuda(), Hkv, Ot, M, r.ws)
    assert code == 0, bd.smoes_status_string(code)
    assert r.device_status()[0] == 0
    torch.cuda.synchronize()
    return r, attn, Ot.float().cpu().numpy(), M.cpu().numpy()


def _check_O(got, ref, Vmax, what):
    err = np.abs(got - ref)
    bad = err > bf16_ulp(ref) + 2.0 ** -8 * Vmax
    assert not np.any(bad), f"{what}: {int(bad.sum())} elements off; worst {err.max():.3e}"
    rel = np.linalg.norm(got - ref) / np.linalg.norm(ref)
    assert rel <= 2e-3 + 2.0 ** -8, f"{what}: rel L2 {rel:.3e}"
    return rel


@pytest.mark.parametrize("B,H,Hkv,S,causal", [(2, 4, 4, 256, 1), (1, 4, 2, 384, 1), (2, 8, 2, 256, 1),
                                              (1, 4, 1, 128, 1), (1, 2, 2, 256, 0)])
def test_attention_forward_with_mass(bd, B, H, Hkv, S, causal):
    aw, K, V = _case(B, H, Hkv, S, seed=200 + S + H, n_image=S // 4)
    _, _, Og, Mg = _run(bd, aw, K, V, Hkv, causal=causal)
    m = aw.is_vision.reshape(B, S).astype(np.float64)
    Oref, mass = O.attention_forward_with_mass(aw.Q.double().numpy(), K.double().numpy(), V.double().numpy(),
                                               m, aw.sm_scale, bool(causal), aw.key_bias.reshape(B, S))
    e = _check_O(Og, Oref, float(V.float().abs().max()), "O")
    assert_tensor_close(Mg[:, 0], mass.reshape(-1), "vision mass")
    np.testing.assert_array_equal(Mg[:, 1], (1.0 - Mg[:, 0]).astype(np.float32))
    print(f"B{B} H{H} Hkv{Hkv} S{S} causal{causal}: O rel L2 {e:.2e}")


def test_carried_float_score_and_residual_blend(bd):
    B, H, Hkv, S = 2, 4, 2, 256
    aw, K, V = _case(B, H, Hkv, S, seed=301, n_image=64)
    rng = np.random.default_rng(3)
    m_prev = rng.uniform(0.0, 1.0, B * S).astype(np.float32)
    an = rng.uniform(0.5, 2.0, B * S).astype(np.float32)
    xn = rng.uniform(0.5, 2.0, B * S).astype(np.float32)
    _, _, Og, Mg = _run(bd, aw, K, V, Hkv, m_prev=m_prev, norms=(an, xn))
    Oref, mass = O.attention_forward_with_mass(aw.Q.double().numpy(), K.double().numpy(), V.double().numpy(),
                                               m_prev.reshape(B, S).astype(np.float64), aw.sm_scale, True,
                                               aw.key_bias.reshape(B, S))
    _check_O(Og, Oref, float(V.float().abs().max()), "O")
    ref = O.residual_score_update(mass.reshape(-1), m_prev, an, xn)
    assert_tensor_close(Mg[:, 0], ref, "blended score (eq. 4)")


def test_score_equals_the_mass_only_kernel(bd):
    # with H_kv = H the score of the forward and of smoes_modality_score(ATTN) are the same quantity
    B, H, S = 2, 4, 512
    aw, _, V = _case(B, H, H, S, seed=302, n_image=128)
    r, attn, _, Mg = _run(bd, aw, aw.K, V, H)
    M2 = torch.empty((B * S, 2), device="cuda")
    r.modality_score(bd.SMOES_SCORE_ATTN, M2, attn=attn)
    torch.cuda.synchronize()
    assert_tensor_close(Mg[:, 0], M2.cpu().numpy()[:, 0], "forward vs mass-only score")


def test_attention_forward_limits(bd):
    aw, K, V = _case(1, 4, 4, 128, seed=303, n_image=32)
    T = aw.S
    r = bd.Router(T, 64, 16, 2, 4, [0, T], np.arange(16) // 4, attn_max_heads=4)
    M = torch.empty((T, 2), device="cuda")
    Ot = torch.empty((1, 4, 128, 128), dtype=torch.bfloat16, device="cuda")
    attn = dict(Q=aw.Q.cuda(), K=K.cuda(), B=1, H=4, S=128, hd=128, sm_scale=aw.sm_scale, causal=1,
                is_vision=torch.from_numpy(aw.is_vision).cuda())
    assert bd.smoes_attention_fwd(r.plan, attn, V.cuda(), 3, Ot, M, r.ws) == -1     # H % H_kv != 0
    assert bd.smoes_attention_fwd(r.plan, dict(attn, hd=64), V.cuda(), 4, Ot, M, r.ws) == -2
