"""Exact ties in the top-k choice (Sec. 3.1), bit for bit against the fp64 oracle.

The paper fixes no tie rule; the reading used on both sides is: descending logit, equal logits
ordered by ascending expert index. Duplicated gate rows (W_a = W_b) give every token two
bit-identical logits, and a negated duplicate (W_c = -W_a) gives bit-identical logits of the
opposite sign, so the rule is exercised for positive and negative ties, inside the top-k and at
its boundary (rank k vs k + 1), within one epilogue group and across the two. Only tokens whose
*distinct* logit values among the top k + 1 come closer than the usual 1e-3 gap are excluded;
exact ties are never excluded. The permutation of the forward's own top-k is compared too.
"""
import numpy as np
import pytest
import torch

from oracle import smoes_oracle as O
from paper_2604_23996_gb300.workloads import random_router_case

from .parity import TIE_GAP, run_gpu

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def bd():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2604_23996_gb300 import binding
    return binding


# name: (seed, T, d, E, k, n_bins, dtype, rows made equal (dst <- src), rows negated (dst <- -src))
CASES = {
    # a pair inside bin 0, a pair across bins, a negated pair; k = 3 puts pairs on the boundary
    "e16_k3": (41, 900, 256, 16, 3, 4, torch.bfloat16, [(1, 0), (9, 4)], [(2, 0), (14, 0)]),
    # every logit in a +/- pair: the top 5 / 6 always reach a negative tied pair
    "e8_k5": (42, 700, 192, 8, 5, 2, torch.bfloat16, [(1, 0), (5, 4)], [(2, 0), (3, 0), (6, 4), (7, 4)]),
    "e8_k6": (43, 700, 192, 8, 6, 4, torch.bfloat16, [(1, 0), (5, 4)], [(2, 0), (3, 0), (6, 4), (7, 4)]),
    # E = 64: the epilogue splits columns 0-31 / 32-63 between two warp groups; pairs straddle it
    "e64_k6_split": (44, 1100, 256, 64, 6, 8, torch.bfloat16, [(40, 5), (33, 31), (62, 1)],
                     [(50, 20), (21, 5), (63, 31)]),
    # the fp32 path
    "f32_e16_k3": (45, 600, 128, 16, 3, 4, torch.float32, [(1, 0), (9, 4)], [(2, 0), (14, 0)]),
}


def _tie_workload(name):
    seed, T, d, E, k, K, dt, dup, neg = CASES[name]
    wl = random_router_case(seed, T, d, E, k, K, [T // 3, T - T // 3], dtype=dt, aligned=True)
    W = wl.W.clone()
    for src in {s for _, s in dup + neg}:       # stronger rows: their pairs reach the top k often
        W[src] = W[src] * 3
    for dst, src in dup:
        W[dst] = W[src]
    for dst, src in neg:
        W[dst] = -W[src]
    wl.W = W
    return wl


def _distinct_gap_ok(z, k):
    """Tokens whose distinct logit values among the top k + 1 are all at least TIE_GAP apart
    (exactly equal logits count as one value)."""
    ok = np.ones(z.shape[0], bool)
    srt = -np.sort(-z, axis=1)[:, :k + 1]
    for j in range(z.shape[0]):
        u = np.unique(srt[j])[::-1]
        if len(u) > 1 and np.any(u[:-1] - u[1:] < TIE_GAP):
            ok[j] = False
    return ok


@pytest.mark.parametrize("name", list(CASES))
@pytest.mark.parametrize("fused", [False, True])
def test_exact_ties_bit_exact(bd, name, fused):
    wl = _tie_workload(name)
    Xd = wl.X.double().numpy()
    z = O.gate_logits(Xd, wl.W.double().numpy())
    _, _, _, _, _, _, _, dup, neg = CASES[name]
    for dst, src in dup:                          # the oracle's logits tie exactly as well
        assert np.array_equal(z[:, dst], z[:, src])
    for dst, src in neg:
        assert np.array_equal(z[:, dst], -z[:, src])
    g = np.exp(z - z.max(1, keepdims=True))
    g /= g.sum(1, keepdims=True)
    idx_ref, w_ref = O.topk_route(z, g, wl.k)
    # tokens on which a tie decides the order or the choice: two equal logits among the top k + 1
    srt = -np.sort(-z, axis=1)[:, :wl.k + 1]
    tied = np.any(srt[:, :-1] == srt[:, 1:], axis=1)
    ok = _distinct_gap_ok(z, wl.k)
    assert (tied & ok).sum() >= 0.3 * wl.T, "the case must exercise ties on many tokens"

    out = run_gpu(wl, bd, mode="gauss", fused=fused, want_dx=False, want_dlogits=False)
    assert out["status"] == 0
    np.testing.assert_array_equal(out["topk_idx"][ok], idx_ref[ok], err_msg="top-k on exact ties")
    # the tied experts carry equal weights
    rel = np.abs(out["topk_w"][ok] - w_ref[ok]) / np.abs(w_ref[ok]).max()
    assert rel.max() < 2e-3
    # the permutation of the GPU's own top-k, bit for bit
    pr = O.bin_permute(out["topk_idx"], wl.expert_bin, wl.n_bins, is_vision=wl.is_vision)
    for key in ("offsets", "perm", "dispatch", "expert_counts"):
        np.testing.assert_array_equal(out[key], pr[key], err_msg=key)
    print(f"{name} fused={fused}: {int((tied & ok).sum())} tokens with exact ties compared, "
          f"{int((~ok).sum())} near-tie tokens excluded")
