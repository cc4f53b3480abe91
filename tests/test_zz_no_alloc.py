"""The permutation entry point that allocates nothing (smoes_bin_permute_noalloc), for callers
that cannot allocate device memory: it must give exactly what the workspace version gives, and
keep doing so on a second call that reuses the library's fixed scratch. This file is collected
last on purpose, so a stop-at-first-failure run has already run every other test."""
import numpy as np
import pytest
import torch

from paper_2604_23996_gb300.workloads import random_router_case

pytestmark = pytest.mark.gpu


def _outputs(T, k, K, E, dev):
    cap = T * min(k, K)
    return dict(bin_offsets=torch.full((K + 1,), -1, dtype=torch.int32, device=dev),
                perm_token=torch.full((cap,), -1, dtype=torch.int32, device=dev),
                perm_mask=torch.full((cap,), -1, dtype=torch.int32, device=dev),
                dispatch=torch.full((K, K), -1, dtype=torch.int32, device=dev),
                expert_counts=torch.full((2, E), -1, dtype=torch.int32, device=dev))


def test_noalloc_permutation_matches_workspace_version_twice():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2604_23996_gb300 import binding as bd
    dev = "cuda"
    wl = random_router_case(31, 3001, 256, 64, 6, 8, [1000, 1500, 501], aligned=True)
    r = bd.Router(wl.T, wl.d, wl.E, wl.k, wl.n_bins, wl.sample_offsets, wl.expert_bin)
    X, W = wl.X.to(dev), wl.W.to(dev)
    r.forward(X, W, mu=wl.mu.to(dev), var=wl.var.to(dev), tau=wl.tau)
    is_vis = torch.from_numpy(wl.is_vision).to(dev)
    r.permute(is_vision=is_vis)                          # the workspace version
    torch.cuda.synchronize()
    n = int(r.bin_offsets[-1].item())
    ref = dict(bin_offsets=r.bin_offsets.cpu().numpy(), perm_token=r.perm_token[:n].cpu().numpy(),
               perm_mask=r.perm_mask[:n].cpu().numpy(), dispatch=r.dispatch.cpu().numpy(),
               expert_counts=r.expert_counts.cpu().numpy())
    for call in range(2):
        out = _outputs(wl.T, wl.k, wl.n_bins, wl.E, dev)
        code = bd.smoes_bin_permute_noalloc(r.plan, r.topk_idx, None, is_vis, out["bin_offsets"],
                                            out["perm_token"], out["perm_mask"], out["dispatch"],
                                            out["expert_counts"])
        assert code == 0, bd.smoes_status_string(code)
        torch.cuda.synchronize()
        for key, want in ref.items():
            got = out[key].cpu().numpy()
            if key in ("perm_token", "perm_mask"):
                got = got[:n]
            np.testing.assert_array_equal(got, want, err_msg=f"call {call}: {key}")
