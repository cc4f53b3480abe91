"""GPU parity of the standalone Gaussian-statistics score (eqs. 8-9) against the fp64 oracle."""
import numpy as np
import pytest
import torch

from oracle import smoes_oracle as O
from paper_2604_23996_gb300.workloads import random_router_case

from .parity import assert_tensor_close

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("dtype,d,tau", [(torch.bfloat16, 264, None), (torch.float32, 128, 1.0),
                                         (torch.bfloat16, 2048, 1.0)])
def test_gauss_score_parity(dtype, d, tau):
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2604_23996_gb300 import binding as bd
    wl = random_router_case(41, 999, d, 16, 2, 4, [500, 499], dtype=dtype, tau=tau)
    r = bd.Router(wl.T, wl.d, wl.E, wl.k, wl.n_bins, wl.sample_offsets, wl.expert_bin,
                  bd.SMOES_BF16 if dtype == torch.bfloat16 else bd.SMOES_F32)
    M = torch.empty((wl.T, 2), dtype=torch.float32, device="cuda")
    r.modality_score(bd.SMOES_SCORE_GAUSS, M, X=wl.X.cuda(), mu=wl.mu.cuda(), var=wl.var.cuda(),
                     tau=wl.tau)
    assert r.device_status()[0] == 0
    ref = O.gaussian_score(wl.X.double().numpy(), wl.mu.double().numpy(), wl.var.double().numpy(),
                           wl.tau)
    assert_tensor_close(M.cpu().numpy(), ref, "M")
    # the fused forward produces the same scores
    r.forward(wl.X.cuda(), wl.W.cuda(), mu=wl.mu.cuda(), var=wl.var.cuda(), tau=wl.tau)
    assert_tensor_close(r.M.cpu().numpy(), ref, "M (fused)")
