"""GPU parity of the Gaussian-mixture modality score (the estimator the paper explores beyond the
single Gaussian of eq. 8) against the fp64 oracle: 1 to 4 components per modality, bf16 and fp32
features, d not a multiple of the 256-feature blocks; one component reproduces the Gaussian score
of eqs. (8)-(9)."""
import numpy as np
import pytest
import torch

from oracle import smoes_oracle as O
from paper_2604_23996_gb300.workloads import random_router_case

from .parity import assert_tensor_close

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def bd():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2604_23996_gb300 import binding
    return binding


def _mixture(wl, C, seed):
    """Per modality, C components around the batch statistics (shifted means, scaled variances)."""
    rng = np.random.default_rng(seed)
    mu = np.repeat(wl.mu.numpy()[:, None, :], C, axis=1) + 0.3 * rng.standard_normal((2, C, wl.d))
    var = np.repeat(wl.var.numpy()[:, None, :], C, axis=1) * rng.uniform(0.7, 1.4, (2, C, wl.d))
    w = rng.uniform(0.3, 1.0, (2, C))
    log_pi = np.log(w / w.sum(axis=1, keepdims=True))
    return log_pi.astype(np.float32), mu.astype(np.float32), var.astype(np.float32)


def _gpu_gmm(bd, wl, log_pi, mu, var, tau):
    dt = bd.SMOES_BF16 if wl.dtype == torch.bfloat16 else bd.SMOES_F32
    r = bd.Router(wl.T, wl.d, 16, 2, 4, [0, wl.T], np.arange(16) // 4, dt)
    M = torch.empty((wl.T, 2), device="cuda")
    C = mu.shape[1]
    g = dict(X=wl.X.cuda(), n_components=C, log_pi=torch.from_numpy(log_pi).cuda(),
             mu=torch.from_numpy(np.ascontiguousarray(mu)).cuda(),
             var=torch.from_numpy(np.ascontiguousarray(var)).cuda(), tau=tau)
    code = bd.smoes_modality_score(r.plan, bd.SMOES_SCORE_GMM, M, r.ws, gmm=g)
    return code, r, M


@pytest.mark.parametrize("C,dtype,d,tau", [(1, torch.bfloat16, 200, 1.0), (2, torch.bfloat16, 520, 1.0),
                                           (3, torch.float32, 136, 2.0), (4, torch.bfloat16, 1288, 0.0),
                                           (2, torch.float32, 64, 1.0)])
def test_gmm_score_parity(bd, C, dtype, d, tau):
    wl = random_router_case(80 + C, 900, d, 16, 2, 4, [900], dtype=dtype, aligned=True)
    log_pi, mu, var = _mixture(wl, C, 90 + C)
    code, r, M = _gpu_gmm(bd, wl, log_pi, mu, var, tau)
    assert code == 0, bd.smoes_status_string(code)
    assert r.device_status()[0] == 0
    ref = O.gmm_score(wl.X.double().numpy(), log_pi, mu, var, tau if tau > 0 else 0.5 * d)
    e = assert_tensor_close(M.cpu().numpy(), ref, f"GMM score C={C}")
    print(f"C={C} d={d}: rel err {e:.2e}, M_v range {ref[:, 0].min():.3f}..{ref[:, 0].max():.3f}")


def test_one_component_matches_the_gaussian_mode(bd):
    wl = random_router_case(85, 700, 256, 16, 2, 4, [700], aligned=True)
    log_pi = np.zeros((2, 1), np.float32)
    mu = wl.mu.numpy()[:, None, :].copy()
    var = wl.var.numpy()[:, None, :].copy()
    code, r, M = _gpu_gmm(bd, wl, log_pi, mu, var, 1.0)
    assert code == 0
    Mg = torch.empty_like(M)
    assert bd.smoes_modality_score(r.plan, bd.SMOES_SCORE_GAUSS, Mg, r.ws, X=wl.X.cuda(),
                                   mu=wl.mu.cuda(), var=wl.var.cuda(), tau=1.0) == 0
    torch.cuda.synchronize()
    np.testing.assert_allclose(M.cpu().numpy(), Mg.cpu().numpy(), rtol=0, atol=2e-6)


def test_gmm_limits(bd):
    wl = random_router_case(86, 128, 64, 16, 2, 4, [128], aligned=True)
    log_pi, mu, var = _mixture(wl, 4, 1)
    lp5 = np.zeros((2, 5), np.float32)
    mu5 = np.zeros((2, 5, 64), np.float32)
    code, _, _ = _gpu_gmm(bd, wl, lp5, mu5, mu5 + 1.0, 1.0)
    assert code == -2                                          # more than 4 components
    var[0, 1, 3] = -1.0                                        # a non-positive variance
    code, r, _ = _gpu_gmm(bd, wl, log_pi, mu, var, 1.0)
    assert code == 0 and r.device_status()[0] == -7
