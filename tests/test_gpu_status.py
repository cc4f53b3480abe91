"""Bounded device waits: a wait that runs out is reported through the workspace status word and
the kernel returns; the context stays usable and the workspace works again after
re-initialisation.

The permutation's grid barrier is the wait under test. With the plan's wait limit at 1 ns, any
block that reaches the barrier before the last one gives up at its first poll (the blocks of a
2^20-token batch reach it microseconds apart), records SMOES_ERR_DEVICE_TIMEOUT and returns
without placing its entries; the last block to arrive resets the barrier words on its way
through, so nothing is left waiting and no state outlives the call.
"""
import numpy as np
import pytest
import torch

from oracle import smoes_oracle as O

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def bd():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2604_23996_gb300 import binding
    return binding


def test_grid_barrier_timeout_is_reported_and_recoverable(bd):
    T, E, k, K = 1 << 20, 64, 8, 8
    rng = np.random.default_rng(5)
    idx = np.argsort(rng.random((T, E)), axis=1)[:, :k].astype(np.int32)    # distinct experts
    r = bd.Router(T, 64, E, k, K, [0, T], np.arange(E) // (E // K))
    top = torch.from_numpy(idx).cuda()
    assert bd.smoes_plan_set_wait_limit(r.plan, 1) == 0
    r.permute(topk_idx=top)
    code, _ = r.device_status()
    assert code == -6, bd.STATUS_NAMES.get(code, code)           # SMOES_ERR_DEVICE_TIMEOUT

    # default limit, fresh status word: the same call completes and is exact
    assert bd.smoes_plan_set_wait_limit(r.plan, 0) == 0
    assert bd.smoes_workspace_init(r.plan, r.ws) == 0
    r.permute(topk_idx=top)
    code, _ = r.device_status()
    assert code == 0
    pr = O.bin_permute(idx, np.arange(E) // (E // K), K)
    n = int(r.bin_offsets[-1].item())
    np.testing.assert_array_equal(r.bin_offsets.cpu().numpy(), pr["offsets"])
    np.testing.assert_array_equal(r.perm_token[:n].cpu().numpy(), pr["perm"])
    np.testing.assert_array_equal(r.dispatch.cpu().numpy(), pr["dispatch"])


def test_wait_limit_rejects_null_plan(bd):
    assert bd.smoes_plan_set_wait_limit(None, 5) == -1
