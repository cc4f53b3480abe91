"""Host-side checks of the C ABI (no GPU needed): the library builds and loads, exports every
entry point include/smoes.h declares, and plan creation validates its arguments."""
import os
import re

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def bd():
    from paper_2604_23996_gb300.build import build_library
    build_library()
    from paper_2604_23996_gb300 import binding
    return binding


def declared_functions():
    text = open(os.path.join(ROOT, "include", "smoes.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(smoes_[a-z_]+)\s*\(", text)))


def test_header_declares_the_four_path_calls():
    fns = declared_functions()
    for name in ("smoes_router_fwd", "smoes_router_bwd", "smoes_modality_score", "smoes_bin_permute"):
        assert name in fns


def test_library_exports_every_declared_symbol(bd):
    import ctypes
    lib = ctypes.CDLL(bd.LIB)
    for name in declared_functions():
        assert hasattr(lib, name), name
    assert set(declared_functions()) == set(bd.exported_symbols())


def _plan(bd, **kw):
    args = dict(T=100, d=64, E=16, k=2, n_bins=4, sample_offsets=[0, 40, 100],
                expert_bin=np.arange(16) // 4, dtype=bd.SMOES_BF16)
    args.update(kw)
    return bd.smoes_plan_create(**args)


def test_plan_create_ok_and_workspace_size(bd):
    code, plan = _plan(bd)
    assert code == 0
    n = bd.smoes_workspace_bytes(plan)
    assert n > 100 * 16 * 4            # at least the saved softmax scores
    bd.smoes_plan_destroy(plan)


@pytest.mark.parametrize("kw,code", [
    (dict(d=60), -1),                                        # d % 8 != 0
    (dict(k=17, E=32, expert_bin=np.arange(32) // 8), -2),   # k > 16
    (dict(E=18, expert_bin=np.arange(18) % 4), -1),          # E % n_bins != 0
    (dict(sample_offsets=[0, 40, 90]), -1),                  # o_B != T
    (dict(sample_offsets=[0, 40, 40, 100]), -1),             # empty sample
    (dict(expert_bin=np.array([0] * 5 + [1] * 3 + [2] * 4 + [3] * 4)), -1),   # unequal bins
    (dict(expert_bin=np.arange(16) // 4 + 1), -1),           # bin out of range
    (dict(n_bins=64, E=64, expert_bin=np.arange(64)), -2),   # more than 32 bins
    (dict(k=0), -1),
    # the limits every later call can run: E <= 128 (bf16), E <= 64 (fp32), T <= 2^20
    (dict(E=256, k=8, n_bins=8, expert_bin=np.arange(256) // 32), -2),
    (dict(E=136, k=8, n_bins=8, expert_bin=np.arange(136) // 17), -2),
    (dict(E=128, k=8, n_bins=16, expert_bin=np.arange(128) // 8, dtype=0), -2),
    (dict(T=(1 << 20) + 1, sample_offsets=[0, (1 << 20) + 1]), -2),
])
def test_plan_create_rejects(bd, kw, code):
    got, plan = _plan(bd, **kw)
    assert got == code


@pytest.mark.parametrize("kw", [
    dict(E=128, k=8, n_bins=16, expert_bin=np.arange(128) // 8),            # largest bf16 plan
    dict(E=64, k=6, n_bins=8, expert_bin=np.arange(64) // 8, dtype=0),      # largest fp32 plan
    dict(T=1 << 20, sample_offsets=[0, 1 << 19, 1 << 20]),                  # largest batch
])
def test_plan_create_accepts_the_limits(bd, kw):
    got, plan = _plan(bd, **kw)
    assert got == 0
    bd.smoes_plan_destroy(plan)


def test_wait_limit_setter(bd):
    code, plan = _plan(bd)
    assert bd.smoes_plan_set_wait_limit(plan, 1000) == 0
    assert bd.smoes_plan_set_wait_limit(plan, 0) == 0        # back to the default
    assert bd.smoes_plan_set_wait_limit(None, 10) == -1
    bd.smoes_plan_destroy(plan)


def test_call_launch_counts(bd):
    # the host's SM count decides the fused permutation: 2 tiles per SM at most (any GPU has more
    # than 8 SMs and fewer than 4096)
    code, small = _plan(bd)                                                 # 1 tile
    assert code == 0
    assert bd.smoes_call_launches(small, bd.SMOES_CALL_ROUTER_FWD) == 1
    assert bd.smoes_call_launches(small, bd.SMOES_CALL_ROUTER_FWD_PERMUTE) == 1
    assert bd.smoes_call_launches(small, bd.SMOES_CALL_ROUTER_BWD) == 3    # dz prep, main, dW sum
    assert bd.smoes_call_launches(small, bd.SMOES_CALL_BIN_PERMUTE) == 1
    assert bd.smoes_call_launches(small, bd.SMOES_CALL_ATTN_SCORE) == 1
    assert bd.smoes_call_launches(small, 99) == -1
    assert bd.smoes_call_launches(None, bd.SMOES_CALL_ROUTER_FWD) == -1
    code, big = _plan(bd, T=1 << 20, sample_offsets=[0, 1 << 20])           # 8192 tiles
    assert code == 0
    assert bd.smoes_call_launches(big, bd.SMOES_CALL_ROUTER_FWD_PERMUTE) == 2
    code, f32 = _plan(bd, dtype=bd.SMOES_F32)
    assert code == 0
    assert bd.smoes_call_launches(f32, bd.SMOES_CALL_ROUTER_FWD_PERMUTE) == 2
    assert bd.smoes_call_launches(f32, bd.SMOES_CALL_ROUTER_BWD) == 2      # main, dW sum
    code, empty = bd.smoes_plan_create(0, 64, 16, 2, 4, [0], np.arange(16) // 4, bd.SMOES_BF16)
    assert code == 0
    assert bd.smoes_call_launches(empty, bd.SMOES_CALL_ROUTER_BWD) == 0
    for p in (small, big, f32, empty):
        bd.smoes_plan_destroy(p)


def test_empty_batch_plan(bd):
    code, plan = bd.smoes_plan_create(0, 64, 16, 2, 4, [0], np.arange(16) // 4, bd.SMOES_BF16)
    assert code == 0
    bd.smoes_plan_destroy(plan)


def test_status_strings(bd):
    assert bd.smoes_status_string(0) == "ok"
    assert "workspace" in bd.smoes_status_string(-4)
