"""Host-side arithmetic of bench.py (no GPU): the algorithmic bytes and flops behind the
roofline fractions, the rule that an ncu traffic record counts only for the sources it was
taken on, and the expert-parallel transfer ratios derived from a dispatch."""
import hashlib
import json
import os
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

bench = pytest.importorskip("bench")
from paper_2604_23996_gb300.workloads import config_workload  # noqa: E402


def test_algorithmic_bytes_dsmoe_vlm():
    # T = 16384, d = 2048, E = 64, k = 6, K = 8, bf16 (b = 2)
    wl = config_workload("dsmoe_vlm")
    step_bytes, step_flops, fwd_bytes, bwd_bytes = bench.algorithmic(wl)
    T, d, E, k, K, b = 16384, 2048, 64, 6, 8, 2
    assert fwd_bytes == T * (d * b + 8 * k + 8 + 8 * min(k, K)) + E * d * b == 69074944
    assert bwd_bytes == T * (2 * d * b + 8) + E * d * (b + 4) == 135135232
    assert step_bytes == T * (3 * d * b + 8 * k + 16 + 4 * k + 8 * min(k, K)) + E * d * (b + 4)
    assert step_flops == 6.0 * T * d * E
    # the step moves at least what its two calls move (the permutation reads the top-k again)
    assert step_bytes >= fwd_bytes + bwd_bytes - E * d * b


def test_traffic_record_only_for_its_source(tmp_path, monkeypatch):
    prof = tmp_path / "profiles"
    src_dir = tmp_path / "paper_2604_23996_gb300" / "csrc"
    prof.mkdir()
    src_dir.mkdir(parents=True)
    src = src_dir / "router_fwd.cu"
    hdr = src_dir / "router_fwd_tc.cuh"
    src.write_text("// kernel v1\n")
    hdr.write_text("// header v1\n")
    sha = hashlib.sha256(src.read_bytes() + hdr.read_bytes()).hexdigest()[:16]
    (prof / "traffic_w_fwd.json").write_text(json.dumps({"source_sha": sha, "dram_bytes_per_launch": 123.0}))
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    files = ["router_fwd.cu", "router_fwd_tc.cuh"]
    assert bench.profile_traffic(files, "w", "fwd") == 123.0
    hdr.write_text("// header v2\n")                     # a source of the kernel changed since
    assert bench.profile_traffic(files, "w", "fwd") is None
    hdr.write_text("// header v1\n")
    assert bench.profile_traffic(files, "other", "fwd") is None
    assert bench.profile_traffic(["router_fwd.cu"], "w", "fwd") is None   # a different source set


def test_dedup_report_counts_remote_transfers():
    # a tiny dispatch through the oracle's permutation, read back by the bench's report, against a
    # brute-force count over the (token, expert) selections with home(j) = floor(j K / T)
    from types import SimpleNamespace

    import torch

    from oracle import smoes_oracle as O
    rng = np.random.default_rng(3)
    T, E, k, K = 37, 12, 3, 4
    eb = np.arange(E) // (E // K)
    topk = np.stack([rng.choice(E, k, replace=False) for _ in range(T)]).astype(np.int32)
    pr = O.bin_permute(topk, eb, K)
    r = SimpleNamespace(dispatch=torch.from_numpy(pr["dispatch"].astype(np.int32)),
                        bin_offsets=torch.from_numpy(pr["offsets"].astype(np.int32)),
                        perm_token=torch.from_numpy(pr["perm"].astype(np.int32)),
                        perm_mask=torch.from_numpy(pr["mask"].astype(np.uint32).view(np.int32)))
    st = SimpleNamespace(r=r, wl=SimpleNamespace(T=T, n_bins=K, k=k))
    rep = bench.dedup_report(st)
    home = (np.arange(T) * K) // T
    remote_sel = sum(int(eb[e] != home[j]) for j in range(T) for e in topk[j])
    remote_pairs = sum(len({int(eb[e]) for e in topk[j]} - {int(home[j])}) for j in range(T))
    assert rep["ratio_without_dedup"] == remote_sel / (T * k)
    assert rep["ratio_with_dedup"] == remote_pairs / T
    assert rep["ratio_with_dedup_per_selection"] == remote_pairs / (T * k)
    assert rep["dedup_saving"] == 1.0 - remote_pairs / remote_sel
    assert rep["check"].endswith("True")
    assert rep["ratio_with_dedup"] <= rep["ratio_without_dedup"] * k


def test_reference_arm_config_names_the_same_workload():
    wl = config_workload("tiny_fp32")
    ours = bench.bench_config("tiny_fp32", wl, 1)
    ref = bench.reference_config("tiny_fp32", wl, 1)
    assert ref["workload"] == ours["workload"] and ref["parallelism"] == ours["parallelism"]
    assert "CUDA graph" in ours["timing"] and "host wall clock" in ref["timing"]
    assert ref["l2"].startswith("not applicable")
