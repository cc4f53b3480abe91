#!/usr/bin/env python
"""Router fwd+bwd throughput of the SMoES hot path on GB300 (one JSON line on stdout).

A step is one pass of the whole router hot path over one batch of the workload:
  smoes_router_fwd_permute (gate GEMM + Gaussian modality score + softmax/top-k/bins + per-sample
  MI + the de-duplicated bin dispatch of the top-k, one launch) -> smoes_router_bwd (MI gradient
  -> dW and dX).
Default workload: the DeepSeekMoE-style VLM layer, T = 16384 tokens (8 x [576 image + 1472 text]),
d = 2048, E = 64 routed experts, top-6, 8 bins, bf16. Inputs are seeded synthetic data.

Timing: W warm-up steps, then K timed steps. The step (all calls) is replayed from one CUDA
graph; before every step the L2 is flushed by writing a 256 MiB buffer (outside the timed
interval), and CUDA events on the launching stream bracket each step. A second pass of K steps
replays a copy of the graph with an event after every call, for the per-call breakdown and the
backward call's duration. --gpus N under torchrun runs N independent
replicas (the path needs no collective); time = max over ranks.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import subprocess
import sys
import threading
import time

import numpy as np
import torch

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "router fwd+bwd tokens/sec per MoE layer on 1 GB300; % of HBM/tensor roofline"
UNIT = "tokens/s"


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--config", default="dsmoe_vlm")
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--profile", action="store_true",
                    help="short run for ncu: no clock load window, no e2e, no CPU baseline")
    args = ap.parse_args()
    if args.profile:
        args.no_e2e = args.no_cpu_baseline = True
    return args


def peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), float(p["bf16_tflops"]), float(p["bf16_tflops_sustained"]), "measured"
    except Exception:
        return 6800.0, 1900.0, 1700.0, "fallback"


WORKLOAD_TEXT = {
    "tiny_fp32": "T=4096 (2458 img + 1638 txt, 1 sample), d=512, E=16 top-2, 4 bins, fp32",
    "dsmoe_vlm": "T=16384 (8x[576 img + 1472 txt]), d=2048, E=64 top-6, 8 bins, bf16",
    "small_hidden": "T=32768 (16x[729 img + 1319 txt]), d=1280, E=64 top-6, 8 bins, bf16",
    "attn_router": "T=32768 (8x[1024 img + 3072 txt]), d=2048, E=64 top-6, 8 bins, bf16",
    "large_fine": "T=131072 (32x[1024 img + 3072 txt]), d=2048, E=128 top-8, 16 bins, bf16",
}


def algorithmic(wl):
    """Algorithmic bytes and flops of one step, and bytes of its forward and backward calls."""
    T, d, E, k, K = wl.T, wl.d, wl.E, wl.k, wl.n_bins
    b = wl.X.element_size()
    per_token = 3 * d * b + 8 * k + 16 + 4 * k + 8 * min(k, K)
    step_bytes = T * per_token + E * d * (b + 4)
    step_flops = 6.0 * T * d * E
    # forward + fused permutation: X read; top-k indices and weights, scores and permutation
    # entries written; W read
    fwd_bytes = T * (d * b + 8 * k + 8 + 8 * min(k, K)) + E * d * b
    bwd_bytes = T * (2 * d * b + 8) + E * d * (b + 4)        # X read, dX write, M read, W read, dW write
    return step_bytes, step_flops, fwd_bytes, bwd_bytes


# Special-function unit: 16 exp2 results per SM and clock (4 per sub-partition), 152 SMs.
SFU_PER_SM_CLK = 16


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled every 200 ms during the timed region."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        vis = os.environ.get("CUDA_VISIBLE_DEVICES")
        if vis:
            try:
                gpu_index = int(vis.split(",")[gpu_index])
            except (ValueError, IndexError):
                pass
        self.idx = gpu_index
        self.proc = None
        self.lines = []

    def start(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.idx), "--query-gpu=" + self.Q,
                                          "--format=csv,noheader,nounits", "-lms", "100"],
                                         stdout=subprocess.PIPE, stderr=subprocess.PIPE, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except Exception:
            self.proc = None

    def wait_first(self, timeout=5.0):
        t0 = time.time()
        while self.proc is not None and not self.lines and time.time() - t0 < timeout:
            time.sleep(0.02)

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            f = [x.strip() for x in ln.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                smax.append(float(f[2]))
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        out = {"sm_mhz": float(np.median(sm)) if sm else None,
               "sm_max_mhz": float(max(smax)) if smax else None,
               "reasons": sorted(reasons), "samples": len(sm)}
        if not sm and self.proc is not None:
            out["error"] = (self.proc.stderr.read() or "")[:200]
        return out


def profile_traffic(kernel_file, workload, call):
    """DRAM bytes per launch of a call (fwd / bwd) from a committed ncu summary, if it was taken on
    the current source."""
    path = os.path.join(ROOT, "profiles", f"traffic_{workload}_{call}.json")
    src = os.path.join(ROOT, "paper_2604_23996_gb300", "csrc", kernel_file)
    try:
        with open(path) as f:
            rec = json.load(f)
        sha = hashlib.sha256(open(src, "rb").read()).hexdigest()[:16]
        if rec.get("source_sha") == sha:
            return float(rec["dram_bytes_per_launch"])
    except Exception:
        pass
    return None


def cpu_oracle_rate(wl, budget_s=10.0):
    """Oracle (fp64 numpy) fwd + bwd + permutation on whole samples of the workload, until the
    time budget is used (at least one sample). Returns (tokens/s, samples, tokens, seconds)."""
    from oracle import smoes_oracle as O
    offs = wl.sample_offsets
    Xd_all = wl.X
    mu = wl.mu.double().numpy()
    var = wl.var.double().numpy()
    Wd = wl.W.double().numpy()
    done_tok, t_used, n = 0, 0.0, 0
    for it in range(10 ** 6):
        i = it % wl.B
        s, e = int(offs[i]), int(offs[i + 1])
        Xd = Xd_all[s:e].double().numpy()
        t0 = time.perf_counter()
        M = O.gaussian_score(Xd, mu, var, wl.tau)
        one = np.array([0, e - s])
        fwd = O.router_forward(Xd, Wd, M, wl.expert_bin, wl.n_bins, one, wl.k)
        O.router_backward(Xd, Wd, M, fwd, wl.expert_bin, one, 1.0)
        O.bin_permute(fwd["topk_idx"], wl.expert_bin, wl.n_bins, is_vision=wl.is_vision[s:e])
        t_used += time.perf_counter() - t0
        done_tok += e - s
        n += 1
        if t_used >= budget_s:
            break
    return done_tok / t_used, n, done_tok, t_used


def cores():
    try:
        return len(os.sched_getaffinity(0))
    except Exception:
        return os.cpu_count() or 1


def run_reference(args, rank, world):
    """The reference arm: the fp64 oracle on the host cores, one bounded sample per step."""
    from paper_2604_23996_gb300.workloads import config_workload
    if rank != 0:
        return
    wl = config_workload(args.config)
    for _ in range(args.warmup):
        cpu_oracle_rate(wl, budget_s=0.0)
    t_tot, tok = 0.0, 0
    for _ in range(args.steps):
        rate, n, ntok, secs = cpu_oracle_rate(wl, budget_s=0.0)
        t_tot += secs
        tok += ntok
    value = tok / t_tot
    line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": 1e3 * t_tot / args.steps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "impl": "reference",
            "config": {"workload": f"{args.config}: {WORKLOAD_TEXT[args.config]}",
                       "sample": "one sample (first of the batch) per step"},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores(), "kind": "oracle",
                             "sample": f"{tok // args.steps} tokens (one sample) per step"},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def rank_env():
    """(rank, world size, local rank) of this process as torchrun sets them (1 process: 0, 1, 0)."""
    return (int(os.environ.get("RANK", "0")), int(os.environ.get("WORLD_SIZE", "1")),
            int(os.environ.get("LOCAL_RANK", "0")))


def max_over_ranks(x, world, device):
    """The largest value of x over all ranks (the job's time is its slowest replica's)."""
    if world <= 1:
        return float(x)
    import torch.distributed as dist
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_rate(tokens_per_replica, world, ms):
    """Whole-job tokens/s: every replica processes tokens_per_replica in ms milliseconds."""
    return world * tokens_per_replica / (ms * 1e-3)


def main():
    args = parse()
    rank, world, local = rank_env()
    if args.impl == "reference":
        run_reference(args, rank, world)
        return
    assert args.warmup >= 3, "at least 3 warm-up steps"
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)

    from paper_2604_23996_gb300 import binding as bd
    from paper_2604_23996_gb300.workloads import attn_workload, config_workload

    wl = config_workload(args.config)
    use_attn = args.config == "attn_router"
    aw = attn_workload() if use_attn else None
    dtype = bd.SMOES_BF16 if wl.dtype == torch.bfloat16 else bd.SMOES_F32
    r = bd.Router(wl.T, wl.d, wl.E, wl.k, wl.n_bins, wl.sample_offsets, wl.expert_bin, dtype,
                  attn_max_heads=aw.H if use_attn else 0)
    X = wl.X.to(dev)
    W = wl.W.to(dev)
    mu, var = wl.mu.to(dev), wl.var.to(dev)
    is_vis = torch.from_numpy(wl.is_vision).to(dev)
    dW = torch.empty((wl.E, wl.d), dtype=torch.float32, device=dev)
    dX = torch.empty_like(X)
    flush = torch.empty(64 * 1024 * 1024, dtype=torch.float32, device=dev)   # 256 MiB > L2
    Ma = torch.empty((wl.T, 2), dtype=torch.float32, device=dev)
    if use_attn:
        attn = dict(Q=aw.Q.to(dev), K=aw.K.to(dev), B=aw.B, H=aw.H, S=aw.S, hd=aw.hd,
                    sm_scale=aw.sm_scale, causal=1, key_bias=torch.from_numpy(aw.key_bias).to(dev),
                    is_vision=torch.from_numpy(aw.is_vision).to(dev))

    def score():
        r.modality_score(bd.SMOES_SCORE_ATTN, Ma, attn=attn)

    def fwd_perm():
        # the forward and the bin permutation of its top-k: one launch on the bf16 path
        if use_attn:
            r.forward_permute(X, W, M_in=Ma, bin_prob=False, is_vision=is_vis)
        else:
            r.forward_permute(X, W, mu=mu, var=var, tau=wl.tau, bin_prob=False, is_vision=is_vis)

    def bwd():
        r.backward(X, W, Ma if use_attn else r.M, dW, dX=dX, loss_scale=1e-4)

    parts = ([("attn", score)] if use_attn else []) + [("fwd+permute", fwd_perm), ("bwd", bwd)]

    # eager warm-up (also checks the device status once), then one CUDA graph for the whole step
    # (the timed object) and a second copy with an event after every call (the per-call breakdown;
    # event nodes between the calls stop the graph from overlapping their launches, so that copy
    # runs a little slower and is timed in a pass of its own)
    for _ in range(2):
        for _, fn in parts:
            fn()
    code, _ = r.device_status()
    assert code == 0, f"device status {code}"
    s = torch.cuda.Stream(device=dev)
    s.wait_stream(torch.cuda.current_stream())
    g_step = torch.cuda.CUDAGraph()
    g_parts, part_graphs = None, []
    with torch.cuda.stream(s):
        with torch.cuda.graph(g_step, stream=s):
            for _, fn in parts:
                fn()
        try:
            ev_in = [torch.cuda.Event(enable_timing=True, external=True) for _ in range(len(parts) + 1)]
            g_parts = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g_parts, stream=s):
                ev_in[0].record()
                for i, (_, fn) in enumerate(parts):
                    fn()
                    ev_in[i + 1].record()
        except Exception:          # no event nodes in graphs: one graph per call instead
            g_parts = None
            for _, fn in parts:
                g = torch.cuda.CUDAGraph()
                with torch.cuda.graph(g, stream=s):
                    fn()
                part_graphs.append(g)
    torch.cuda.current_stream().wait_stream(s)
    torch.cuda.synchronize()
    # our kernels per step: attention 1; fwd + permutation 1 (one cooperative launch; fp32:
    # Gaussian coefficients 1, forward 1, permutation 1); bwd 3 (dz prep, main, dW reduce; fp32:
    # main, dW reduce)
    f32 = dtype != bd.SMOES_BF16
    fwd_launches = ((0 if use_attn else 1) + 2) if f32 else 1
    launches_per_step = (1 if use_attn else 0) + fwd_launches + (2 if f32 else 3)

    def step_timed():
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        g_step.replay()
        b.record()
        return a, b

    def parts_timed():
        """Durations (ms) of the step's calls, one step."""
        if g_parts is not None:
            g_parts.replay()
            torch.cuda.synchronize()
            return [ev_in[i].elapsed_time(ev_in[i + 1]) for i in range(len(parts))]
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(len(parts) + 1)]
        ev[0].record()
        for i, g in enumerate(part_graphs):
            g.replay()
            ev[i + 1].record()
        torch.cuda.synchronize()
        return [ev[i].elapsed_time(ev[i + 1]) for i in range(len(parts))]

    for _ in range(args.warmup):
        flush.zero_()
        step_timed()
    torch.cuda.synchronize()
    if world > 1:
        import torch.distributed as dist
        dist.barrier()
    torch.cuda.synchronize()
    # clocks: sampled from a load window that starts ~0.5 s before the timed steps (the timed
    # steps alone last a few ms, shorter than the sampling period) and ends after them
    clocks = ClockSampler(local)
    if not args.profile:
        clocks.start()
        clocks.wait_first()
        t_load = time.time()
        while time.time() - t_load < 0.5:
            flush.zero_()
            step_timed()
            torch.cuda.synchronize()
    evs = []
    for _ in range(args.steps):
        flush.zero_()
        evs.append(step_timed())
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    clk = clocks.stop() if not args.profile else {"sm_mhz": None, "note": "profile run"}
    t_step = [a.elapsed_time(b) for a, b in evs]
    # per-call breakdown: the same steps again, each call bracketed by events
    t_part = {name: [] for name, _ in parts}
    for _ in range(args.steps):
        flush.zero_()
        for (name, _), t in zip(parts, parts_timed()):
            t_part[name].append(t)
    total_ms = max_over_ranks(float(np.sum(t_step)), world, dev)
    ms_per_step = total_ms / args.steps
    value = job_rate(wl.T, world, ms_per_step)

    total_ms = max_over_ranks(float(np.sum(t_step)), world, dev)
    ms_per_step = total_ms / args.steps
    value = job_rate(wl.T, world, ms_per_step)

    # end to end through the public API: every step's inputs come from pinned host memory and its
    # loss goes back to the host, all inside the timed region. As in a training loop that
    # prefetches, step i+1's inputs are copied on a second stream into the other of two device
    # buffers while step i computes (a copy waits until the step that last used its buffer is
    # done); the calls are the eager API calls. L2 is not flushed here: each step's inputs arrive
    # by copy, as they would in deployment.
    e2e = None
    if not args.no_e2e:
        Xh = wl.X.pin_memory()
        Wh = wl.W.pin_memory()
        muh, varh = wl.mu.pin_memory(), wl.var.pin_memory()
        n_loss = args.steps + 3
        lossh = torch.empty(n_loss, dtype=torch.float32).pin_memory()
        h2d = (Xh.numel() * Xh.element_size() + Wh.numel() * Wh.element_size() +
               muh.numel() * 4 + varh.numel() * 4)
        d2h = 4
        bufs = [dict(X=X, W=W, mu=mu, var=var),
                dict(X=torch.empty_like(X), W=torch.empty_like(W), mu=torch.empty_like(mu),
                     var=torch.empty_like(var))]
        if use_attn:
            Qh, Kh = aw.Q.pin_memory(), aw.K.pin_memory()
            h2d += 2 * Qh.numel() * Qh.element_size()
            bufs[0].update(Q=attn["Q"], K=attn["K"])
            bufs[1].update(Q=torch.empty_like(attn["Q"]), K=torch.empty_like(attn["K"]))
        cs = torch.cuda.Stream(device=dev)
        main = torch.cuda.current_stream()
        copied = [torch.cuda.Event(), torch.cuda.Event()]
        done = [torch.cuda.Event(), torch.cuda.Event()]

        def issue_copy(i):
            bb = bufs[i & 1]
            with torch.cuda.stream(cs):
                cs.wait_event(done[i & 1])             # the step that last read this buffer
                bb["X"].copy_(Xh, non_blocking=True)
                bb["W"].copy_(Wh, non_blocking=True)
                bb["mu"].copy_(muh, non_blocking=True)
                bb["var"].copy_(varh, non_blocking=True)
                if use_attn:
                    bb["Q"].copy_(Qh, non_blocking=True)
                    bb["K"].copy_(Kh, non_blocking=True)
                copied[i & 1].record(cs)

        def compute(i):
            bb = bufs[i & 1]
            main.wait_event(copied[i & 1])
            if use_attn:
                a_args = dict(attn, Q=bb["Q"], K=bb["K"])
                r.modality_score(bd.SMOES_SCORE_ATTN, Ma, attn=a_args)
                r.forward_permute(bb["X"], bb["W"], M_in=Ma, bin_prob=False, is_vision=is_vis)
                r.backward(bb["X"], bb["W"], Ma, dW, dX=dX, loss_scale=1e-4)
            else:
                r.forward_permute(bb["X"], bb["W"], mu=bb["mu"], var=bb["var"], tau=wl.tau,
                                  bin_prob=False, is_vision=is_vis)
                r.backward(bb["X"], bb["W"], r.M, dW, dX=dX, loss_scale=1e-4)
            lossh[i:i + 1].copy_(r.loss, non_blocking=True)
            done[i & 1].record(main)

        def pipeline(n, first, start_ev=None):
            if start_ev is not None:
                cs.wait_event(start_ev)
            issue_copy(first)
            for i in range(first, first + n):
                if i + 1 < first + n:
                    issue_copy(i + 1)
                compute(i)

        pipeline(3, 0)                                 # warm-up
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(main)
        pipeline(args.steps, 3, start_ev=a)
        b.record(main)
        b.synchronize()
        t_e2e = max_over_ranks(a.elapsed_time(b), world, dev)
        e2e = {"value": job_rate(wl.T, world, t_e2e / args.steps), "unit": UNIT,
               "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h),
               "note": "inputs of step i+1 copied while step i computes (two device buffers)"}

    if rank != 0:
        if world > 1:
            dist.destroy_process_group()
        return

    hbm, tf_burst, tf_sus, peak_kind = peaks()
    step_bytes, step_flops, fwd_bytes, bwd_bytes = algorithmic(wl)
    if use_attn:   # causal Q K^T of the attention score: B H S^2 hd flops; Q and K read once
        attn_flops = float(aw.B) * aw.H * aw.S * aw.S * aw.hd
        attn_bytes = 2.0 * aw.Q.numel() * aw.Q.element_size()
    else:
        attn_flops = attn_bytes = 0.0
    t_roof = (max(step_bytes / (hbm * 1e9), step_flops / (tf_sus * 1e12)) +
              max(attn_bytes / (hbm * 1e9), attn_flops / (tf_sus * 1e12)))
    # roofline of every call of the step; `roofline` is the one of the longest call (the
    # dominant kernel). The forward and backward are HBM-bound streams; the attention score
    # evaluates one exponential per unmasked score on the special-function unit.
    sm_mhz = float(clk.get("sm_max_mhz") or 2070.0)
    rooflines = {}
    for name in t_part:
        ms = float(np.mean(t_part[name]))
        if name == "attn":
            n_exp = float(aw.B) * aw.H * aw.S * (aw.S + 1) / 2.0
            peak = SFU_PER_SM_CLK * torch.cuda.get_device_properties(dev).multi_processor_count * sm_mhz * 1e-3
            ach = n_exp / (ms * 1e-3) / 1e9
            rooflines[name] = {"bound": "alu", "achieved": ach, "peak": peak, "unit": "Gexp/s",
                               "frac": ach / peak, "traffic": None, "kernel": "k_attn_mass",
                               "peak_source": "derived: 16 exp2 per SM and clock x SMs x max SM clock"}
        else:
            call = "fwd" if name.startswith("fwd") else "bwd"
            by = fwd_bytes if call == "fwd" else bwd_bytes
            ach = by / (ms * 1e-3) / 1e9
            kern = ("smoes_router_fwd_permute (k_router_fwd_tc, one launch)" if call == "fwd" and not f32
                    else "smoes_router_bwd (k_dz_prep + k_router_bwd_tc + k_dw_reduce)" if not f32
                    else f"smoes_router_{call} (fp32 path)")
            rooflines[name] = {"bound": "hbm", "achieved": ach, "peak": hbm, "unit": "GB/s",
                               "frac": ach / hbm, "bytes": by,
                               "traffic": profile_traffic(f"router_{call}.cu", args.config, call),
                               "kernel": kern, "peak_source": peak_kind}
    dominant = max(t_part, key=lambda n: float(np.mean(t_part[n])))
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16" if wl.dtype == torch.bfloat16 else "f32",
        "data": "synthetic (seeded; shapes of the paper's MoE-VLM router layers)",
        "config": {"workload": f"{args.config}: {WORKLOAD_TEXT[args.config]}; "
                               + ("attention score (8x4096, 16 heads, hd 128, causal) + " if use_attn
                                  else "Gaussian score; ")
                               + "fwd + bwd (dW, dX) + bin permutation",
                   "l2": "flushed before every step (256 MiB write, outside the timed interval)",
                   "timing": "one CUDA graph per step, events around each replay; breakdown_us and "
                             "the backward duration from a second pass with events between calls",
                   "clocks": "nvidia-smi every 100 ms over a load window of ~0.5 s of steps "
                             "ending with the timed steps",
                   "parallelism": f"replicas x{world}"},
        "roofline": dict(rooflines[dominant], call=dominant),
        "rooflines": rooflines,
        "step_roofline": {"t_roof_us": t_roof * 1e6, "t_step_us": ms_per_step * 1e3,
                          "frac": t_roof / (ms_per_step * 1e-3),
                          "bytes": step_bytes + attn_bytes, "flops": step_flops + attn_flops},
        "breakdown_us": {name: 1e3 * float(np.mean(v)) for name, v in t_part.items()},
        "gpu_launches": launches_per_step * args.steps,
        "clocks": clk,
        "e2e": e2e,
    }
    if not args.no_cpu_baseline and world == 1:
        rate, n, ntok, secs = cpu_oracle_rate(wl)
        line["cpu_baseline"] = {"value": rate, "unit": UNIT, "cores": cores(), "kind": "oracle",
                                "sample": f"{n} whole samples of {wl.B} ({ntok} tokens, repeated), {secs:.1f} s"}
    print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
