#!/usr/bin/env python
"""Router fwd+bwd throughput of the SMoES hot path on GB300 (one JSON line on stdout).

A step is one pass of the whole router hot path over one batch of the workload:
  smoes_router_fwd_permute (gate GEMM + Gaussian modality score + softmax/top-k/bins + per-sample
  MI + the de-duplicated bin dispatch of the top-k, one launch) -> smoes_router_bwd (MI gradient
  -> dW and dX); the attention workload adds smoes_modality_score(ATTN) in front.
Default workload: the large fine-grained router layer, T = 131072 tokens (32 x [1024 image +
3072 text]), d = 2048, E = 128 routed experts, top-8, 16 bins, bf16 (the largest single-GPU
configuration). --tokens T runs the same layer on the first T / 4096 samples; the default run
also reports the throughput sweep over T in {8K, 32K, 131K}. Inputs are seeded synthetic data.

Timing: W warm-up steps, then K timed steps. The step (all calls) is replayed from one CUDA
graph; before every step the L2 is flushed by writing a 256 MiB buffer (outside the timed
interval), and CUDA events on the launching stream bracket each step. A second pass of K steps
replays a copy of the graph with an event after every call, for the per-call breakdown.
--gpus N under torchrun runs N independent replicas (the path needs no collective); time = max
over ranks. --impl reference times the fp64 oracle on the host cores on the same workload.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import platform
import subprocess
import sys
import tempfile
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "router fwd+bwd tokens/sec per MoE layer on 1 GB300; % of HBM/tensor roofline"
UNIT = "tokens/s"
DEFAULT_CONFIG = "large_fine"
SWEEP_TOKENS = (8192, 32768, 131072)


def parse(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--config", default=DEFAULT_CONFIG)
    ap.add_argument("--tokens", type=int, default=None,
                    help="tokens of the batch (a multiple of the workload's sample length)")
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-sweep", action="store_true")
    ap.add_argument("--no-next", action="store_true",
                    help="skip the timings of the next rows' kernels (statistics, binning, "
                         "balance, GMM score, attention forward)")
    ap.add_argument("--profile", action="store_true",
                    help="short run for ncu: no clock load window, no e2e, no CPU baseline, no sweep")
    ap.add_argument("--oracle-child", default=None, help=argparse.SUPPRESS)
    args = ap.parse_args(argv)
    if args.profile:
        args.no_e2e = args.no_cpu_baseline = args.no_sweep = args.no_next = True
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


def samples_for(config, tokens):
    """Samples of the workload for a batch of `tokens` tokens (None: the configured batch)."""
    from paper_2604_23996_gb300.workloads import CONFIGS
    c = CONFIGS[config]
    per = c["T_img"] + c["T_txt"]
    if tokens is None:
        return c["n_samples"]
    if tokens <= 0 or tokens % per:
        raise SystemExit(f"--tokens must be a positive multiple of {per} for {config}")
    return tokens // per


def workload_text(config, wl):
    base = WORKLOAD_TEXT[config]
    if wl is not None and wl.B != samples_for(config, None):
        from paper_2604_23996_gb300.workloads import CONFIGS
        c = CONFIGS[config]
        base = (f"T={wl.T} ({wl.B}x[{c['T_img']} img + {c['T_txt']} txt]), d={wl.d}, E={wl.E} "
                f"top-{wl.k}, {wl.n_bins} bins, " + ("bf16" if wl.X.element_size() == 2 else "fp32"))
    return base


def bench_config(config, wl, world):
    """The `config` object of the JSON line. Both arms print the same workload; the reference arm
    replaces the two keys that describe how the device is timed."""
    use_attn = config == "attn_router"
    return {"workload": f"{config}: {workload_text(config, wl)}; "
                        + (f"attention score ({wl.B if wl is not None else 8}x4096, 16 heads, hd 128, "
                           "causal) + " if use_attn
                           else "Gaussian score; ")
                        + "fwd + bwd (dW, dX) + bin permutation",
            "l2": "flushed before every step (256 MiB write, outside the timed interval)",
            "timing": "one CUDA graph per step, events around each replay; breakdown_us from a "
                      "second pass with events between calls",
            "parallelism": f"replicas x{world}"}



def reference_config(config, wl, world):
    """The reference arm's `config`: our arm's workload and parallelism, with the two keys that
    describe the device timing replaced by how the oracle is timed."""
    return dict(bench_config(config, wl, world), l2="not applicable (host cores)",
                timing="host wall clock (time.perf_counter) around each sample's oracle evaluation")

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
    """nvidia-smi clocks and throttle reasons sampled every 100 ms during the timed region."""
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


# the sources whose code a call's kernels are compiled from (a traffic record counts only for them)
TRAFFIC_SOURCES = {
    "fwd": ["router_fwd.cu", "router_fwd_tc.cuh", "router_fwd_var.cu", "ptx.cuh", "device_common.cuh",
            "smoes_internal.cuh"],
    "bwd": ["router_bwd.cu", "ptx.cuh", "device_common.cuh", "smoes_internal.cuh"],
}


def sources_sha(files):
    """First 16 hex digits of the sha256 of the files' bytes, in order."""
    h = hashlib.sha256()
    for name in files:
        with open(os.path.join(ROOT, "paper_2604_23996_gb300", "csrc", name), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def profile_traffic(kernel_files, workload, call):
    """DRAM bytes per launch of a call (fwd / bwd) from a committed ncu summary, if it was taken on
    the current sources."""
    path = os.path.join(ROOT, "profiles", f"traffic_{workload}_{call}.json")
    try:
        with open(path) as f:
            rec = json.load(f)
        if rec.get("source_sha") == sources_sha(kernel_files):
            return float(rec["dram_bytes_per_launch"])
    except Exception:
        pass
    return None


# ------------------------------------------------------------------------------ the oracle legs

def _oracle_sample(O, Xd, Wd, mu, var, tau, expert_bin, n_bins, k, is_vision):
    """One sample through the oracle: score, forward, backward, permutation."""
    M = O.gaussian_score(Xd, mu, var, tau)
    one = np.array([0, Xd.shape[0]])
    fwd = O.router_forward(Xd, Wd, M, expert_bin, n_bins, one, k)
    O.router_backward(Xd, Wd, M, fwd, expert_bin, one, 1.0)
    O.bin_permute(fwd["topk_idx"], expert_bin, n_bins, is_vision=is_vision)


def oracle_samples(wl, samples):
    """Times the oracle over the given sample indices; returns (tokens, seconds)."""
    from oracle import smoes_oracle as O
    offs = wl.sample_offsets
    mu, var, Wd = wl.mu.double().numpy(), wl.var.double().numpy(), wl.W.double().numpy()
    tok, secs = 0, 0.0
    for i in samples:
        s, e = int(offs[i]), int(offs[i + 1])
        Xd = wl.X[s:e].double().numpy()
        t0 = time.perf_counter()
        _oracle_sample(O, Xd, Wd, mu, var, wl.tau, wl.expert_bin, wl.n_bins, wl.k, wl.is_vision[s:e])
        secs += time.perf_counter() - t0
        tok += e - s
    return tok, secs


def cpu_oracle_rate(wl, budget_s=10.0):
    """Oracle (fp64 numpy) fwd + bwd + permutation on whole samples of the workload, until the
    time budget is used (at least one sample). Returns (tokens/s, samples, tokens, seconds)."""
    done_tok, t_used, n = 0, 0.0, 0
    while True:
        tok, secs = oracle_samples(wl, [n % wl.B])
        done_tok += tok
        t_used += secs
        n += 1
        if t_used >= budget_s:
            break
    return done_tok / t_used, n, done_tok, t_used


def oracle_child(path):
    """Single-threaded oracle leg (run in a child process whose BLAS was limited to one thread
    before numpy loaded): the sample in `path`, repeated until its budget is used."""
    from oracle import smoes_oracle as O
    a = np.load(path)
    budget = float(a["budget"])
    tok, secs = 0, 0.0
    while secs < budget or tok == 0:
        t0 = time.perf_counter()
        _oracle_sample(O, a["X"], a["W"], a["mu"], a["var"], float(a["tau"]), a["expert_bin"],
                       int(a["n_bins"]), int(a["k"]), a["is_vision"])
        secs += time.perf_counter() - t0
        tok += a["X"].shape[0]
    print(json.dumps({"tokens": tok, "seconds": secs}))


def single_thread_oracle_rate(wl, budget_s=5.0):
    """The oracle on one core: one sample repeated for ~budget_s in a child process with every
    BLAS / OpenMP pool limited to one thread. Returns (tokens/s, tokens, seconds) or None."""
    s, e = int(wl.sample_offsets[0]), int(wl.sample_offsets[1])
    with tempfile.TemporaryDirectory() as td:
        path = os.path.join(td, "sample.npz")
        np.savez(path, X=wl.X[s:e].double().numpy(), W=wl.W.double().numpy(),
                 mu=wl.mu.double().numpy(), var=wl.var.double().numpy(), tau=wl.tau,
                 expert_bin=wl.expert_bin, n_bins=wl.n_bins, k=wl.k, is_vision=wl.is_vision[s:e],
                 budget=budget_s)
        env = dict(os.environ)
        for v in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS", "BLIS_NUM_THREADS",
                  "VECLIB_MAXIMUM_THREADS", "NUMEXPR_NUM_THREADS"):
            env[v] = "1"
        try:
            out = subprocess.run([sys.executable, os.path.abspath(__file__), "--oracle-child", path],
                                 capture_output=True, text=True, env=env, timeout=600)
            rec = json.loads(out.stdout.strip().splitlines()[-1])
            return rec["tokens"] / rec["seconds"], rec["tokens"], rec["seconds"]
        except Exception:
            return None


def cores():
    try:
        return len(os.sched_getaffinity(0))
    except Exception:
        return os.cpu_count() or 1


def cpu_model():
    """The host CPU's model name (lscpu, else /proc/cpuinfo, else the platform string)."""
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for ln in out.splitlines():
            if ln.strip().lower().startswith("model name"):
                return ln.split(":", 1)[1].strip()
    except Exception:
        pass
    try:
        with open("/proc/cpuinfo") as f:
            for ln in f:
                if ln.lower().startswith("model name"):
                    return ln.split(":", 1)[1].strip()
    except Exception:
        pass
    return platform.processor() or platform.machine()


def run_reference(args, rank, world):
    """The reference arm: the fp64 oracle on the host cores, every step the whole batch of the
    same workload (its samples one after another); rank 0 only."""
    if rank != 0:
        return
    from paper_2604_23996_gb300.workloads import config_workload
    wl = config_workload(args.config, n_samples=samples_for(args.config, args.tokens))
    for w in range(args.warmup):                 # untimed: one sample each
        oracle_samples(wl, [w % wl.B])
    t_tot, tok = 0.0, 0
    for _ in range(args.steps):
        ntok, secs = oracle_samples(wl, range(wl.B))
        t_tot += secs
        tok += ntok
    value = tok / t_tot
    line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": 1e3 * t_tot / args.steps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "impl": "reference",
            "config": reference_config(args.config, wl, world),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores(), "kind": "oracle",
                             "cpu_model": cpu_model(),
                             "sample": f"the whole batch ({wl.B} samples, {wl.T} tokens) per step; "
                                       "warm-up steps one sample each"},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# ------------------------------------------------------------------------------ our arm

def rank_env():
    """(rank, world size, local rank) of this process as torchrun sets them (1 process: 0, 1, 0)."""
    return (int(os.environ.get("RANK", "0")), int(os.environ.get("WORLD_SIZE", "1")),
            int(os.environ.get("LOCAL_RANK", "0")))


def max_over_ranks(x, world, device):
    """The largest value of x over all ranks (the job's time is its slowest replica's)."""
    if world <= 1:
        return float(x)
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_rate(tokens_per_replica, world, ms):
    """Whole-job tokens/s: every replica processes tokens_per_replica in ms milliseconds."""
    return world * tokens_per_replica / (ms * 1e-3)


class Step:
    """One router layer's step on the device: the plan, resident inputs and outputs, the calls of
    the step, and its CUDA graphs (the timed one and one with events between the calls)."""

    def __init__(self, bd, wl, aw, dev, X=None):
        import torch
        self.bd, self.wl, self.aw, self.dev = bd, wl, aw, dev
        self.use_attn = aw is not None
        self.f32 = wl.dtype != torch.bfloat16
        dtype = bd.SMOES_F32 if self.f32 else bd.SMOES_BF16
        self.r = bd.Router(wl.T, wl.d, wl.E, wl.k, wl.n_bins, wl.sample_offsets, wl.expert_bin, dtype,
                           attn_max_heads=aw.H if self.use_attn else 0)
        self.X = wl.X.to(dev) if X is None else X
        self.W = wl.W.to(dev)
        self.mu, self.var = wl.mu.to(dev), wl.var.to(dev)
        self.is_vis = torch.from_numpy(wl.is_vision).to(dev)
        self.dW = torch.empty((wl.E, wl.d), dtype=torch.float32, device=dev)
        self.dX = torch.empty_like(self.X)
        self.Ma = torch.empty((wl.T, 2), dtype=torch.float32, device=dev)
        if self.use_attn:
            self.attn = dict(Q=aw.Q.to(dev), K=aw.K.to(dev), B=aw.B, H=aw.H, S=aw.S, hd=aw.hd,
                             sm_scale=aw.sm_scale, causal=1,
                             key_bias=torch.from_numpy(aw.key_bias).to(dev),
                             is_vision=torch.from_numpy(aw.is_vision).to(dev))
        self.parts = (([("attn", self.score)] if self.use_attn else [])
                      + [("fwd+permute", self.fwd_perm), ("bwd", self.bwd)])
        # our kernels per step, as the library reports them for this plan: the attention score,
        # the forward with the permutation (one launch when the permutation is fused into the
        # forward kernel, else two), the backward (dz prep, main, dW sum; fp32: main, dW sum)
        plan = self.r.plan
        self.fwd_launches = bd.smoes_call_launches(plan, bd.SMOES_CALL_ROUTER_FWD_PERMUTE)
        self.launches = ((bd.smoes_call_launches(plan, bd.SMOES_CALL_ATTN_SCORE) if self.use_attn else 0)
                         + self.fwd_launches + bd.smoes_call_launches(plan, bd.SMOES_CALL_ROUTER_BWD))
        assert min(self.fwd_launches, self.launches) > 0

    def score(self, X=None, Q=None, K=None):
        a = self.attn if Q is None else dict(self.attn, Q=Q, K=K)
        self.r.modality_score(self.bd.SMOES_SCORE_ATTN, self.Ma, attn=a)

    def fwd_perm(self, X=None, W=None, mu=None, var=None):
        # the forward and the bin permutation of its top-k
        X = self.X if X is None else X
        W = self.W if W is None else W
        if self.use_attn:
            self.r.forward_permute(X, W, M_in=self.Ma, bin_prob=False, is_vision=self.is_vis)
        else:
            self.r.forward_permute(X, W, mu=self.mu if mu is None else mu,
                                   var=self.var if var is None else var, tau=self.wl.tau,
                                   bin_prob=False, is_vision=self.is_vis)

    def bwd(self, X=None, W=None):
        X = self.X if X is None else X
        W = self.W if W is None else W
        self.r.backward(X, W, self.Ma if self.use_attn else self.r.M, self.dW, dX=self.dX,
                        loss_scale=1e-4)

    def capture(self):
        """Eager warm-up (checks the device status once), then one CUDA graph for the whole step
        (the timed object) and a second copy with an event after every call (the per-call
        breakdown; event nodes between the calls stop the graph from overlapping their launches,
        so that copy runs a little slower and is timed in a pass of its own)."""
        import torch
        for _ in range(2):
            for _, fn in self.parts:
                fn()
        code, _ = self.r.device_status()
        assert code == 0, f"device status {code}"
        s = torch.cuda.Stream(device=self.dev)
        s.wait_stream(torch.cuda.current_stream())
        self.g_step = torch.cuda.CUDAGraph()
        self.g_parts, self.part_graphs = None, []
        with torch.cuda.stream(s):
            with torch.cuda.graph(self.g_step, stream=s):
                for _, fn in self.parts:
                    fn()
            try:
                self.ev_in = [torch.cuda.Event(enable_timing=True, external=True)
                              for _ in range(len(self.parts) + 1)]
                g = torch.cuda.CUDAGraph()
                with torch.cuda.graph(g, stream=s):
                    self.ev_in[0].record()
                    for i, (_, fn) in enumerate(self.parts):
                        fn()
                        self.ev_in[i + 1].record()
                self.g_parts = g
            except Exception:          # no event nodes in graphs: one graph per call instead
                self.g_parts = None
                for _, fn in self.parts:
                    g = torch.cuda.CUDAGraph()
                    with torch.cuda.graph(g, stream=s):
                        fn()
                    self.part_graphs.append(g)
        torch.cuda.current_stream().wait_stream(s)
        torch.cuda.synchronize()

    def step_timed(self):
        import torch
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        self.g_step.replay()
        b.record()
        return a, b

    def parts_timed(self):
        """Durations (ms) of the step's calls, one step."""
        import torch
        if self.g_parts is not None:
            self.g_parts.replay()
            torch.cuda.synchronize()
            return [self.ev_in[i].elapsed_time(self.ev_in[i + 1]) for i in range(len(self.parts))]
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(len(self.parts) + 1)]
        ev[0].record()
        for i, g in enumerate(self.part_graphs):
            g.replay()
            ev[i + 1].record()
        torch.cuda.synchronize()
        return [ev[i].elapsed_time(ev[i + 1]) for i in range(len(self.parts))]


def time_steps(st, flush, steps):
    """K graph replays, L2 flushed before each (outside the events); per-step ms."""
    import torch
    evs = []
    for _ in range(steps):
        flush.zero_()
        evs.append(st.step_timed())
    torch.cuda.synchronize()
    return [a.elapsed_time(b) for a, b in evs]


def time_parts(st, flush, steps):
    out = {name: [] for name, _ in st.parts}
    for _ in range(steps):
        flush.zero_()
        for (name, _), t in zip(st.parts, st.parts_timed()):
            out[name].append(t)
    return out


def run_e2e(st, args, world, dev, rate_of):
    """End to end through the public API: every step's inputs come from pinned host memory and
    its results (the loss, dW, the top-k and the permutation with its offsets and dispatch
    counts) go back to pinned host memory, all inside the timed region. As in a training loop
    that prefetches, step i+1's inputs are copied on a second stream into the other of two
    device buffers while step i computes (a copy waits until the step that last used its
    buffer is done); the calls are the eager API calls. L2 is not flushed here: each step's
    inputs arrive by copy, as they would in deployment."""
    import torch
    wl, aw, r = st.wl, st.aw, st.r
    pin = lambda t: t.pin_memory()
    Xh, Wh = pin(wl.X), pin(wl.W)
    muh, varh = pin(wl.mu), pin(wl.var)
    h2d = (Xh.numel() * Xh.element_size() + Wh.numel() * Wh.element_size() + muh.numel() * 4 +
           varh.numel() * 4)
    bufs = [dict(X=st.X, W=st.W, mu=st.mu, var=st.var),
            dict(X=torch.empty_like(st.X), W=torch.empty_like(st.W), mu=torch.empty_like(st.mu),
                 var=torch.empty_like(st.var))]
    if st.use_attn:
        Qh, Kh = pin(aw.Q), pin(aw.K)
        h2d += 2 * Qh.numel() * Qh.element_size()
        bufs[0].update(Q=st.attn["Q"], K=st.attn["K"])
        bufs[1].update(Q=torch.empty_like(st.attn["Q"]), K=torch.empty_like(st.attn["K"]))
    outs = [("loss", r.loss), ("dW", st.dW), ("topk_idx", r.topk_idx), ("topk_w", r.topk_w),
            ("bin_offsets", r.bin_offsets), ("perm_token", r.perm_token),
            ("perm_mask", r.perm_mask), ("dispatch", r.dispatch)]
    host = {n: torch.empty(t.shape, dtype=t.dtype).pin_memory() for n, t in outs}
    d2h = sum(t.numel() * t.element_size() for _, t in outs)
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
            if st.use_attn:
                bb["Q"].copy_(Qh, non_blocking=True)
                bb["K"].copy_(Kh, non_blocking=True)
            copied[i & 1].record(cs)

    def compute(i):
        bb = bufs[i & 1]
        main.wait_event(copied[i & 1])
        if st.use_attn:
            st.score(Q=bb["Q"], K=bb["K"])
        st.fwd_perm(X=bb["X"], W=bb["W"], mu=bb["mu"], var=bb["var"])
        st.bwd(X=bb["X"], W=bb["W"])
        for n, t in outs:
            host[n].copy_(t, non_blocking=True)
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
    return {"value": rate_of(t_e2e / args.steps), "unit": UNIT,
            "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h),
            "d2h": "loss, dW, top-k indices and weights, bin offsets, permutation (tokens, masks; "
                   "full capacity), dispatch counts",
            "note": "inputs of step i+1 copied while step i computes (two device buffers)"}


def dedup_report(st):
    """Expert-parallel transfer ratios of the step's dispatch (Sec. 4.5), from the permutation the
    GPU produced: with the bins as devices and a token's home device floor(j K / T) (a contiguous
    data-parallel split), w/o DeDup = remote (token, expert) selections / (T k), w/ DeDup = remote
    unique (token, bin) pairs / T (also per selection, / (T k), and the share of remote copies
    that DeDup saves). The dispatch matrix gives the remote pairs directly."""
    import torch
    r, wl = st.r, st.wl
    if torch.cuda.is_available():
        torch.cuda.synchronize()
    T, K, k = wl.T, wl.n_bins, wl.k
    D = r.dispatch.cpu().numpy().astype(np.int64)                 # [home, bin] unique pairs
    off = r.bin_offsets.cpu().numpy().astype(np.int64)
    P = int(off[-1])
    tok = r.perm_token[:P].cpu().numpy().astype(np.int64)
    mask = r.perm_mask[:P].cpu().numpy().view(np.uint32).astype(np.uint64)
    b = np.repeat(np.arange(K), np.diff(off))
    home = (tok * K) // T
    sel = np.zeros(P, dtype=np.int64)                             # selected experts per entry
    m = mask.copy()
    while np.any(m):
        sel += (m & 1).astype(np.int64)
        m >>= np.uint64(1)
    remote_pairs = int(D.sum() - np.trace(D))
    remote_sel = int(sel[home != b].sum())
    return {"home": "floor(j K / T)", "devices": K,
            "ratio_without_dedup": remote_sel / float(T * k),
            "ratio_with_dedup": remote_pairs / float(T),
            "ratio_with_dedup_per_selection": remote_pairs / float(T * k),
            "dedup_saving": 1.0 - remote_pairs / float(remote_sel) if remote_sel else 0.0,
            "unique_pairs_per_token": P / float(T),
            "check": "remote pairs from the dispatch matrix = remote entries of the permutation: "
                     + str(remote_pairs == int((home != b).sum()))}


def graph_time(fn, steps, flush):
    """Mean device time (ms) of fn replayed from a CUDA graph, L2 flushed before each replay."""
    import torch
    fn()
    torch.cuda.synchronize()
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    g = torch.cuda.CUDAGraph()
    with torch.cuda.stream(s):
        with torch.cuda.graph(g, stream=s):
            fn()
    torch.cuda.current_stream().wait_stream(s)
    torch.cuda.synchronize()
    for _ in range(3):
        g.replay()
    ts = []
    for _ in range(steps):
        flush.zero_()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        g.replay()
        b.record()
        b.synchronize()
        ts.append(a.elapsed_time(b))
    return float(np.mean(ts))


def measure_next(bd, st, dev, flush, steps, hbm, tf_sus, sm_mhz, n_sms):
    """Timings of the next rows' kernels beside the hot path (one layer's worth each), with their
    rooflines: the Gaussian statistics update and the GMM score over this batch's X, the
    bin-level balance loss over its saved softmax, the adaptive binning, and the attention
    forward with the vision score on the attention workload (8 x 16 heads x 4096, hd 128), with
    H_kv = 16 and with grouped-query heads (H_kv = 4)."""
    import torch
    from paper_2604_23996_gb300.workloads import attn_workload
    wl, r = st.wl, st.r
    T, d, E, k, K = wl.T, wl.d, wl.E, wl.k, wl.n_bins
    b = wl.X.element_size()
    out = {}

    def hbm_entry(ms, by, kern):
        ach = by / (ms * 1e-3) / 1e9
        return {"us": 1e3 * ms, "bound": "hbm", "bytes": by, "achieved": ach, "peak": hbm,
                "unit": "GB/s", "frac": ach / hbm, "kernel": kern}

    N = torch.zeros(2, dtype=torch.float64, device=dev)
    S_mu = torch.zeros((2, d), dtype=torch.float64, device=dev)
    S_var = torch.zeros((2, d), dtype=torch.float64, device=dev)
    mu, var = torch.empty((2, d), device=dev), torch.empty((2, d), device=dev)
    ms = graph_time(lambda: bd.smoes_gaussian_stats_update(r.plan, st.X, st.is_vis, 0.99, N, S_mu, S_var,
                                                           mu, var, r.ws), steps, flush)
    out["gaussian_stats_update"] = hbm_entry(ms, T * d * b + T, "k_stats_partial + k_stats_finalize")
    C_bar = torch.zeros((2, E), dtype=torch.float64, device=dev)
    eb = torch.empty(E, dtype=torch.int32, device=dev)
    st.fwd_perm()
    ms = graph_time(lambda: bd.smoes_adaptive_bins(r.plan, r.expert_counts, 0.99, C_bar, eb), steps, flush)
    out["adaptive_bins"] = {"us": 1e3 * ms, "bound": "latency", "kernel": "k_adaptive_bins (one block)"}
    lb = torch.empty(1, device=dev)
    ms = graph_time(lambda: bd.smoes_bin_balance(r.plan, r.topk_idx, 1e-3, lb, r.ws), steps, flush)
    out["bin_balance"] = hbm_entry(ms, T * E * 4 + T * k * 4, "k_bal_partial + k_bal_finalize")
    if wl.dtype == torch.bfloat16:
        C = 2
        lp = torch.log(torch.full((2, C), 0.5, device=dev))
        mu2 = st.mu[:, None, :].repeat(1, C, 1).contiguous()
        var2 = st.var[:, None, :].repeat(1, C, 1).contiguous()
        Mg = torch.empty((T, 2), device=dev)
        gmm = dict(X=st.X, n_components=C, log_pi=lp, mu=mu2, var=var2, tau=wl.tau)
        ms = graph_time(lambda: bd.smoes_modality_score(r.plan, bd.SMOES_SCORE_GMM, Mg, r.ws, gmm=gmm),
                        steps, flush)
        out["gmm_score_2"] = hbm_entry(ms, T * d * b + 8 * T, "k_gmm_coef + k_gmm_score (2 components)")
    aw = attn_workload()
    Ta = aw.B * aw.S
    ra = bd.Router(Ta, 64, 16, 2, 4, [0, Ta], np.arange(16) // 4, attn_max_heads=aw.H)
    Ma = torch.empty((Ta, 2), device=dev)
    Q = aw.Q.to(dev)
    rng = np.random.default_rng(11)
    for hkv in (aw.H, aw.H // 4):
        Kt = aw.K.to(dev) if hkv == aw.H else aw.K[:, :hkv].contiguous().to(dev)
        V = torch.from_numpy(rng.standard_normal((aw.B, hkv, aw.S, aw.hd), dtype=np.float32)).to(torch.bfloat16).to(dev)
        Oo = torch.empty((aw.B, aw.H, aw.S, aw.hd), dtype=torch.bfloat16, device=dev)
        attn = dict(Q=Q, K=Kt, B=aw.B, H=aw.H, S=aw.S, hd=aw.hd, sm_scale=aw.sm_scale, causal=1,
                    key_bias=torch.from_numpy(aw.key_bias).to(dev), is_vision=torch.from_numpy(aw.is_vision).to(dev))
        ms = graph_time(lambda: bd.smoes_attention_fwd(ra.plan, attn, V, hkv, Oo, Ma, ra.ws), steps, flush)
        pairs = float(aw.B) * aw.H * aw.S * (aw.S + 1) / 2.0
        flops = 4.0 * pairs * aw.hd                            # causal Q K^T and P V
        ach = flops / (ms * 1e-3) / 1e12
        exp_peak = 16 * n_sms * sm_mhz * 1e-3                  # Gexp/s on the special-function unit
        out[f"attention_fwd_hkv{hkv}"] = {
            "us": 1e3 * ms, "bound": "tensor", "flops": flops, "achieved": ach, "peak": tf_sus,
            "unit": "TFLOP/s", "frac": ach / tf_sus, "exp_rate_frac": pairs / (ms * 1e-3) / 1e9 / exp_peak,
            "kernel": "k_attn_fwd (8x16x4096, hd 128, causal)"}
        del V, Oo, Kt
    return out


def main():
    args = parse()
    if args.oracle_child:
        oracle_child(args.oracle_child)
        return
    rank, world, local = rank_env()
    if args.impl == "reference":
        run_reference(args, rank, world)
        return
    assert args.warmup >= 3, "at least 3 warm-up steps"
    import torch
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)

    from paper_2604_23996_gb300 import binding as bd
    from paper_2604_23996_gb300.workloads import attn_workload, config_workload

    wl = config_workload(args.config, n_samples=samples_for(args.config, args.tokens))
    use_attn = args.config == "attn_router"
    aw = attn_workload(B=wl.B) if use_attn else None       # one sequence per sample
    st = Step(bd, wl, aw, dev)
    st.capture()
    flush = torch.empty(64 * 1024 * 1024, dtype=torch.float32, device=dev)   # 256 MiB > L2

    for _ in range(args.warmup):
        flush.zero_()
        st.step_timed()
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    # clocks: sampled from a load window that starts ~0.5 s before the timed steps (the timed
    # steps alone may be shorter than the sampling period) and ends after them
    clocks = ClockSampler(local)
    if not args.profile:
        clocks.start()
        clocks.wait_first()
        t_load = time.time()
        while time.time() - t_load < 0.5:
            flush.zero_()
            st.step_timed()
            torch.cuda.synchronize()
    t_step = time_steps(st, flush, args.steps)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    clk = clocks.stop() if not args.profile else {"sm_mhz": None, "note": "profile run"}
    t_part = time_parts(st, flush, args.steps)
    total_ms = max_over_ranks(float(np.sum(t_step)), world, dev)
    ms_per_step = total_ms / args.steps
    value = job_rate(wl.T, world, ms_per_step)
    hbm, tf_burst, tf_sus, peak_kind = peaks()

    def step_roof(w):
        sb, sf, _, _ = algorithmic(w)
        return max(sb / (hbm * 1e9), sf / (tf_sus * 1e12)), sb, sf

    # throughput sweep over the batch size (the same layer on the first T / 4096 samples)
    sweep = None
    if (not args.no_sweep and args.config == DEFAULT_CONFIG and args.tokens is None):
        sweep = {}
        for T in SWEEP_TOKENS:
            if T == wl.T:
                ms, w = ms_per_step, wl
            else:
                w = config_workload(args.config, n_samples=samples_for(args.config, T))
                ss = Step(bd, w, None, dev)
                ss.capture()
                for _ in range(args.warmup):
                    flush.zero_()
                    ss.step_timed()
                ms = max_over_ranks(float(np.sum(time_steps(ss, flush, args.steps))), world, dev) / args.steps
                del ss
            t_roof = step_roof(w)[0]
            sweep[str(T)] = {"tokens_per_s": job_rate(T, world, ms), "us_per_step": 1e3 * ms,
                             "step_frac": t_roof / (ms * 1e-3)}

    e2e = None if args.no_e2e else run_e2e(st, args, world, dev, lambda ms: job_rate(wl.T, world, ms))
    nxt = None
    if not args.no_next and rank == 0 and args.config == DEFAULT_CONFIG and args.tokens is None:
        nxt = measure_next(bd, st, dev, flush, args.steps, peaks()[0], peaks()[2],
                           float(clk.get("sm_max_mhz") or 2070.0),
                           torch.cuda.get_device_properties(dev).multi_processor_count)

    if rank != 0:
        if world > 1:
            dist.destroy_process_group()
        return

    step_bytes, step_flops, fwd_bytes, bwd_bytes = algorithmic(wl)
    if use_attn:   # causal Q K^T of the attention score: B H S^2 hd flops; Q and K read once
        attn_flops = float(aw.B) * aw.H * aw.S * aw.S * aw.hd
        attn_bytes = 2.0 * aw.Q.numel() * aw.Q.element_size()
    else:
        attn_flops = attn_bytes = 0.0
    t_roof = step_roof(wl)[0] + max(attn_bytes / (hbm * 1e9), attn_flops / (tf_sus * 1e12))
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
            fwd_kern = ("smoes_router_fwd_permute (k_router_fwd_tc, one launch)" if st.fwd_launches == 1
                        else "smoes_router_fwd_permute (k_router_fwd_tc + k_perm)")
            kern = (fwd_kern if call == "fwd" and not st.f32
                    else "smoes_router_bwd (k_dz_prep + k_router_bwd_tc + k_dw_reduce)" if not st.f32
                    else f"smoes_router_{call} (fp32 path)")
            tkey = args.config if args.tokens is None else f"{args.config}_T{wl.T}"
            rooflines[name] = {"bound": "hbm", "achieved": ach, "peak": hbm, "unit": "GB/s",
                               "frac": ach / hbm, "bytes": by,
                               "traffic": profile_traffic(TRAFFIC_SOURCES[call], tkey, call),
                               "kernel": kern, "peak_source": peak_kind + " (burst copy)"}
    dominant = max(t_part, key=lambda n: float(np.mean(t_part[n])))
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16" if not st.f32 else "f32",
        "data": "synthetic (seeded; shapes of the paper's MoE-VLM router layers)",
        "config": bench_config(args.config, wl, world),
        "roofline": dict(rooflines[dominant], call=dominant),
        "rooflines": rooflines,
        "step_roofline": {"t_roof_us": t_roof * 1e6, "t_step_us": ms_per_step * 1e3,
                          "frac": t_roof / (ms_per_step * 1e-3),
                          "bytes": step_bytes + attn_bytes, "flops": step_flops + attn_flops},
        "breakdown_us": {name: 1e3 * float(np.mean(v)) for name, v in t_part.items()},
        "gpu_launches": st.launches * args.steps,
        "clocks": clk,
        "e2e": e2e,
    }
    if sweep is not None:
        line["sweep"] = sweep
    line["dedup"] = dedup_report(st)
    if nxt is not None:
        line["next_rows"] = nxt
    if not args.no_cpu_baseline and world == 1:
        rate, n, ntok, secs = cpu_oracle_rate(wl)
        one = single_thread_oracle_rate(wl)
        line["cpu_baseline"] = {"value": rate, "unit": UNIT, "cores": cores(), "kind": "oracle",
                                "cpu_model": cpu_model(),
                                "sample": f"{n} whole samples of {wl.B} ({ntok} tokens, repeated), "
                                          f"{secs:.1f} s, numpy with its default thread pool",
                                "single_thread": None if one is None else
                                {"value": one[0], "unit": UNIT, "cores": 1,
                                 "sample": f"sample 0 repeated ({one[1]} tokens), {one[2]:.1f} s, "
                                           "every BLAS/OpenMP pool limited to one thread"}}
    print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
