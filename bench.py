"""Benchmark of the SAO loss head on GB300: one step = one pass of the whole
hot path over one packed batch:

    sao_advantages -> sao_value_loss -> sao_token_logprobs_fwd ->
    sao_policy_loss_fwd -> sao_policy_loss_bwd -> sao_token_logprobs_bwd

on the MoE-policy head shape (hidden 2048, vocabulary 151936, bf16, 65536
packed tokens of single-rollout agentic trajectories). Prints one JSON line.

    python bench.py [--gpus N --steps K --warmup W] [--impl reference]

Under torchrun each rank processes its own batch (weak scaling, trajectories
sharded across ranks, no collective on the data path); rank 0 prints the
whole-job tokens/s over the slowest rank's time.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "loss-head tokens/s (fwd+bwd) at h=2048,V=151936 bf16; % bf16 tensor peak"
UNIT = "tokens/s"
WORKLOAD = "moe"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}


def stored_traffic(kernel: str, rows: int, cols: float):
    """DRAM bytes per launch of `kernel` from the committed small-case ncu
    capture (profiles/dram_traffic_tc_gemm_moe8k.txt: the moe shape at 8,192
    tokens), scaled by rows x vocabulary columns per launch to a launch of
    `rows` rows and `cols` columns (the dZ writes and operand reads dominate
    and grow with both), or None for a missing capture or kernel sources
    changed since it was taken."""
    from paper_2607_07508_gb300.build import kernel_source_hash
    path = os.path.join(ROOT, "profiles", "dram_traffic_tc_gemm_moe8k.txt")
    try:
        lines = [l.split() for l in open(path) if l.strip() and not l.startswith("#")]
    except OSError:
        return None
    src = kernel_source_hash()
    for f in lines:
        if len(f) == 6 and f[0] == kernel and f[1] == src:
            cap_rows, cap_cols, rd, wr = int(f[2]), int(f[3]), float(f[4]), float(f[5])
            return (rd + wr) * (rows * cols) / (cap_rows * cap_cols)
    return None


def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return d, "measured"
    except (OSError, ValueError):
        return dict(FALLBACK_PEAKS), "fallback"


# ---------------------------------------------------------------------------
# clocks sampled with nvidia-smi during the timed region
# ---------------------------------------------------------------------------
class ClockSampler:
    FIELDS = ("timestamp,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.lines = []
        self.thread = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "100"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
            return
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self, t_begin=None, t_end=None):
        """Median clocks over the samples taken between t_begin and t_end
        (host wall-clock seconds); all samples if none falls inside."""
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        if self.thread:
            self.thread.join(timeout=2)
        return summarise_clocks(self.lines, t_begin, t_end)


THROTTLE_NAMES = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
# a timed region that saw one of these is not a measurement of the kernels
REJECTING_REASONS = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown")
# median SM clock below this share of its maximum with no throttle reason
# active: a clock lock left behind by an earlier user
LOCKED_CLOCK_SHARE = 0.8


def summarise_clocks(lines, t_begin=None, t_end=None):
    """Median SM clock, maximum clock, peak power and the throttle reasons seen
    in nvidia-smi's `--query-gpu=ClockSampler.FIELDS --format=csv,noheader,nounits`
    lines, over the samples taken between t_begin and t_end (host wall-clock
    seconds; all samples if none falls inside)."""
    import datetime
    samples = []
    for line in lines:
        parts = [p.strip() for p in line.split(",")]
        if len(parts) < 9:
            continue
        try:
            ts = datetime.datetime.strptime(parts[0], "%Y/%m/%d %H:%M:%S.%f").timestamp()
            samples.append((ts, float(parts[1]), float(parts[2]), float(parts[3]), parts[5:9]))
        except ValueError:
            continue
    inside = [x for x in samples if t_begin is not None and t_begin <= x[0] <= t_end]
    used = inside or samples
    sm = [x[1] for x in used]
    mx = [x[2] for x in used]
    power = [x[3] for x in used]
    reasons = set()
    for x in used:
        for name, val in zip(THROTTLE_NAMES, x[4]):
            if val.lower().startswith("active"):
                reasons.add(name)
    if not sm:
        return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
    return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "samples": len(sm),
            "samples_in_timed_region": len(inside), "power_w_max": max(power) if power else None,
            "reasons": sorted(reasons)}


def clocks_rejection(clk):
    """Why a timed region's clock record makes its number invalid, or None:
    a hardware or thermal slowdown, or the SM clock held well below its
    maximum with no throttle reason (a leftover clock lock). sw_power_cap is a
    normal state of a dense GEMM step on a 1.4 kW part and is kept."""
    seen = [r for r in clk.get("reasons", []) if r in REJECTING_REASONS]
    if seen:
        return "throttled: " + ", ".join(seen)
    sm, mx = clk.get("sm_mhz"), clk.get("sm_max_mhz")
    if sm and mx and sm < LOCKED_CLOCK_SHARE * mx and not any(r in THROTTLE_NAMES for r in clk.get("reasons", [])):
        return f"SM clock {sm:.0f} of {mx:.0f} MHz with no throttle reason (clock lock suspected)"
    return None


# ---------------------------------------------------------------------------
# the step
# ---------------------------------------------------------------------------
class LossHeadStep:
    """Device buffers and the six ABI calls of one loss-head step."""

    def __init__(self, wl, device, torch, cached=False):
        from paper_2607_07508_gb300 import sao
        self.sao = sao
        self.torch = torch
        self.wl = wl
        N, h, V = wl.N, wl.h, wl.V
        f32 = torch.float32
        dev = device
        self.H = wl.H
        self.W = wl.W
        self.y = torch.as_tensor(wl.y).to(dev)
        self.mask = torch.as_tensor(wl.loss_mask).to(dev)
        self.values = torch.as_tensor(wl.values).to(dev)
        self.rewards = torch.as_tensor(wl.rewards).to(dev)
        self.cu = torch.as_tensor(wl.cu_seqlens).to(dev)
        self.adv = torch.empty(N, dtype=f32, device=dev)
        self.ret = torch.empty(N, dtype=f32, device=dev)
        self.logp = torch.empty(N, dtype=f32, device=dev)
        self.lse = torch.empty(N, dtype=f32, device=dev)
        self.coef = torch.empty(N, dtype=f32, device=dev)
        self.flags = torch.empty(N, dtype=torch.uint8, device=dev)
        self.G = torch.empty(N, dtype=f32, device=dev)
        self.dV = torch.empty(N, dtype=f32, device=dev)
        self.loss = torch.empty(1, dtype=f32, device=dev)
        self.vloss = torch.empty(1, dtype=f32, device=dev)
        self.counts = torch.empty(4, dtype=torch.int64, device=dev)
        self.ev = torch.empty(4, dtype=torch.float64, device=dev)
        self.one = torch.ones(1, dtype=f32, device=dev)
        self.dH = torch.empty_like(self.H)
        self.dW = torch.empty(V, h, dtype=f32, device=dev)
        self.ws = sao.workspace(N, h, V, self.H.dtype, device=dev)
        # The rollout policy's log-probs: the current policy's, perturbed by the
        # workload's staleness noise (prepared once, outside any timing).
        sao.sao_token_logprobs_fwd(self.H, self.W, self.y, self.logp, self.lse, self.ws)
        self.old = (self.logp + torch.as_tensor(wl.xi).to(dev)).contiguous()
        # The default path is vocabulary-chunked with the logits recomputed in
        # the backward: no [N, V] buffer of any dtype exists. Only on request
        # (cached=True) does the forward keep its bf16 probabilities (about
        # 2*N*V bytes) for the backward.
        self.cache = None
        if cached:
            if self.H.dtype != torch.bfloat16:
                raise ValueError("the probability cache is for bf16 workloads only")
            self.cache = sao.logprob_cache(N, V, device=dev)

    def run(self):
        s, wl = self.sao, self.wl
        s.sao_advantages(self.values, self.rewards, self.mask, self.cu, wl.gamma, wl.lam, wl.lam_critic, wl.alpha,
                         self.adv, self.ret, self.ws)
        s.sao_value_loss(self.values, self.ret, self.mask, self.vloss, self.dV, self.ws, ev_sums=self.ev)
        # log-probs of observation tokens are never read: skip those rows
        if self.cache is not None:
            s.sao_token_logprobs_fwd_cached(self.H, self.W, self.y, self.logp, self.lse, self.cache, self.ws,
                                            row_mask=self.mask)
        else:
            s.sao_token_logprobs_fwd(self.H, self.W, self.y, self.logp, self.lse, self.ws, row_mask=self.mask)
        s.sao_policy_loss_fwd(self.logp, self.old, self.adv, self.mask, wl.eps_low, wl.eps_high, self.loss,
                              self.counts, self.ws, coef=self.coef, flags=self.flags)
        s.sao_policy_loss_bwd(self.logp, self.old, self.adv, self.mask, wl.eps_low, wl.eps_high, self.one, self.G,
                              self.ws)
        if self.cache is not None:
            s.sao_token_logprobs_bwd_cached(self.H, self.W, self.y, self.lse, self.G, self.dH, self.dW, self.cache,
                                            self.ws)
        else:
            s.sao_token_logprobs_bwd(self.H, self.W, self.y, self.lse, self.G, self.dH, self.dW, self.ws)


# Algorithmic work per step of each tensor-core kernel, in flops: the forward
# computes the rows with loss_mask = 1, the backward kernels the rows with a
# non-zero incoming gradient (over all vocabulary chunks and row blocks of the
# step; a launch does its share of it).
def kernel_bytes(name, h, rows, cols):
    """Bytes one launch of a log-prob GEMM must move at least (operands read
    once, outputs written once) for `rows` token rows and `cols` vocabulary
    columns: the yardstick for its DRAM traffic."""
    if name == "tc_logits_lse_fwd":  # H_c, W, per-tile (max, sum) partials
        return 2 * rows * h + 2 * cols * h + 8 * rows * -(-cols // 256)
    if name == "tc_dlogits":  # H_c, W chunk -> bf16 dZ chunk
        return 2 * rows * h + 2 * cols * h + 2 * rows * cols
    if name == "tc_dH_gemm":  # dZ chunk, W chunk -> fp32 dH
        return 2 * rows * cols + 2 * cols * h + 4 * rows * h
    if name == "tc_dW_gemm":  # dZ chunk, H_c -> fp32 dW rows of the chunk
        return 2 * rows * cols + 2 * rows * h + 4 * cols * h
    return None


def kernel_flops(name, h, V, rows_fwd, rows_bwd):
    if name == "tc_logits_lse_fwd":
        return 2.0 * rows_fwd * h * V
    if name in ("tc_dlogits", "tc_dH_gemm", "tc_dW_gemm"):
        return 2.0 * rows_bwd * h * V
    return None


# ---------------------------------------------------------------------------
# CPU baseline: the fp64 oracle on a bounded sample of the same workload
# ---------------------------------------------------------------------------
POOL_ROWS = 4096


def sample_pool(wl, H_cpu):
    """A seeded pool of up to POOL_ROWS token rows (random order) and their
    hidden states: every CPU-baseline sample is a prefix of it."""
    rng = np.random.default_rng(0)
    pool = rng.choice(wl.N, size=min(POOL_ROWS, wl.N), replace=False)
    import torch
    return pool, H_cpu[torch.as_tensor(pool)]


def cpu_baseline(wl, rows: int, pool, H_pool, W_cpu, threads_note: str):
    """Times the oracle on `rows` sampled tokens (all three GEMMs over the full
    vocabulary) and on all N tokens for the O(N) parts; returns tokens/s
    extrapolated to the N-token step."""
    from oracle import sao_oracle as O
    rows = min(rows, len(pool))
    order = np.argsort(pool[:rows])
    idx = pool[:rows][order]
    import torch
    Hs = H_pool[:rows][torch.as_tensor(order)]
    ys = wl.y[idx]
    t0 = time.perf_counter()
    adv, ret = O.advantages(wl.values, wl.rewards, wl.loss_mask, wl.cu_seqlens, wl.gamma, wl.lam, wl.lam_critic,
                            wl.alpha)
    O.value_loss(wl.values, ret, wl.loss_mask)
    t_on = time.perf_counter() - t0
    t1 = time.perf_counter()
    logp, lse = O.token_logprobs(Hs, W_cpu, ys)
    old = logp + wl.xi[idx]
    O.policy_loss(logp, old, adv[idx], wl.loss_mask[idx], wl.eps_low, wl.eps_high)
    G = O.policy_loss_bwd(logp, old, adv[idx], wl.loss_mask[idx], wl.eps_low, wl.eps_high, 0, 1.0)
    O.token_logprobs_bwd(Hs, W_cpu, ys, lse, G)
    t_gemm = time.perf_counter() - t1
    t_step = t_on + t_gemm * (wl.N / rows)
    return {"value": wl.N / t_step, "unit": UNIT, "kind": "oracle",
            "sample": (f"fp64 numpy oracle: advantages + value loss on all {wl.N} tokens ({t_on:.2f} s), "
                       f"log-prob fwd + policy loss + log-prob bwd on {rows} sampled tokens over the full "
                       f"vocabulary ({t_gemm:.2f} s), extrapolated linearly to {wl.N} tokens; {threads_note}"),
            "measured_s": t_on + t_gemm, "rows": rows, "t_on": t_on, "t_gemm": t_gemm, "threads_note": threads_note}


def two_point(wl, a, b):
    """Whole-step tokens/s from two sample sizes: the GEMM part's time as a
    fixed part (the oracle's per-call fp64 copy of W) plus a per-row part, fit
    through both samples, then extrapolated to all N rows."""
    per_row = (b["t_gemm"] - a["t_gemm"]) / (b["rows"] - a["rows"])
    if per_row <= 0:
        return b
    fixed = max(0.0, a["t_gemm"] - per_row * a["rows"])
    t_step = b["t_on"] + fixed + per_row * wl.N
    out = dict(b)
    out["value"] = wl.N / t_step
    out["sample"] = (f"fp64 numpy oracle: advantages + value loss on all {wl.N} tokens ({b['t_on']:.2f} s), "
                     f"log-prob fwd + policy loss + log-prob bwd on {a['rows']} and {b['rows']} sampled tokens "
                     f"over the full vocabulary ({a['t_gemm']:.2f} s, {b['t_gemm']:.2f} s), fit as {fixed:.2f} s "
                     f"per call + {1e3 * per_row:.2f} ms per token and extrapolated to {wl.N} tokens; "
                     f"{b['threads_note']}")
    return out


def sized_cpu_baseline(wl, pool, H_pool, W_cpu, threads_note, budget_s=15.0, first_rows=64):
    """The oracle on samples of 4x more tokens each time until one takes at
    least 40 % of `budget_s` (or the pool is used up); the last two samples
    give the fixed and per-token parts of the time (two_point)."""
    prev, cur = None, cpu_baseline(wl, first_rows, pool, H_pool, W_cpu, threads_note)
    while cur["measured_s"] < 0.4 * budget_s and cur["rows"] < len(pool):
        prev, cur = cur, cpu_baseline(wl, min(len(pool), 4 * cur["rows"]), pool, H_pool, W_cpu, threads_note)
    return two_point(wl, prev, cur) if prev is not None else cur


def cpu_baseline_child(args):
    """--cpu-baseline-child FILE: the oracle on the sample the parent saved,
    in a process whose BLAS thread count the parent fixed through the
    environment before numpy loaded; prints one JSON object."""
    import torch
    from paper_2607_07508_gb300 import synthetic as S
    d = torch.load(args.cpu_baseline_child)
    wl = S.make_workload(d["config"], dense=False, seed=d["seed"], N_override=d["N_override"])
    note = f"BLAS threads = {d['threads']} (OPENBLAS/OMP/MKL_NUM_THREADS)"
    cb = sized_cpu_baseline(wl, d["pool"].numpy(), d["H_pool"], d["W"], note, budget_s=d["budget_s"], first_rows=8)
    print(json.dumps({k: cb[k] for k in ("value", "unit", "kind", "sample", "rows")}))
    return 0


def cpu_baselines(wl, H_cpu, W_cpu, config, seed, N_override, budget_s=12.0):
    """The oracle timed on the host cores twice: with numpy's BLAS on every
    core (in this process) and on one thread (a child process started with
    the BLAS thread count fixed, since it cannot change once numpy is
    loaded). Reported: all-cores value as `value`, both figures by name."""
    import tempfile
    import torch
    pool, H_pool = sample_pool(wl, H_cpu)
    cores = os.cpu_count() or 1
    allc = sized_cpu_baseline(wl, pool, H_pool, W_cpu, f"BLAS threads = host cores ({cores})", budget_s=budget_s)
    one = None
    fd, path = tempfile.mkstemp(suffix=".pt", prefix="sao_cpu_baseline_")
    os.close(fd)
    try:
        torch.save({"config": config, "seed": seed, "N_override": N_override, "pool": torch.as_tensor(pool),
                    "H_pool": H_pool,
                    "W": W_cpu, "threads": 1, "budget_s": budget_s}, path)
        env = dict(os.environ, OPENBLAS_NUM_THREADS="1", OMP_NUM_THREADS="1", MKL_NUM_THREADS="1")
        r = subprocess.run([sys.executable, os.path.abspath(__file__), "--cpu-baseline-child", path], env=env,
                           capture_output=True, text=True, timeout=600)
        if r.returncode == 0 and r.stdout.strip():
            one = json.loads(r.stdout.strip().splitlines()[-1])
    except (subprocess.TimeoutExpired, OSError, ValueError):
        one = None
    finally:
        os.unlink(path)
    out = {"value": allc["value"], "unit": UNIT, "cores": cores, "kind": "oracle", "sample": allc["sample"],
           "sample_rows": allc["rows"],
           "value_all_cores": allc["value"], "cores_all": cores,
           "value_1thread": one["value"] if one else None, "sample_1thread": one["sample"] if one else None}
    return out


# ---------------------------------------------------------------------------
def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def run_reference(args):
    rank, world, _ = dist_env()
    if rank != 0:
        return 0
    from paper_2607_07508_gb300 import synthetic as S
    wl = S.make_workload(args.config, device="cpu")
    H_cpu, W_cpu = wl.H, wl.W
    pool, H_pool = sample_pool(wl, H_cpu)
    cores = os.cpu_count() or 1
    note = f"BLAS threads = host cores ({cores})"
    # each step is a bounded sample: the row count a 4-second budget gives
    rows = sized_cpu_baseline(wl, pool, H_pool, W_cpu, note, budget_s=4.0, first_rows=16)["rows"]
    vals, walls = [], []
    cb = None
    for _ in range(args.steps):
        cb = cpu_baseline(wl, rows, pool, H_pool, W_cpu, note)
        vals.append(cb["value"])
        walls.append(cb["measured_s"])
    value = statistics.median(vals)
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup,
            # the time each bounded sample step took; `value` extrapolates it to the whole batch
            "ms_per_step": 1000.0 * statistics.median(walls),
            "ms_per_step_is": f"wall time of one bounded sample step ({rows} sampled tokens for the GEMMs, all "
                              f"{wl.N} for the O(N) parts)",
            "ms_per_step_extrapolated": 1000.0 * wl.N / value,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": workload_config(wl),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                             "sample": cb["sample"]},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line))
    return 0


def workload_config(wl, cached=False):
    if wl.name == "moe":
        what = (f"moe: MoE-policy head, {wl.N} packed tokens in {wl.B} single-rollout agentic trajectories "
                f"(lognormal lengths, median 4k, max 32k), 25% observation tokens")
    else:
        what = f"{wl.name}: {wl.N} packed tokens in {wl.B} trajectories; {wl.recipe}"
    if cached:
        what += ("; VARIANT: the forward stores bf16 probabilities of every computed row over the whole "
                 "vocabulary (2*N*V bytes) for the backward")
    else:
        what += "; log-probs vocabulary-chunked, logits recomputed in the backward (no [N, V] buffer)"
    return {"workload": what, "logprob_path": "cached" if cached else "recompute",
            "tokens": wl.N, "trajectories": wl.B, "hidden": wl.h, "vocab": wl.V, "dtype": wl.dtype,
            "gamma": wl.gamma, "lambda": wl.lam, "eps_low": wl.eps_low, "eps_high": wl.eps_high,
            "l2": (f"inputs larger than L2 (H {wl.N * wl.h * 2 / 1e6:.0f} MB + W {wl.V * wl.h * 2 / 1e6:.0f} MB per step, "
                   f"L2 126 MB); no flush")}


# Algorithmic bytes per token of each O(N) kernel (reads + writes).
ON_BYTES = {"gae_scan": 13, "gae_telescoped": 13, "policy_loss_fwd": 18, "policy_loss_bwd": 17, "value_loss": 13, "count_mask": 1,
            "gae_count": 1, "decoupled_loss_fwd": 22, "decoupled_loss_bwd": 21}


def bandwidth_study(args):
    """HBM study of the O(N) kernels on the 2^27-token workload (inputs far
    above L2): achieved algorithmic GB/s per kernel from the library's own
    CUDA-event timing, against the measured HBM copy bandwidth."""
    import torch
    from paper_2607_07508_gb300 import sao, synthetic as S
    torch.cuda.set_device(0)
    sao.load()
    peaks, src = load_peaks()
    N = args.tokens or (1 << 27)
    wl = S.bandwidth_workload(N=N, B=max(1, N >> 13))
    dev = "cuda"
    t = lambda a: torch.as_tensor(a).to(dev)
    v, m, cu, R = t(wl.values), t(wl.loss_mask), t(wl.cu_seqlens), t(wl.rewards)
    lp, old = t(wl.logp_syn), t(wl.old_logp_syn)
    f = lambda: torch.empty(N, dtype=torch.float32, device=dev)
    adv, ret, coef, grad, dV = f(), f(), f(), f(), f()
    flags = torch.empty(N, dtype=torch.uint8, device=dev)
    loss = torch.empty(1, device=dev)
    counts = torch.empty(4, dtype=torch.int64, device=dev)
    ev = torch.empty(4, dtype=torch.float64, device=dev)
    one = torch.ones(1, device=dev)
    ws = sao.workspace(N)

    # decoupled three-policy objective: pi_old = the stale log-probs, pi_rollout
    # = pi_old with an engine mismatch (the generator's xi)
    roll = t((wl.old_logp_syn + wl.xi).astype("float32"))
    counts6 = torch.empty(6, dtype=torch.int64, device=dev)

    def calls():
        sao.sao_advantages(v, R, m, cu, wl.gamma, wl.lam, wl.lam_critic, 0.0, adv, ret, ws)
        sao.sao_advantages(v, R, m, cu, 1.0, 1.0, 1.0, 1.5, adv, ret, ws)
        sao.sao_policy_loss_fwd(lp, old, adv, m, wl.eps_low, wl.eps_high, loss, counts, ws, coef=coef, flags=flags)
        sao.sao_policy_loss_bwd(lp, old, adv, m, wl.eps_low, wl.eps_high, one, grad, ws)
        sao.sao_value_loss(v, ret, m, loss, dV, ws, ev_sums=ev)
        sao.sao_decoupled_loss_fwd(lp, old, roll, adv, m, 0.2, 0.28, 0.5, 2.0, loss, counts6, ws, coef=coef,
                                   flags=flags)
        sao.sao_decoupled_loss_bwd(lp, old, roll, adv, m, 0.2, 0.28, 0.5, 2.0, one, grad, ws)

    # the follow-on rows (App. A.1 step GAE, clipped surrogate, GRPO and running-mean advantages)
    vm = torch.empty(N, dtype=torch.uint8, device=dev)
    B = wl.B
    gid = t((np.arange(B) // 8).astype(np.int32))              # groups of 8 trajectories
    pid = t((np.arange(B) % 64).astype(np.int32))              # 64 prompts
    hist = torch.zeros(64, 8, dtype=torch.float32, device=dev)
    seen = torch.zeros(64, dtype=torch.int64, device=dev)

    n_act = int(wl.loss_mask.astype(np.int64).sum())
    # whole calls with their algorithmic bytes per token (reads + writes)
    whole = {
        "sao_advantages": (13, lambda: sao.sao_advantages(v, R, m, cu, wl.gamma, wl.lam, wl.lam_critic, 0.0,
                                                          adv, ret, ws)),
        "sao_advantages (gamma = lambda = 1)": (13, lambda: sao.sao_advantages(v, R, m, cu, 1.0, 1.0, 1.0, 0.0,
                                                                               adv, ret, ws)),
        "sao_step_advantages": (14, lambda: sao.sao_step_advantages(v, R, m, cu, wl.gamma, wl.lam, wl.lam_critic,
                                                                    0.0, sao.SAO_STEP_AVERAGE, adv, ret, ws,
                                                                    value_mask=vm)),
        "sao_policy_loss_fwd": (18, lambda: sao.sao_policy_loss_fwd(lp, old, adv, m, wl.eps_low, wl.eps_high, loss,
                                                                    counts, ws, coef=coef, flags=flags)),
        # a trainer that knows its normaliser (the data-parallel action-token
        # total) passes it: the forward then needs no count pass
        "sao_policy_loss_fwd (n_norm given)": (18, lambda: sao.sao_policy_loss_fwd(
            lp, old, adv, m, wl.eps_low, wl.eps_high, loss, counts, ws, coef=coef, flags=flags, n_norm=n_act)),
        "sao_value_loss": (13, lambda: sao.sao_value_loss(v, ret, m, loss, dV, ws, ev_sums=ev)),
        "sao_value_loss (n_norm given)": (13, lambda: sao.sao_value_loss(v, ret, m, loss, dV, ws, ev_sums=ev,
                                                                         n_norm=n_act)),
        "sao_clip_loss_fwd": (18, lambda: sao.sao_clip_loss_fwd(lp, old, adv, m, cu, 0.2, 0.28,
                                                                sao.SAO_NORM_SEQUENCE, loss, counts, ws, coef=coef,
                                                                flags=flags)),
        "sao_clip_loss_bwd": (17, lambda: sao.sao_clip_loss_bwd(lp, old, adv, m, cu, 0.2, 0.28,
                                                                sao.SAO_NORM_SEQUENCE, one, grad, ws)),
        "sao_decoupled_loss_fwd": (22, lambda: sao.sao_decoupled_loss_fwd(lp, old, roll, adv, m, 0.2, 0.28, 0.5,
                                                                          2.0, loss, counts6, ws, coef=coef,
                                                                          flags=flags)),
        "sao_decoupled_loss_fwd (n_norm given)": (22, lambda: sao.sao_decoupled_loss_fwd(
            lp, old, roll, adv, m, 0.2, 0.28, 0.5, 2.0, loss, counts6, ws, coef=coef, flags=flags, n_norm=n_act)),
        "sao_group_advantages": (5, lambda: sao.sao_group_advantages(R, gid, m, cu, 1e-6, adv, ws)),
        "sao_running_mean_advantages": (5, lambda: sao.sao_running_mean_advantages(R, pid, hist, seen, m, cu, adv,
                                                                                   ws)),
    }

    for _ in range(max(3, args.warmup)):
        calls()
        for _, fn in whole.values():
            fn()
    torch.cuda.synchronize()
    sao.sao_profile_enable(True)
    sao.sao_profile_reset()
    for _ in range(args.steps):
        calls()
    torch.cuda.synchronize()
    prof = sao.sao_profile_read()
    sao.sao_profile_enable(False)
    per_call = {}
    stream = torch.cuda.current_stream()
    for name, (b, fn) in whole.items():
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(args.steps):
            fn()
        e1.record(stream)
        torch.cuda.synchronize()
        us = 1000 * e0.elapsed_time(e1) / args.steps
        gbs = b * N / (us / 1e6) / 1e9
        # the call's kernels, timed separately by the library (one more round)
        sao.sao_profile_enable(True)
        sao.sao_profile_reset()
        fn()
        torch.cuda.synchronize()
        ks = {k: round(1000 * t / n, 1) for k, (n, t) in sao.sao_profile_read().items()}
        sao.sao_profile_enable(False)
        per_call[name] = {"avg_us": us, "bytes_per_token": b, "achieved_gbs": gbs,
                          "frac_of_hbm": gbs / peaks["hbm_gbs"], "kernels_us": ks}
    out = {}
    names = {"policy_loss_fwd": "policy_loss_fwd", "policy_loss_bwd": "policy_loss_bwd"}
    for k, (n, ms) in prof.items():
        b = ON_BYTES.get(names.get(k, k))
        avg = ms / n
        row = {"launches": n, "avg_us": 1000 * avg}
        if b is not None:
            gbs = b * N / (avg / 1000) / 1e9
            row.update({"bytes_per_token": b, "achieved_gbs": gbs, "frac_of_hbm": gbs / peaks["hbm_gbs"]})
        out[k] = row
    print(json.dumps({"study": "O(N) kernels, HBM", "tokens": N, "trajectories": wl.B,
                      "peak_hbm_gbs": peaks["hbm_gbs"], "peak_source": src, "kernels": out,
                      "calls": per_call}))
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="native", choices=["native", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--tokens", type=int, default=None,
                    help="override the packed token count (smaller cases for profiling captures)")
    ap.add_argument("--config", default=WORKLOAD, choices=["tiny", "small", "moe", "long", "large"],
                    help="workload (the metric is quoted on moe; the others are the parity configurations)")
    ap.add_argument("--cached", action="store_true",
                    help="time the variant whose forward stores bf16 probabilities for all computed rows "
                         "(2*N*V bytes) instead of the default vocabulary-chunked recompute path")
    ap.add_argument("--dz-budget-gib", type=float, default=None,
                    help="bound on the backward's bf16 dZ buffer (default: the library's, 4 GiB)")
    ap.add_argument("--cta-pairs", type=int, choices=[0, 1], default=None,
                    help="tile the tensor-core GEMMs over CTA pairs (1) or single CTAs (0); default: the library's")
    ap.add_argument("--cpu-baseline-child", default=None, help=argparse.SUPPRESS)
    ap.add_argument("--bandwidth-study", action="store_true",
                    help="time the O(N) kernels alone on the 2^27-token bandwidth workload")
    args = ap.parse_args()
    if args.cpu_baseline_child:
        return cpu_baseline_child(args)
    if args.impl == "reference":
        return run_reference(args)
    if args.bandwidth_study:
        return bandwidth_study(args)

    import torch
    from paper_2607_07508_gb300 import sao, synthetic as S

    rank, world, local = dist_env()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
    sao.load()
    peaks, peak_src = load_peaks()
    if args.dz_budget_gib is not None:
        sao.sao_set_dz_budget_bytes(int(args.dz_budget_gib * (1 << 30)))
    if args.cta_pairs is not None:
        sao.sao_set_cta_pairs(bool(args.cta_pairs))

    seed = S.SEED_BASE + S.CONFIG_NAMES.index(args.config) + 97 * rank
    wl = S.make_workload(args.config, device=dev, seed=seed, N_override=args.tokens)
    step = LossHeadStep(wl, dev, torch, cached=args.cached)
    stream = torch.cuda.current_stream()
    for _ in range(max(3, args.warmup)):
        step.run()
    torch.cuda.synchronize()

    def barrier():
        if world > 1:
            torch.distributed.barrier()

    # ---- timed region (device-resident inputs) --------------------------------
    def timed_region():
        sao.sao_profile_enable(True)
        sao.sao_profile_reset()
        clocks = ClockSampler(local)
        clocks.start()
        time.sleep(0.3)
        barrier()
        torch.cuda.synchronize()
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        t_begin = time.time()
        e0.record(stream)
        for _ in range(args.steps):
            step.run()
        e1.record(stream)
        torch.cuda.synchronize()
        t_end = time.time()
        barrier()
        clk = clocks.stop(t_begin, t_end)
        ms = e0.elapsed_time(e1) / args.steps
        prof = sao.sao_profile_read()
        sao.sao_profile_enable(False)
        if world > 1:
            t = torch.tensor([ms], device=dev)
            torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
            ms = float(t.item())
        return ms, clk, prof

    ms, clk, prof = timed_region()
    # a region that ran throttled or under a leftover clock lock is measured
    # once more (every rank, if any rank's was); the second one is reported
    why = clocks_rejection(clk)
    redo = why is not None
    if world > 1:
        t = torch.tensor([1 if redo else 0], device=dev)
        torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
        redo = bool(t.item())
    if redo:
        first = {"ms_per_step": ms, "clocks": clk, "rejected_because": why or "another rank's clocks"}
        ms, clk, prof = timed_region()
        clk = dict(clk, remeasured_after=first)
    total_tokens = wl.N * world
    value = total_tokens / (ms / 1000.0)

    # ---- roofline of the dominant kernel --------------------------------------
    rows_fwd = int(step.mask.sum().item())
    rows_bwd = int((step.G != 0).sum().item())
    launches = sum(n for n, _ in prof.values())
    dom = max(prof.items(), key=lambda kv: kv[1][1])
    dom_name, (dom_n, dom_ms) = dom
    avg_ms = dom_ms / dom_n
    fl_step = kernel_flops(dom_name, wl.h, wl.V, rows_fwd, rows_bwd)
    per_step = dom_n / args.steps
    fl = fl_step / per_step if fl_step is not None else None
    burst = peaks.get("bf16_tflops", FALLBACK_PEAKS["bf16_tflops"])
    sustained = peaks.get("bf16_tflops_sustained", FALLBACK_PEAKS["bf16_tflops_sustained"])
    peak_mhz = (peaks.get("clocks_under_load") or {}).get("sm_mhz_median")
    bench_mhz = clk.get("sm_mhz")
    cached = step.cache is not None
    if fl is not None:
        achieved = fl / (avg_ms / 1000.0) / 1e12
        # the cached backward's GEMMs run over the forward rows (zero-gradient rows scaled by 0)
        dom_rows = rows_fwd if (dom_name == "tc_logits_lse_fwd" or cached) else rows_bwd
        roofline = {"bound": "tensor", "kernel": dom_name, "achieved": achieved, "peak": burst,
                    "unit": "TFLOP/s", "frac": achieved / burst,
                    "traffic": (stored_traffic(dom_name, dom_rows, wl.V / per_step)
                                if wl.name == "moe" and args.tokens is None else None),
                    "algorithmic_bytes_per_launch": kernel_bytes(dom_name, wl.h, dom_rows, wl.V / per_step),
                    "traffic_unit": ("bytes per launch (dram read + write from the 8k-token ncu capture, scaled by "
                                     "rows x vocabulary columns per launch)"),
                    "algorithmic_per_launch": (f"2*rows*h*V = {fl_step:.4g} flop per step over {per_step:g} "
                                               f"launches = {fl:.4g} flop per launch"),
                    "avg_launch_ms": avg_ms, "launches_per_step": per_step,
                    "peak_source": f"{peak_src} bf16_tflops (burst)",
                    "frac_of_sustained_peak": achieved / sustained}
    else:
        roofline = {"bound": "hbm", "kernel": dom_name, "achieved": None, "peak": peaks.get("hbm_gbs"),
                    "unit": "GB/s", "frac": None, "traffic": None}
    step_alg = 2.0 * wl.h * wl.V * (rows_fwd + 2 * rows_bwd)
    step_exec = 2.0 * wl.h * wl.V * (3 * rows_fwd if cached else rows_fwd + 3 * rows_bwd)
    alg_t = step_alg / (ms / 1000) / 1e12
    exe_t = step_exec / (ms / 1000) / 1e12
    step_roof = {"algorithmic_tflops": alg_t,
                 "frac_of_burst_peak": alg_t / burst,
                 "executed_tflops": exe_t,
                 "executed_frac_of_burst_peak": exe_t / burst,
                 # the sustained peak was taken at its own clocks: compare flops per SM clock
                 "executed_frac_of_sustained_peak_per_clock": (
                     (exe_t / bench_mhz) / (sustained / peak_mhz) if bench_mhz and peak_mhz else None),
                 "clocks_mhz": {"this_step_median": bench_mhz, "sustained_peak_run_median": peak_mhz},
                 "algorithmic_flops_per_step": f"2hV per forward row ({rows_fwd} action tokens) + 4hV per row "
                                               f"with a non-zero gradient ({rows_bwd}); 6*N*h*V = "
                                               f"{6.0 * wl.N * wl.h * wl.V:.4g} if no row were skipped",
                 "executed_flops_per_step": ("2hV per forward row, three times: the backward's two GEMMs read "
                                             "the forward's stored bf16 probabilities (no logit recompute) and "
                                             "run over the forward rows, a zero-gradient row scaled by 0"
                                             if cached else
                                             "algorithmic + 2hV per backward row (the logits are recomputed)"),
                 "logprob_path": "cached" if cached else "recompute",
                 "gemm_tiling": "CTA pairs (tcgen05 cta_group::2, M = 256)" if sao.sao_get_cta_pairs()
                                else "single CTAs (M = 128)",
                 "largest_logit_buffer": (f"[{rows_fwd}, {wl.V}] bf16 probabilities ({2.0 * rows_fwd * wl.V / 1e9:.1f} GB)"
                                          if cached else
                                          f"bf16 dZ of one row block x vocabulary chunk, at most "
                                          f"{sao.sao_get_dz_budget_bytes() / 2**30:.2f} GiB"),
                 "rows_forward": rows_fwd, "rows_backward": rows_bwd,
                 "peak_source": peak_src}
    kernels = {k: {"launches": n, "avg_ms": t / n} for k, (n, t) in sorted(prof.items(), key=lambda kv: -kv[1][1])}

    # ---- end to end through the ABI with host buffers ---------------------------
    e2e = None
    if not args.no_e2e:
        host = {
            "H": torch.empty(step.H.shape, dtype=step.H.dtype, pin_memory=True),
            "y": torch.empty(wl.N, dtype=torch.int32, pin_memory=True),
            "old": torch.empty(wl.N, dtype=torch.float32, pin_memory=True),
            "values": torch.empty(wl.N, dtype=torch.float32, pin_memory=True),
            "rewards": torch.empty(wl.B, dtype=torch.float32, pin_memory=True),
            "mask": torch.empty(wl.N, dtype=torch.uint8, pin_memory=True),
            "cu": torch.empty(wl.B + 1, dtype=torch.int32, pin_memory=True),
        }
        host["H"].copy_(step.H)
        host["y"].copy_(step.y)
        host["old"].copy_(step.old)
        host["values"].copy_(step.values)
        host["rewards"].copy_(step.rewards)
        host["mask"].copy_(step.mask)
        host["cu"].copy_(step.cu)
        out = torch.empty(1 + 1 + 4 * 2, dtype=torch.float32, pin_memory=True)
        # Two device input sets: step i+1's inputs are copied on a second
        # stream into one set while step i runs on the other.
        names = ("H", "y", "old", "values", "rewards", "mask", "cu")
        sets = [{k: getattr(step, k) for k in names}, {k: torch.empty_like(getattr(step, k)) for k in names}]
        copy_stream = torch.cuda.Stream(device=dev)
        copied = [torch.cuda.Event(), torch.cuda.Event()]  # set j holds the next inputs
        freed = [torch.cuda.Event(), torch.cuda.Event()]   # the step that read set j is done
        h2d = sum(t.numel() * t.element_size() for t in host.values())
        d2h = out.numel() * out.element_size()
        res = torch.empty(10, dtype=torch.float32, device=dev)
        torch.cuda.synchronize()
        barrier()
        e2 = torch.cuda.Event(enable_timing=True)
        e3 = torch.cuda.Event(enable_timing=True)
        t_wall = time.perf_counter()

        def stage(i):
            j = i % 2
            with torch.cuda.stream(copy_stream):
                copy_stream.wait_event(e2 if i == 0 else freed[j])  # i = 1: freed[1] not yet recorded
                for k in names:
                    sets[j][k].copy_(host[k], non_blocking=True)
                copied[j].record(copy_stream)

        e2.record(stream)
        stage(0)
        for i in range(args.steps):
            if i + 1 < args.steps:
                stage(i + 1)
            stream.wait_event(copied[i % 2])
            for k in names:
                setattr(step, k, sets[i % 2][k])
            step.run()
            freed[i % 2].record(stream)
            res[0:1].copy_(step.loss)
            res[1:2].copy_(step.vloss)
            res[2:10].copy_(step.counts.view(torch.float32))
            out.copy_(res, non_blocking=True)
        e3.record(stream)
        torch.cuda.synchronize()
        barrier()
        for k in names:
            setattr(step, k, sets[0][k])
        ms_e2e = e2.elapsed_time(e3) / args.steps
        if world > 1:
            t = torch.tensor([ms_e2e], device=dev)
            torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
            ms_e2e = float(t.item())
        e2e = {"value": total_tokens / (ms_e2e / 1000.0), "unit": UNIT, "h2d_bytes_per_step": h2d,
               "d2h_bytes_per_step": d2h, "ms_per_step": ms_e2e,
               "note": "pinned host H, token ids, rollout log-probs, values, rewards, mask and cu_seqlens copied in, "
                       "loss, value loss and counts copied out, every step; W stays resident (model weight); "
                       "the inputs of step i+1 are copied on a second stream into a second buffer set while step "
                       "i runs"}

    # ---- CPU baseline (rank 0, single GPU only) ---------------------------------
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_baselines(wl, step.H.cpu(), step.W.cpu(), args.config, seed, args.tokens)

    if rank == 0:
        line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
                "warmup": max(3, args.warmup), "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
                "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
                "config": workload_config(wl, cached=step.cache is not None),
                "roofline": roofline, "step_roofline": step_roof, "cpu_baseline": cpu, "e2e": e2e,
                "clocks": clk, "gpu_launches": launches * 1, "gpu_launches_per_step": launches / args.steps,
                "kernels": kernels}
        print(json.dumps(line))
    if world > 1:
        torch.distributed.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
