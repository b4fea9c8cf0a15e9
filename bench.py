#!/usr/bin/env python3
"""Benchmark of the CPDP hot path on GB300: HBM GB/s of the local step and the
fused reconcile, ResNet-50 / CIFAR-100 parameter shape, W=8 workers, K=4.

One benchmark step is one synchronization period (one K-cycle): K-1 local
momentum-SGD steps and one reconcile, dispatched through the library's
schedule (cpdp_step), each mini-batch with its own gradient buffer. Inputs are
seeded synthetic tensors of the model's parameter shapes, resident in HBM.

Metric: algorithmic bytes / device time, where per parameter and worker a
local step moves 12 + 8 bytes (theta, buf, g read; theta, buf written; float32
gradients) and a reconcile moves 20 W + 16 bytes per parameter (W rows of g,
theta, buf read; buf, theta written; theta_ref, v read and written).

Launch (one process per GPU):
  python bench.py [--gpus 1] [--steps K] [--warmup W]
  torchrun ... bench.py --gpus N      # N independent replicas, weak scaling
  python bench.py --impl reference    # the fp64 CPU oracle on the same metric
"""
from __future__ import annotations

import argparse
import csv
import io
import json
import math
import os
import statistics
import subprocess
import sys
import tempfile
import time
from pathlib import Path

ROOT = Path(__file__).resolve().parent
METRIC = "CPDP reconcile+local-step HBM GB/s (% of GB300 peak), ResNet-50 shape, W=8"
DEFAULT_WORKLOAD = "resnet50_cifar100"
NOMINAL_HBM_GBS = 8000.0
# The paper's own figures, quoted as context only (other hardware, end-to-end training): it times no
# hot-path kernel. Sec. 5.1 and 6.1, Table 5.
PAPER_CONTEXT = ("context only, not a target: the paper times no optimizer or reconcile kernel; on Grid'5000 "
                 "(8 RTX 2080 Ti across two sites, 10/1 GbE, about 16.6 ms round trip, NCCL over TCP), CPDP "
                 "at K=4 trains ResNet-50/CIFAR-100 in 4275 s against DDP's 4959 s (13.8 % less wall-clock)")
FALLBACK_HBM_GBS = 6800.0
L2_BYTES = 129 * 10**6


# ---------------------------------------------------------------------------
# algorithmic bytes (host arithmetic; tested on CPU)
# ---------------------------------------------------------------------------
def local_step_bytes(W: int, N: int, grad_bytes: int, state_arrays: int = 2) -> int:
    """Per element: each [W][N] state array read and written (8 B; SGD has
    theta and buf, AdamW adds the second moments) and one gradient read."""
    return (8 * state_arrays + grad_bytes) * W * N


def reconcile_bytes(W: int, N: int, grad_bytes: int, state_arrays: int = 2) -> int:
    """W rows of g and of every state array read, the state arrays written;
    theta_ref and v read and written once per parameter."""
    return ((8 * state_arrays + grad_bytes) * W + 16) * N


def sync_bytes(W: int, N: int, grad_bytes: int, method: str = "cpdp", state_arrays: int = 2) -> int:
    """One synchronization step of `method`: CPDP's reconcile; LocalSGD's and
    DDP's sync steps touch no anchor or velocity (the local step's bytes)."""
    if method == "cpdp":
        return reconcile_bytes(W, N, grad_bytes, state_arrays)
    return local_step_bytes(W, N, grad_bytes, state_arrays)


def cycle_bytes(W: int, N: int, K: int, grad_bytes: int, method: str = "cpdp", state_arrays: int = 2) -> int:
    """K steps: K-1 local steps and one sync step (DDP: K sync steps)."""
    if method == "ddp":
        return K * sync_bytes(W, N, grad_bytes, method, state_arrays)
    return ((K - 1) * local_step_bytes(W, N, grad_bytes, state_arrays)
            + sync_bytes(W, N, grad_bytes, method, state_arrays))


def measured_peak() -> tuple[float, str]:
    p = ROOT / "MEASURED_PEAKS.json"
    try:
        return float(json.loads(p.read_text())["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


def strip_comments(source: str) -> str:
    """C++ source without its comments and with whitespace runs collapsed (the
    kernel headers hold no string literal with a comment marker in it)."""
    import re
    source = re.sub(r"/\*.*?\*/", " ", source, flags=re.S)
    source = re.sub(r"//[^\n]*", " ", source)
    return " ".join(source.split())


def kernel_source_sha() -> str:
    """Hash of the code (comments and layout left out) of the files that define
    the kernels and their launch shapes."""
    import hashlib
    h = hashlib.sha256()
    for name in ("cpdp_kernels.cuh", "cpdp_shapes.cuh"):
        h.update(strip_comments((ROOT / "paper_2607_21224_gb300" / "csrc" / name).read_text()).encode())
    return h.hexdigest()[:16]


def ncu_traffic(kernel: str) -> float | None:
    """DRAM bytes per launch of `kernel` from the committed ncu summary, if it
    was taken on the current kernel source (else None)."""
    f = ROOT / "profiles" / "ncu_traffic.txt"
    if not f.exists():
        return None
    sha = kernel_source_sha()
    for line in f.read_text().splitlines():
        parts = dict(kv.split("=", 1) for kv in line.split() if "=" in kv)
        if parts.get("kernel") == kernel and parts.get("source_sha") == sha:
            return float(parts["bytes_per_launch"])
    return None


# ---------------------------------------------------------------------------
# clocks sampled during the timed region
# ---------------------------------------------------------------------------
CLOCK_FIELDS = ("timestamp,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
                "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
                "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")


class ClockSampler:
    def __init__(self, gpu_id: str | None):
        self.proc = None
        self.file = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
        cmd = ["nvidia-smi", f"--query-gpu={CLOCK_FIELDS}", "--format=csv,noheader,nounits", "-lms", "100"]
        if gpu_id:
            cmd.insert(1, f"--id={gpu_id}")
        try:
            self.proc = subprocess.Popen(cmd, stdout=self.file, stderr=subprocess.DEVNULL)
        except (OSError, ValueError):
            self.proc = None
        self.t0 = self.t1 = None

    def mark_start(self):
        self.t0 = time.time()

    def mark_end(self):
        self.t1 = time.time()

    def stop(self) -> dict:
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"], "samples": 0}
        time.sleep(0.25)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.file.flush()
        text = Path(self.file.name).read_text()
        os.unlink(self.file.name)
        return summarize_clocks(text, self.t0, self.t1)


def _parse_ts(s: str) -> float | None:
    from datetime import datetime
    for fmt in ("%Y/%m/%d %H:%M:%S.%f", "%Y/%m/%d %H:%M:%S"):
        try:
            return datetime.strptime(s.strip(), fmt).timestamp()
        except ValueError:
            pass
    return None


def summarize_clocks(text: str, t0: float | None, t1: float | None) -> dict:
    rows = []
    for r in csv.reader(io.StringIO(text)):
        if len(r) < 9:
            continue
        try:
            rows.append(dict(ts=_parse_ts(r[0]), sm=float(r[1]), smax=float(r[2]),
                             power=float(r[3]) if r[3].strip() not in ("", "[N/A]") else None,
                             reasons={"hw_slowdown": r[5], "hw_thermal_slowdown": r[6],
                                      "sw_thermal_slowdown": r[7], "sw_power_cap": r[8]}))
        except ValueError:
            continue
    if not rows:
        return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"], "samples": 0}
    inside = [r for r in rows if r["ts"] is not None and t0 is not None and t1 is not None
              and t0 - 0.05 <= r["ts"] <= t1 + 0.05]
    used = inside or rows
    reasons = sorted({k for r in used for k, v in r["reasons"].items() if v.strip().lower() == "active"})
    return {"sm_mhz": statistics.median(r["sm"] for r in used),
            "sm_max_mhz": max(r["smax"] for r in used),
            "reasons": reasons,
            "samples": len(used),
            "window": "timed region" if inside else "whole run (timed region shorter than the sampling period)"}


# ---------------------------------------------------------------------------
# multi-rank helpers (replicas only; the path has no data exchange)
# ---------------------------------------------------------------------------
def dist_env() -> tuple[int, int, int]:
    return (int(os.environ.get("RANK", "0")), int(os.environ.get("WORLD_SIZE", "1")),
            int(os.environ.get("LOCAL_RANK", "0")))


def max_over_ranks(x: float, device=None) -> float:
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()):
        return x
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def barrier(device=None):
    import torch.distributed as dist
    if dist.is_available() and dist.is_initialized():
        if device is not None and device.type == "cuda":
            dist.barrier(device_ids=[device.index])
        else:
            dist.barrier()


# ---------------------------------------------------------------------------
# CPU oracle timing (baseline and reference arm)
# ---------------------------------------------------------------------------
def oracle_cycle_sample(wl, n_cols: int, seed: int = 42):
    """Inputs for one K-cycle of `wl` restricted to its first n_cols columns."""
    from paper_2607_21224_gb300 import workloads as wls
    cols = slice(0, n_cols)
    theta0 = wls.make_theta0(wl, seed)[cols].double().numpy()
    grads = [wls.make_grads(wl, t, seed, columns=cols).float().double().numpy() for t in range(1, wl.K + 1)]
    return theta0, grads


def time_oracle_cycle(wl, theta0, grads, split: dict | None = None, method: str = "cpdp",
                      state_sync: bool = False) -> float:
    """Seconds for one K-cycle of the oracle (K-1 local steps + 1 reconcile;
    DDP: K synchronized steps) of `method`, with the workload's optimizer. With
    `split`, each step's seconds are also appended to split["local"] or
    split["sync"] (the cycle's last step syncs)."""
    import oracle
    import numpy as np
    f = lambda x: float(np.float32(x))  # noqa: E731
    algo = oracle.default()
    if wl.optimizer == "adamw":
        algo = oracle.AdamWOracle(algo, f(wl.adam_beta1), f(wl.adam_beta2), f(wl.adam_eps))
    hp = oracle.Hyper(lr=f(wl.lr), momentum=f(wl.momentum), weight_decay=f(wl.weight_decay), K=wl.K,
                      beta=f(wl.beta), alpha=f(wl.alpha))
    st = algo.init(wl.W, theta0)
    t0 = time.perf_counter()
    for t in range(1, wl.K + 1):
        ts = time.perf_counter()
        algo.step(st, grads[t - 1], hp, t, wl.K, method, state_sync)
        if split is not None:
            split["sync" if t == wl.K else "local"].append(time.perf_counter() - ts)
    return time.perf_counter() - t0


def calibrate_oracle_cols(wl, seconds: float) -> int:
    """Columns of the workload one oracle K-cycle covers in about `seconds`."""
    probe = min(wl.N, 1 << 14)
    th, gr = oracle_cycle_sample(wl, probe)
    dt = min(time_oracle_cycle(wl, th, gr) for _ in range(2))
    n = int(probe * seconds / max(dt, 1e-9))
    return max(256, min(wl.N, n - n % 4))


def cpu_baseline(wl, target_s: float = 15.0) -> dict:
    n_cols = calibrate_oracle_cols(wl, target_s / 3)
    th, gr = oracle_cycle_sample(wl, n_cols)
    reps, total = 0, 0.0
    split: dict = {"local": [], "sync": []}
    while total < target_s and reps < 50:
        total += time_oracle_cycle(wl, th, gr, split)
        reps += 1
    gbytes = cycle_bytes(wl.W, n_cols, wl.K, wl.grad_bytes, "cpdp", wl.state_arrays) * reps
    scale = wl.N / n_cols  # per-column work: seconds scale with the columns
    per_step = {}
    for kind, nbytes in (("local_step", local_step_bytes(wl.W, n_cols, wl.grad_bytes, wl.state_arrays)),
                         ("reconcile", reconcile_bytes(wl.W, n_cols, wl.grad_bytes, wl.state_arrays))):
        xs = split["local" if kind == "local_step" else "sync"]
        if xs:
            mean = statistics.fmean(xs)
            per_step[kind] = {"s_full_N": round(mean * scale, 4), "GB_s": round(nbytes / mean / 1e9, 4)}
    return {"value": round(gbytes / total / 1e9, 4), "unit": "GB/s", "cores": 1, "kind": "oracle",
            "per_step": per_step,
            "sample": (f"{reps} K-cycles (K-1={wl.K - 1} local steps + 1 reconcile) of {wl.name} "
                       f"(W={wl.W}) on its first {n_cols} of {wl.N} parameter columns, fp64, "
                       f"single thread, {total:.1f} s"),
            "host_cpus": os.cpu_count()}


def run_reference(args) -> None:
    rank, world, _ = dist_env()
    if rank != 0:
        return
    from paper_2607_21224_gb300 import workloads as wls
    wl = wls.get(args.workload)
    # each step's sample is sized so that warm-up and timed steps together take about
    # --ref-total-seconds (at most --ref-step-seconds per step)
    per_step = min(args.ref_step_seconds, args.ref_total_seconds / (args.steps + args.warmup))
    n_cols = calibrate_oracle_cols(wl, per_step)
    th, gr = oracle_cycle_sample(wl, n_cols)
    run = lambda: time_oracle_cycle(wl, th, gr, method=args.method, state_sync=args.state_reconcile)  # noqa: E731
    for _ in range(args.warmup):
        run()
    times = [run() for _ in range(args.steps)]
    total = sum(times)
    gbytes = cycle_bytes(wl.W, n_cols, wl.K, wl.grad_bytes, args.method, wl.state_arrays) * args.steps
    value = gbytes / total / 1e9
    sample = (f"each step one K-cycle ({args.method}) of {wl.name} (W={wl.W}, K={wl.K}) on its first {n_cols} of "
              f"{wl.N} parameter columns, fp64, single thread")
    line = {
        "impl": "reference", "metric": METRIC, "value": round(value, 4), "unit": "GB/s",
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(1e3 * total / args.steps, 3), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": f"synthetic (seeded; {wl.data})",
        "paper_context": PAPER_CONTEXT,
        "config": arm_config(wl, args),
        "cpu_baseline": {"value": round(value, 4), "unit": "GB/s", "cores": 1, "kind": "oracle",
                         "sample": sample, "host_cpus": os.cpu_count()},
        "e2e": {"value": round(value, 4), "unit": "GB/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def resident_bytes(wl) -> int:
    """Device bytes the benchmark keeps resident: the state arrays, K gradient
    buffers, anchor and velocity."""
    return 4 * wl.state_arrays * wl.W * wl.N + wl.K * wl.grad_bytes * wl.W * wl.N + 8 * wl.N


def needs_l2_flush(wl) -> bool:
    """Whether the workload's resident data could stay in L2 between steps."""
    return resident_bytes(wl) <= 4 * L2_BYTES


def workload_config(wl) -> dict:
    res = resident_bytes(wl)
    if not needs_l2_flush(wl):
        l2 = (f"inputs larger than L2: {res / 1e9:.2f} GB resident, "
              f"{cycle_bytes(wl.W, wl.N, wl.K, wl.grad_bytes, 'cpdp', wl.state_arrays) / 1e9:.2f} GB streamed per step vs "
              f"{L2_BYTES / 1e6:.0f} MB L2, no flush needed")
    else:
        l2 = (f"working set {res / 1e6:.0f} MB vs {L2_BYTES / 1e6:.0f} MB L2: the L2 is scrubbed (a "
              f"{2 * L2_BYTES / 1e6:.0f} MB write) before every timed K-cycle and every timed launch, outside "
              f"their CUDA events; the step time is the sum of the per-K-cycle event times")
    return {"workload": wl.name, "W": wl.W, "N": wl.N, "num_tensors": len(wl.tensors), "K": wl.K,
            "steps_per_epoch": wl.T, "grad_dtype": wl.grad_dtype,
            "step": f"one K-cycle: {wl.K - 1} local steps + 1 reconcile",
            "optimizer": wl.optimizer,
            "bytes_per_step": cycle_bytes(wl.W, wl.N, wl.K, wl.grad_bytes, "cpdp", wl.state_arrays), "l2": l2,
            "parallelism": "replicas"}


def arm_config(wl, args) -> dict:
    """The `config` both arms print (the GPU arm and the reference arm), so the
    two lines name the same workload and options."""
    return {**workload_config(wl), "method": args.method, "state_reconcile": args.state_reconcile,
            "programmatic_launch": not args.no_pdl, "reconcile_staging": args.reconcile_staging,
            "reconcile_shuffle": args.reconcile_shuffle,
            "bytes_per_step": cycle_bytes(wl.W, wl.N, wl.K, wl.grad_bytes, args.method, wl.state_arrays)}


# ---------------------------------------------------------------------------
# GPU arm
# ---------------------------------------------------------------------------
def run_native(args) -> None:
    import torch
    import torch.distributed as dist

    rank, world, local_rank = dist_env()
    if world > 1 and not dist.is_initialized():
        dist.init_process_group("nccl", device_id=torch.device("cuda", local_rank))
    device = torch.device("cuda", local_rank)
    torch.cuda.set_device(device)

    from paper_2607_21224_gb300 import build, workloads as wls
    from paper_2607_21224_gb300.state import CPDPState

    build.build_library()  # no-op when up to date
    wl = wls.get(args.workload)
    W, N, K = wl.W, wl.N, wl.K
    seed = args.seed + 1000 * rank
    stream = torch.cuda.Stream(device)

    theta0 = wls.make_theta0(wl, seed, device)
    grads = [wls.make_grads(wl, t, seed, device) for t in range(1, K + 1)]
    st = CPDPState(W, N, wl.offsets, device=device, **wl.hyper())
    if wl.optimizer == "adamw":
        st.set_adamw(wl.adam_beta1, wl.adam_beta2, wl.adam_eps)
    with torch.cuda.stream(stream):
        st.init_params(theta0)
    stream.synchronize()

    st.set_method(args.method)
    st.set_state_reconcile(args.state_reconcile)
    st.set_pdl(not args.no_pdl)
    st.set_reconcile_staging(args.reconcile_staging)
    st.set_reconcile_shuffle(args.reconcile_shuffle)
    S = wl.state_arrays

    flush = needs_l2_flush(wl)
    scrub = torch.empty(2 * L2_BYTES // 4, dtype=torch.float32, device=device) if flush else None

    def scrub_l2(i: int) -> None:
        with torch.cuda.stream(stream):
            scrub.fill_(float(i % 7))

    def cycle(c: int, ev=None):
        base = (c * K) % wl.T
        for k in range(K):
            t = base + k + 1
            if ev is not None:
                if flush:
                    scrub_l2(k)
                e0 = torch.cuda.Event(enable_timing=True)
                e0.record(stream)
            synced = st.step(grads[k], t, wl.T, stream=stream)
            if ev is not None:
                e1 = torch.cuda.Event(enable_timing=True)
                e1.record(stream)
                ev.append((e0, e1, synced))

    gpu_id = None
    try:
        gpu_id = "GPU-" + str(torch.cuda.get_device_properties(device).uuid)
    except Exception:
        gpu_id = None
    clocks = ClockSampler(gpu_id) if rank == 0 else None

    for c in range(args.warmup):
        cycle(c)
    torch.cuda.synchronize(device)

    # timed region: exactly args.steps K-cycles, launched back to back (no
    # event between launches, which would stop programmatic launch overlap)
    barrier(device)
    torch.cuda.synchronize(device)
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    per_cycle = []
    if clocks:
        clocks.mark_start()
    start.record(stream)
    for c in range(args.steps):
        if flush:  # L2-sized data: scrub, then time the K-cycle on its own
            scrub_l2(c)
            c0, c1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            c0.record(stream)
            cycle(args.warmup + c)
            c1.record(stream)
            per_cycle.append((c0, c1))
        else:
            cycle(args.warmup + c)
    end.record(stream)
    torch.cuda.synchronize(device)
    if clocks:
        clocks.mark_end()
    barrier(device)
    elapsed_ms = sum(a.elapsed_time(b) for a, b in per_cycle) if flush else start.elapsed_time(end)
    elapsed_ms = max_over_ranks(elapsed_ms, device)

    # per-kernel launch durations: the same K-cycles again, right after, with
    # CUDA events around each launch on the launching stream
    kev: list = []
    for c in range(args.steps):
        cycle(args.warmup + args.steps + c, kev)
    torch.cuda.synchronize(device)
    local_ms, recon_ms = [], []
    for e0, e1, synced in kev:
        (recon_ms if synced else local_ms).append(e0.elapsed_time(e1))

    # end to end through the public API from pinned host memory
    e2e = None if args.no_e2e else run_e2e(args, wl, st, device, stream, seed)
    graph = run_graph(args, wl, st, grads, device, stream) if args.graph else None

    clock_info = clocks.stop() if clocks else None
    timeouts = st.wait_timeouts()
    recon_kernel = st.reconcile_kernel()
    # the floors (of small, L2-scrubbed workloads, and of any workload with
    # --floor): run last, they overwrite the state
    floor = (run_floor(args, wl, st, grads, device, stream, scrub_l2 if flush else None)
             if flush or args.floor else None)
    st.close()
    if rank != 0:
        return

    step_bytes = cycle_bytes(W, N, K, wl.grad_bytes, args.method, S)
    value = world * step_bytes * args.steps / (elapsed_ms / 1e3) / 1e9
    peak, peak_kind = measured_peak()
    lb, rb = local_step_bytes(W, N, wl.grad_bytes, S), sync_bytes(W, N, wl.grad_bytes, args.method, S)
    l_avg, r_avg = statistics.fmean(local_ms) if local_ms else None, statistics.fmean(recon_ms)

    def roof(nbytes, avg_ms, kernel):
        ach = nbytes / (avg_ms / 1e3) / 1e9
        # the committed ncu traffic is per launch of the CPDP method's SGD kernels at the benchmark's
        # default (ResNet-50, W=8) size: other workloads and variants report none
        tr = (ncu_traffic(kernel) if wl.name == DEFAULT_WORKLOAD and args.method == "cpdp"
              and wl.optimizer == "sgd" and not args.state_reconcile else None)
        return {"bound": "hbm", "achieved": round(ach, 1), "peak": peak, "unit": "GB/s",
                "frac": round(ach / peak, 4), "traffic": tr, "kernel": kernel,
                "algorithmic_bytes_per_launch": nbytes, "avg_launch_ms": round(avg_ms, 4),
                "launches": len(local_ms) if kernel.startswith("local") else len(recon_ms),
                "peak_source": f"{peak_kind} (MEASURED_PEAKS.json hbm_gbs)" if peak_kind == "measured"
                else "fallback 6.8 TB/s", "frac_of_nominal_8TBs": round(ach / NOMINAL_HBM_GBS, 4),
                "timing": ("CUDA events around each launch on the launching stream, over a second pass of the "
                           "same --steps K-cycles run right after the timed region (the events end launch "
                           "overlap at each boundary, so these durations include each launch's ramp)")}

    rl = roof(lb, l_avg, "local_step_kernel") if l_avg else None
    rr = roof(rb, r_avg, recon_kernel)
    dominant = rl if (rl and l_avg * len(local_ms) >= r_avg * len(recon_ms)) else rr
    other = rr if dominant is rl else rl

    line = {
        "metric": METRIC, "value": round(value, 1), "unit": "GB/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(elapsed_ms / args.steps, 4),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
        "data": f"synthetic (seeded; {wl.data})", "paper_context": PAPER_CONTEXT,
        "config": arm_config(wl, args),
        "pct_of_nominal_8TBs": round(100 * value / world / NOMINAL_HBM_GBS, 2),
        "pct_of_measured_peak": round(100 * value / world / peak, 2),
        "params_per_s": round(world * W * N * K * args.steps / (elapsed_ms / 1e3), 1),
        "roofline": dominant, "roofline_other": other,
        "gpu_launches": K * args.steps,
        "e2e": e2e, "clocks": clock_info, "kernel_wait_timeouts": timeouts,
    }
    if floor is not None:
        floor["frac_of_stream_floor"] = round(value / world / floor["stream_GB_s"], 4)
        line["floor"] = floor
        for r in (rl, rr):
            if r is not None:
                f = floor["stream_local_GB_s" if r is rl else "stream_reconcile_GB_s"]
                r["floor_GB_s"], r["frac_of_floor"] = f, round(r["achieved"] / f, 4)
        if rr is not None:
            f = floor["columns_reconcile_GB_s"]
            rr["column_walk_GB_s"], rr["frac_of_column_walk"] = f, round(rr["achieved"] / f, 4)
    if graph is not None:
        line["graph_replay"] = graph
    if not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(wl, args.cpu_baseline_seconds)
    print(json.dumps(line), flush=True)


def floor_rows(wl, st, g, kind: str):
    """The rows (float32 inputs, bf16 inputs, outputs, columns) one launch of
    `kind` ("local" or "sync", CPDP) touches, for the plain streaming floor
    kernel: the same buffers, in place, the gradient rows among the bf16
    inputs where the gradients are bf16."""
    states = [st.params, st.mom] + ([st.exp_avg_sq] if wl.state_arrays == 3 else [])
    half = wl.grad_dtype == "bf16"
    if kind == "local":
        flat = [x.view(-1) for x in states]
        grad = [g.view(-1)]
        return flat + ([] if half else grad), grad if half else [], flat, wl.W * wl.N
    rows = [x[i] for x in states for i in range(wl.W)]
    grad = [g[i] for i in range(wl.W)]
    return (([] if half else grad) + rows + [st.anchor, st.slow_v], grad if half else [],
            rows + [st.anchor, st.slow_v], wl.N)


# the compiled shapes of the column-walk floor: (rows per chunk, resident blocks per SM)
COLUMN_FLOOR_SHAPES = ((2, 4), (3, 3), (4, 2))


def run_floor(args, wl, st, grads, device, stream, scrub_l2) -> dict | None:
    """What the K-cycle would take if only launches and data movement cost
    time, under the same L2 scrub as the timed region (none for data larger
    than L2): (1) K empty launches; (2) K launches of a plain streaming kernel
    (cpdp_floor_stream) that move the same bytes with the same read:write mix
    over the same buffers, in place, with no optimizer arithmetic, walking a
    reconcile's rows column by column as the reconcile does; the better of two
    grids (one group of 4 columns per thread, or 8 blocks per SM looping).
    Timed K-cycle by K-cycle like the timed region, and launch by launch with
    CUDA events around each launch like the kernels' roofline durations (the
    local and reconcile floors). CPDP only, and N a multiple of 4 (the kernel
    moves groups of 4 columns, and its rows must start 16 bytes apart);
    overwrites the state."""
    if args.method != "cpdp" or wl.N % 4:
        return None
    import torch
    from paper_2607_21224_gb300 import cpdp
    K = wl.K
    sms = torch.cuda.get_device_properties(device).multi_processor_count
    s = stream.cuda_stream
    shapes = {}
    for kind, g in (("local", grads[0]), ("sync", grads[-1])):
        ins, ins16, outs, n = floor_rows(wl, st, g, kind)
        shapes[kind] = (cpdp.FloorRows(ins, outs, ins16), n)

    def timed(launch_cycle) -> float:
        evs = []
        for c in range(args.warmup + args.steps):
            if scrub_l2 is not None:
                scrub_l2(c)
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            launch_cycle()
            e1.record(stream)
            if c >= args.warmup:
                evs.append((e0, e1))
        torch.cuda.synchronize(device)
        return sum(a.elapsed_time(b) for a, b in evs) / args.steps

    def stream_cycle(grid):
        def go():
            for k in range(K):
                rows, n = shapes["sync" if k == K - 1 else "local"]
                cpdp.cpdp_floor_stream(rows, None, n, grid, s)
        return go

    def one_launch(kind, grid):
        rows, n = shapes[kind]
        return lambda: cpdp.cpdp_floor_stream(rows, None, n, grid, s)

    def columns_launch(rows, blocks):
        sq = st.exp_avg_sq if wl.state_arrays == 3 else None
        dt = cpdp.CPDP_BF16 if wl.grad_dtype == "bf16" else cpdp.CPDP_F32
        return lambda: cpdp.cpdp_floor_columns(st.params, st.mom, sq, grads[-1], dt, st.anchor, st.slow_v, wl.W, wl.N,
                                               rows, blocks, s)

    best = min((timed(stream_cycle(g)), g) for g in (0, 8 * sms))
    empty_grid = max(1, (wl.W * wl.N // 4 + 511) // 512)  # the local step's grid
    empty_ms = timed(lambda: [cpdp.cpdp_floor_empty(empty_grid, s) for _ in range(K)])
    nbytes = cycle_bytes(wl.W, wl.N, K, wl.grad_bytes, "cpdp", wl.state_arrays)
    per_launch = {kind: min(timed(one_launch(kind, g)) for g in (0, 8 * sms)) for kind in ("local", "sync")}
    columns = min((timed(columns_launch(r, b)), r, b) for r, b in COLUMN_FLOOR_SHAPES)
    lb = local_step_bytes(wl.W, wl.N, wl.grad_bytes, wl.state_arrays)
    rb = sync_bytes(wl.W, wl.N, wl.grad_bytes, "cpdp", wl.state_arrays)
    return {"stream_ms_per_step": round(best[0], 5), "stream_GB_s": round(nbytes / (best[0] / 1e3) / 1e9, 1),
            "stream_grid": "one group of 4 columns per thread" if best[1] == 0 else f"{best[1]} blocks (8 per SM)",
            "stream_local_GB_s": round(lb / (per_launch["local"] / 1e3) / 1e9, 1),
            "stream_reconcile_GB_s": round(rb / (per_launch["sync"] / 1e3) / 1e9, 1),
            "columns_reconcile_GB_s": round(rb / (columns[0] / 1e3) / 1e9, 1),
            "columns_shape": f"{columns[1]}-row chunks, {columns[2]} blocks per SM",
            "empty_ms_per_step": round(empty_ms, 5), "empty_grid": empty_grid,
            "scrub": "L2 scrubbed before each timed K-cycle and launch" if scrub_l2 is not None
            else "none: the data is larger than L2",
            "how": ("K launches per K-cycle, timed K-cycle by K-cycle over --steps K-cycles after --warmup, and "
                    "single launches of each kind timed the same way (the local and reconcile floors): plain "
                    "streaming kernels moving each launch's bytes with its read:write mix in place over the same "
                    "buffers (no optimizer arithmetic; a reconcile's rows walked column by column), and empty "
                    "kernels; columns_reconcile: the reconcile's rows read and written chunk by chunk in its own "
                    "order with no sums and no dependency between rows (cpdp_floor_columns, best of its shapes)")}


def sweep_cpu_baseline(wl, target_s: float) -> dict:
    """The oracle on a sweep point, timed on an instance of the same point with
    at most 2^18 columns (the sweep's single flat tensor has independent,
    identically distributed columns at any N, and every column is an
    independent problem), with seconds scaled to the full N."""
    from paper_2607_21224_gb300 import workloads as wls
    n = min(wl.N, 1 << 18)
    cb = cpu_baseline(wls.sweep_point(n, wl.W, wl.K), target_s)
    cycle_s = cycle_bytes(wl.W, wl.N, wl.K, wl.grad_bytes) / (cb["value"] * 1e9)
    cb["sample"] += f"; an instance of this point with {n} of its {wl.N} columns, seconds scaled to N"
    cb["s_per_cycle_full_N"] = round(cycle_s, 4)
    for v in cb.get("per_step", {}).values():
        v["s_full_N"] = round(v["s_full_N"] * wl.N / n, 4)
    return cb


def run_sweep(args) -> None:
    """Roofline sweep: one JSON line per (N, W, K) point. Every launch of a
    K-cycle is timed with its own CUDA events, after about 0.25 s of warm-up
    cycles and over about 1 s of timed ones (10-200 and 20-200 cycles); the
    cycle time is (K-1) times the median local step plus the median reconcile. Gradient buffers alternate
    between two resident ones. When one launch's data (12 W N bytes) is under
    4x the L2 size, the L2 is scrubbed (a 2x-L2 write) before every launch,
    outside its events, so the point measures HBM rather than L2; each line
    says which."""
    import torch
    from paper_2607_21224_gb300 import build, workloads as wls
    from paper_2607_21224_gb300.state import CPDPState

    build.build_library()
    device = torch.device("cuda", 0)
    stream = torch.cuda.Stream(device)
    scrub = torch.empty(2 * L2_BYTES // 4, dtype=torch.float32, device=device)
    peak, _ = measured_peak()
    pts = wls.sweep_points()
    if args.sweep_max_n:
        pts = [p for p in pts if p[0] <= args.sweep_max_n]
    for N, W, K in pts:
        wl = wls.sweep_point(N, W, K)
        theta0 = wls.make_theta0(wl, args.seed, device)
        grads = [wls.make_grads(wl, t, args.seed, device) for t in range(1, min(K, 2) + 1)]
        st = CPDPState(W, N, wl.offsets, device=device, **wl.hyper())
        with torch.cuda.stream(stream):
            st.init_params(theta0)
        nbytes = cycle_bytes(W, N, K, 4)
        flush = 12 * W * N < 4 * L2_BYTES
        # warm up for about 0.25 s and time about 1 s of K-cycles (the first tens of ms after
        # allocating and filling tens of GB ran up to 4 % slow)
        t_est = nbytes / 7.0e12
        warm = int(min(200, max(10, 0.25 / t_est)))
        reps = int(min(200, max(20, 1.0 / t_est)))
        loc_ev, rec_ev = [], []
        for r in range(warm + reps):
            for k in range(K):
                if flush:
                    with torch.cuda.stream(stream):
                        scrub.fill_(float(r + k))
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                e0.record(stream)
                st.step(grads[k % len(grads)], k + 1, K, stream=stream)
                e1.record(stream)
                if r >= warm:
                    (rec_ev if k == K - 1 else loc_ev).append((e0, e1))
        torch.cuda.synchronize(device)
        rec_ms = statistics.median(a.elapsed_time(b) for a, b in rec_ev)
        loc_ms = statistics.median(a.elapsed_time(b) for a, b in loc_ev) if loc_ev else 0.0
        ms = (K - 1) * loc_ms + rec_ms
        gbs = nbytes / (ms / 1e3) / 1e9
        floor = sweep_floor(wl, st, grads, stream, scrub, reps) if flush else None
        line = {"sweep_point": wl.name, "N": N, "W": W, "K": K, "GB_s": round(gbs, 1),
                "ms_per_cycle": round(ms, 4), "frac_of_measured_peak": round(gbs / peak, 4),
                "pct_of_nominal_8TBs": round(100 * gbs / NOMINAL_HBM_GBS, 2),
                "reconcile_GB_s": round(reconcile_bytes(W, N, 4) / (rec_ms / 1e3) / 1e9, 1),
                "local_GB_s": round(local_step_bytes(W, N, 4) / (loc_ms / 1e3) / 1e9, 1) if loc_ev else None,
                "warmup": warm, "reps": reps,
                "l2": "scrubbed before every launch" if flush else "inputs larger than L2"}
        if floor is not None:
            floor["frac_of_stream_floor"] = round(floor["stream_ms_per_cycle"] / ms, 4)
            line["floor"] = floor
        if not args.no_cpu_baseline:
            line["cpu_baseline"] = sweep_cpu_baseline(wl, args.sweep_cpu_seconds)
        print(json.dumps(line), flush=True)
        st.close()
        del theta0, grads
        torch.cuda.empty_cache()


def sweep_floor(wl, st, grads, stream, scrub, reps: int) -> dict:
    """A sweep point's floors, each launch timed on its own after an L2 scrub
    like the point's own launches (median of `reps`): the plain streaming
    kernel moving one local step's and one reconcile's bytes with their
    read:write mix in place over the same buffers (the better of two grids),
    and an empty launch. Overwrites the state."""
    import torch
    from paper_2607_21224_gb300 import cpdp
    s = stream.cuda_stream
    sms = torch.cuda.get_device_properties(stream.device).multi_processor_count

    def median_ms(go) -> float:
        evs = []
        for r in range(reps + 3):
            with torch.cuda.stream(stream):
                scrub.fill_(float(r))
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            go()
            e1.record(stream)
            if r >= 3:
                evs.append((e0, e1))
        torch.cuda.synchronize(stream.device)
        return statistics.median(a.elapsed_time(b) for a, b in evs)

    out = {}
    for kind in ("local", "sync"):
        ins, ins16, outs, n = floor_rows(wl, st, grads[0], kind)
        rows = cpdp.FloorRows(ins, outs, ins16)
        out[kind] = min(median_ms(lambda: cpdp.cpdp_floor_stream(rows, None, n, g, s)) for g in (0, 8 * sms))
    empty = median_ms(lambda: cpdp.cpdp_floor_empty(max(1, (wl.W * wl.N // 4 + 511) // 512), s))
    cyc = (wl.K - 1) * out["local"] + out["sync"]
    return {"stream_ms_per_cycle": round(cyc, 5),
            "stream_GB_s": round(cycle_bytes(wl.W, wl.N, wl.K, 4) / (cyc / 1e3) / 1e9, 1),
            "stream_local_GB_s": round(local_step_bytes(wl.W, wl.N, 4) / (out["local"] / 1e3) / 1e9, 1),
            "stream_reconcile_GB_s": round(reconcile_bytes(wl.W, wl.N, 4) / (out["sync"] / 1e3) / 1e9, 1),
            "empty_launch_ms": round(empty, 5)}


def run_graph(args, wl, st, grads, device, stream) -> dict:
    """The same K-cycle captured once into a CUDA graph and replayed per step
    (removes per-launch host overhead; matters for small N)."""
    import torch
    K = wl.K
    if wl.optimizer == "adamw":
        return {"unavailable": "AdamW steps are refused under stream capture: the bias correction moves with the step "
                               "count, so a replay would repeat a stale step"}
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        for k in range(K):
            st.step(grads[k], k + 1, K, stream=stream)
    for _ in range(args.warmup):
        g.replay()
    torch.cuda.synchronize(device)
    flush = needs_l2_flush(wl)
    scrub = torch.empty(2 * L2_BYTES // 4, dtype=torch.float32, device=device) if flush else None
    s, e = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    per_replay = []
    with torch.cuda.stream(stream):
        s.record(stream)
        for i in range(args.steps):
            if flush:  # L2-sized data: scrub, then time the replay on its own
                scrub.fill_(float(i % 7))
                r0, r1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                r0.record(stream)
                g.replay()
                r1.record(stream)
                per_replay.append((r0, r1))
            else:
                g.replay()
        e.record(stream)
    torch.cuda.synchronize(device)
    ms = sum(a.elapsed_time(b) for a, b in per_replay) if flush else s.elapsed_time(e)
    ms = max_over_ranks(ms, device)
    _, world, _ = dist_env()
    nbytes = world * cycle_bytes(wl.W, wl.N, K, wl.grad_bytes, args.method, wl.state_arrays) * args.steps
    return {"value": round(nbytes / (ms / 1e3) / 1e9, 1), "unit": "GB/s", "ms_per_step": round(ms / args.steps, 5),
            "steps": args.steps, "how": "one K-cycle captured into a CUDA graph, replayed once per step"}


def run_e2e(args, wl, st, device, stream, seed) -> dict:
    """The same metric end to end: every step copies its K gradient buffers
    from pinned host memory to the device, runs the K-cycle through the public
    API, and reads the reconciled model (theta_ref) back to pinned host memory.
    The copies run on their own stream, overlapped with earlier steps' kernels
    (paper_2607_21224_gb300.pipeline.HostGradientPipeline)."""
    import torch
    from paper_2607_21224_gb300 import workloads as wls
    from paper_2607_21224_gb300.pipeline import HostGradientPipeline
    K = wl.K
    host = [wls.make_grads(wl, t, seed, "cpu").pin_memory() for t in range(1, K + 1)]
    feed = HostGradientPipeline(st, dtype=wl.torch_grad_dtype)
    out = torch.empty(wl.N, dtype=torch.float32).pin_memory()
    h2d = sum(h.numel() * h.element_size() for h in host)
    d2h = out.numel() * out.element_size()
    steps = max(1, min(args.steps, args.e2e_steps))

    def one(c):
        base = (c * K) % wl.T
        for k in range(K):
            feed.step(host[k], base + k + 1, wl.T, stream=stream)
        with torch.cuda.stream(stream):
            out.copy_(st.anchor, non_blocking=True)

    for c in range(min(args.warmup, 3)):
        one(c)
    torch.cuda.synchronize(device)
    link = host_link_ceiling(host, device)
    # an event after each step's read-back (already a stream-ordered copy between
    # K-cycles) also gives each step's own time
    marks = [torch.cuda.Event(enable_timing=True) for _ in range(steps + 1)]
    marks[0].record(stream)
    for c in range(steps):
        one(c)
        marks[c + 1].record(stream)
    torch.cuda.synchronize(device)
    ms = max_over_ranks(marks[0].elapsed_time(marks[-1]), device)
    step_ms = [marks[c].elapsed_time(marks[c + 1]) for c in range(steps)]
    # the link rate moves from second to second on this machine: measured again right after
    after = host_link_ceiling(host, device)
    best = max(link["h2d_GB_s"], after["h2d_GB_s"])
    _, world, _ = dist_env()
    nbytes = world * cycle_bytes(wl.W, wl.N, K, wl.grad_bytes, args.method, wl.state_arrays) * steps
    h2d_rate = h2d * steps / (ms / 1e3) / 1e9
    # the e2e figure if the gradients' host-to-device copies were the only limit
    link_bound = nbytes / steps / (h2d / (best * 1e9)) / 1e9
    return {"value": round(nbytes / (ms / 1e3) / 1e9, 1), "unit": "GB/s", "h2d_bytes_per_step": h2d,
            "d2h_bytes_per_step": d2h, "steps": steps, "ms_per_step": round(ms / steps, 3),
            "h2d_GB_s": round(h2d_rate, 1),
            "ms_per_step_median": round(statistics.median(step_ms), 3),
            "ms_per_step_max": round(max(step_ms), 3),
            "value_at_median_step": round(nbytes / steps / (statistics.median(step_ms) / 1e3) / 1e9, 1),
            "link_h2d_GB_s": best, "frac_of_link": round(h2d_rate / best, 4),
            "link_h2d_before_GB_s": link["h2d_GB_s"], "link_h2d_after_GB_s": after["h2d_GB_s"],
            "link_bound_value": round(link_bound, 1),
            "link_how": link["how"] + "; measured again right after it; link_h2d_GB_s is the higher of the two",
            "path": "cpdp_step_host x K from pinned host buffers (the library copies on its own stream into 2 "
                    "rotating staging buffers, overlapped with the kernels), anchor -> pinned host"}


def host_link_ceiling(host: list, device, reps: int = 3) -> dict:
    """The host link's rate for one step's gradients, measured in the same run
    just before the e2e timed region: plain pinned host-to-device copies of
    the step's K gradient buffers in turn (the bytes and host buffers the e2e
    step copies) on a stream of its own, nothing else running, timed with CUDA
    events; the median over `reps` steps' worth."""
    import torch
    dst = torch.empty(host[0].shape, dtype=host[0].dtype, device=device)
    s = torch.cuda.Stream(device)
    with torch.cuda.stream(s):
        for h in host:  # warm-up
            dst.copy_(h, non_blocking=True)
        evs = []
        for _ in range(reps):
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(s)
            for h in host:
                dst.copy_(h, non_blocking=True)
            b.record(s)
            evs.append((a, b))
    s.synchronize()
    ms = statistics.median(a.elapsed_time(b) for a, b in evs)
    nbytes = sum(h.numel() * h.element_size() for h in host)
    del dst
    return {"h2d_GB_s": round(nbytes / (ms / 1e3) / 1e9, 1),
            "how": (f"pinned host-to-device copies of one step's {len(host)} gradient buffers ({nbytes} B) on a "
                    f"stream of their own, nothing else running, median of {reps} steps' worth, CUDA events, "
                    f"same run, just before the e2e timed region")}


def main(argv=None) -> None:
    ap = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=400)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=("native", "reference"), default="native")
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD)
    ap.add_argument("--seed", type=int, default=42)
    ap.add_argument("--e2e-steps", type=int, default=40)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true", help="skip the end-to-end leg (profiling runs)")
    ap.add_argument("--sweep", action="store_true", help="run the roofline sweep instead (one line per point)")
    ap.add_argument("--graph", action="store_true", help="also time the K-cycle replayed from a CUDA graph")
    ap.add_argument("--floor", action="store_true",
                    help="also time the plain streaming floors for data larger than L2 (always timed for L2-sized "
                         "data; CPDP only; overwrites the state after the timed region)")
    ap.add_argument("--method", choices=("cpdp", "localsgd", "ddp"), default="cpdp",
                    help="synchronization method (the paper's method or one of its baselines)")
    ap.add_argument("--state-reconcile", action="store_true",
                    help="also average the optimizer states at every synchronization")
    ap.add_argument("--sweep-max-n", type=int, default=0, help="limit the sweep to N <= this")
    ap.add_argument("--no-pdl", action="store_true",
                    help="launch with plain stream order instead of programmatic dependent launch")
    ap.add_argument("--reconcile-shuffle", action="store_true",
                    help="the reconcile with worker rows split across a warp's lanes and warp-shuffle sums, the "
                         "measured alternative to per-thread register sums")
    ap.add_argument("--reconcile-staging", type=int, default=0, metavar="STAGES",
                    help="0: the reconcile loads its rows directly (default); 2-8: rows staged through that many "
                         "shared-memory slots by bulk copies (TMA), the measured alternative")
    ap.add_argument("--cpu-baseline-seconds", type=float, default=15.0)
    ap.add_argument("--sweep-cpu-seconds", type=float, default=0.6,
                    help="oracle seconds per sweep point (--no-cpu-baseline skips them)")
    ap.add_argument("--ref-step-seconds", type=float, default=1.0)
    ap.add_argument("--ref-total-seconds", type=float, default=120.0,
                    help="reference arm: about this much oracle time over warm-up and timed steps together")
    args = ap.parse_args(argv)
    args.warmup = max(args.warmup, 3)  # at least 3 untimed warm-up steps
    if args.impl == "reference":
        run_reference(args)
    elif args.sweep:
        run_sweep(args)
    else:
        run_native(args)


if __name__ == "__main__":
    main()
