#!/usr/bin/env python3
"""Benchmark of the SS2D selective-scan hot path (full and VMeanba channel-mean).

One step = one SS2D pass over one synthetic batch, both paths:
    cross-scan x -> xs;  full scan xs -> y_full;  channel-mean scan xs -> y_mean;
    cross-merge y_full -> out_full;  cross-merge y_mean -> out_mean
all through the C ABI of libvmb.  The default workload is the largest
single-GPU configuration: batch 128, D=256, N=16, 56x56 maps, fp32, channel
noise 0.05 (5.1 GB of scan operands per call, far larger than L2, so the
steps run back to back without an L2 flush; smaller workloads given with
--workload flush L2 before every step).

Prints ONE JSON line (rank 0).  `value` is the step's algorithmic HBM bytes
(sum over its five kernels) per second of device time, with inputs resident
in HBM; `e2e` is the same metric with the inputs copied from pinned host
memory and both outputs copied back inside the timed region (every step; the
copies of one step overlap the kernels of its neighbours).  `configs` times
every workload of the scan's configuration list (inputs drawn on the device
with the same recipe), kernel by kernel.  `--impl reference` times the fp64
CPU oracle on a one-batch-element slice of the workload instead.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference] [--workload NAME]
"""
from __future__ import annotations

import argparse
import ctypes
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import workloads  # noqa: E402

METRIC = ("selective-scan HBM GB/s and (B·K·D·L)/s, full vs channel-mean, "
          "% of GB300 HBM peak")
DEFAULT_WORKLOAD = "batch128_d256_n16_56x56_sigma0.05_f32"
FALLBACK_HBM_GBS = 6800.0
KERNELS = ["cross_scan", "full_scan", "mean_scan", "cross_merge_full", "cross_merge_mean"]
SOURCES = {"full_scan": "full_scan.cu", "mean_scan": "mean_scan.cu", "cross_scan": "cross_scan_merge.cu",
           "cross_merge_full": "cross_scan_merge.cu", "cross_merge_mean": "cross_scan_merge.cu"}


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=250)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD, choices=sorted(workloads.WORKLOADS))
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-paper-style", action="store_true",
                    help="skip the timing of the paper's split (discretise, then scan alone)")
    ap.add_argument("--no-grouped", action="store_true", help="skip the timing of the grouped basis")
    ap.add_argument("--no-selection", action="store_true", help="skip the timing of the Eq. 6 selection functions")
    ap.add_argument("--no-backward", action="store_true", help="skip the timing of the mean scan's backward")
    ap.add_argument("--e2e-steps", type=int, default=20)
    ap.add_argument("--no-configs", action="store_true", help="skip the per-workload timing table")
    ap.add_argument("--extra-steps", type=int, default=20,
                    help="timed calls of each extra measurement (fused path, grouped, selection, paper split)")
    ap.add_argument("--batch", type=int, default=None,
                    help="override the workload's batch size (smaller captures for profiling)")
    return ap.parse_args()


def kernel_bytes(wl: workloads.Workload) -> dict:
    return {"cross_scan": wl.csm_bytes(), "full_scan": wl.scan_bytes(), "mean_scan": wl.scan_bytes(),
            "cross_merge_full": wl.csm_bytes(), "cross_merge_mean": wl.csm_bytes()}


def measured_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


def src_hash(kernel: str) -> str:
    p = os.path.join(ROOT, "paper_2412_16602_gb300", "csrc", SOURCES[kernel])
    with open(p, "rb") as f:
        return hashlib.sha256(f.read()).hexdigest()[:16]


def committed_traffic(kernel: str, workload: str):
    """DRAM bytes per launch from the committed ncu summary, if it was taken on
    the current source of that kernel (else None)."""
    path = os.path.join(ROOT, "profiles", "dram_traffic.txt")
    if not os.path.exists(path):
        return None
    want = src_hash(kernel)
    for line in open(path):
        if line.startswith("#") or not line.strip():
            continue
        kv = dict(tok.split("=", 1) for tok in line.split() if "=" in tok)
        if kv.get("kernel") == kernel and kv.get("workload") == workload and kv.get("src_sha") == want:
            return float(kv["dram_bytes_per_launch"])
    return None


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled while the timed region runs."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None
        return self

    def __exit__(self, *a):
        self.out = ""
        if self.proc is not None:
            time.sleep(0.25)
            self.proc.terminate()
            try:
                self.out, _ = self.proc.communicate(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        rows = []
        for line in (self.out or "").splitlines():
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                rows.append((float(parts[1]), float(parts[2]), parts[5:9]))
            except ValueError:
                continue
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unavailable"], "samples": 0}
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for _, _, r in rows for i, v in enumerate(r) if v.lower() == "active"})
        return {"sm_mhz": statistics.median(r[0] for r in rows), "sm_max_mhz": max(r[1] for r in rows),
                "reasons": reasons, "samples": len(rows)}


# ----------------------------------------------------------------------------- ranks


def rank_seed(wl: workloads.Workload, rank: int) -> int:
    """Every rank draws its own batch (weak scaling: per-rank work is fixed)."""
    return wl.seed + 7919 * rank


def max_over_ranks(values, world: int, device=None):
    """Element-wise max of a list of floats over all ranks (the step time of the
    slowest rank); identity on one rank.  Only timings cross ranks: the path
    itself has no exchange step."""
    if world <= 1:
        return list(values)
    import torch
    t = torch.tensor(list(values), dtype=torch.float64, device=device)
    torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
    return [float(v) for v in t.tolist()]


def job_throughput(step_bytes: int, world: int, max_ms_per_step: float) -> float:
    """Whole-job GB/s: every rank moves step_bytes per step; the job takes as
    long as its slowest rank."""
    return world * step_bytes / (max_ms_per_step / 1e3) / 1e9


# ----------------------------------------------------------------------------- CPU oracle


def oracle_step(inp, nthreads):
    import oracle
    oracle.ss2d_full(inp, nthreads=nthreads)
    oracle.ss2d_mean(inp, nthreads=nthreads)


def time_oracle(inp, target_s=10.0, max_steps=None):
    """Run whole oracle steps until about target_s seconds have passed."""
    import oracle
    nth = oracle.default_threads()
    times = []
    t_end = time.perf_counter() + target_s
    while True:
        t0 = time.perf_counter()
        oracle_step(inp, nth)
        times.append(time.perf_counter() - t0)
        if time.perf_counter() >= t_end or (max_steps and len(times) >= max_steps):
            break
    return times, nth


# ----------------------------------------------------------------------------- GPU arm


class Step:
    """Pre-marshalled C-ABI calls of one SS2D step (pointers, shapes, stream)."""

    def __init__(self, vmb, wl, g, outs, stream_handle):
        self.vmb = vmb
        lib = vmb.lib
        self.lib = lib
        B, D, N, H, W = wl.B, wl.D, wl.N, wl.H, wl.W
        K = 4
        dt = vmb.VMB_BF16 if wl.dtype == "bf16" else vmb.VMB_F32
        P = lambda t: ctypes.c_void_p(t.data_ptr())  # noqa: E731
        s = ctypes.c_void_p(stream_handle)
        fl = vmb.VMB_FLAG_SOFTPLUS
        wsf = outs["ws_full"]
        wsm = outs["ws_mean"]
        self.calls = [
            ("cross_scan", lib.vmb_cross_scan, (P(g["x"]), P(outs["xs"]), B, D, H, W, dt, s)),
            ("full_scan", lib.vmb_selective_scan_fwd,
             (P(outs["xs"]), P(g["draw"]), P(g["A"]), P(g["Bs"]), P(g["Cs"]), P(g["Dskip"]), P(g["bias"]),
              P(outs["yf"]), B, K, D, N, H, W, fl, dt, P(wsf), wsf.numel(), s)),
            ("mean_scan", lib.vmb_mean_scan_fwd,
             (P(outs["xs"]), P(g["draw"]), P(g["A"]), P(g["Bs"]), P(g["Cs"]), P(g["Dskip"]), P(g["bias"]),
              P(outs["ym"]), ctypes.c_void_p(0), B, K, D, N, H, W, fl, dt, P(wsm), wsm.numel(), s)),
            ("cross_merge_full", lib.vmb_cross_merge, (P(outs["yf"]), P(outs["of"]), B, D, H, W, dt, s)),
            ("cross_merge_mean", lib.vmb_cross_merge, (P(outs["ym"]), P(outs["om"]), B, D, H, W, dt, s)),
        ]
        # the channel-mean path with the broadcast fused into the merge (timed on
        # its own, next to the unfused mean scan + cross-merge of the step)
        self.fused = ("mean_scan_merge", lib.vmb_mean_scan_merge_fwd,
                      (P(outs["xs"]), P(g["draw"]), P(g["A"]), P(g["Bs"]), P(g["Cs"]), P(g["Dskip"]), P(g["bias"]),
                       P(g["x"]), P(outs["ofused"]), P(outs["ybar"]), B, D, N, H, W, fl, dt, P(wsm), wsm.numel(), s))
        # the scan side of the block straight from the map (no cross-scan, no y)
        self.gathered = ("ss2d_mean", lib.vmb_ss2d_mean_fwd,
                         (P(g["x"]), P(outs["xt"]), P(g["draw"]), P(g["A"]), P(g["Bs"]), P(g["Cs"]), P(g["Dskip"]),
                          P(g["bias"]), P(outs["ofused"]), P(outs["ybar"]), B, D, N, H, W, fl, dt, P(wsm),
                          wsm.numel(), s))
        # the full-channel scan side of the block from the map (no cross-scan)
        self.gathered_full = ("ss2d_full", lib.vmb_ss2d_full_fwd,
                              (P(g["x"]), P(outs["xt"]), P(g["draw"]), P(g["A"]), P(g["Bs"]), P(g["Cs"]),
                               P(g["Dskip"]), P(g["bias"]), P(outs["yf"]), P(outs["of"]), B, D, N, H, W, fl, dt,
                               P(wsf), wsf.numel(), s))
        # kernels each call launches (the chunked full scan launches three)
        self.launches = sum(int(lib.vmb_scan_kernel_count(path, B, K, D, N, H, W, dt)) if path >= 0 else 1
                            for path in (-1, 0, 1, -1, -1))
        self.fused_launches = int(lib.vmb_scan_kernel_count(1, B, K, D, N, H, W, dt)) + 1

    def run_fused(self):
        name, fn, args = self.fused
        st = fn(*args)
        if st != 0:
            raise RuntimeError(f"{name}: {self.vmb.status_string(st)}")

    def run_gathered(self):
        name, fn, args = self.gathered
        st = fn(*args)
        if st != 0:
            raise RuntimeError(f"{name}: {self.vmb.status_string(st)}")

    def run_gathered_full(self):
        name, fn, args = self.gathered_full
        st = fn(*args)
        if st != 0:
            raise RuntimeError(f"{name}: {self.vmb.status_string(st)}")

    def run(self, events=None):
        for i, (name, fn, args) in enumerate(self.calls):
            st = fn(*args)
            if st != 0:
                raise RuntimeError(f"{name}: {self.vmb.status_string(st)}")
            if events is not None:
                events[i + 1].record()


def time_paper_style(vmb, B, K, D, N, H, W, dev, prelude, steps, warmup):
    """The paper's kernel split (Sec. 4): discretisation into materialised fp32
    operands, then the scan alone, for the full channel axis and for the
    channel means; each call timed alone after an L2 flush (synthetic inputs)."""
    import torch
    L = H * W
    gen = torch.Generator(device=dev)
    gen.manual_seed(7)
    u = torch.randn(B, K, D, L, device=dev, generator=gen)
    draw = 0.5 * torch.randn(B, K, D, L, device=dev, generator=gen)
    Bs = torch.randn(B, K, N, L, device=dev, generator=gen)
    Cs = torch.randn(B, K, N, L, device=dev, generator=gen)
    A = -torch.arange(1, N + 1, device=dev, dtype=torch.float32).repeat(K * D, 1).contiguous()
    bias = torch.full((K * D,), -3.0, device=dev)
    dA = torch.empty(B, K, D, N, L, device=dev)
    dBu = torch.empty_like(dA)
    dAm = torch.empty(B, K, N, L, device=dev)
    dBum = torch.empty_like(dAm)
    y = torch.empty(B, K, D, L, device=dev)
    yb = torch.empty(B, K, L, device=dev)
    calls = {
        "discretise": lambda: vmb.vmb_discretise_fwd(u, draw, A, Bs, bias, H, W, dA=dA, dBu=dBu),
        "scan_only_full": lambda: vmb.vmb_scan_only_fwd(dA, dBu, Cs, H, W, y=y),
        "discretise_mean": lambda: vmb.vmb_discretise_mean_fwd(u, draw, A, Bs, bias, H, W, dAm=dAm, dBum=dBum),
        "scan_only_mean": lambda: vmb.vmb_scan_only_fwd(dAm, dBum, Cs, H, W, y=yb),
    }
    ops, res = B * K * D * N * L, {}
    byt = {"discretise": 4 * (2 * ops + 2 * B * K * D * L + B * K * N * L),
           "scan_only_full": 4 * (2 * ops + B * K * N * L + B * K * D * L),
           "discretise_mean": 4 * (2 * B * K * D * L + 3 * B * K * N * L),
           "scan_only_mean": 4 * (3 * B * K * N * L + B * K * L)}
    for name, fn in calls.items():
        for _ in range(warmup):
            prelude()
            fn()
        evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(steps)]
        for e0, e1 in evs:
            prelude()
            e0.record()
            fn()
            e1.record()
        torch.cuda.synchronize()
        us = 1e3 * statistics.median(e0.elapsed_time(e1) for e0, e1 in evs)
        res[name] = {"us": us, "algorithmic_bytes": byt[name], "gbs": byt[name] / (us / 1e6) / 1e9}
    res["shape"] = {"B": B, "K": K, "D": D, "N": N, "L": L}
    res["scan_only_speedup_mean_over_full"] = res["scan_only_full"]["us"] / res["scan_only_mean"]["us"]
    return res


def needs_flush(wl, l2_bytes: int) -> bool:
    """Flush L2 between steps unless one step's inputs are far larger than L2."""
    return wl.scan_bytes() < 4 * l2_bytes


def make_outs(wl, dev, tdt, vmb):
    import torch
    B, D, N, H, W, L = wl.B, wl.D, wl.N, wl.H, wl.W, wl.L
    return {
        "xs": torch.empty((B, 4, D, L), dtype=tdt, device=dev),
        "yf": torch.empty((B, 4, D, L), dtype=tdt, device=dev),
        "ym": torch.empty((B, 4, D, L), dtype=tdt, device=dev),
        "of": torch.empty((B, D, H, W), dtype=tdt, device=dev),
        "om": torch.empty((B, D, H, W), dtype=tdt, device=dev),
        "ws_full": torch.zeros(vmb.vmb_scan_workspace_bytes(0, B, 4, D, N, H, W, tdt), dtype=torch.uint8, device=dev),
        "ws_mean": torch.zeros(vmb.vmb_scan_workspace_bytes(1, B, 4, D, N, H, W, tdt), dtype=torch.uint8, device=dev),
        "ofused": torch.empty((B, D, H, W), dtype=tdt, device=dev),
        "ybar": torch.empty((B, 4, L), dtype=torch.float32, device=dev),
        "xt": torch.empty((B, D, W, H), dtype=tdt, device=dev),
    }


def check_status(vmb, outs, where):
    if vmb.vmb_read_status(outs["ws_full"]) != 0 or vmb.vmb_read_status(outs["ws_mean"]) != 0:
        raise RuntimeError(f"device error word set {where}")


def time_breakdown(step, n, prelude):
    """n steps with an event after every call: per-kernel durations (ms lists),
    the fused channel-mean path and the gathered one (from the map) timed alone
    (ms lists)."""
    import torch
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(len(KERNELS) + 1)] for _ in range(n)]
    for i in range(n):
        prelude()
        evs[i][0].record()
        step.run(evs[i])
    fev = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(n)]
    for i in range(n):
        prelude()
        fev[i][0].record()
        step.run_fused()
        fev[i][1].record()
    gev = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(n)]
    for i in range(n):
        prelude()
        gev[i][0].record()
        step.run_gathered()
        gev[i][1].record()
    hev = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(n)]
    for i in range(n):
        prelude()
        hev[i][0].record()
        step.run_gathered_full()
        hev[i][1].record()
    torch.cuda.synchronize()
    per_kernel = {k: [e[j].elapsed_time(e[j + 1]) for e in evs] for j, k in enumerate(KERNELS)}
    return per_kernel, ([e[0].elapsed_time(e[1]) for e in fev], [e[0].elapsed_time(e[1]) for e in gev],
                        [e[0].elapsed_time(e[1]) for e in hev])


def kernel_table(wl, per_kernel_ms, fused_pair, peak):
    fused_ms, gathered_ms, gathered_full_ms = fused_pair
    kb = kernel_bytes(wl)
    per = {}
    for k in KERNELS:
        avg = statistics.mean(per_kernel_ms[k])
        gbs = kb[k] / (avg / 1e3) / 1e9
        per[k] = {"us": avg * 1e3, "gbs": gbs, "frac_of_peak": gbs / peak}
    fused_us = 1e3 * statistics.mean(fused_ms)
    fb = wl.fused_mean_bytes()
    fused = {"us": fused_us, "gbs": fb / (fused_us / 1e6) / 1e9, "frac_of_peak": fb / (fused_us / 1e6) / 1e9 / peak,
             "algorithmic_bytes": fb,
             "unfused_us": per["mean_scan"]["us"] + per["cross_merge_mean"]["us"],
             "speedup_over_unfused": (per["mean_scan"]["us"] + per["cross_merge_mean"]["us"]) / fused_us,
             "speedup_over_full_path": (per["full_scan"]["us"] + per["cross_merge_full"]["us"]) / fused_us}
    g_us = 1e3 * statistics.mean(gathered_ms)
    gb = wl.gathered_mean_bytes()
    unfused_all = per["cross_scan"]["us"] + per["mean_scan"]["us"] + per["cross_merge_mean"]["us"]
    fused["gathered_from_map"] = {
        "us": g_us, "algorithmic_bytes": gb, "gbs": gb / (g_us / 1e6) / 1e9,
        "frac_of_peak": gb / (g_us / 1e6) / 1e9 / peak,
        "calls": "vmb_ss2d_mean_fwd: cross-scan, channel-mean scan and cross-merge, no xs and no y",
        "speedup_over_cross_scan_plus_fused": (per["cross_scan"]["us"] + fused_us) / g_us,
        "speedup_over_unfused_mean_path": unfused_all / g_us,
        "speedup_over_full_path": (per["cross_scan"]["us"] + per["full_scan"]["us"] + per["cross_merge_full"]["us"]) / g_us}
    h_us = 1e3 * statistics.mean(gathered_full_ms)
    hb = wl.gathered_full_bytes()
    three = per["cross_scan"]["us"] + per["full_scan"]["us"] + per["cross_merge_full"]["us"]
    fused["full_path_from_map"] = {
        "us": h_us, "algorithmic_bytes": hb, "gbs": hb / (h_us / 1e6) / 1e9,
        "frac_of_peak": hb / (h_us / 1e6) / 1e9 / peak,
        "calls": "vmb_ss2d_full_fwd: cross-scan, full scan and cross-merge, no xs",
        "three_calls_us": three, "speedup_over_three_calls": three / h_us,
        "gathered_mean_speedup_over_it": h_us / g_us}
    return per, fused


def sweep_configs(vmb, dev, peak, prelude_flush, warmup):
    """Every workload of the configuration list, kernel by kernel (inputs drawn on
    the device with the workload recipe; about 50 ms of timed calls each)."""
    import torch
    l2 = torch.cuda.get_device_properties(dev).L2_cache_size
    stream = torch.cuda.current_stream()
    table = {}
    for name, wl in workloads.WORKLOADS.items():
        tdt = torch.bfloat16 if wl.dtype == "bf16" else torch.float32
        g = workloads.make_device_inputs(wl, dev)
        outs = make_outs(wl, dev, tdt, vmb)
        step = Step(vmb, wl, g, outs, stream.cuda_stream)
        flush = needs_flush(wl, l2)
        prelude = prelude_flush if flush else (lambda: None)
        for _ in range(warmup):
            prelude()
            step.run()
            step.run_fused()
            step.run_gathered()
        torch.cuda.synchronize()
        est_s = sum(kernel_bytes(wl).values()) / 3e12
        n = int(min(50, max(5, 0.05 / est_s)))
        per_kernel, fused_ms = time_breakdown(step, n, prelude)
        check_status(vmb, outs, f"in the {name} sweep")
        per, fused = kernel_table(wl, per_kernel, fused_ms, peak)
        table[name] = {"B": wl.B, "D": wl.D, "N": wl.N, "H": wl.H, "W": wl.W, "storage": wl.dtype,
                       "sigma": wl.sigma, "calls": n, "l2": "flushed before every step" if flush else
                       "not flushed (inputs far larger than L2)",
                       "kernels": per, "mean_speedup_over_full": per["full_scan"]["us"] / per["mean_scan"]["us"],
                       "full_path_from_map": fused.pop("full_path_from_map"),
                       "mean_path_fused": fused, "gpu_launches_per_step": step.launches}
        del g, outs, step
        torch.cuda.empty_cache()
    return table


def run_ours(args, wl, rank, world, local_rank):
    import torch
    import paper_2412_16602_gb300 as vmb

    dev = torch.device("cuda", local_rank)
    torch.cuda.set_device(dev)
    # the workload recipe drawn on the device (seeded per rank); a pinned host
    # copy feeds the end-to-end leg
    tdt = torch.bfloat16 if wl.dtype == "bf16" else torch.float32
    g = workloads.make_device_inputs(wl, dev, seed=rank_seed(wl, rank))
    host = {k: v.cpu().pin_memory() for k, v in g.items()}
    outs = make_outs(wl, dev, tdt, vmb)
    stream = torch.cuda.current_stream()
    step = Step(vmb, wl, g, outs, stream.cuda_stream)
    l2 = torch.cuda.get_device_properties(dev).L2_cache_size
    flush_buf = torch.empty(max(2 * l2, 256 << 20) // 4, dtype=torch.float32, device=dev)

    def prelude_flush():
        flush_buf.fill_(1.0)       # evict the inputs from L2
        torch.cuda._sleep(100000)  # let the host enqueue the whole step before the GPU reaches it

    flush = needs_flush(wl, l2)
    prelude = prelude_flush if flush else (lambda: None)

    for _ in range(args.warmup):
        prelude()
        step.run()
    torch.cuda.synchronize()
    check_status(vmb, outs, "during warm-up")

    # the timed steps.  Inputs far larger than L2: the steps run back to back,
    # an event before every step and one after the last (nothing else on the
    # stream).  Smaller inputs: L2 is flushed before every step, outside the
    # step's own pair of events.
    if flush:
        sev = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(args.steps)]
    else:
        sev = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps + 1)]
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    with ClockSampler(local_rank) as clk:
        if flush:
            for i in range(args.steps):
                prelude()
                sev[i][0].record()
                step.run()
                sev[i][1].record()
        else:
            sev[0].record()
            for i in range(args.steps):
                step.run()
                sev[i + 1].record()
        torch.cuda.synchronize()
    if world > 1:
        torch.distributed.barrier()
    check_status(vmb, outs, "during the timed steps")
    if flush:
        step_ms = [e0.elapsed_time(e1) for e0, e1 in sev]
    else:
        step_ms = [sev[i].elapsed_time(sev[i + 1]) for i in range(args.steps)]
    total_ms = float(sum(step_ms))

    # per-kernel breakdown and the fused channel-mean path (separate steps with
    # an event after every call; each event costs the stream a few microseconds)
    for _ in range(2):
        prelude()
        step.run_fused()
        step.run_gathered()
    per_kernel, fused_ms = time_breakdown(step, min(args.steps, 50), prelude)
    check_status(vmb, outs, "during the breakdown steps")

    # ---- end-to-end leg: pinned host inputs -> device -> step -> host outputs.
    # Every step copies all its inputs from pinned host memory (packed in one
    # buffer: one copy) and both merged outputs back.  Two device buffer sets
    # let a step's copies overlap its neighbours' kernels: H2D on one stream,
    # the kernels on the compute stream, D2H on a third, ordered by events (a
    # step's inputs are not overwritten before the kernels that read them ran,
    # its outputs not before they were read back).
    names = list(host.keys())
    offs, off = {}, 0
    for k in names:
        nb = host[k].numel() * host[k].element_size()
        offs[k] = (off, nb)
        off = (off + nb + 255) // 256 * 256
    h2d = off
    h_in = torch.empty(h2d, dtype=torch.uint8).pin_memory()
    for k in names:
        o, nb = offs[k]
        h_in[o:o + nb].copy_(host[k].reshape(-1).view(torch.uint8))
    sets = []
    for _ in range(2):
        d_in = torch.empty(h2d, dtype=torch.uint8, device=dev)
        gv = {k: d_in[offs[k][0]:offs[k][0] + offs[k][1]].view(host[k].dtype).view(host[k].shape) for k in names}
        o2 = dict(outs)
        o2["of"], o2["om"] = torch.empty_like(outs["of"]), torch.empty_like(outs["om"])
        hout = {k: torch.empty(o2[k].shape, dtype=tdt).pin_memory() for k in ("of", "om")}
        ev = {k: torch.cuda.Event() for k in ("h2d", "comp", "d2h")}
        sets.append((d_in, o2, hout, ev, Step(vmb, wl, gv, o2, stream.cuda_stream)))
    d2h = sum(t.numel() * t.element_size() for t in sets[0][2].values())
    cs, ds = torch.cuda.Stream(device=dev), torch.cuda.Stream(device=dev)

    def e2e_steps(n):
        for i in range(n):
            d_in, o2, hout, ev, st = sets[i % 2]
            cs.wait_event(ev["comp"])  # the kernels that read this buffer two steps ago ran
            with torch.cuda.stream(cs):
                d_in.copy_(h_in, non_blocking=True)
            ev["h2d"].record(cs)
            stream.wait_event(ev["h2d"])
            stream.wait_event(ev["d2h"])  # this set's outputs of two steps ago were read back
            st.run()
            ev["comp"].record(stream)
            ds.wait_event(ev["comp"])
            with torch.cuda.stream(ds):
                hout["of"].copy_(o2["of"], non_blocking=True)
                hout["om"].copy_(o2["om"], non_blocking=True)
            ev["d2h"].record(ds)

    e2e_steps(4)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    e0.record(stream)
    cs.wait_event(e0)
    e2e_steps(args.e2e_steps)
    for _, _, _, ev, _ in sets:
        stream.wait_event(ev["d2h"])
    e1.record(stream)
    torch.cuda.synchronize()
    e2e_ms = e0.elapsed_time(e1)
    check_status(vmb, outs, "during the end-to-end steps")
    del sets, h_in

    nx = max(3, args.extra_steps)

    def time_alone(fn):
        for _ in range(args.warmup):
            prelude()
            fn()
        ev2 = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(nx)]
        for a0, a1 in ev2:
            prelude()
            a0.record()
            fn()
            a1.record()
        torch.cuda.synchronize()
        return 1e3 * statistics.mean(a0.elapsed_time(a1) for a0, a1 in ev2)

    # the grouped basis (d channel groups, each its own mean and recurrence) on the step's inputs
    grouped = {}
    for G in ((4, 16) if not args.no_grouped else ()):
        if wl.D % G:
            continue
        wsg = torch.zeros(vmb.vmb_scan_workspace_bytes(1, wl.B, 4 * G, wl.D // G, wl.N, wl.H, wl.W, tdt),
                          dtype=torch.uint8, device=dev)
        yg = outs["ym"]

        def fn():
            vmb.vmb_mean_scan_grouped_fwd(outs["xs"], g["draw"], g["A"], g["Bs"], g["Cs"], g["Dskip"], g["bias"],
                                          wl.H, wl.W, G, y=yg, workspace=wsg, stream=stream)
        grouped[G] = time_alone(fn)
        if vmb.vmb_read_status(wsg) != 0:
            raise RuntimeError("device error word set in the grouped mean scan")
    # the selection functions of Eq. 6 (B, C, raw Delta from the cross-scanned
    # input; rank-6 Delta projection as in VMamba-T) on the step's input
    sel_us = None
    if not args.no_selection:
        gsel = torch.Generator(device=dev)
        gsel.manual_seed(11)
        R = 6
        sw = [torch.randn(sz, device=dev, generator=gsel) / math.sqrt(wl.D)
              for sz in ((4, wl.N, wl.D), (4, wl.N, wl.D), (4, R, wl.D), (4, wl.D, R))]
        sdr, sB, sC = outs["yf"], torch.empty_like(g["Bs"]), torch.empty_like(g["Cs"])

        def sel():
            vmb.vmb_selection_fwd(outs["xs"], *sw, wl.H, wl.W, delta_raw=sdr, Bs=sB, Cs=sC, stream=stream)
        sel_us = time_alone(sel)
        # the same with the Delta branch left low-rank: the selection writes z
        # [B, 4, R, L] and the full scan forms the raw Deltas Wup z itself
        sz = torch.empty((wl.B, 4, R, wl.L), dtype=torch.float32, device=dev)
        ylr = outs["ym"]
        wsf = outs["ws_full"]

        def sel_lr():
            vmb.vmb_selection_lowrank_fwd(outs["xs"], sw[0], sw[1], sw[2], wl.H, wl.W, z=sz, Bs=sB, Cs=sC,
                                          stream=stream)

        def scan_lr():
            vmb.vmb_selective_scan_lowrank_fwd(outs["xs"], sz, sw[3], g["A"], sB, sC, g["Dskip"], g["bias"],
                                               wl.H, wl.W, y=ylr, workspace=wsf, stream=stream)

        def scan_raw():
            vmb.vmb_selective_scan_fwd(outs["xs"], sdr, g["A"], sB, sC, g["Dskip"], g["bias"], wl.H, wl.W,
                                       y=ylr, workspace=wsf, stream=stream)
        wsm = outs["ws_mean"]

        def mean_lr():
            vmb.vmb_mean_scan_lowrank_fwd(outs["xs"], sz, sw[3], g["A"], sB, sC, g["Dskip"], g["bias"],
                                          wl.H, wl.W, y=ylr, workspace=wsm, stream=stream)

        def mean_raw():
            vmb.vmb_mean_scan_fwd(outs["xs"], sdr, g["A"], sB, sC, g["Dskip"], g["bias"], wl.H, wl.W,
                                  y=ylr, workspace=wsm, stream=stream)
        sel()
        lowrank = {"selection_us": time_alone(sel_lr), "scan_us": time_alone(scan_lr),
                   "scan_raw_deltas_us": time_alone(scan_raw), "rank": R,
                   "mean_scan_us": time_alone(mean_lr), "mean_scan_raw_deltas_us": time_alone(mean_raw)}
        sel_us = (sel_us, lowrank)
    # the backward of the channel-mean scan on the step's inputs (dLoss/dy drawn
    # on the device), with its workspace allocated once
    bwd_us = None
    if not args.no_backward:
        gy = torch.randn(outs["ym"].shape, device=dev, dtype=torch.float32).to(tdt)
        bws = torch.empty(max(256, vmb.vmb_mean_scan_bwd_workspace_bytes(wl.B, 4, wl.D, wl.N, wl.H, wl.W, 1, tdt)),
                          dtype=torch.uint8, device=dev)
        gouts = dict(u=torch.empty_like(outs["xs"]), delta=torch.empty_like(outs["xs"]),
                     A=torch.empty_like(g["A"]), Bs=torch.empty_like(g["Bs"]), Cs=torch.empty_like(g["Cs"]),
                     Dskip=torch.empty_like(g["Dskip"]), bias=torch.empty_like(g["bias"]))
        PP = lambda t: ctypes.c_void_p(t.data_ptr()) if t is not None else ctypes.c_void_p(0)  # noqa: E731
        # the training forward: the mean scan that also keeps its group means
        saved = torch.empty((wl.B, 4, 1, wl.N + 1, wl.L), dtype=torch.float32, device=dev)
        wst = vmb.default_workspace(dev)

        def train_fwd():
            vmb.vmb_mean_scan_train_fwd(outs["xs"], g["draw"], g["A"], g["Bs"], g["Cs"], g["Dskip"], g["bias"],
                                        wl.H, wl.W, y=outs["ym"], saved=saved, stream=stream)
        train_us = time_alone(train_fwd)

        def bwd_with(sv):
            def bwd():
                st = vmb.lib.vmb_mean_scan_bwd(
                    PP(outs["xs"]), PP(g["draw"]), PP(g["A"]), PP(g["Bs"]), PP(g["Cs"]), PP(g["Dskip"]),
                    PP(g["bias"]), PP(gy), PP(sv), PP(gouts["u"]), PP(gouts["delta"]), PP(gouts["A"]),
                    PP(gouts["Bs"]), PP(gouts["Cs"]), PP(gouts["Dskip"]), PP(gouts["bias"]), wl.B, 4, wl.D, wl.N,
                    wl.H, wl.W, 1, vmb.VMB_FLAG_SOFTPLUS, vmb.VMB_BF16 if wl.dtype == "bf16" else vmb.VMB_F32,
                    PP(bws), bws.numel(), ctypes.c_void_p(stream.cuda_stream))
                if st != 0:
                    raise RuntimeError(f"vmb_mean_scan_bwd: {vmb.status_string(st)}")
            return bwd
        train_fwd()
        bwd_us = {"saved": time_alone(bwd_with(saved)), "recompute": time_alone(bwd_with(None)),
                  "train_fwd": train_us}
        if vmb.vmb_read_status(wst) != 0:
            raise RuntimeError("device error word set in the training forward")
        del gy, bws, gouts, saved
    # the materialised operands of the bench workload: 2 x B*4*D*N*L fp32
    small_enough = 8 * wl.B * 4 * wl.D * wl.N * wl.L <= (32 << 30)
    paper = None if args.no_paper_style else {
        "bench_workload": (time_paper_style(vmb, wl.B, 4, wl.D, wl.N, wl.H, wl.W, dev, prelude_flush, nx,
                                            args.warmup) if small_enough else
                           "not timed: the materialised operands exceed 32 GB"),
        # Table 1 / Table 2 "Base" row of the paper: inner dimension 512, L = 3136,
        # batch 128, d_state 1 (the byte counts of Table 2 fix batch x N = 128)
        "paper_table_base_512x3136": time_paper_style(vmb, 128, 4, 128, 1, 56, 56, dev, prelude_flush,
                                                      min(nx, 10), args.warmup),
    }
    res = {"total_ms": total_ms, "step_ms": step_ms, "per_kernel": per_kernel, "e2e_ms": e2e_ms,
           "paper_style": paper, "grouped_us": grouped, "selection_us": sel_us,
           "h2d": h2d, "d2h": d2h, "clocks": clk.summary(), "fused_ms": fused_ms,
           "launches_per_step": step.launches, "fused_launches": step.fused_launches,
           "flushed": flush, "backward_us": bwd_us}
    del g, outs, step, flush_buf
    torch.cuda.empty_cache()
    peak, _ = measured_peaks()
    res["configs"] = None if args.no_configs else sweep_configs(vmb, dev, peak, prelude_flush_factory(dev),
                                                                 min(args.warmup, 3))
    res["total_ms"], res["e2e_ms"] = max_over_ranks([total_ms, e2e_ms], world, dev)
    return res, None


def prelude_flush_factory(dev):
    import torch
    l2 = torch.cuda.get_device_properties(dev).L2_cache_size
    buf = torch.empty(max(2 * l2, 256 << 20) // 4, dtype=torch.float32, device=dev)

    def prelude():
        buf.fill_(1.0)
        torch.cuda._sleep(100000)
    return prelude


# The paper's own scan-only kernel times on one RTX A6000 (Table 1, "Base"
# rows; VMeanba about 0.02 ms in every row), for context next to the split
# measured here.  Different hardware: not a target.
PAPER_A6000_BASE_512x3136 = {"scan_only_full_ms": 5.86, "scan_only_mean_ms": 0.02, "speedup": 293}


# ALU ceilings of the state updates (b, k, d, n, l) on one GB300 (152 SMs,
# 2.07 GHz; ex2 at 32 results/clk/SM and FP32 at 128 lanes/clk/SM, both
# measured; 4 warp-instruction issues/clk/SM).  Full scan: one ex2 and four
# FP32 operations per update (delta*A, delta*u*B, the state FMA, the output
# FMA), five warp instructions per 32 updates: issue-bound at 8.05e12/s.
# Channel-mean scan: one ex2 and two FP32 operations per (d, n) term of the
# reduction: ex2-bound at 1.01e13/s.
ALU_UPDATES_PER_S = {"full_scan": 4 * 152 * 2.07e9 * 32 / 5, "mean_scan": 32 * 152 * 2.07e9}
ALU_BASIS = {"full_scan": "5 warp instructions per 32 state updates, 4 issues/clk/SM, 152 SMs, 2.07 GHz",
             "mean_scan": "one ex2 per (d, n) term, 32 ex2/clk/SM, 152 SMs, 2.07 GHz"}


def alu_view(kernel, wl, ms):
    """The dominant kernel against the ALU ceiling of its state updates."""
    if kernel not in ALU_UPDATES_PER_S:
        return None
    achieved = wl.B * 4 * wl.D * wl.N * wl.L / (ms / 1e3)
    peak = ALU_UPDATES_PER_S[kernel]
    return {"bound": "alu", "unit": "state updates/s", "achieved": achieved, "peak": peak, "frac": achieved / peak,
            "basis": ALU_BASIS[kernel]}


def selection_summary(us_pair, wl, peak, R=6):
    """Eq. 6 selection on the step's input: reads u, writes B, C and the raw Delta.
    "lowrank": the same with the Delta branch left low-rank (the selection writes
    z, fp32 [B, 4, R, L]; the full scan forms the raw Deltas Wup z itself),
    timed next to the selection + full scan on its raw Deltas."""
    if us_pair is None:
        return None
    us, lr = us_pair
    s = 2 if wl.dtype == "bf16" else 4
    bkdl, bknl, bkrl = wl.B * 4 * wl.D * wl.L, wl.B * 4 * wl.N * wl.L, wl.B * 4 * R * wl.L
    bytes_ = s * (2 * bkdl + 2 * bknl) + 4 * 4 * (2 * wl.N + 2 * R) * wl.D
    gbs = bytes_ / (us / 1e6) / 1e9
    sel_lr_bytes = s * (bkdl + 2 * bknl) + 4 * bkrl + 4 * 4 * (2 * wl.N + R) * wl.D
    scan_lr_bytes = s * (2 * bkdl + 2 * bknl) + 4 * bkrl + 4 * 4 * wl.D * (wl.N + 2 + R)
    pair_lr = lr["selection_us"] + lr["scan_us"]
    pair_raw = us + lr["scan_raw_deltas_us"]
    lowrank = {"rank": R, "selection_us": lr["selection_us"], "scan_us": lr["scan_us"],
               "scan_algorithmic_bytes": scan_lr_bytes,
               "scan_gbs": scan_lr_bytes / (lr["scan_us"] / 1e6) / 1e9,
               "scan_frac_of_peak": scan_lr_bytes / (lr["scan_us"] / 1e6) / 1e9 / peak,
               "pair_us": pair_lr, "pair_bytes": sel_lr_bytes + scan_lr_bytes,
               "raw_deltas_pair_us": pair_raw, "raw_deltas_pair_bytes": bytes_ + wl.scan_bytes(),
               "speedup_over_raw_deltas": pair_raw / pair_lr,
               "mean_scan_us": lr["mean_scan_us"], "mean_scan_raw_deltas_us": lr["mean_scan_raw_deltas_us"],
               "mean_pair_us": lr["selection_us"] + lr["mean_scan_us"],
               "mean_raw_deltas_pair_us": us + lr["mean_scan_raw_deltas_us"],
               "mean_speedup_over_raw_deltas": (us + lr["mean_scan_raw_deltas_us"]) /
                                               (lr["selection_us"] + lr["mean_scan_us"])}
    return {"us": us, "algorithmic_bytes": bytes_, "gbs": gbs, "frac_of_peak": gbs / peak, "rank": R,
            "kernel": "tcgen05.mma kind::tf32 (three-product tf32 split for fp32 accuracy), accumulator in TMEM",
            "lowrank": lowrank}


def backward_summary(us, wl, peak):
    """The channel-mean scan's backward: reads u, the raw Delta, dLoss/dy, B and C,
    writes the gradients of u, Delta, B and C (and the small parameter gradients).
    "us": given the group means the training forward kept (which it also reads,
    fp32 [B, K, N + 1, L]); "us_recompute": recomputing them (N exponentials per
    element).  "train_fwd_us": that forward (the mean scan plus the kept means)."""
    if us is None:
        return None
    s = 2 if wl.dtype == "bf16" else 4
    bkdl = wl.B * 4 * wl.D * wl.L
    bknl = wl.B * 4 * wl.N * wl.L
    base = s * (5 * bkdl + 4 * bknl) + 2 * 4 * 4 * wl.D * (wl.N + 2)
    bytes_ = base + 4 * wl.B * 4 * (wl.N + 1) * wl.L
    gbs = bytes_ / (us["saved"] / 1e6) / 1e9
    return {"us": us["saved"], "algorithmic_bytes": bytes_, "gbs": gbs, "frac_of_peak": gbs / peak,
            "launches": 6, "us_recompute": us["recompute"],
            "frac_of_peak_recompute": base / (us["recompute"] / 1e6) / 1e9 / peak,
            "train_fwd_us": us["train_fwd"]}


def paper_style_summary(ps, peak):
    if ps is None:
        return None
    out = {}
    for key, r in ps.items():
        if not isinstance(r, dict):
            out[key] = r
            continue
        out[key] = {k: (dict(v, frac_of_peak=v["gbs"] / peak) if isinstance(v, dict) and "gbs" in v else v)
                    for k, v in r.items()}
    out["paper_a6000_base_512x3136"] = PAPER_A6000_BASE_512x3136
    return out


def main():
    args = parse()
    wl = workloads.WORKLOADS[args.workload]
    if args.batch is not None:
        wl = wl.replace(B=args.batch, name=f"{wl.name}@batch{args.batch}")
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    step_bytes = sum(kernel_bytes(wl).values())
    elems = wl.scan_elements()
    config = {"workload": wl.name, "B": wl.B, "K": 4, "D": wl.D, "N": wl.N, "H": wl.H, "W": wl.W, "L": wl.L,
              "storage": wl.dtype, "sigma": wl.sigma,
              "step": "cross_scan + full_scan + mean_scan + 2 x cross_merge"}
    # The oracle (fp64, host cores) runs on a bounded sample of the workload:
    # one batch element (the same recipe with B = 1); its throughput is the
    # sample's algorithmic bytes per second.
    cpu_wl = wl.replace(B=1, name=f"{wl.name}[one batch element]") if wl.B > 1 else wl
    cpu_bytes = sum(kernel_bytes(cpu_wl).values())
    cpu_sample = (f"one batch element of {wl.name} (B = 1 of {wl.B}, same recipe) per oracle step, "
                  "full + mean paths with the cross-scan and both merges")

    if args.impl == "reference":
        if rank != 0:
            return
        inp = workloads.make_inputs(cpu_wl)
        import oracle
        nth = oracle.default_threads()
        for _ in range(min(args.warmup, 1)):
            oracle_step(inp, nth)
        times = []
        for _ in range(args.steps):
            t0 = time.perf_counter()
            oracle_step(inp, nth)
            times.append(time.perf_counter() - t0)
        ms = 1e3 * sum(times) / len(times)
        v = cpu_bytes / (ms / 1e3) / 1e9
        line = {"impl": "reference", "metric": METRIC, "value": v, "unit": "GB/s", "n_gpus": args.gpus,
                "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
                "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic", "config": config,
                "elements_per_s": 2 * cpu_wl.scan_elements() / (ms / 1e3),
                "cpu_baseline": {"value": v, "unit": "GB/s", "cores": nth, "kind": "oracle", "sample": cpu_sample},
                "e2e": {"value": v, "unit": "GB/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
        print(json.dumps(line))
        return

    if world > 1:
        import torch
        torch.distributed.init_process_group("nccl", device_id=torch.device("cuda", local_rank))
    res, _ = run_ours(args, wl, rank, world, local_rank)
    if rank != 0:
        if world > 1:
            import torch
            torch.distributed.destroy_process_group()
        return

    ms = res["total_ms"] / args.steps
    value = job_throughput(step_bytes, world, ms)
    config["l2"] = ("flushed before every step (2x L2 write, outside the timed events)" if res["flushed"] else
                    "not flushed: a step's inputs are far larger than L2; steps run back to back")
    config["timed_region_s"] = res["total_ms"] / 1e3
    kb = kernel_bytes(wl)
    peak, peak_src = measured_peaks()
    per, fused_table = kernel_table(wl, res["per_kernel"], res["fused_ms"], peak)
    dominant = max(KERNELS, key=lambda k: statistics.mean(res["per_kernel"][k]))
    dom_ms = statistics.mean(res["per_kernel"][dominant])
    achieved = kb[dominant] / (dom_ms / 1e3) / 1e9
    traffic = committed_traffic(dominant, wl.name)
    line = {
        "metric": METRIC, "value": value, "unit": "GB/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f32",
        "data": "synthetic (seeded; shared map + per-channel noise, the workload recipe drawn on the device)",
        "config": config,
        "elements_per_s": world * 2 * elems / (ms / 1e3),
        "frac_of_peak": value / peak,
        "full": {"us": per["full_scan"]["us"], "gbs": per["full_scan"]["gbs"],
                 "elements_per_s": elems / (per["full_scan"]["us"] / 1e6),
                 "frac_of_peak": per["full_scan"]["frac_of_peak"]},
        "mean": {"us": per["mean_scan"]["us"], "gbs": per["mean_scan"]["gbs"],
                 "elements_per_s": elems / (per["mean_scan"]["us"] / 1e6),
                 "frac_of_peak": per["mean_scan"]["frac_of_peak"]},
        "mean_speedup_over_full": per["full_scan"]["us"] / per["mean_scan"]["us"],
        "kernels": per,
        "roofline": {"kernel": dominant, "bound": "hbm", "achieved": achieved, "peak": peak,
                     "peak_source": f"{peak_src} hbm_gbs (MEASURED_PEAKS.json)" if peak_src == "measured"
                     else "fallback 6.8 TB/s", "unit": "GB/s", "frac": achieved / peak,
                     "algorithmic_bytes_per_launch": kb[dominant], "traffic": traffic,
                     "alu_view": alu_view(dominant, wl, dom_ms)},
        # the fused channel-mean path (broadcast inside the merge) and the same
        # from the map (no cross-scan either), timed separately
        "full_path_from_map": fused_table.pop("full_path_from_map"),
        "mean_path_fused": fused_table,
        "gpu_launches": res["launches_per_step"] * args.steps,
        "paper_style": paper_style_summary(res["paper_style"], peak),
        # grouped basis: d channel groups per direction, each its own channel mean
        # and recurrence (same algorithmic bytes as the mean scan)
        "selection": selection_summary(res["selection_us"], wl, peak),
        "mean_backward": backward_summary(res["backward_us"], wl, peak),
        "mean_grouped": {str(G): {"groups": G, "us": us, "gbs": kb["mean_scan"] / (us / 1e6) / 1e9,
                                  "frac_of_peak": kb["mean_scan"] / (us / 1e6) / 1e9 / peak}
                         for G, us in res["grouped_us"].items()},
        "clocks": res["clocks"],
        # every workload of the configuration list, kernel by kernel (inputs drawn
        # on the device with the same recipe; the headline above is one of them)
        "configs": res["configs"],
        "e2e": {"value": job_throughput(step_bytes, world, res["e2e_ms"] / args.e2e_steps), "unit": "GB/s",
                "ms_per_step": res["e2e_ms"] / args.e2e_steps,
                "h2d_bytes_per_step": res["h2d"], "d2h_bytes_per_step": res["d2h"],
                "pipelined": "one packed H2D copy and two D2H copies per step, overlapping the neighbouring "
                             "steps' kernels (two buffer sets, copy streams ordered by events)"},
    }
    if not args.no_cpu_baseline and world == 1 and rank == 0:
        times, nth = time_oracle(workloads.make_inputs(cpu_wl), target_s=10.0)
        cms = 1e3 * statistics.mean(times)
        line["cpu_baseline"] = {"value": cpu_bytes / (cms / 1e3) / 1e9, "unit": "GB/s", "cores": nth,
                                "kind": "oracle", "ms_per_step": cms,
                                "sample": f"{len(times)} oracle steps, ~10 s: {cpu_sample}"}
    print(json.dumps(line))
    if world > 1:
        import torch
        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
