#!/usr/bin/env python3
"""Benchmark of the exact Gauss kernel sum on one GB300 (or N replicas).

A step is one full pass of the path -- centring mean, centre/cast/norm
prep, value prep, fused tcgen05 kernel, finalise -- over one batch of the
MMD-style workload: M = N = 65536 points in D = 64 (fp16, q = k), C = 1,
v = +-1/N, tau = 1/64, i.e. 4.29e9 pair interactions per step.  The metric
is pair interactions per second; the roofline of the fused kernel is the
slower of dense fp16 tensor work 2 M N (D + C) and M N exponentials on the
MUFU unit.

Usage:
  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl own|reference]
Under torchrun (N > 1) each rank runs an independent replica on its own
GPU (no data exchange); the ranks agree on the max step time.
"""
from __future__ import annotations

import argparse
import glob
import hashlib
import json
import math
import os
import re
import signal
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "Gauss-sum pair-interactions/s and % of tensor/SFU roofline on 1 GB300"
UNIT = "pairs/s"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
L2_FLUSH_BYTES = 512 << 20


def parse_args(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=400)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["own", "reference"], default="own")
    ap.add_argument("--workload", default="mmd_d64")
    ap.add_argument("--cpu-seconds", type=float, default=15.0,
                    help="target CPU time of the oracle baseline sample")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-clocks", action="store_true")
    return ap.parse_args(argv)


def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", str(rank)))
    return rank, world, local


def reduce_max(value, device):
    """Largest `value` over the ranks of the default process group (the
    value itself when no group of more than one rank is initialised)."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return float(value)
    t = torch.tensor([float(value)], device=device, dtype=torch.float64)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def replica_value(world, pairs_per_rank, ms):
    """Whole-job rate of `world` replicas that each process `pairs_per_rank`
    pairs per step, from the slowest rank's step time in ms."""
    return world * pairs_per_rank / (ms * 1e-3)


def workload_config(w):
    return {
        "workload": f"{w.name}: M={w.M}, N={w.N}, D={w.D}, C={w.C}, {w.dtype}, tau={w.tau:g}"
                    + (", q=k" if w.q_is_k else "") + (", forward+grad_q" if w.grad else ""),
        "M": w.M, "N": w.N, "D": w.D, "C": w.C, "input_dtype": w.dtype, "tau": w.tau,
        "pairs_per_step": w.pairs, "seed": 0,
        "l2": "flushed (512 MiB write) before every timed step",
    }


# ---------------------------------------------------------------- CPU oracle
def time_oracle(inp, seconds, max_rows=None):
    """Oracle (float64, all host cores) on a seeded row sample sized to take
    about `seconds`; returns (pairs/s, rows, elapsed, threads)."""
    from oracle import oracle_grad_q, oracle_sum
    from paper_2609_04910_gb300.workloads import sample_rows
    w = inp["workload"]
    threads = max(1, len(os.sched_getaffinity(0)))
    fn = (lambda rows: oracle_grad_q(inp["q64"], inp["k64"], inp["v64"], w.tau, rows=rows,
                                     nthreads=threads)) if w.grad else \
        (lambda rows: oracle_sum(inp["q64"], inp["k64"], inp["v64"], w.tau, rows=rows,
                                 nthreads=threads))
    probe = sample_rows(w.M, threads, seed=1)
    t0 = time.perf_counter()
    fn(probe)
    t_probe = max(time.perf_counter() - t0, 1e-4)
    rows_n = int(max(threads, min(w.M, seconds / t_probe * len(probe))))
    if max_rows:
        rows_n = min(rows_n, max_rows)
    rows = sample_rows(w.M, rows_n, seed=1)
    t0 = time.perf_counter()
    fn(rows)
    el = time.perf_counter() - t0
    return len(rows) * w.N / el, len(rows), el, threads


# ---------------------------------------------------------------- reference arm
def run_reference(args):
    rank, world, _ = dist_env()
    if rank != 0:
        return 0
    from paper_2609_04910_gb300.workloads import WORKLOADS, generate
    w = WORKLOADS[args.workload]
    inp = generate(w, seed=0)
    steps, warm = max(1, args.steps), max(0, args.warmup)
    budget = 150.0 / (steps + warm)  # keep the whole run within a few minutes
    per_step = min(5.0, budget)
    from oracle import build_oracle
    build_oracle()
    rate, rows, el, threads = time_oracle(inp, per_step)
    from oracle import oracle_sum, oracle_grad_q
    from paper_2609_04910_gb300.workloads import sample_rows
    times = []
    for i in range(warm + steps):
        r = sample_rows(w.M, rows, seed=1 + i)
        t0 = time.perf_counter()
        if w.grad:
            oracle_grad_q(inp["q64"], inp["k64"], inp["v64"], w.tau, rows=r, nthreads=threads)
        else:
            oracle_sum(inp["q64"], inp["k64"], inp["v64"], w.tau, rows=r, nthreads=threads)
        if i >= warm:
            times.append(time.perf_counter() - t0)
    t = statistics.mean(times)
    value = rows * w.N / t
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
        "steps": steps, "warmup": warm, "ms_per_step": t * 1e3, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": workload_config(w),
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": threads, "kind": "oracle",
                         "sample": f"{rows} seeded query rows x all {w.N} keys per step"},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
        "note": "float64 CPU oracle (plain double loop over Eq. 1) on the host cores; "
                "no reference implementation of the paper exists",
    }
    print(json.dumps(line), flush=True)
    return 0


# ---------------------------------------------------------------- clocks
class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index, enabled=True):
        self.proc = None
        self.path = None
        self.gpu = gpu_index
        if not enabled:
            return
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={gpu_index}", f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except (OSError, ValueError):
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.send_signal(signal.SIGTERM)
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        rows = []
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) >= 9:
                    rows.append(parts)
        os.unlink(self.path)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"], "samples": 0}
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        reasons = set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for r in rows:
            for name, val in zip(names, r[5:9]):
                if val.lower().startswith("active"):
                    reasons.add(name)
        pw = [float(r[3]) for r in rows if re.match(r"^[0-9.]+$", r[3])]
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": sorted(reasons),
                "samples": len(rows), "power_w_max": max(pw) if pw else None}


# ---------------------------------------------------------------- helpers
def measured_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return d, "measured"
    except (OSError, ValueError):
        return dict(FALLBACK_PEAKS), "fallback"


def kernel_source_hash():
    """Hash of every library source file: a profile taken on other sources
    no longer describes the kernel."""
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2609_04910_gb300", "csrc")
    for name in sorted(os.listdir(csrc)):
        if name.endswith((".cu", ".cuh", ".h")):
            with open(os.path.join(csrc, name), "rb") as f:
                h.update(name.encode())
                h.update(f.read())
    return h.hexdigest()[:16]


def main_kernel_name(w):
    """Fused kernel the library picks for this workload (plan in csrc)."""
    if w.dtype == "fp32":
        # fp32 forward sums with C <= 4, D <= 32 from 2^25 pairs: 3xTF32 variant.
        tf32 = not w.grad and w.C <= 4 and w.D <= 32 and w.M * w.N >= 2 ** 25
        return "tc_gauss_fma_kernel" if tf32 else "simt_gauss_kernel"
    return "tc_gauss_fma_kernel" if (not w.grad and w.C <= 4) else "tc_gauss_kernel"


def profiled_traffic(w):
    """DRAM bytes per launch of the fused kernel from the committed ncu
    summary, if it was taken on the current library sources."""
    src = kernel_source_hash()
    for path in glob.glob(os.path.join(ROOT, "profiles", f"{main_kernel_name(w)}_{w.name}*.md")):
        text = open(path).read()
        m_h = re.search(r"source_sha256_16:\s*([0-9a-f]+)", text)
        m_t = re.search(r"dram_bytes_per_launch:\s*([0-9.eE+]+)", text)
        if m_h and m_t and m_h.group(1) == src:
            return float(m_t.group(1)), os.path.relpath(path, ROOT)
    return None, None


# ---------------------------------------------------------------- own arm
def run_own(args):
    import torch
    rank, world, local = dist_env()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)

    from paper_2609_04910_gb300.build import build_library
    build_library()
    import paper_2609_04910_gb300 as gs
    from paper_2609_04910_gb300.workloads import WORKLOADS, device_inputs, generate

    w = WORKLOADS[args.workload]
    inp = generate(w, seed=0)
    q, k, v = device_inputs(inp, dev)
    M, N, D, C = w.M, w.N, w.D, w.C
    out = torch.empty((M, D if w.grad else C), dtype=torch.float32, device=dev)
    s_out = torch.empty((M,), dtype=torch.float32, device=dev) if w.grad else None
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream()

    def step(main_events=None):
        if w.grad:
            gs.gauss_sum_grad_q(q, k, v, w.tau, grad=out, s_out=s_out, main_events=main_events)
        else:
            gs.gauss_sum(q, k, v, w.tau, out=out, main_events=main_events)

    def barrier():
        if world > 1:
            import torch.distributed as dist
            dist.barrier()

    # Roofline denominators.
    peaks, peak_src = measured_peaks()
    r_x = gs.gauss_sum_probe_ex2_rate()
    props = torch.cuda.get_device_properties(dev)
    sms = props.multi_processor_count
    sm_max_mhz = float(peaks.get("sm_max_mhz", 2070.0))
    r_x_nominal = 32.0 * sms * sm_max_mhz * 1e6

    K, W = max(1, args.steps), max(3, args.warmup)
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(K)]
    mev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
           for _ in range(K)]
    for a, b in ev + mev:  # create the CUDA events before handing them to the library
        a.record(stream)
        b.record(stream)
    for _ in range(W):
        flush.zero_()
        step()
    gs.gauss_sum_device_status()
    torch.cuda.synchronize()

    sampler = ClockSampler(local, enabled=not args.no_clocks)
    time.sleep(0.3 if not args.no_clocks else 0.0)
    barrier()
    torch.cuda.synchronize()
    wall0 = time.perf_counter()
    launches0 = gs.gauss_sum_kernel_launches()
    for i in range(K):
        flush.zero_()
        ev[i][0].record(stream)
        step(main_events=mev[i])
        ev[i][1].record(stream)
    launches = gs.gauss_sum_kernel_launches() - launches0
    torch.cuda.synchronize()
    barrier()
    wall = time.perf_counter() - wall0
    gs.gauss_sum_device_status()
    step_ms = [a.elapsed_time(b) for a, b in ev]
    main_ms = [a.elapsed_time(b) for a, b in mev]
    ms = statistics.mean(step_ms)
    main_mean = statistics.mean(main_ms)
    ms = reduce_max(ms, dev)

    # End to end through the public API with host buffers: H2D of the
    # inputs, the call, D2H of the result, every step.
    e2e = None
    if not args.no_e2e:
        import numpy as np
        kh = torch.from_numpy(np.ascontiguousarray(inp["k"]).view(np.int16 if w.dtype == "bf16" else inp["k"].dtype)).pin_memory()
        vh = torch.from_numpy(np.ascontiguousarray(inp["v"]).view(np.int16 if w.dtype == "bf16" else inp["v"].dtype)).pin_memory()
        qh = kh if w.q_is_k else torch.from_numpy(
            np.ascontiguousarray(inp["q"]).view(np.int16 if w.dtype == "bf16" else inp["q"].dtype)).pin_memory()
        kd = torch.empty_like(kh, device=dev)
        vd = torch.empty_like(vh, device=dev)
        qd = kd if w.q_is_k else torch.empty_like(qh, device=dev)
        outh = torch.empty(tuple(out.shape), dtype=torch.float32).pin_memory()
        sh = torch.empty((M,), dtype=torch.float32).pin_memory() if w.grad else None
        conv = (lambda t: t.view(torch.bfloat16)) if w.dtype == "bf16" else (lambda t: t)
        e_ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                for _ in range(min(K, 200))]
        h2d = kh.numel() * kh.element_size() + vh.numel() * vh.element_size() + \
            (0 if w.q_is_k else qh.numel() * qh.element_size())
        d2h = outh.numel() * 4 + (M * 4 if w.grad else 0)
        for i in range(len(e_ev) + W):
            flush.zero_()
            if i >= W:
                e_ev[i - W][0].record(stream)
            kd.copy_(kh, non_blocking=True)
            vd.copy_(vh, non_blocking=True)
            if not w.q_is_k:
                qd.copy_(qh, non_blocking=True)
            if w.grad:
                g, s_ = gs.gauss_sum_grad_q(conv(qd), conv(kd), conv(vd), w.tau)
                outh.copy_(g, non_blocking=True)
                sh.copy_(s_, non_blocking=True)
            else:
                o = gs.gauss_sum(conv(qd), conv(kd), conv(vd), w.tau)
                outh.copy_(o, non_blocking=True)
            if i >= W:
                e_ev[i - W][1].record(stream)
        torch.cuda.synchronize()
        e_ms = statistics.mean(a.elapsed_time(b) for a, b in e_ev)
        e_ms = reduce_max(e_ms, dev)
        e2e = {"value": replica_value(world, w.pairs, e_ms), "unit": UNIT, "ms_per_step": e_ms,
               "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h),
               "steps": len(e_ev)}
    clocks = sampler.stop() if sampler is not None else None

    # Roofline of the fused kernel (algorithmic work, unpadded D and C;
    # the gradient evaluates C' = D + 1 value channels).
    Ceff = D + 1 if w.grad else C
    flops = 2.0 * M * N * (D + Ceff)
    exps = float(M) * N
    r_t = float(peaks.get("bf16_tflops", FALLBACK_PEAKS["bf16_tflops"])) * 1e12  # fp16 = bf16 rate
    t_tensor = flops / r_t
    t_sfu = exps / r_x
    t_main = main_mean * 1e-3
    traffic, traffic_src = profiled_traffic(w)
    if w.dtype == "fp32":
        roof = None
    elif t_sfu >= t_tensor:
        # Bound by the MUFU exp2 issue rate: peak from unit count x SMs x
        # maximum SM clock (32 ex2 per clock per SM, the rate the probe
        # reaches at the maximum clock).
        roof = {"bound": "alu", "achieved": exps / t_main / 1e12, "peak": r_x_nominal / 1e12,
                "unit": "Texp/s", "frac": exps / r_x_nominal / t_main}
    else:
        roof = {"bound": "tensor", "achieved": flops / t_main / 1e12, "peak": r_t / 1e12,
                "unit": "TFLOP/s", "frac": (t_tensor / t_main)}
    if roof is not None:
        roof.update({
            "traffic": traffic, "traffic_source": traffic_src,
            "kernel": main_kernel_name(w), "kernel_ms": main_mean,
            "t_roof_ms": max(t_tensor, exps / r_x_nominal) * 1e3,
            "peak_note": ("alu = MUFU ex2.approx: 32/clk/SM x "
                          f"{sms} SMs x {sm_max_mhz:.0f} MHz = {r_x_nominal:.4g}/s "
                          f"(the library's probe measured {r_x:.4g}/s live); tensor peak = "
                          f"{peak_src} bf16 dense {r_t/1e12:.1f} TFLOP/s (fp16 runs at the bf16 "
                          "rate)"),
            "tensor": {"achieved": flops / t_main / 1e12, "peak": r_t / 1e12, "unit": "TFLOP/s",
                       "frac": t_tensor / t_main},
            "sfu": {"achieved": exps / t_main / 1e12, "peak": r_x_nominal / 1e12,
                    "unit": "Texp/s", "frac": exps / r_x_nominal / t_main,
                    "probe_ex2_per_s": r_x},
        })

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        from oracle import build_oracle
        build_oracle()
        rate, rows, el, threads = time_oracle(inp, args.cpu_seconds)
        cpu = {"value": rate, "unit": UNIT, "cores": threads, "kind": "oracle",
               "sample": f"{rows} seeded query rows x all {w.N} keys ({el:.1f} s, float64, "
                         f"{threads} threads)"}

    if rank == 0:
        line = {
            "metric": METRIC, "value": replica_value(world, w.pairs, ms), "unit": UNIT,
            "n_gpus": world, "steps": K, "warmup": W, "ms_per_step": ms,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "fp16" if w.dtype == "fp16" else w.dtype, "data": "synthetic",
            "config": workload_config(w),
            "roofline": roof, "cpu_baseline": cpu, "e2e": e2e,
            "gpu_launches": launches,
            "clocks": clocks, "wall_s_timed": wall,
            "main_kernel_ms": main_mean,
            "main_kernel_ms_min": min(main_ms),
            "step_ms_min": min(step_ms),
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()
    return 0


def main(argv=None):
    args = parse_args(argv)
    if args.impl == "reference":
        return run_reference(args)
    return run_own(args)


if __name__ == "__main__":
    sys.exit(main())
