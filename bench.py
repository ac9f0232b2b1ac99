#!/usr/bin/env python3
"""Benchmark of the exact Gauss kernel sum on one GB300 (or N replicas).

A step is one full pass of the path -- centring mean, centre/cast/norm
prep, value prep, fused tcgen05 kernel, finalise -- over one batch of the
MMD-style workload: M = N = 65536 points in D = 64 (fp16; q and k drawn
independently from N(0, 1)), C = 1, v = +-1/N, tau = 1/64, i.e. 4.29e9 pair
interactions per step.  The metric is pair interactions per second; the
roofline of the fused kernel is the slower of dense fp16 tensor work
2 M N (D + C) and M N exponentials on the MUFU unit.  The same run also
times the other configurations (fewer steps) and reports them under
"other_workloads".

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
    ap.add_argument("--no-other-workloads", action="store_true",
                    help="skip timing the other four configurations")
    ap.add_argument("--no-peak-probe", action="store_true")
    ap.add_argument("--batched", action="store_true",
                    help="time gauss_sum_batched on the paper's benchmark shapes "
                         "(B = 64 clouds of 16384 points, D = 16..128) and smaller "
                         "batches; one JSON line per case, instead of the step")
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
                         "cpu_model": cpu_model(),
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


def strip_comments(src):
    """C/C++ source without its comments and with every run of whitespace
    outside string and character literals reduced to one space: two
    sources give the same text when they differ only in comments and
    layout."""
    out, i, n = [], 0, len(src)
    space = False
    while i < n:
        c = src[i]
        if c in "\"'":
            j = i + 1
            while j < n and src[j] != c:
                j += 2 if src[j] == "\\" else 1
            out.append(src[i:j + 1])
            i = j + 1
            space = False
            continue
        if src.startswith("//", i):
            j = src.find("\n", i)
            i = n if j < 0 else j
            c = " "
        elif src.startswith("/*", i):
            j = src.find("*/", i + 2)
            i = n if j < 0 else j + 2
            c = " "
        else:
            i += 1
        if c.isspace():
            if not space:
                out.append(" ")
            space = True
        else:
            out.append(c)
            space = False
    return "".join(out)


def kernel_source_hash():
    """Hash of every library source file with its comments removed: a
    profile taken on other code no longer describes the kernel, while a
    comment changes nothing that runs."""
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2609_04910_gb300", "csrc")
    for name in sorted(os.listdir(csrc)):
        if name.endswith((".cu", ".cuh", ".h")):
            with open(os.path.join(csrc, name), encoding="utf-8") as f:
                h.update(name.encode())
                h.update(strip_comments(f.read()).encode())
    return h.hexdigest()[:16]


def main_kernel_name(w):
    """Fused kernel the library picks for this workload (plan in csrc)."""
    if w.dtype == "fp32":
        # fp32 forward sums with C <= 4, D <= 32 from 2^25 pairs: 3xTF32 variant.
        tf32 = not w.grad and w.C <= 4 and w.D <= 32 and w.M * w.N >= 2 ** 25
        return "tc_gauss_fma_kernel" if tf32 else "simt_gauss_kernel"
    if w.grad or w.C > 4:
        return "tc_gauss_kernel"
    # Three or four channels on augmented rows (D + 4 <= 128 for fp16, + 6
    # for bf16) go to the two-MMA kernel from 2^28 pairs.
    aug = w.D + (4 if w.dtype == "fp16" else 6) <= 128
    return "tc_gauss_kernel" if (w.C >= 3 and aug and w.M * w.N >= 2 ** 28) else "tc_gauss_fma_kernel"


def profiled_traffic(w):
    """DRAM bytes per launch of the fused kernel from the committed ncu
    summary, if it was taken on the current library sources."""
    src = kernel_source_hash()
    for path in glob.glob(os.path.join(ROOT, "profiles", f"{main_kernel_name(w)}_{w.name}.md")):
        text = open(path).read()
        m_h = re.search(r"source_sha256_16:\s*([0-9a-f]+)", text)
        m_t = re.search(r"dram_bytes_per_launch:\s*([0-9.eE+]+)", text)
        if m_h and m_t and m_h.group(1) == src:
            return float(m_t.group(1)), os.path.relpath(path, ROOT)
    return None, None


# ---------------------------------------------------------------- own arm
def cpu_model():
    """Host CPU model name (lscpu, else /proc/cpuinfo), or None."""
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.lower().startswith("model name"):
                return line.split(":", 1)[1].strip()
    except (OSError, subprocess.SubprocessError):
        pass
    try:
        for line in open("/proc/cpuinfo"):
            if line.lower().startswith("model name"):
                return line.split(":", 1)[1].strip()
    except OSError:
        pass
    return None


def probe_fp16_tflops(dev):
    """Dense fp16 matmul throughput (torch, 8192^3, best of 10): context for
    the tensor peak, measured the way the bf16 peak in MEASURED_PEAKS.json
    is.  Not a library kernel."""
    import torch
    n = 8192
    a = torch.randn(n, n, device=dev, dtype=torch.float16)
    b = torch.randn(n, n, device=dev, dtype=torch.float16)
    for _ in range(3):
        torch.matmul(a, b)
    best = 0.0
    for _ in range(10):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        torch.matmul(a, b)
        e1.record()
        e1.synchronize()
        best = max(best, 2.0 * n ** 3 / (e0.elapsed_time(e1) * 1e-3) / 1e12)
    del a, b
    torch.cuda.empty_cache()
    return best


def roofline_of(w, main_ms, peaks, peak_src, sms, r_x, traffic=None, traffic_src=None,
                r_mix=None):
    """Roofline of the fused kernel (algorithmic work, unpadded D and C; the
    gradient evaluates C' = D + 1 value channels): the slower of dense tensor
    work 2 M N (D + C) at the measured bf16 peak (fp16 runs at the bf16
    rate) and M N exponentials at the MUFU rate (32 ex2 per clock per SM at
    the maximum SM clock)."""
    M, N, D, C = w.M, w.N, w.D, w.C
    Ceff = D + 1 if w.grad else C
    flops = 2.0 * M * N * (D + Ceff)
    exps = float(M) * N
    r_t = float(peaks.get("bf16_tflops", FALLBACK_PEAKS["bf16_tflops"])) * 1e12
    sm_max_mhz = float(peaks.get("sm_max_mhz", 2070.0))
    r_x_nominal = 32.0 * sms * sm_max_mhz * 1e6
    t_tensor = flops / r_t
    t_sfu = exps / r_x_nominal
    t_main = main_ms * 1e-3
    if w.dtype == "fp32":
        return None            # fp32_d16 runs on the SIMT kernel: launch and latency bound
    if t_sfu >= t_tensor:
        roof = {"bound": "alu", "achieved": exps / t_main / 1e12, "peak": r_x_nominal / 1e12,
                "unit": "Texp/s", "frac": t_sfu / t_main}
    else:
        roof = {"bound": "tensor", "achieved": flops / t_main / 1e12, "peak": r_t / 1e12,
                "unit": "TFLOP/s", "frac": t_tensor / t_main}
    roof.update({
        "traffic": traffic, "traffic_source": traffic_src,
        "kernel": main_kernel_name(w), "kernel_ms": main_ms,
        "t_roof_ms": max(t_tensor, t_sfu) * 1e3,
        "peak_note": ("alu = MUFU ex2.approx: 32/clk/SM x "
                      f"{sms} SMs x {sm_max_mhz:.0f} MHz = {r_x_nominal:.4g}/s "
                      f"(the library's probe measured {r_x:.4g}/s live); tensor peak = "
                      f"{peak_src} bf16 dense {r_t/1e12:.1f} TFLOP/s (fp16 at the bf16 rate, "
                      "the nominal ratio 1)"),
        "tensor": {"achieved": flops / t_main / 1e12, "peak": r_t / 1e12, "unit": "TFLOP/s",
                   "frac": t_tensor / t_main},
        "sfu": {"achieved": exps / t_main / 1e12, "peak": r_x_nominal / 1e12,
                "unit": "Texp/s", "frac": t_sfu / t_main, "probe_ex2_per_s": r_x},
    })
    r_ts = peaks.get("bf16_tflops_sustained")
    if r_ts:
        # A tensor-bound kernel that runs for a whole timed loop meets the
        # power cap like the sustained cuBLAS loop that measured this peak;
        # its fraction of that peak is reported beside the burst fraction.
        r_ts = float(r_ts) * 1e12
        roof["tensor"]["peak_sustained"] = r_ts / 1e12
        roof["tensor"]["frac_of_sustained"] = flops / r_ts / t_main
        if roof["bound"] == "tensor":
            roof["peak_sustained"] = r_ts / 1e12
            roof["frac_of_sustained"] = flops / r_ts / t_main
    if r_mix and main_kernel_name(w) == "tc_gauss_fma_kernel" and roof["bound"] == "alu":
        # The exp2 rate that the FMA kernel's own exponent-loop instruction
        # mix reaches without tiles, barriers or tensor-memory traffic
        # (gauss_sum_probe_ex2_mix_rate): the practical ceiling of that loop.
        roof["sfu"]["mix_ceiling_per_s"] = r_mix
        roof["sfu"]["frac_of_mix_ceiling"] = exps / t_main / r_mix
    return roof


class Runner:
    """One workload's inputs on the device and its timed steps."""

    def __init__(self, w, dev, flush):
        import torch
        from paper_2609_04910_gb300.workloads import device_inputs, generate
        self.w = w
        self.dev = dev
        self.flush = flush
        self.inp = generate(w, seed=0)
        self.q, self.k, self.v = device_inputs(self.inp, dev)
        M, D, C = w.M, w.D, w.C
        self.out = torch.empty((M, D if w.grad else C), dtype=torch.float32, device=dev)
        self.s_out = torch.empty((M,), dtype=torch.float32, device=dev) if w.grad else None

    def step(self, main_events=None):
        import paper_2609_04910_gb300 as gs
        w = self.w
        if w.grad:
            gs.gauss_sum_grad_q(self.q, self.k, self.v, w.tau, grad=self.out, s_out=self.s_out,
                                main_events=main_events)
        else:
            gs.gauss_sum(self.q, self.k, self.v, w.tau, out=self.out, main_events=main_events)

    def timed(self, K, W, before=None, after=None):
        """W warm-up steps, then K timed steps, each after an L2 flush, with
        CUDA events around the step; then up to 50 more steps with events
        that the library records around its main kernel (kept out of the
        timed steps: an event between two kernels of a call makes the later
        one launch without overlapping the earlier one's tail).  Returns
        (step ms list, main-kernel ms list, launches in the timed steps)."""
        import torch
        import paper_2609_04910_gb300 as gs
        stream = torch.cuda.current_stream()
        Km = min(K, 50)
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
              for _ in range(K)]
        mev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
               for _ in range(Km)]
        for a, b in ev + mev:  # create the CUDA events before handing them to the library
            a.record(stream)
            b.record(stream)
        for _ in range(W):
            self.flush.zero_()
            self.step()
        gs.gauss_sum_device_status()
        torch.cuda.synchronize()
        if before is not None:
            before()
        launches0 = gs.gauss_sum_kernel_launches()
        for i in range(K):
            self.flush.zero_()
            ev[i][0].record(stream)
            self.step()
            ev[i][1].record(stream)
        launches = gs.gauss_sum_kernel_launches() - launches0
        torch.cuda.synchronize()
        if after is not None:
            after()
        for i in range(Km):
            self.flush.zero_()
            self.step(main_events=mev[i])
        torch.cuda.synchronize()
        gs.gauss_sum_device_status()
        return ([a.elapsed_time(b) for a, b in ev], [a.elapsed_time(b) for a, b in mev],
                launches)

    def e2e(self, K, W, world):
        """The same step from pinned host buffers through the public API:
        H2D of the step's inputs and D2H of its result inside the timed
        region, every step."""
        import numpy as np
        import torch
        import paper_2609_04910_gb300 as gs
        w, inp, dev = self.w, self.inp, self.dev
        stream = torch.cuda.current_stream()

        # The step's inputs live in one pinned host buffer and travel in one
        # copy (q, k and v at 256-byte aligned offsets); the result comes
        # back into a pinned host buffer.
        arrays = [np.ascontiguousarray(inp["k"]), np.ascontiguousarray(inp["v"])]
        if not w.q_is_k:
            arrays.append(np.ascontiguousarray(inp["q"]))
        offs, total = [], 0
        for a in arrays:
            offs.append(total)
            total += (a.nbytes + 255) // 256 * 256
        host = torch.empty(total, dtype=torch.uint8).pin_memory()
        for a, o in zip(arrays, offs):
            host[o:o + a.nbytes].copy_(torch.from_numpy(a.view(np.uint8).reshape(-1)))
        devbuf = torch.empty(total, dtype=torch.uint8, device=dev)
        tdt = {"fp16": torch.float16, "bf16": torch.bfloat16, "fp32": torch.float32}[w.dtype]

        def view(i):
            a = arrays[i]
            return devbuf[offs[i]:offs[i] + a.nbytes].view(tdt).view(a.shape)

        kd, vd = view(0), view(1)
        qd = kd if w.q_is_k else view(2)
        outh = torch.empty(tuple(self.out.shape), dtype=torch.float32).pin_memory()
        sh = torch.empty((w.M,), dtype=torch.float32).pin_memory() if w.grad else None
        outd = torch.empty(tuple(self.out.shape), dtype=torch.float32, device=dev)
        sd = torch.empty((w.M,), dtype=torch.float32, device=dev) if w.grad else None
        e_ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                for _ in range(K)]
        h2d = sum(a.nbytes for a in arrays)
        d2h = outh.numel() * 4 + (w.M * 4 if w.grad else 0)
        for i in range(K + W):
            self.flush.zero_()
            if i >= W:
                e_ev[i - W][0].record(stream)
            devbuf.copy_(host, non_blocking=True)
            if w.grad:
                gs.gauss_sum_grad_q(qd, kd, vd, w.tau, grad=outd, s_out=sd)
                outh.copy_(outd, non_blocking=True)
                sh.copy_(sd, non_blocking=True)
            else:
                gs.gauss_sum(qd, kd, vd, w.tau, out=outd)
                outh.copy_(outd, non_blocking=True)
            if i >= W:
                e_ev[i - W][1].record(stream)
        torch.cuda.synchronize()
        e_ms = statistics.mean(a.elapsed_time(b) for a, b in e_ev)
        e_ms = reduce_max(e_ms, dev)
        return {"value": replica_value(world, w.pairs, e_ms), "unit": UNIT, "ms_per_step": e_ms,
                "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h),
                "steps": K}


OTHER_WORKLOADS = ("svgd_d32", "multi_c64", "offset_d256", "fp32_d16", "mmd_d64_qk")


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
    from paper_2609_04910_gb300.workloads import WORKLOADS

    w = WORKLOADS[args.workload]
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)
    run = Runner(w, dev, flush)

    def barrier():
        if world > 1:
            import torch.distributed as dist
            dist.barrier()

    # Roofline denominators.
    peaks, peak_src = measured_peaks()
    r_x = gs.gauss_sum_probe_ex2_rate()
    r_mix = gs.gauss_sum_probe_ex2_mix_rate()
    props = torch.cuda.get_device_properties(dev)
    sms = props.multi_processor_count

    K, W = max(1, args.steps), max(3, args.warmup)
    sampler = ClockSampler(local, enabled=not args.no_clocks)

    def start():
        time.sleep(0.3 if not args.no_clocks else 0.0)
        barrier()
        torch.cuda.synchronize()

    wall = {}

    def t0():
        start()
        wall["t0"] = time.perf_counter()

    def t1():
        barrier()
        wall["t"] = time.perf_counter() - wall["t0"]

    step_ms, main_ms, launches = run.timed(K, W, before=t0, after=t1)
    wall = wall["t"]
    ms = reduce_max(statistics.mean(step_ms), dev)
    main_mean = statistics.mean(main_ms)
    e2e = None if args.no_e2e else run.e2e(min(K, 200), W, world)
    clocks = sampler.stop() if sampler is not None else None

    traffic, traffic_src = profiled_traffic(w)
    roof = roofline_of(w, main_mean, peaks, peak_src, sms, r_x, traffic, traffic_src, r_mix)

    # The other configurations, measured the same way (fewer steps) so that
    # every configuration has a number from this run.
    others = None
    if rank == 0 and world == 1 and not args.no_other_workloads:
        others = {}
        del run
        torch.cuda.empty_cache()
        for name in OTHER_WORKLOADS:
            wo = WORKLOADS[name]
            try:
                ro = Runner(wo, dev, flush)
                s_ms, m_ms, n_l = ro.timed(min(K, 20), W)
                tr, tr_src = profiled_traffic(wo)
                rf = roofline_of(wo, statistics.mean(m_ms), peaks, peak_src, sms, r_x, tr,
                                 tr_src, r_mix=r_mix)
                others[name] = {
                    "config": workload_config(wo), "steps": len(s_ms),
                    "ms_per_step": statistics.mean(s_ms), "value": wo.pairs / (statistics.mean(s_ms) * 1e-3),
                    "unit": UNIT, "main_kernel_ms": statistics.mean(m_ms),
                    "main_kernel_ms_min": min(m_ms), "gpu_launches": n_l, "roofline": rf}
                del ro
                torch.cuda.empty_cache()
            except Exception as exc:  # report, keep the headline line
                others[name] = {"error": f"{type(exc).__name__}: {exc}"}

    fp16_tf = None
    if rank == 0 and not args.no_peak_probe:
        fp16_tf = probe_fp16_tflops(dev)

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        from oracle import build_oracle
        from paper_2609_04910_gb300.workloads import generate
        build_oracle()
        rate, rows, el, threads = time_oracle(generate(w, seed=0), args.cpu_seconds)
        cpu = {"value": rate, "unit": UNIT, "cores": threads, "kind": "oracle",
               "cpu_model": cpu_model(),
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
            "fp16_matmul_tflops_probe": fp16_tf,
            "other_workloads": others,
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()
    return 0


BATCHED_CASES = ((64, 16384, 16), (64, 16384, 32), (64, 16384, 64), (64, 16384, 128),
                 (4, 65536, 64), (64, 4096, 64), (256, 1024, 64))


def run_batched(args):
    """gauss_sum_batched on the benchmark shape of Sec. 4 (B independent
    Gaussian clouds, M = N = n points each, C = 1, fp16, tau = 1/D): 3
    warm-up calls, then 8 timed calls (the paper's protocol), each after an
    L2 flush, CUDA events around the whole call.  The roofline is the
    slower of the dense tensor work 2 B n^2 (D + 1) at the measured bf16
    peak and the B n^2 exponentials at the MUFU rate."""
    import torch
    from paper_2609_04910_gb300.build import build_library
    build_library()
    import paper_2609_04910_gb300 as gs
    from paper_2609_04910_gb300.workloads import batched_clouds, to_device
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    peaks, peak_src = measured_peaks()
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    r_x = 32.0 * sms * float(peaks.get("sm_max_mhz", 2070.0)) * 1e6
    r_t = float(peaks.get("bf16_tflops", FALLBACK_PEAKS["bf16_tflops"])) * 1e12
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream()
    sampler = ClockSampler(0, enabled=not args.no_clocks)
    for B, n, D in BATCHED_CASES:
        inp = batched_clouds(B, n, D)
        q, k, v = (to_device(inp[x], "fp16", dev) for x in ("q", "k", "v"))
        out = torch.empty((B, n, 1), dtype=torch.float32, device=dev)
        for _ in range(3):
            gs.gauss_sum_batched(q, k, v, inp["tau"], out=out)
        torch.cuda.synchronize()
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
              for _ in range(8)]
        for a, b in ev:
            flush.zero_()
            a.record(stream)
            gs.gauss_sum_batched(q, k, v, inp["tau"], out=out)
            b.record(stream)
        torch.cuda.synchronize()
        gs.gauss_sum_device_status()
        ms = [a.elapsed_time(b) for a, b in ev]
        t = statistics.mean(ms) * 1e-3
        pairs = float(B) * n * n
        t_x, t_t = pairs / r_x, 2.0 * pairs * (D + 1) / r_t
        print(json.dumps({
            "case": f"batched B={B} M=N={n} D={D} C=1 fp16", "B": B, "n": n, "D": D,
            "ms_mean": statistics.mean(ms), "ms_std": statistics.pstdev(ms), "ms_min": min(ms),
            "pairs_per_s": pairs / t, "tflops": 2.0 * pairs * (D + 1) / t / 1e12,
            "bound": "alu" if t_x >= t_t else "tensor", "roofline_frac": max(t_x, t_t) / t,
            "ex2_frac": t_x / t, "tensor_frac": t_t / t,
            "peaks": f"MUFU 32/clk/SM x {sms} SMs at max clock; {peak_src} bf16 {r_t / 1e12:.1f} TFLOP/s",
            "l2": "flushed (512 MiB write) before every timed call", "timing": "whole call, CUDA events"}),
            flush=True)
        del q, k, v, out
        torch.cuda.empty_cache()
    clocks = sampler.stop() if sampler is not None else None
    print(json.dumps({"batched_clocks": clocks}), flush=True)


def main(argv=None):
    args = parse_args(argv)
    if args.impl == "reference":
        return run_reference(args)
    if args.batched:
        return run_batched(args)
    return run_own(args)


if __name__ == "__main__":
    sys.exit(main())
