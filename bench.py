#!/usr/bin/env python3
"""Benchmark: whole benchmarking commands per second on GB300.

A step is one benchmarking command (the paper's Section 2.1): generate the
seeded inputs, run the reference, run the candidate once, check it, then time
the candidate in a critical region (drain, L2 flush, warm-up, timed
iterations each preceded by an L2-flush write).  Every step is one
``krex_command_run`` call into libkrex.so.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME]
  python bench.py --impl reference ...   # the CPU oracle, timed on host cores

The JSON line carries: value (commands/s, device-timed with inputs resident),
e2e (the same metric with host-resident inputs and outputs copied inside the
timed region), roofline (the GEMM kernel, from the per-iteration CUDA events
of the commands' timed loops), kernels (each kernel of the path timed alone
with CUDA events), cpu_baseline (the oracle on a bounded sample), clocks.
Under torchrun (N > 1) every rank runs independent commands on its own GPU
(replicas; no data-path collective) and rank 0 reports the aggregate.
"""
from __future__ import annotations

import argparse
import csv
import ctypes
import hashlib
import io
import json
import math
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "GEMM TFLOP/s & fill/flush/softmax/check GB/s vs roofline; bench cmds/s, 1 GB300"
DEFAULT_WORKLOAD = "gemm_bf16_4096"
SOFTMAX_WORKLOAD = "softmax_f32_65536x8192"
# 32-bit integer-ALU operations the uniform generator's definition takes per
# 16-bit element: per SplitMix64 draw (two elements) a 64-bit add (2) and three
# 64-bit xor-shifts (2 funnel shifts + 2 xors each: 12); per element the 24-bit
# field to [-1, 1) (a shift, two masks, an integer subtract: 4).  The two 64-bit
# multiplies per draw run on the multiply-add pipe and are not counted.
FILL_ALU_OPS_PER_ELEMENT = (2 + 12) / 2 + 4


def _peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return {"hbm_gbs": d["hbm_gbs"], "bf16_tflops": d["bf16_tflops"],
                "bf16_tflops_sustained": d.get("bf16_tflops_sustained"), "source": "measured"}
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0, "source": "fallback"}


# ------------------------------------------------------------ clocks --------

class ClockSampler:
    """nvidia-smi sampling of SM clocks and throttle reasons during the timed region."""
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index: int):
        self.dev = device_index
        self.proc = None
        self.out = b""

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits", "-lms", "100",
                 "-i", str(self.dev)], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None
        time.sleep(0.3)
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            time.sleep(0.2)
            self.proc.terminate()
            try:
                self.out, _ = self.proc.communicate(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
                self.out, _ = self.proc.communicate()

    def summary(self):
        if self.proc is None:
            return None
        rows = []
        for r in csv.reader(io.StringIO(self.out.decode(errors="replace"))):
            if len(r) < 8:
                continue
            try:
                rows.append([x.strip() for x in r])
            except ValueError:
                pass
        if not rows:
            return None
        sm = [float(r[0]) for r in rows if r[0].replace(".", "", 1).isdigit()]
        mx = [float(r[1]) for r in rows if r[1].replace(".", "", 1).isdigit()]
        pw = [float(r[2]) for r in rows if r[2].replace(".", "", 1).isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[4 + i].lower() == "active"})
        loaded = sorted(sm)[len(sm) // 2:] if sm else []
        return {"sm_mhz": statistics.median(loaded) if loaded else None, "sm_max_mhz": max(mx) if mx else None,
                "power_w_max": max(pw) if pw else None, "samples": len(rows), "reasons": reasons}


# ------------------------------------------------------------ helpers -------

def _src_hash(path: str) -> str:
    with open(path, "rb") as f:
        return hashlib.sha256(f.read()).hexdigest()[:16]


def _ncu_traffic(kernel: str, workload: str):
    """DRAM bytes per launch of `kernel` from the committed ncu summary, or None
    if the kernel source changed since the capture."""
    p = os.path.join(ROOT, "profiles", "ncu_traffic.json")
    if not os.path.exists(p):
        return None
    with open(p) as f:
        d = json.load(f)
    e = d.get(kernel, {}).get(workload)
    if not e:
        return None
    src = os.path.join(ROOT, e["source"])
    if not os.path.exists(src) or _src_hash(src) != e["source_sha256_16"]:
        return None
    return e["dram_bytes_per_launch"]


def _time_launches(fn, n, stream, flush=None):
    """Mean device time of `fn` over n launches, CUDA events on `stream`; an
    L2-flush write (not timed) precedes each launch when `flush` is given."""
    import torch
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(n)]
    for i in range(n):
        if flush is not None:
            flush()
        evs[i][0].record(stream)
        fn()
        evs[i][1].record(stream)
    stream.synchronize()
    return statistics.fmean(a.elapsed_time(b) for a, b in evs)


def kernel_table(ws, w, peaks, stream):
    """Each kernel of the path timed alone (after warm-up, L2 flushed before
    every launch), with its algorithmic bytes or flops per launch."""
    import torch
    import paper_2609_30057_gb300 as krex
    from paper_2609_30057_gb300.command import WORKLOADS, Workspace
    if not w.is_gemm:               # the GEMM rows run at the GEMM workload's size
        w = WORKLOADS[DEFAULT_WORKLOAD]
        ws = Workspace(w)
    flush_t = ws.flush
    flush = lambda: krex.krex_flush_l2(flush_t, stream=stream)  # noqa: E731
    out = {}

    # integer-ALU roofline of the uniform fill: 64 ALU lanes per clock per SM
    # at the 2070 MHz maximum SM clock (the clock the runs see under load)
    alu_peak = torch.cuda.get_device_properties(stream.device).multi_processor_count * 64 * 2.070e9

    def rec(name, fn, nbytes=None, flops=None, alu_ops=None, n=20, do_flush=True):
        for _ in range(3):
            fn()
        ms = _time_launches(fn, n, stream, flush if do_flush else None)
        e = {"ms": ms}
        if nbytes is not None:
            gbs = nbytes / ms / 1e6
            e.update({"GB/s": gbs, "frac_hbm": gbs / peaks["hbm_gbs"], "bytes": nbytes})
        if flops is not None:
            tf = flops / ms / 1e9
            e.update({"TFLOP/s": tf, "frac_bf16": tf / peaks["bf16_tflops"], "flops": flops})
        if alu_ops is not None:
            e.update({"bound": "alu", "alu_ops": alu_ops, "Tops/s": alu_ops / ms / 1e9,
                      "frac_alu": alu_ops / ms * 1e3 / alu_peak})
        out[name] = e

    A, B = ws.inputs
    rec("fill_uniform_bf16", lambda: krex.krex_gen_inputs(w.seed, 0, 0, 0.0, A, stream), nbytes=A.numel() * 2,
        alu_ops=A.numel() * FILL_ALU_OPS_PER_ELEMENT)
    big = torch.empty(16384, 16384, dtype=torch.bfloat16, device=A.device)   # steady state, 512 MiB
    rec("fill_uniform_bf16_16384", lambda: krex.krex_gen_inputs(w.seed, 0, 0, 0.0, big, stream),
        nbytes=big.numel() * 2, alu_ops=big.numel() * FILL_ALU_OPS_PER_ELEMENT, n=10)
    del big
    rec("flush_l2", flush, nbytes=flush_t.numel(), do_flush=False)
    rec("gemm_ref_simt", lambda: krex.krex_run_reference(w.op, ws.inputs, ws.ref, stream), flops=w.flops, n=3)
    rec("gemm_tcgen05", lambda: krex.krex_run_candidate_ws(w.op, ws.inputs, ws.out, ws.gemm_ws, stream),
        flops=w.flops)
    scratch = ws.check_scratch
    rec("check_bf16_f32", lambda: krex.krex_check_launch(ws.out, ws.ref, w.atol, w.rtol, scratch, stream),
        nbytes=ws.out.numel() * 6, n=10)
    # the bandwidth-bound candidate at its own workload size
    sw = WORKLOADS[SOFTMAX_WORKLOAD]
    x = torch.empty(sw.M, sw.N, dtype=torch.float32, device=A.device)
    y = torch.empty_like(x)
    rec("fill_normal_f32", lambda: krex.krex_gen_inputs(sw.seed, 0, 1, sw.sigma, x, stream), nbytes=x.numel() * 4,
        n=10)
    rec("softmax_f32", lambda: krex.krex_run_candidate(1, [x], y, stream), nbytes=x.numel() * 8, n=10)
    rec("check_f32_f32", lambda: krex.krex_check_launch(y, x, 1e-6, 0.0, scratch, stream), nbytes=x.numel() * 8, n=5)
    del x, y
    # the fp16 form of the GEMM candidate at the same size
    fw = WORKLOADS["gemm_f16_4096"]
    a16 = torch.empty(fw.M, fw.K, dtype=torch.float16, device=A.device)
    b16 = torch.empty(fw.K, fw.N, dtype=torch.float16, device=A.device)
    c16 = torch.empty(fw.M, fw.N, dtype=torch.float16, device=A.device)
    rec("fill_uniform_f16", lambda: krex.krex_gen_inputs(fw.seed, 0, 0, 0.0, a16, stream), nbytes=a16.numel() * 2,
        alu_ops=a16.numel() * FILL_ALU_OPS_PER_ELEMENT)
    krex.krex_gen_inputs(fw.seed, 1, 0, 0.0, b16, stream)
    rec("gemm_tcgen05_f16", lambda: krex.krex_run_candidate_ws(fw.op, [a16, b16], c16, ws.gemm_ws, stream),
        flops=fw.flops)
    del a16, b16, c16
    torch.cuda.empty_cache()
    return out


# ---------------------------------------------------------- CPU oracle ------

def oracle_command_cost(w, budget_s: float = 10.0):
    """Seconds one benchmarking command of workload `w` takes when the oracle
    does its arithmetic on the host: generate the inputs, the GEMM once for the
    reference and once per candidate run (1 + warm-up + iters), the check.
    Bounded sample: the GEMM is timed on a block of output rows and scaled by
    M / rows; generation and the check run in full.  Returns (seconds, info)."""
    import numpy as np
    from oracle import gen, ref
    t0 = time.perf_counter()
    if w.is_gemm:
        a = gen.uniform(w.dtype, w.seed, 0, w.M, w.K)
        b = gen.uniform(w.dtype, w.seed, 1, w.K, w.N)
    else:
        x = gen.normal_f32(w.seed, 0, min(w.M, 2048), w.N, w.sigma)
    t_gen = time.perf_counter() - t0
    if not w.is_gemm:
        t_gen *= w.M / min(w.M, 2048)
    rows = 0
    t_work = 0.0
    reps = 0
    tb = time.perf_counter()
    block = 64 if w.is_gemm else 256
    while time.perf_counter() - tb < budget_s * 0.6 and rows < w.M:
        t1 = time.perf_counter()
        if w.is_gemm:
            c = ref.gemm_f64(a[rows % w.M:rows % w.M + block], b, dtype=w.dtype)
        else:
            c = ref.softmax_rows_f64(x[:block].astype(np.float64))
        t_work += time.perf_counter() - t1
        rows += block
        reps += 1
    per_full = t_work * (w.M / rows)
    t1 = time.perf_counter()
    n_chk = min(w.M, 2048)
    o32 = c[:1].astype(np.float32).repeat(n_chk, axis=0)
    ref.check_f32(o32, o32, w.atol, w.rtol)
    t_chk = (time.perf_counter() - t1) * (w.M / n_chk)
    runs = 1 + 1 + w.warmup + w.iters
    total = t_gen + runs * per_full + t_chk
    info = (f"oracle command of {w.name}: input generation in full (single thread), "
            f"{'fp64 GEMM' if w.is_gemm else 'fp64 softmax'} on {rows} of {w.M} output rows scaled to the full "
            f"output and counted {runs}x (reference + check run + {w.warmup} warm-up + {w.iters} timed), "
            f"fp32 check on {n_chk} rows scaled; sample wall {time.perf_counter() - t0:.1f} s")
    in_bytes = (w.M * w.K + w.K * w.N) * 2 if w.is_gemm else w.M * w.N * 4
    comp = {"gen_GB_per_s": in_bytes / t_gen / 1e9, "check_GB_per_s": w.M * w.N * (6 if w.is_gemm else 8) / t_chk / 1e9}
    if w.is_gemm:
        comp["gemm_fp64_GFLOP_per_s"] = 2.0 * w.M * w.N * w.K / per_full / 1e9
    else:
        comp["softmax_fp64_rows_per_s"] = w.M / per_full
    return total, info, comp


def _p95(xs) -> float:
    """Linear-interpolation percentile 0.95 (the percentile method of the timed loop)."""
    v = sorted(xs)
    h = (len(v) - 1) * 0.95
    lo = int(h)
    return v[lo] if lo + 1 >= len(v) else v[lo] + (h - lo) * (v[lo + 1] - v[lo])


def cpu_cores() -> int:
    return len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else (os.cpu_count() or 1)


def cpu_model() -> str:
    """The host CPU's model name as lscpu reports it (the machine type if lscpu is missing)."""
    import platform
    import subprocess
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.strip().lower().startswith("model name:"):
                return line.split(":", 1)[1].strip()
    except (OSError, subprocess.SubprocessError):
        pass
    return platform.machine()


# ------------------------------------------------------------- main ---------

def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD)
    ap.add_argument("--no-kernels", action="store_true", help="skip the per-kernel table")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--kernel-only", default=None,
                    choices=["gemm", "gemm_ref", "fill_uniform", "fill_normal", "flush", "check", "softmax"],
                    help="launch one kernel of the workload --launches times and exit (for ncu captures)")
    ap.add_argument("--launches", type=int, default=3)
    args = ap.parse_args()

    from paper_2609_30057_gb300 import replicas
    rank, world, local_rank = replicas.rank_world()

    if args.impl == "reference":
        return reference_arm(args, rank, world)
    if args.kernel_only:
        return kernel_only(args)

    import torch
    import paper_2609_30057_gb300 as krex
    from paper_2609_30057_gb300.command import WORKLOADS, Workspace

    torch.cuda.set_device(local_rank)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local_rank))
    if rank == 0 or world > 1:
        krex.build()
    if world > 1:
        dist.barrier()

    w = WORKLOADS[args.workload]
    peaks = _peaks()
    ws = Workspace(w)
    stream = torch.cuda.current_stream()

    def barrier():
        replicas.barrier(dist)

    for _ in range(args.warmup):
        r = ws.run()
        if not r.passed:
            raise SystemExit(f"check failed during warm-up: {r.check.n_violations} violations")

    # ------------------------------------------------ timed region (value)
    gemm_ms, p50s, p95s, phases = [], [], [], []
    clocks = ClockSampler(torch.cuda.current_device())
    barrier()
    torch.cuda.synchronize()
    launches0 = krex.krex_launch_count()
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with clocks:
        ev0.record(stream)
        t0 = time.perf_counter()
        for _ in range(args.steps):
            r = ws.run()
            if not r.passed:
                raise SystemExit(f"check failed: {r.check.n_violations} violations")
            gemm_ms.extend(ws.durations[: r.n_iters])
            p50s.append(r.p50_ms)
            p95s.append(r.p95_ms)
            phases.append(list(r.phase_ms))
        ev1.record(stream)
        torch.cuda.synchronize()
        wall = time.perf_counter() - t0
    barrier()
    launches = int(replicas.sum_over_ranks(dist, krex.krex_launch_count() - launches0, device="cuda"))
    # a kernel whose bounded wait ran out returned early: no valid number
    status = krex.krex_device_status()
    if status:
        raise SystemExit(f"a kernel reported device status {status:#x} during the timed region")
    elapsed_ms = replicas.max_over_ranks(dist, ev0.elapsed_time(ev1), device="cuda")
    value = replicas.aggregate_throughput(args.steps, world, elapsed_ms / 1e3)

    # ------------------------------------------------ e2e (host buffers)
    e2e = None
    if not args.no_e2e:
        host_in = [torch.empty(t.shape, dtype=t.dtype).pin_memory() for t in ws.inputs]
        for h, t in zip(host_in, ws.inputs):
            h.copy_(t)
        host_out = torch.empty(ws.out.shape, dtype=ws.out.dtype).pin_memory()
        ptrs = [h.data_ptr() for h in host_in]
        for _ in range(max(1, args.warmup)):
            ws.run(host_in=ptrs, host_out=host_out.data_ptr())
        barrier()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(args.steps):
            r = ws.run(host_in=ptrs, host_out=host_out.data_ptr())
            if not r.passed:
                raise SystemExit("check failed (e2e)")
        e1.record(stream)
        torch.cuda.synchronize()
        barrier()
        te_ms = replicas.max_over_ranks(dist, e0.elapsed_time(e1), device="cuda")
        e2e = {"value": replicas.aggregate_throughput(args.steps, world, te_ms / 1e3), "unit": "cmds/s",
               "h2d_bytes_per_step": sum(h.numel() * h.element_size() for h in host_in),
               "d2h_bytes_per_step": host_out.numel() * host_out.element_size() + 16}

    kernels = None if args.no_kernels or rank != 0 else kernel_table(ws, w, peaks, stream)

    if rank != 0:
        if dist is not None:
            dist.destroy_process_group()
        return

    # ------------------------------------------------ roofline (GEMM kernel)
    mean_gemm_ms = statistics.fmean(gemm_ms)
    if w.is_gemm:
        achieved = w.flops / (mean_gemm_ms / 1e3) / 1e12
        roofline = {"bound": "tensor", "achieved": achieved, "peak": peaks["bf16_tflops"], "unit": "TFLOP/s",
                    "frac": achieved / peaks["bf16_tflops"], "traffic": _ncu_traffic("gemm_tcgen05", w.name),
                    "peak_kind": f"bf16 dense burst, {peaks['source']} (MEASURED_PEAKS.json)",
                    "frac_of_sustained": (achieved / peaks["bf16_tflops_sustained"]
                                          if peaks.get("bf16_tflops_sustained") else None),
                    "kernel": "gemm_tcgen05_2sm", "launches_timed": len(gemm_ms),
                    "algorithmic_flops_per_launch": w.flops}
    else:
        # the bandwidth-bound candidate: one read and one write of the matrix
        achieved = w.candidate_bytes / (mean_gemm_ms / 1e3) / 1e9
        roofline = {"bound": "hbm", "achieved": achieved, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                    "frac": achieved / peaks["hbm_gbs"], "traffic": _ncu_traffic("softmax_rows", w.name),
                    "peak_kind": f"HBM copy, {peaks['source']} (MEASURED_PEAKS.json)",
                    "kernel": "softmax_rows_reg", "launches_timed": len(gemm_ms),
                    "algorithmic_bytes_per_launch": w.candidate_bytes}

    cpu = None
    if not args.no_cpu_baseline and world == 1:   # the host baseline is a single-GPU figure
        secs, info, comp = oracle_command_cost(w)
        cpu = {"value": 1.0 / secs, "unit": "cmds/s", "cores": cpu_cores(), "kind": "oracle", "sample": info,
               "components": comp, "cpu_model": cpu_model()}

    cs = clocks.summary()
    ph = [statistics.fmean(p[i] for p in phases) for i in range(5)]
    line = {
        "metric": METRIC, "value": value, "unit": "cmds/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": elapsed_ms / args.steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": {"bf16": "bf16", "f16": "f16"}.get(w.dtype, "f32"), "data": "synthetic",
        "config": {"workload": w.name, "M": w.M, "N": w.N, "K": w.K, "seed": w.seed, "timed_iters": w.iters,
                   "warmup_iters": w.warmup, "flush_bytes": w.flush_bytes,
                   "l2": "flushed: a flush_bytes write precedes every timed candidate iteration and region entry",
                   "parallelism": f"replicas{world}"},
        "roofline": roofline,
        "cpu_baseline": cpu,
        "e2e": e2e,
        "gpu_launches": launches,
        "clocks": cs,
        "timing_spread": {"p50_ms_median": statistics.median(p50s), "p95_ms_median": statistics.median(p95s),
                          "p95_over_p50_minus_1": statistics.median(p95s) / statistics.median(p50s) - 1.0,
                          # Eq. 1 across the commands: p95 of (command median / overall median) - 1
                          "P_across_commands": _p95([p / statistics.median(p50s) for p in p50s]) - 1.0},
        "phase_ms": dict(zip(["inputs", "reference", "candidate", "check", "timed_loop"], ph)),
        "kernels": kernels,
        "host_wall_s": wall,
    }
    print(json.dumps(line))
    if dist is not None:
        dist.destroy_process_group()


def kernel_only(args):
    """Set up the workload (or the softmax workload for softmax / fill_normal),
    then launch one kernel --launches times; used for ncu captures."""
    import torch
    import paper_2609_30057_gb300 as krex
    from paper_2609_30057_gb300.command import WORKLOADS, Workspace
    krex.build()
    torch.cuda.set_device(0)
    stream = torch.cuda.current_stream()
    name = args.workload
    if args.kernel_only in ("softmax", "fill_normal") and WORKLOADS[name].is_gemm:
        name = SOFTMAX_WORKLOAD
    w = WORKLOADS[name]
    ws = Workspace(w)
    k = args.kernel_only
    # minimal set-up: inputs, and for the check the two outputs it compares
    if w.is_gemm:
        krex.krex_gen_inputs(w.seed, 0, 0, 0.0, ws.inputs[0], stream)
        krex.krex_gen_inputs(w.seed, 1, 0, 0.0, ws.inputs[1], stream)
    else:
        krex.krex_gen_inputs(w.seed, 0, 1, w.sigma, ws.inputs[0], stream)
    if k == "check":
        krex.krex_run_reference(w.op, ws.inputs, ws.ref, stream)
        krex.krex_run_candidate(w.op, ws.inputs, ws.out, stream)
    fn = {
        "gemm": lambda: krex.krex_run_candidate_ws(w.op, ws.inputs, ws.out, ws.gemm_ws, stream),
        "gemm_ref": lambda: krex.krex_run_reference(w.op, ws.inputs, ws.ref, stream),
        "fill_uniform": lambda: krex.krex_gen_inputs(w.seed, 0, 0, 0.0, ws.inputs[0], stream),
        "fill_normal": lambda: krex.krex_gen_inputs(w.seed, 0, 1, w.sigma, ws.inputs[0], stream),
        "flush": lambda: krex.krex_flush_l2(ws.flush, stream=stream),
        "check": lambda: krex.krex_check(ws.out, ws.ref, w.atol, w.rtol, ws.check_scratch, stream),
        "softmax": lambda: krex.krex_run_candidate(1, ws.inputs, ws.out, stream),
    }[k]
    for _ in range(args.launches):
        if k != "flush":
            krex.krex_flush_l2(ws.flush, stream=stream)
        fn()
    torch.cuda.synchronize()
    assert krex.krex_device_status() == 0
    print(json.dumps({"kernel_only": k, "workload": w.name, "launches": args.launches}))


def reference_arm(args, rank, world):
    """The oracle as the reference arm: each step is one bounded-sample oracle
    command on the host cores; rank 0 alone runs it."""
    if rank != 0:
        return
    from paper_2609_30057_gb300.command import WORKLOADS
    w = WORKLOADS[args.workload]
    budget = max(1.0, min(10.0, 150.0 / max(1, args.steps + args.warmup)))
    for _ in range(args.warmup):
        oracle_command_cost(w, budget)
    secs = []
    info = ""
    comp = {}
    for _ in range(args.steps):
        s, info, comp = oracle_command_cost(w, budget)
        secs.append(s)
    value = args.steps / sum(secs)
    line = {"metric": METRIC, "value": value, "unit": "cmds/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": 1e3 * sum(secs) / args.steps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": w.name, "M": w.M, "N": w.N, "K": w.K, "seed": w.seed, "timed_iters": w.iters,
                       "parallelism": "host"},
            "impl": "reference",
            "cpu_baseline": {"value": value, "unit": "cmds/s", "cores": cpu_cores(), "kind": "oracle",
                             "sample": info, "components": comp, "cpu_model": cpu_model()},
            "e2e": {"value": value, "unit": "cmds/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line))


if __name__ == "__main__":
    main()
