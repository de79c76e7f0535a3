#!/usr/bin/env python3
"""Benchmark: whole benchmarking commands per second on GB300.

A step is one benchmarking command (the paper's Section 2.1): generate the
seeded inputs, run the candidate once and the reference, check it, then time
the candidate in a critical region (drain, L2 flush, warm-up, timed
iterations each preceded by an L2-flush write).  Every step is one
``krex_command_run`` call into libkrex.so.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME]
  python bench.py --impl reference ...   # the CPU oracle, timed on host cores

The default workload is the 16384^3 GEMM command, 32 commands per
measurement.  The JSON line carries: value (commands/s, device-timed with
inputs resident), e2e (the same metric with host-resident inputs and outputs
copied inside the timed region), roofline (the command's dominant kernel by device
time: the CUDA-core reference GEMM on the FP32 FMA pipe at 16384^3, the
tcgen05 GEMM candidate at 4096^3 and 8192^3; from CUDA events in the timed
commands), roofline_other_gemm (the other of the two),
configs (one sub-record per workload of the configuration list: commands/s,
the candidate's roofline, p50/p95, P across commands), kernels (each kernel
of the path timed alone with CUDA events), cpu_baseline (the oracle on a
bounded sample, measured), clocks.
Under torchrun (N > 1) every rank runs independent commands on its own GPU
(replicas; no data-path collective) and rank 0 reports the aggregate.
"""
from __future__ import annotations

import argparse
import csv
import hashlib
import io
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "GEMM TFLOP/s & fill/flush/softmax/check GB/s vs roofline; bench cmds/s, 1 GB300"
# the headline: the 16384^3 GEMM command, repeated 32 times to report commands/s
DEFAULT_WORKLOAD = "gemm_bf16_16384"
# every workload of the configuration list, each measured as a sub-record, with
# the number of commands timed for it
CONFIG_WORKLOADS = {"gemm_bf16_256": 32, "gemm_bf16_4096": 20, "softmax_f32_65536x8192": 10,
                    "gemm_bf16_8192": 8, "gemm_bf16_16384": 32}
SOFTMAX_WORKLOAD = "softmax_f32_65536x8192"
SMALL_GEMM_WORKLOAD = "gemm_bf16_4096"
# Output bytes per SplitMix64 draw: two bf16 (uniform) or two fp32 (normal).
DRAW_BYTES = {0: 4, 1: 8}
# FP32 fused multiply-add lanes per SM (the CUDA-core reference GEMM's pipe)
FMA_LANES_PER_SM = 128


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

def code_text(src: str) -> str:
    """C/C++/CUDA source with its comments removed and every run of whitespace
    made one space: what the compiler sees, so an edit of comments or layout
    leaves it unchanged and any other edit changes it.  String and character
    literals are kept whole (a // inside one is not a comment)."""
    out, i, n = [], 0, len(src)
    while i < n:
        c = src[i]
        if c in "\"'":
            j = i + 1
            while j < n and src[j] != c:
                j += 2 if src[j] == "\\" else 1
            out.append(src[i:j + 1])
            i = j + 1
        elif src.startswith("//", i):
            j = src.find("\n", i)
            i = n if j < 0 else j
        elif src.startswith("/*", i):
            j = src.find("*/", i + 2)
            i = n if j < 0 else j + 2
            out.append(" ")
        else:
            out.append(c)
            i += 1
    return " ".join("".join(out).split())


def code_hash(path: str) -> str:
    """First 16 hex digits of the sha256 of code_text(path)."""
    with open(path, encoding="utf-8") as f:
        return hashlib.sha256(code_text(f.read()).encode()).hexdigest()[:16]


def _ncu_traffic(kernel: str, workload: str):
    """DRAM bytes per launch of `kernel` from the committed ncu summary, or None
    if the kernel's code changed since the capture (the record keeps the hash
    of the code it was taken on; edits of comments alone keep it valid)."""
    p = os.path.join(ROOT, "profiles", "ncu_traffic.json")
    if not os.path.exists(p):
        return None
    with open(p) as f:
        d = json.load(f)
    e = d.get(kernel, {}).get(workload)
    if not e:
        return None
    src = os.path.join(ROOT, e["source"])
    if not os.path.exists(src) or code_hash(src) != e["code_sha256_16"]:
        return None
    return e["dram_bytes_per_launch"]


def _time_launches(fn, n, stream, flush=None, best=False):
    """Mean (best=True: shortest) device time of `fn` over n launches, CUDA
    events on `stream`; an L2-flush write (not timed) precedes each launch
    when `flush` is given."""
    import torch
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(n)]
    for i in range(n):
        if flush is not None:
            flush()
        evs[i][0].record(stream)
        fn()
        evs[i][1].record(stream)
    stream.synchronize()
    times = [a.elapsed_time(b) for a, b in evs]
    return min(times) if best else statistics.fmean(times)


def kernel_table(peaks, stream, gemm_names=(SMALL_GEMM_WORKLOAD, DEFAULT_WORKLOAD)):
    """Each kernel of the path timed alone (after warm-up, L2 flushed before
    every launch), with its algorithmic bytes or flops per launch: the GEMM
    path's kernels at the sizes of `gemm_names`, the softmax path's at its
    workload's size.  The fills come first and the largest GEMMs last: after
    seconds of those the power controller holds the SM clock down for a while
    (GB300, sw_power_cap), which would charge the next kernels for it."""
    import torch
    import paper_2609_30057_gb300 as krex
    from paper_2609_30057_gb300.command import WORKLOADS, Workspace
    out = {}
    dev = torch.cuda.current_device()
    n_sm = torch.cuda.get_device_properties(dev).multi_processor_count
    # the fills at the headline sizes beside their compute ceilings, first
    # (before seconds of GEMMs leave the clock under the power cap), each
    # launched alternately with its generator probe
    sw = WORKLOADS[SOFTMAX_WORKLOAD]
    flush_buf = torch.empty(256 << 20, dtype=torch.uint8, device="cuda")
    flush0 = lambda: krex.krex_flush_l2(flush_buf, stream=stream)  # noqa: E731
    ceiling, fill_ms = {}, {}
    big = torch.empty(16384, 16384, dtype=torch.bfloat16, device="cuda")
    ceiling[0], fill_ms[0] = fill_beside_ceiling(
        0, n_sm, stream, lambda: krex.krex_gen_inputs(1, 0, 0, 0.0, big, stream), big.numel(), flush0)
    del big
    big = torch.empty(sw.M, sw.N, dtype=torch.float32, device="cuda")
    ceiling[1], fill_ms[1] = fill_beside_ceiling(
        1, n_sm, stream, lambda: krex.krex_gen_inputs(sw.seed, 0, 1, sw.sigma, big, stream), big.numel(), flush0)
    del big, flush_buf
    torch.cuda.empty_cache()
    out["generator_probe_uniform@16384"] = ceiling[0]
    out["generator_probe_normal@65536x8192"] = ceiling[1]
    for dist, name, nbytes in ((0, "fill_uniform_bf16@16384", 16384 * 16384 * 2),
                               (1, "fill_normal_f32", sw.M * sw.N * 4)):
        gbs = nbytes / fill_ms[dist] / 1e6
        out[name] = {"ms": fill_ms[dist], "launches": 10, "GB/s": gbs, "frac_hbm": gbs / peaks["hbm_gbs"],
                     "bytes": nbytes, "bound": "alu", "peak_GB/s": ceiling[dist]["GB/s"],
                     "frac_alu": gbs / ceiling[dist]["GB/s"]}

    def rec(name, fn, flush, nbytes=None, flops=None, gen_dist=None, n=20, fma_peak=None):
        for _ in range(3):
            fn()
        ms = _time_launches(fn, n, stream, flush)
        e = {"ms": ms, "launches": n}
        if nbytes is not None:
            gbs = nbytes / ms / 1e6
            e.update({"GB/s": gbs, "frac_hbm": gbs / peaks["hbm_gbs"], "bytes": nbytes})
        if flops is not None:
            tf = flops / ms / 1e9
            e.update({"TFLOP/s": tf, "flops": flops})
            if fma_peak is None:
                e["frac_bf16"] = tf / peaks["bf16_tflops"]
            else:
                e.update({"bound": "fp32 fma", "frac_fma": tf * 1e12 / fma_peak})
        if gen_dist is not None:
            # compute-bound generator: its roofline is the measured rate of
            # its own per-draw arithmetic (fill_beside_ceiling)
            c = ceiling[gen_dist]["GB/s"]
            e.update({"bound": "alu", "peak_GB/s": c, "frac_alu": (nbytes / ms / 1e6) / c})
        out[name] = e

    # the bandwidth-bound candidate at its own workload size
    sws = Workspace(sw)
    flush = lambda: krex.krex_flush_l2(sws.flush, stream=stream)  # noqa: E731
    x, y = sws.inputs[0], sws.out
    krex.krex_gen_inputs(sw.seed, 0, 1, sw.sigma, x, stream)
    rec("softmax_f32", lambda: krex.krex_run_candidate(1, [x], y, stream), flush, nbytes=x.numel() * 8, n=10)
    rec("check_f32_f32", lambda: krex.krex_check_launch(y, x, 1e-6, 0.0, sws.check_scratch, stream), flush,
        nbytes=x.numel() * 8, n=5)
    del sws, x, y
    # the fp16 form of the GEMM candidate at 4096^3
    fw = WORKLOADS["gemm_f16_4096"]
    fws = Workspace(fw)
    flush = lambda: krex.krex_flush_l2(fws.flush, stream=stream)  # noqa: E731
    a16, b16 = fws.inputs
    rec("fill_uniform_f16@4096", lambda: krex.krex_gen_inputs(fw.seed, 0, 0, 0.0, a16, stream), flush,
        nbytes=a16.numel() * 2)
    krex.krex_gen_inputs(fw.seed, 1, 0, 0.0, b16, stream)
    rec("gemm_tcgen05_f16@4096", lambda: krex.krex_run_candidate_ws(fw.op, fws.inputs, fws.out, fws.gemm_ws, stream),
        flush, flops=fw.flops)
    del fws, a16, b16
    torch.cuda.empty_cache()
    for gname in gemm_names:
        w = WORKLOADS[gname]
        ws = Workspace(w)
        sfx = f"@{w.M}"
        flush = lambda ws=ws: krex.krex_flush_l2(ws.flush, stream=stream)  # noqa: E731
        A, B = ws.inputs
        if w.M != 16384:   # (the 16384^2 fill is timed above, beside its ceiling)
            rec("fill_uniform_bf16" + sfx, lambda: krex.krex_gen_inputs(w.seed, 0, 0, 0.0, A, stream), flush,
                nbytes=A.numel() * 2, gen_dist=0, n=10)
        krex.krex_gen_inputs(w.seed, 0, 0, 0.0, A, stream)
        krex.krex_gen_inputs(w.seed, 1, 0, 0.0, B, stream)
        if gname == gemm_names[0]:
            rec("flush_l2", flush, None, nbytes=ws.flush.numel())
        rec(reference_kernel(w) + sfx, lambda: krex.krex_run_reference(w.op, ws.inputs, ws.ref, stream), flush,
            flops=w.flops, n=2 if w.M >= 16384 else 10, fma_peak=n_sm * FMA_LANES_PER_SM * 2 * 2.070e9)
        rec("gemm_tcgen05" + sfx, lambda: krex.krex_run_candidate_ws(w.op, ws.inputs, ws.out, ws.gemm_ws, stream),
            flush, flops=w.flops, n=10 if w.M >= 16384 else 20)
        rec("check_bf16_f32" + sfx,
            lambda: krex.krex_check_launch(ws.out, ws.ref, w.atol, w.rtol, ws.check_scratch, stream), flush,
            nbytes=ws.out.numel() * 6, n=10)
        del ws, A, B
        torch.cuda.empty_cache()
    return out


def fill_beside_ceiling(dist: int, n_sm: int, stream, fill, n_elements: int, flush, n: int = 10):
    """A fill and its generator probe launched alternately, so both see the
    same clock and power state.  The probe (krex_probe_generator) runs the
    fill kernel's loop over as many elements on the fills' residency (8 blocks
    of 256 threads per SM) with folds instead of stores: the rate at which
    this GPU computes the generator, the fill's compute roofline.  Returns the
    probe's best of n launches (a peak, like the driver's) as output GB/s and
    the fill's mean of n launches, each fill after an L2 flush."""
    import torch
    import paper_2609_30057_gb300 as krex
    blocks = n_sm * 8
    sink = torch.empty(blocks * 256, dtype=torch.int32, device="cuda")
    probe = lambda: krex.krex_probe_generator(dist, n_elements, blocks, sink, stream=stream)  # noqa: E731
    for _ in range(3):
        probe()
        fill()
    pe = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(n)]
    fe = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(n)]
    for i in range(n):
        pe[i][0].record(stream)
        probe()
        pe[i][1].record(stream)
        flush()
        fe[i][0].record(stream)
        fill()
        fe[i][1].record(stream)
    stream.synchronize()
    p_ms = min(a.elapsed_time(b) for a, b in pe)
    f_ms = statistics.fmean(a.elapsed_time(b) for a, b in fe)
    draws = n_elements // 2
    ceiling = {"ms": p_ms, "elements": n_elements, "Gdraws/s": draws / p_ms / 1e6,
               "GB/s": draws * DRAW_BYTES[dist] / p_ms / 1e6, "blocks": blocks}
    return ceiling, f_ms


# ---------------------------------------------------------- CPU oracle ------

def _oracle_block(w):
    """The block of one workload's output that one oracle step computes:
    (rows, cols) of C for a GEMM (cols = N for the small GEMM, whose whole
    command is one step), rows for the softmax."""
    if w.is_gemm:
        if w.M * w.N <= 256 * 256:
            return w.M, w.N
        return 256, 256
    return 128, w.N


def oracle_command_fraction(w, step: int):
    """One step of the oracle as a benchmarking command's program on the host:
    the work of a block of the command's output, executed in full.  For block
    b of C (r rows, c columns): generate the r rows of A and c columns of B the
    block needs; compute the block with the oracle's fp64 GEMM once for the
    reference, once for the candidate's checked run and once per warm-up and
    timed candidate run; check the block (fp32, oracle check).  The softmax
    does the same on r rows.  The block is a fraction f = r*c / (M*N) of the
    command's output; the step's generation covers more than f of the inputs
    (whole operand rows and columns), so f / seconds understates the oracle's
    command rate.  Blocks walk the output in order with `step`.
    Returns (f, seconds, description)."""
    import numpy as np
    from oracle import gen, ref
    r, c = _oracle_block(w)
    runs = 1 + 1 + w.warmup + w.iters
    t0 = time.perf_counter()
    if w.is_gemm:
        nbr, nbc = w.M // r, w.N // c
        br, bc = (step // max(1, nbc)) % max(1, nbr), step % max(1, nbc)
        r0, c0 = br * r, bc * c
        kk = np.arange(w.K, dtype=np.int64)
        a_idx = (r0 + np.arange(r, dtype=np.int64))[:, None] * w.K + kk[None, :]
        b_idx = kk[:, None] * w.N + (c0 + np.arange(c, dtype=np.int64))[None, :]
        a = gen.uniform_at(w.dtype, w.seed, 0, a_idx.ravel()).reshape(r, w.K)
        b = gen.uniform_at(w.dtype, w.seed, 1, b_idx.ravel()).reshape(w.K, c)
        for _ in range(runs):
            blk = ref.gemm_f64(a, b, dtype=w.dtype)
        what = f"a {r}x{c} block of C (K = {w.K}): {r} rows of A and {c} columns of B generated"
    else:
        r0 = (step * r) % w.M
        x = gen.normal_f32_at(w.seed, 0, (r0 * w.N + np.arange(r * w.N, dtype=np.int64)), w.sigma).reshape(r, w.N)
        for _ in range(runs):
            blk = ref.softmax_rows_f64(x.astype(np.float64))
        what = f"{r} rows of {w.N} generated"
    b32 = blk.astype(np.float32)
    ref.check_f32(b32, b32, w.atol, w.rtol)
    secs = time.perf_counter() - t0
    frac = (r * c) / (w.M * w.N)
    info = (f"{what}, computed {runs} times in fp64 (reference + checked run + {w.warmup} warm-up + {w.iters} "
            f"timed) and checked in fp32; a fraction {frac:.3g} of one command's output, executed in full")
    return frac, secs, info


def oracle_rate(w, budget_s: float, first_step: int = 0):
    """Commands/s of the oracle over consecutive steps until `budget_s` of
    host time has passed (at least one step): total fraction / total time."""
    f_tot = t_tot = 0.0
    step = first_step
    info = ""
    while True:
        f, t, info = oracle_command_fraction(w, step)
        f_tot += f
        t_tot += t
        step += 1
        if t_tot >= budget_s:
            break
    return f_tot / t_tot, step - first_step, t_tot, info


def oracle_full_command(w):
    """The oracle running one whole command of a small workload, unextrapolated:
    generate A and B, the fp64 GEMM for the reference, the checked run, the
    warm-up and the timed runs, the fp32 check.  Returns seconds."""
    from oracle import gen, ref
    t0 = time.perf_counter()
    a = gen.uniform(w.dtype, w.seed, 0, w.M, w.K)
    b = gen.uniform(w.dtype, w.seed, 1, w.K, w.N)
    for _ in range(1 + 1 + w.warmup + w.iters):
        c = ref.gemm_f64(a, b, dtype=w.dtype)
    c32 = c.astype("float32")
    ref.check_f32(c32, c32, w.atol, w.rtol)
    return time.perf_counter() - t0


def cpu_baseline_record(w, budget_s: float = 12.0):
    """The oracle as it stands on the host cores (a bounded sample of the
    workload), plus one whole small command timed in full and each oracle
    routine timed on its own."""
    from paper_2609_30057_gb300.command import WORKLOADS
    rate, steps, secs, info = oracle_rate(w, budget_s)
    small = WORKLOADS["gemm_bf16_256"]
    full_s = oracle_full_command(small)
    return {"value": rate, "unit": "cmds/s", "cores": cpu_cores(), "kind": "oracle",
            "sample": (f"{steps} oracle steps of {w.name}, {secs:.1f} s of host time measured; each step: {info}; "
                       f"value = fractions of a command executed / measured seconds"),
            "measured_wall_s": secs, "steps": steps,
            "threads": "fp64 GEMM through numpy's BLAS on all host cores; generation and check single-threaded",
            "cpu_model": cpu_model(),
            "full_command_unextrapolated": {"workload": small.name, "seconds": full_s, "cmds_per_s": 1.0 / full_s},
            "components": oracle_components()}


_ONE_THREAD_GEMM = r"""
import json, sys, time
sys.path.insert(0, sys.argv[1])
from oracle import gen, ref
n = int(sys.argv[2])
a, b = gen.uniform_bf16(2, 0, n, n), gen.uniform_bf16(2, 1, n, n)
ref.gemm_f64(a, b)
t = time.perf_counter()
ref.gemm_f64(a, b)
print(json.dumps({"seconds": time.perf_counter() - t}))
"""


def oracle_components() -> dict:
    """Baseline only: each oracle routine timed once on the host, with the
    threads it runs on.  Generation (GB/s of output: the 4096^2 bf16 operand,
    2^21 Box-Muller values), the fp64 GEMM (GFLOP/s: the 4096^3 workload in
    full on all cores through numpy's BLAS, and 1024^3 on one thread in a
    child process with the BLAS limited to one thread), the fp64 softmax (rows
    of 8192 per second) and the fp32 check (GB/s of a 16-bit output and an
    fp32 reference, 6 B per element, 4096^2 elements)."""
    import subprocess
    import sys
    import numpy as np
    from oracle import gen, ref

    def timed(fn):
        t = time.perf_counter()
        r = fn()
        return r, time.perf_counter() - t

    out = {"label": "baseline only"}
    a, s = timed(lambda: gen.uniform_bf16(2, 0, 4096, 4096))
    out["gen_uniform_bf16"] = {"GB/s": a.nbytes / s / 1e9, "elements": int(a.size), "threads": 1}
    x, s = timed(lambda: gen.normal_f32(3, 0, 256, 8192, 2.0))
    out["gen_normal_f32"] = {"GB/s": x.nbytes / s / 1e9, "elements": int(x.size), "threads": 1}
    b = gen.uniform_bf16(2, 1, 4096, 4096)
    c, s = timed(lambda: ref.gemm_f64(a, b))
    out["gemm_f64_4096"] = {"GFLOP/s": 2 * 4096 ** 3 / s / 1e9, "seconds": s, "threads": cpu_cores()}
    env = dict(os.environ, OPENBLAS_NUM_THREADS="1", OMP_NUM_THREADS="1", MKL_NUM_THREADS="1")
    try:
        r = subprocess.run([sys.executable, "-c", _ONE_THREAD_GEMM, os.path.dirname(os.path.abspath(__file__)),
                            "1024"], env=env, capture_output=True, text=True, timeout=300)
        one = json.loads(r.stdout.strip().splitlines()[-1])["seconds"]
        out["gemm_f64_1024_one_thread"] = {"GFLOP/s": 2 * 1024 ** 3 / one / 1e9, "seconds": one, "threads": 1}
    except (subprocess.SubprocessError, ValueError, IndexError, KeyError) as e:
        out["gemm_f64_1024_one_thread"] = {"error": str(e)[:200]}
    y, s = timed(lambda: ref.softmax_rows_f64(x.astype(np.float64)))
    out["softmax_f64_8192"] = {"rows/s": x.shape[0] / s, "rows": int(x.shape[0]), "threads": 1}
    c32 = c.astype(np.float32)
    _, s = timed(lambda: ref.check_f32(c32, c32, 2.0 ** -6, 2.0 ** -7))
    out["check_f32_4096"] = {"GB/s": c32.size * 6 / s / 1e9, "elements": int(c32.size), "threads": 1}
    return out


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


def workload_config(w, world: int) -> dict:
    """The `config` object of a JSON line (the same keys for both arms)."""
    return {"workload": w.name, "M": w.M, "N": w.N, "K": w.K, "seed": w.seed, "timed_iters": w.iters,
            "warmup_iters": w.warmup, "flush_bytes": w.flush_bytes, "commands_per_measurement": w.repeat,
            "l2": "flushed: a flush_bytes write precedes every timed candidate iteration and region entry",
            "parallelism": f"replicas{world}"}


# ------------------------------------------------------------- main ---------

def candidate_roofline(w, mean_ms: float, peaks) -> dict:
    """The candidate kernel's roofline from its mean CUDA-event duration."""
    if w.is_gemm:
        achieved = w.flops / (mean_ms / 1e3) / 1e12
        return {"bound": "tensor", "achieved": achieved, "peak": peaks["bf16_tflops"], "unit": "TFLOP/s",
                "frac": achieved / peaks["bf16_tflops"], "traffic": _ncu_traffic("gemm_tcgen05", w.name),
                "peak_kind": f"bf16 dense burst, {peaks['source']} (MEASURED_PEAKS.json)",
                "frac_of_sustained": (achieved / peaks["bf16_tflops_sustained"]
                                      if peaks.get("bf16_tflops_sustained") else None),
                "kernel": "gemm_tcgen05_2sm", "algorithmic_flops_per_launch": w.flops}
    # the bandwidth-bound candidate: one read and one write of the matrix
    achieved = w.candidate_bytes / (mean_ms / 1e3) / 1e9
    return {"bound": "hbm", "achieved": achieved, "peak": peaks["hbm_gbs"], "unit": "GB/s",
            "frac": achieved / peaks["hbm_gbs"], "traffic": _ncu_traffic("softmax_rows", w.name),
            "peak_kind": f"HBM copy, {peaks['source']} (MEASURED_PEAKS.json)",
            "kernel": "softmax_rows_reg", "algorithmic_bytes_per_launch": w.candidate_bytes}


def fma_rate(n_sm: int, stream) -> dict:
    """The FP32 FMA pipe's rate measured with the library's probe (16
    independent FMA chains per thread, 8 blocks of 256 threads per SM), as
    TFLOP/s: the measured counterpart of the derived FMA peak."""
    import torch
    import paper_2609_30057_gb300 as krex
    blocks, iters = n_sm * 8, 4096
    sink = torch.empty(blocks * 256, dtype=torch.float32, device="cuda")
    fn = lambda: krex.krex_probe_fma(iters, blocks, sink, stream=stream)  # noqa: E731
    for _ in range(3):
        fn()
    ms = _time_launches(fn, 10, stream, best=True)   # a peak: best of 10
    flops = 2 * 16 * iters * blocks * 256
    return {"ms": ms, "TFLOP/s": flops / ms / 1e9, "blocks": blocks, "iters": iters}


def reference_kernel(w) -> str:
    """The reference GEMM kernel the library runs for this shape: one output
    per thread for at most 16 tiles of 128x128, the unchecked kernel for
    whole tiles, else the general tiled one."""
    if ((w.M + 127) // 128) * ((w.N + 127) // 128) <= 16:
        return "gemm_ref_small"
    if w.M % 128 == 0 and w.N % 128 == 0 and w.K % 16 == 0:
        return "gemm_ref_whole"
    return "gemm_ref_simt"


def reference_roofline(w, mean_ms: float, n_sm: int, sm_mhz, fma_measured=None) -> dict | None:
    """The CUDA-core reference GEMM on the FP32 fused multiply-add pipe: peak =
    SMs x 128 FMA lanes x 2 flops x clock (the 2070 MHz maximum; also at the
    median SM clock sampled during the run), beside the probe's measured rate."""
    if not w.is_gemm:
        return None
    achieved = w.flops / (mean_ms / 1e3) / 1e12
    peak = n_sm * FMA_LANES_PER_SM * 2 * 2.070e9 / 1e12
    r = {"bound": "alu", "pipe": "fp32 fma", "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
         "frac": achieved / peak, "traffic": _ncu_traffic(reference_kernel(w), w.name),
         "peak_kind": f"derived: {n_sm} SMs x {FMA_LANES_PER_SM} FP32 FMA lanes x 2 flops x 2070 MHz",
         "kernel": reference_kernel(w), "algorithmic_flops_per_launch": w.flops, "ms_per_launch": mean_ms}
    if sm_mhz:
        r["frac_at_sampled_clock"] = achieved / (peak * sm_mhz / 2070.0)
    if fma_measured:
        r["peak_measured"] = fma_measured["TFLOP/s"]
        r["frac_of_measured"] = achieved / fma_measured["TFLOP/s"]
    return r


def measure_commands(ws, n: int, stream):
    """n back-to-back commands timed with CUDA events on `stream`; returns
    (elapsed ms, candidate durations, p50s, p95s, phases)."""
    import torch
    cand, p50s, p95s, phases = [], [], [], []
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    ev0.record(stream)
    for _ in range(n):
        r = ws.run()
        if not r.passed:
            raise SystemExit(f"{ws.w.name}: check failed: {r.check.n_violations} violations")
        cand.extend(ws.durations[: r.n_iters])
        p50s.append(r.p50_ms)
        p95s.append(r.p95_ms)
        phases.append(list(r.phase_ms))
    ev1.record(stream)
    torch.cuda.synchronize()
    return ev0.elapsed_time(ev1), cand, p50s, p95s, phases


def spread(p50s, p95s) -> dict:
    m50 = statistics.median(p50s)
    return {"p50_ms_median": m50, "p95_ms_median": statistics.median(p95s),
            "p95_over_p50_minus_1": statistics.median(p95s) / m50 - 1.0,
            # Eq. 1 across the commands: p95 of (command median / overall median) - 1
            "P_across_commands": _p95([p / m50 for p in p50s]) - 1.0}


def config_records(names, peaks, stream, n_sm, skip=()):
    """One sub-record per workload of the configuration list: commands/s,
    the candidate's roofline, p50/p95 and P across commands."""
    import torch
    from paper_2609_30057_gb300.command import WORKLOADS, Workspace
    out = {}
    for name in names:
        if name in skip:
            continue
        w = WORKLOADS[name]
        n = CONFIG_WORKLOADS[name]
        ws = Workspace(w)
        for _ in range(2):
            ws.run()
        torch.cuda.synchronize()
        ms, cand, p50s, p95s, phases = measure_commands(ws, n, stream)
        ph = [statistics.fmean(p[i] for p in phases) for i in range(5)]
        rl = candidate_roofline(w, statistics.fmean(cand), peaks)
        rec = {"commands": n, "cmds_per_s": n / (ms / 1e3), "ms_per_command": ms / n,
               "candidate": {k: rl[k] for k in ("kernel", "achieved", "unit", "peak", "frac")},
               "phase_ms": dict(zip(["inputs", "reference", "candidate", "check", "timed_loop"], ph))}
        rr = reference_roofline(w, ph[1], n_sm, None)
        if rr:
            rec["reference"] = {k: rr[k] for k in ("kernel", "achieved", "unit", "peak", "frac")}
        rec.update(spread(p50s, p95s))
        out[name] = rec
        del ws
        torch.cuda.empty_cache()
    return out


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=None,
                    help="commands timed (default: the workload's commands per measurement, else 20)")
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD)
    ap.add_argument("--no-kernels", action="store_true", help="skip the per-kernel table")
    ap.add_argument("--no-configs", action="store_true", help="skip the per-configuration sub-records")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--kernel-only", default=None,
                    choices=["gemm", "gemm_ref", "fill_uniform", "fill_normal", "flush", "check", "softmax",
                             "cublas"],
                    help="launch one kernel of the workload --launches times and exit (for ncu captures); "
                         "cublas: torch.matmul on the same operands, a library comparison outside the command")
    ap.add_argument("--launches", type=int, default=3)
    ap.add_argument("--tuning", action="append", default=[], metavar="FIELD=VALUE",
                    help="with --kernel-only: set a field of the library's tuning record first (repeatable)")
    args = ap.parse_args()

    from paper_2609_30057_gb300 import replicas
    from paper_2609_30057_gb300.command import WORKLOADS
    rank, world, local_rank = replicas.rank_world()
    w = WORKLOADS[args.workload]
    if args.steps is None:
        args.steps = w.repeat if w.repeat > 1 else 20

    if args.impl == "reference":
        return reference_arm(args, w, rank, world)
    if args.kernel_only:
        return kernel_only(args)

    import torch
    import paper_2609_30057_gb300 as krex
    from paper_2609_30057_gb300.command import Workspace

    torch.cuda.set_device(local_rank)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local_rank))
    if rank == 0 or world > 1:
        krex.build()
    if world > 1:
        dist.barrier()

    peaks = _peaks()
    ws = Workspace(w)
    stream = torch.cuda.current_stream()
    n_sm = torch.cuda.get_device_properties(local_rank).multi_processor_count

    def barrier():
        replicas.barrier(dist)

    for _ in range(args.warmup):
        r = ws.run()
        if not r.passed:
            raise SystemExit(f"check failed during warm-up: {r.check.n_violations} violations")

    # ------------------------------------------------ timed region (value)
    clocks = ClockSampler(torch.cuda.current_device())
    barrier()
    torch.cuda.synchronize()
    launches0 = krex.krex_launch_count()
    with clocks:
        t0 = time.perf_counter()
        elapsed, cand_ms, p50s, p95s, phases = measure_commands(ws, args.steps, stream)
        wall = time.perf_counter() - t0
    barrier()
    launches = int(replicas.sum_over_ranks(dist, krex.krex_launch_count() - launches0, device="cuda"))
    # a kernel whose bounded wait ran out returned early: no valid number
    status = krex.krex_device_status()
    if status:
        raise SystemExit(f"a kernel reported device status {status:#x} during the timed region")
    elapsed_ms = replicas.max_over_ranks(dist, elapsed, device="cuda")
    value = replicas.aggregate_throughput(args.steps, world, elapsed_ms / 1e3)

    # ------------------------------------------------ e2e (host buffers)
    e2e = None
    if not args.no_e2e:
        # page-locked, huge-page-backed host buffers (krex_host_alloc)
        host_in = [krex.host_buffer(t.shape, t.dtype) for t in ws.inputs]
        for h, t in zip(host_in, ws.inputs):
            h.copy_(t)
        host_out = krex.host_buffer(ws.out.shape, ws.out.dtype)
        ptrs = [h.data_ptr() for h in host_in]
        for _ in range(max(1, min(args.warmup, 2))):
            ws.run(host_in=ptrs, host_out=host_out.data_ptr())
        barrier()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e_phases = []
        e_clocks = ClockSampler(torch.cuda.current_device())
        with e_clocks:
            e0.record(stream)
            for _ in range(args.steps):
                r = ws.run(host_in=ptrs, host_out=host_out.data_ptr())
                if not r.passed:
                    raise SystemExit("check failed (e2e)")
                e_phases.append(list(r.phase_ms))
            e1.record(stream)
            torch.cuda.synchronize()
        barrier()
        te_ms = replicas.max_over_ranks(dist, e0.elapsed_time(e1), device="cuda")
        e2e = {"value": replicas.aggregate_throughput(args.steps, world, te_ms / 1e3), "unit": "cmds/s",
               "h2d_bytes_per_step": sum(h.numel() * h.element_size() for h in host_in),
               "d2h_bytes_per_step": host_out.numel() * host_out.element_size() + 16,
               "ms_per_step": te_ms / args.steps,
               # the phases of these commands (inputs = the host-to-device copies)
               "phase_ms": dict(zip(["inputs", "reference", "candidate", "check", "timed_loop"],
                                    [statistics.fmean(p[i] for p in e_phases) for i in range(5)])),
               "clocks": e_clocks.summary()}
        del host_in, host_out

    cs = clocks.summary()
    ph = [statistics.fmean(p[i] for p in phases) for i in range(5)]
    headline = {"commands": args.steps, "cmds_per_s": args.steps / (elapsed / 1e3),
                "ms_per_command": elapsed / args.steps}
    rl_c = candidate_roofline(w, statistics.fmean(cand_ms), peaks)
    rl_c["launches_timed"] = len(cand_ms)
    rl_r = reference_roofline(w, ph[1], n_sm, cs.get("sm_mhz") if cs else None,
                              fma_rate(n_sm, stream) if w.is_gemm else None)
    if rl_r:
        rl_r["launches_timed"] = len(phases)
    # device time per command of each GEMM: the candidate runs once for the
    # check and once per warm-up and timed iteration, the reference once
    cand_share_ms = statistics.fmean(cand_ms) * (1 + w.warmup + w.iters)
    rl_c["device_ms_per_command"] = cand_share_ms
    if rl_r:
        rl_r["device_ms_per_command"] = ph[1]
    # the line's roofline is the command's dominant kernel (most device time)
    dominant, other = (rl_r, rl_c) if rl_r and ph[1] > cand_share_ms else (rl_c, rl_r)
    del ws
    torch.cuda.empty_cache()

    configs = None
    kernels = None
    if rank == 0:
        if not args.no_configs:
            configs = config_records(list(CONFIG_WORKLOADS), peaks, stream, n_sm, skip=(w.name,))
            hl = dict(headline)
            hl["candidate"] = {k: rl_c[k] for k in ("kernel", "achieved", "unit", "peak", "frac")}
            if rl_r:
                hl["reference"] = {k: rl_r[k] for k in ("kernel", "achieved", "unit", "peak", "frac")}
            hl["phase_ms"] = dict(zip(["inputs", "reference", "candidate", "check", "timed_loop"], ph))
            hl.update(spread(p50s, p95s))
            configs[w.name] = {"headline": True, **hl}
        if not args.no_kernels:
            # the small size first: right after seconds of the large GEMMs the
            # power controller holds the clock down for the next launches
            gnames = (SMALL_GEMM_WORKLOAD, w.name) if w.is_gemm and w.name != SMALL_GEMM_WORKLOAD \
                else (SMALL_GEMM_WORKLOAD,)
            kernels = kernel_table(peaks, stream, gnames)

    if rank != 0:
        if dist is not None:
            dist.destroy_process_group()
        return

    cpu = None
    if not args.no_cpu_baseline and world == 1:   # the host baseline is a single-GPU figure
        cpu = cpu_baseline_record(w)

    line = {
        "metric": METRIC, "value": value, "unit": "cmds/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": elapsed_ms / args.steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": {"bf16": "bf16", "f16": "f16"}.get(w.dtype, "f32"),
        "data": "synthetic",
        "config": workload_config(w, world),
        "roofline": dominant,
        "roofline_other_gemm": other,
        "cpu_baseline": cpu,
        "e2e": e2e,
        "gpu_launches": launches,
        "clocks": cs,
        "timing_spread": spread(p50s, p95s),
        "phase_ms": dict(zip(["inputs", "reference", "candidate", "check", "timed_loop"], ph)),
        "configs": configs,
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
    if args.tuning:
        krex.krex_set_tuning(**{k: int(v) for k, v in (t.split("=", 1) for t in args.tuning)})
    stream = torch.cuda.current_stream()
    name = args.workload
    if args.kernel_only in ("softmax", "fill_normal") and WORKLOADS[name].is_gemm:
        name = SOFTMAX_WORKLOAD
    w = WORKLOADS[name]
    k = args.kernel_only
    if k == "cublas" and not w.is_gemm:
        raise SystemExit("--kernel-only cublas needs a GEMM workload")
    ws = Workspace(w)
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
        "cublas": lambda: torch.matmul(ws.inputs[0], ws.inputs[1], out=ws.out),
    }[k]
    for _ in range(args.launches):
        if k != "flush":
            krex.krex_flush_l2(ws.flush, stream=stream)
        fn()
    torch.cuda.synchronize()
    assert krex.krex_device_status() == 0
    print(json.dumps({"kernel_only": k, "workload": w.name, "launches": args.launches}))


def reference_arm(args, w, rank, world):
    """The oracle as the reference arm: each step executes a block of one
    command of the workload in full on the host cores (oracle_command_fraction);
    value = fractions of a command executed / measured seconds.  Rank 0 alone
    runs it."""
    if rank != 0:
        return
    for i in range(args.warmup):
        oracle_command_fraction(w, i)
    fr, secs = [], []
    info = ""
    for i in range(args.steps):
        f, t, info = oracle_command_fraction(w, args.warmup + i)
        fr.append(f)
        secs.append(t)
    value = sum(fr) / sum(secs)
    line = {"metric": METRIC, "value": value, "unit": "cmds/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": 1e3 * sum(secs) / args.steps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": workload_config(w, world),
            "impl": "reference",
            "cpu_baseline": {"value": value, "unit": "cmds/s", "cores": cpu_cores(), "kind": "oracle",
                             "sample": f"each step: {info}; value = fractions of a command executed / measured "
                                       f"seconds",
                             "measured_wall_s": sum(secs), "fraction_per_step": fr[0],
                             "threads": "fp64 GEMM through numpy's BLAS on all host cores; generation and check "
                                        "single-threaded",
                             "cpu_model": cpu_model()},
            "e2e": {"value": value, "unit": "cmds/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line))


if __name__ == "__main__":
    main()
