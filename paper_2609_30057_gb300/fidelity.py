"""Measurement-fidelity experiment on one GPU (the paper's Section 6.4, in-process).

Candidate kernels (tcgen05 GEMMs of several sizes, row softmaxes) are timed the
way a benchmarking command times them (region, warm-up, flushed iterations,
median) in four conditions:

* ``native``   — nothing else on the GPU;
* ``repeat``   — a second native run (run-to-run variation);
* ``ungated``  — background tenants keep launching work on their own streams;
* ``gated``    — the same background tenants, but they submit through the
                 in-region gate and the measuring region enters it, so their
                 submissions are blocked and their queued work drained while
                 the timed loop runs (Section 4.2).

Reported per condition, against the first native run: P = p95(r) − 1 with
r = t_measured / t_native per candidate (Eq. 1), the median ratio, the share
of ratios within 5 %, the pairwise ordering-flip rate grouped by native gap
(pairs whose durations differ by less than 2 %, 2–10 %, more than 10 %), and
Kendall's τ_b between measured and native rankings.

    python -m paper_2609_30057_gb300.fidelity [--tenants 2] [--iters 20] [--processes] [--json out.json]

With ``--processes`` the background tenants run in their own processes (own
CUDA contexts) and the gate lives in shared memory (``run_xproc``).
"""
from __future__ import annotations

import argparse
import json
import math
import threading
import time

from . import (KREX_OP_GEMM_BF16, KREX_OP_SOFTMAX_F32, Gate, KrexError, build, krex_bench_candidate,
               krex_device_status, krex_device_status_detail, krex_gen_inputs, krex_run_candidate, tuning)


def _device_status(details: dict | None = None, phase: str = "") -> int:
    """The kernels' status word (non-zero: a bounded wait ran out); read and
    cleared.  Where a wait ran out is added to `details` under `phase`."""
    detail = krex_device_status_detail()
    try:
        return krex_device_status()
    except KrexError as e:
        if details is not None:
            details[phase] = detail
        return int(str(e).split("status 0x")[-1].rstrip(")"), 16) if "status 0x" in str(e) else -1


# ------------------------------------------------------------- statistics --

def percentile(xs, q: float) -> float:
    """Linear interpolation between order statistics."""
    v = sorted(xs)
    h = (len(v) - 1) * q
    lo = int(math.floor(h))
    if lo >= len(v) - 1:
        return v[-1]
    return v[lo] + (h - lo) * (v[lo + 1] - v[lo])


def inflation_p95(measured, native) -> float:
    """Eq. 1: P = p95(r) − 1, r = t_measured / t_native."""
    return percentile([m / n for m, n in zip(measured, native)], 0.95) - 1.0


def kendall_tau_b(x, y) -> float:
    conc = disc = tx = ty = 0
    n = len(x)
    for i in range(n):
        for j in range(i + 1, n):
            dx = (x[i] > x[j]) - (x[i] < x[j])
            dy = (y[i] > y[j]) - (y[i] < y[j])
            if dx == 0 and dy == 0:
                continue
            if dx == 0:
                tx += 1
            elif dy == 0:
                ty += 1
            elif dx == dy:
                conc += 1
            else:
                disc += 1
    d = math.sqrt((conc + disc + tx) * (conc + disc + ty))
    return (conc - disc) / d if d else float("nan")


GAP_GROUPS = ((0.0, 0.02), (0.02, 0.10), (0.10, float("inf")))


def flip_rates(measured, native):
    """Fraction of candidate pairs whose order differs from the native order,
    grouped by the native gap |a − b| / min(a, b) (Section 6.4)."""
    out = {}
    for lo, hi in GAP_GROUPS:
        flips = total = 0
        for i in range(len(native)):
            for j in range(i + 1, len(native)):
                a, b = native[i], native[j]
                gap = abs(a - b) / min(a, b)
                if not (lo <= gap < hi) or a == b:
                    continue
                total += 1
                flips += (measured[i] < measured[j]) != (a < b)
        out[f"{lo:.2f}-{hi:.2f}"] = {"pairs": total, "flip_rate": flips / total if total else None}
    return out


def summarize(measured, native) -> dict:
    r = [m / n for m, n in zip(measured, native)]
    return {"P_p95_inflation": inflation_p95(measured, native), "median_ratio": percentile(r, 0.5),
            "within_5pct": sum(abs(x - 1) <= 0.05 for x in r) / len(r), "kendall_tau_b": kendall_tau_b(measured, native),
            "flips": flip_rates(measured, native)}


# ------------------------------------------------------------- candidates --

def candidates(device="cuda", quick: bool = False):
    """(name, op, inputs, out) for candidate kernels of mixed lengths with
    near-tied pairs, like an agent's trajectory: tcgen05 GEMMs whose sizes
    differ by 16 (about 1-2 % more work) and row softmaxes."""
    import torch
    cands = []
    sizes = (2048, 2064, 4096) if quick else (2048, 2064, 3072, 3088, 4096, 4112, 5120, 5136, 6144)
    for n in sizes:
        a = torch.empty(n, n, dtype=torch.bfloat16, device=device)
        b = torch.empty(n, n, dtype=torch.bfloat16, device=device)
        krex_gen_inputs(n, 0, 0, 0.0, a)
        krex_gen_inputs(n, 1, 0, 0.0, b)
        cands.append((f"gemm{n}", KREX_OP_GEMM_BF16, [a, b], torch.empty(n, n, dtype=torch.bfloat16, device=device)))
    for rows in ((16384,) if quick else (16384, 16512, 32768)):
        x = torch.empty(rows, 8192, dtype=torch.float32, device=device)
        krex_gen_inputs(rows, 0, 1, 2.0, x)
        cands.append((f"softmax{rows}x8192", KREX_OP_SOFTMAX_F32, [x], torch.empty_like(x)))
    return cands


# Variants of the tcgen05 kernel on one 4096^3 GEMM, as an agent tuning it
# would produce: K depth per ring stage, pair-tile width, the raster group and
# the ring depth (fields of the library's tuning record, krex_set_tuning).
TILE_VARIANTS = (
    ("sm2_k128_n256", {}),
    ("sm2_k64_n256", {"gemm_stage_k": 64}),
    ("sm2_k128_n192", {"gemm_pair_tile_n": 192}),
    ("sm2_k128_n128", {"gemm_pair_tile_n": 128}),
    ("sm2_k128_g8", {"gemm_raster_group": 8}),
    ("sm2_k64_st5", {"gemm_stage_k": 64, "gemm_ring_stages": 5}),
    ("sm2_k128_g2", {"gemm_raster_group": 2}),
)


def tile_variant_candidates(device="cuda"):
    """(name, op, inputs, out, tuning) for the kernel variants above on one
    4096^3 GEMM; timing sets each variant's tuning in this process only, so
    it is used where no thread of this process launches GEMMs concurrently."""
    import torch
    n = 4096
    a = torch.empty(n, n, dtype=torch.bfloat16, device=device)
    b = torch.empty(n, n, dtype=torch.bfloat16, device=device)
    krex_gen_inputs(7, 0, 0, 0.0, a)
    krex_gen_inputs(7, 1, 0, 0.0, b)
    c = torch.empty(n, n, dtype=torch.bfloat16, device=device)
    return [(f"gemm4096_{name}", KREX_OP_GEMM_BF16, [a, b], c, knobs) for name, knobs in TILE_VARIANTS]


def time_candidates(cands, flush, iters, stream, gate=None, tenant=0, per_iter=None):
    """Median of `iters` flushed, timed iterations of each candidate (the
    command's timed loop), optionally inside a gated region.  `per_iter`, if
    a list, receives every candidate's iteration durations.  A candidate's
    optional fifth field is a dict of tuning fields set while it is timed."""
    out = []
    for cand in cands:
        name, op, ins, o = cand[:4]
        knobs = cand[4] if len(cand) > 4 else {}
        with tuning(**knobs):
            d, p50, _ = krex_bench_candidate(op, ins, o, warmup=3, iters=iters, flush_scratch=flush,
                                             flush_bytes=flush.numel(), stream=stream, gate=gate, tenant=tenant)
        out.append(p50)
        if per_iter is not None:
            per_iter.append(list(d))
    return out


def iteration_stats(per_iter, native) -> dict:
    """Interference seen by single iterations rather than by medians: every
    iteration's duration over its candidate's native median."""
    r = [x / n for d, n in zip(per_iter, native) for x in d]
    return {"iter_p95_inflation": percentile(r, 0.95) - 1.0, "iter_max_ratio": max(r),
            "iter_share_over_1_5x": sum(x > 1.5 for x in r) / len(r)}


# ------------------------------------------------------------- background --

class Background:
    """Tenant threads that keep the GPU busy with their own streams: each
    repeatedly launches a 4096^3 GEMM and a 16384x8192 softmax, bracketing
    every submission with the gate when one is given."""

    def __init__(self, n: int, gate: Gate | None, device="cuda"):
        import torch
        self.stop = threading.Event()
        self.threads = []
        self.launched = [0] * n
        self.work = []
        for i in range(n):
            s = torch.cuda.Stream(device=device)
            a = torch.empty(4096, 4096, dtype=torch.bfloat16, device=device)
            b = torch.empty_like(a)
            c = torch.empty_like(a)
            x = torch.empty(16384, 8192, dtype=torch.float32, device=device)
            y = torch.empty_like(x)
            with torch.cuda.stream(s):
                krex_gen_inputs(100 + i, 0, 0, 0.0, a, stream=s)
                krex_gen_inputs(100 + i, 1, 0, 0.0, b, stream=s)
                krex_gen_inputs(100 + i, 2, 1, 2.0, x, stream=s)
            t = gate.register(s) if gate is not None else None
            self.work.append((s, t, a, b, c, x, y))
        self.gate = gate

    def _loop(self, i):
        s, t, a, b, c, x, y = self.work[i]
        while not self.stop.is_set():
            if self.gate is not None:
                self.gate.submit_begin(t, timeout_us=30_000_000)
            try:
                krex_run_candidate(KREX_OP_GEMM_BF16, [a, b], c, stream=s)
                krex_run_candidate(KREX_OP_SOFTMAX_F32, [x], y, stream=s)
            finally:
                if self.gate is not None:
                    self.gate.submit_end(t)
            self.launched[i] += 2
            if s.query() is False:       # keep at most a short queue per tenant
                s.synchronize()

    def __enter__(self):
        for i in range(len(self.work)):
            th = threading.Thread(target=self._loop, args=(i,), daemon=True)
            th.start()
            self.threads.append(th)
        time.sleep(0.2)
        return self

    def __exit__(self, *exc):
        self.stop.set()
        for th in self.threads:
            th.join(30)
        for s, *_ in self.work:
            s.synchronize()
        if self.gate is not None:
            for _, t, *_ in self.work:
                self.gate.unregister(t)


def run(tenants: int = 2, iters: int = 20, quick: bool = False) -> dict:
    import torch
    build()
    torch.cuda.set_device(0)
    stream = torch.cuda.Stream()
    flush = torch.empty(256 << 20, dtype=torch.uint8, device="cuda")
    cands = candidates(quick=quick)
    names = [c[0] for c in cands]
    status, details = {}, {}
    it = {k: [] for k in ("repeat", "ungated", "gated")}
    time_candidates(cands, flush, 3, stream)                       # warm everything up
    native = time_candidates(cands, flush, iters, stream)
    repeat = time_candidates(cands, flush, iters, stream, per_iter=it["repeat"])
    status["native"] = _device_status(details, "native")
    with Background(tenants, None) as bg:
        ungated = time_candidates(cands, flush, iters, stream, per_iter=it["ungated"])
        ungated_bg = sum(bg.launched)
    status["ungated"] = _device_status(details, "ungated")
    gate = Gate(16)
    holder = gate.register(stream)
    with Background(tenants, gate) as bg:
        gated = time_candidates(cands, flush, iters, stream, gate=gate, tenant=holder, per_iter=it["gated"])
        gated_bg = sum(bg.launched)
    gate.unregister(holder)
    gate.close()
    status["gated"] = _device_status(details, "gated")
    return {
        "device_status": status, "device_status_detail": details,
        "candidates": names, "native_ms": native,
        "conditions": {"repeat": {"ms": repeat, **summarize(repeat, native), **iteration_stats(it["repeat"], native)},
                       "ungated": {"ms": ungated, "background_launches": ungated_bg, **summarize(ungated, native),
                                   **iteration_stats(it["ungated"], native)},
                       "gated": {"ms": gated, "background_launches": gated_bg, **summarize(gated, native),
                                 **iteration_stats(it["gated"], native)}},
        "tenants": tenants, "iters": iters,
    }


# ------------------------------------------------- tenants in processes --

# control words (int64) after the shared gate: stop, pause, then per tenant
# ready, launches, device status
_X_STOP, _X_PAUSE, _X_BASE = 0, 1, 2


def _xproc_tenant(path: str, nbytes: int, gate_bytes: int, idx: int):
    """A tenant in its own process (own CUDA context): attaches to the shared
    gate and keeps launching a 4096^3 GEMM and a 16384x8192 softmax on its
    stream, each submission bracketed by the gate, until told to stop."""
    import ctypes
    import torch
    from . import SharedMap
    m = SharedMap(path, nbytes)
    ctl = (ctypes.c_int64 * 32).from_address(m.addr + gate_bytes)
    torch.cuda.set_device(0)
    build()
    g = Gate.attach(m.addr, gate_bytes)
    s = torch.cuda.Stream()
    a = torch.empty(4096, 4096, dtype=torch.bfloat16, device="cuda")
    b, c = torch.empty_like(a), torch.empty_like(a)
    x = torch.empty(16384, 8192, dtype=torch.float32, device="cuda")
    y = torch.empty_like(x)
    krex_gen_inputs(100 + idx, 0, 0, 0.0, a, stream=s)
    krex_gen_inputs(100 + idx, 1, 0, 0.0, b, stream=s)
    krex_gen_inputs(100 + idx, 2, 1, 2.0, x, stream=s)
    s.synchronize()
    t = g.register(s)
    base = _X_BASE + 3 * idx
    ctl[base] = 1
    launched = 0
    while not ctl[_X_STOP]:
        if ctl[_X_PAUSE]:
            s.synchronize()
            time.sleep(0.002)
            continue
        g.submit_begin(t, timeout_us=60_000_000)
        try:
            krex_run_candidate(KREX_OP_GEMM_BF16, [a, b], c, stream=s)
            krex_run_candidate(KREX_OP_SOFTMAX_F32, [x], y, stream=s)
        finally:
            g.submit_end(t)
        launched += 2
        if s.query() is False:
            s.synchronize()
    s.synchronize()
    ctl[base + 1] = launched
    ctl[base + 2] = _device_status()
    g.unregister(t)
    g.close()


def run_xproc(tenants: int = 2, iters: int = 20, quick: bool = False, shm_dir: str = "/dev/shm") -> dict:
    """The fidelity experiment with the background tenants in other processes
    (each its own CUDA context, as the paper's tenants are) and the gate in
    shared memory: native, repeat, ungated, gated."""
    import ctypes
    import multiprocessing as mp
    import os
    import torch
    from . import SharedMap, gate_shared_bytes, gate_shared_init
    build()
    torch.cuda.set_device(0)
    gate_bytes = (gate_shared_bytes(16) + 63) // 64 * 64
    nbytes = gate_bytes + 32 * 8
    path = os.path.join(shm_dir if os.path.isdir(shm_dir) else "/tmp", f"krex_fid_{os.getpid()}_{time.monotonic_ns()}")
    m = SharedMap(path, nbytes, create=True)
    try:
        gate_shared_init(m.addr, gate_bytes, 16)
        ctl = (ctypes.c_int64 * 32).from_address(m.addr + gate_bytes)
        ctl[_X_PAUSE] = 1
        procs = [mp.get_context("spawn").Process(target=_xproc_tenant, args=(path, nbytes, gate_bytes, i), daemon=True)
                 for i in range(tenants)]
        for p in procs:
            p.start()
        stream = torch.cuda.Stream()
        flush = torch.empty(256 << 20, dtype=torch.uint8, device="cuda")
        # tenants run in other processes, so the tile variants' knobs can be
        # set in this one while they are timed
        cands = candidates(quick=quick) + ([] if quick else tile_variant_candidates())
        t0 = time.monotonic()
        while not all(ctl[_X_BASE + 3 * i] for i in range(tenants)):
            if time.monotonic() - t0 > 120 or any(p.exitcode not in (None, 0) for p in procs):
                raise RuntimeError("tenant processes did not start")
            time.sleep(0.05)
        status, details = {}, {}
        it = {k: [] for k in ("repeat", "ungated", "gated")}
        time_candidates(cands, flush, 3, stream)
        native = time_candidates(cands, flush, iters, stream)
        repeat = time_candidates(cands, flush, iters, stream, per_iter=it["repeat"])
        status["native"] = _device_status(details, "native")
        ctl[_X_PAUSE] = 0
        time.sleep(0.5)
        ungated = time_candidates(cands, flush, iters, stream, per_iter=it["ungated"])
        status["ungated"] = _device_status(details, "ungated")
        g = Gate.attach(m.addr, gate_bytes)
        holder = g.register(stream)
        gated = time_candidates(cands, flush, iters, stream, gate=g, tenant=holder, per_iter=it["gated"])
        status["gated"] = _device_status(details, "gated")
        ctl[_X_STOP] = 1
        for p in procs:
            p.join(120)
        g.unregister(holder)
        g.close()
        tenant_launches = [int(ctl[_X_BASE + 3 * i + 1]) for i in range(tenants)]
        tenant_status = [int(ctl[_X_BASE + 3 * i + 2]) for i in range(tenants)]
        return {
            "device_status": status, "device_status_detail": details,
            "tenant_exitcodes": [p.exitcode for p in procs], "tenant_launches": tenant_launches,
            "tenant_device_status": tenant_status,
            "candidates": [c[0] for c in cands], "native_ms": native,
            "conditions": {k: {"ms": v, **summarize(v, native), **iteration_stats(it[k], native)}
                           for k, v in (("repeat", repeat), ("ungated", ungated), ("gated", gated))},
            "tenants": tenants, "iters": iters, "tenant_form": "processes",
        }
    finally:
        os.unlink(path)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--tenants", type=int, default=2)
    ap.add_argument("--iters", type=int, default=20)
    ap.add_argument("--json", default=None)
    ap.add_argument("--processes", action="store_true", help="tenants in their own processes, gate in shared memory")
    args = ap.parse_args()
    res = run_xproc(args.tenants, args.iters) if args.processes else run(args.tenants, args.iters)
    text = json.dumps(res, indent=1)
    if args.json:
        with open(args.json, "w") as f:
            f.write(text)
    print(json.dumps({k: {kk: vv for kk, vv in v.items() if kk != "ms"} for k, v in res["conditions"].items()}))


if __name__ == "__main__":
    main()
