"""bench.py's JSON line: the reference arm on the CPU (the oracle on the host
cores), and our arm on the GPU, carry every key the measurement contract
names, with consistent values."""
import json
import os
import subprocess
import sys

import pytest

from conftest import ROOT

BASE_KEYS = {"metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better", "scaling",
             "vs_baseline", "dtype", "data", "config", "e2e", "cpu_baseline"}


def _bench(*args, timeout=600):
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), *args], capture_output=True, text=True,
                       timeout=timeout, cwd=ROOT)
    assert r.returncode == 0, r.stdout[-2000:] + r.stderr[-2000:]
    return json.loads(r.stdout.strip().splitlines()[-1])


def test_reference_arm_line():
    d = _bench("--impl", "reference", "--steps", "1", "--warmup", "0", "--workload", "gemm_bf16_256")
    assert BASE_KEYS <= set(d)
    assert d["impl"] == "reference" and d["value"] > 0 and d["unit"] == "cmds/s" and d["higher_is_better"]
    assert d["e2e"] == {"value": d["value"], "unit": d["unit"], "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["value"] == d["value"] and cb["cores"] >= 1 and cb["sample"]
    # measured, not extrapolated: the small command is one whole command per step
    assert cb["fraction_per_step"] == 1.0
    assert abs(d["value"] - 1e3 / d["ms_per_step"]) < 1e-9 * d["value"]
    assert abs(cb["measured_wall_s"] - d["ms_per_step"] / 1e3) < 1e-9
    assert d["config"]["workload"] == "gemm_bf16_256"


def test_reference_arm_config_keys_match_our_arm():
    sys.path.insert(0, ROOT)
    import bench
    from paper_2609_30057_gb300.command import WORKLOADS
    d = _bench("--impl", "reference", "--steps", "2", "--warmup", "1", "--workload", "gemm_bf16_4096")
    assert d["config"] == bench.workload_config(WORKLOADS["gemm_bf16_4096"], 1)
    f = d["cpu_baseline"]["fraction_per_step"]
    assert f == (256 * 256) / (4096 * 4096)
    # value = fractions executed / measured time, and the steps' time is real
    assert abs(d["value"] - 2 * f / (d["ms_per_step"] * 2 / 1e3)) < 1e-9 * d["value"]


def test_oracle_components_are_labelled_timings():
    # cpu_baseline.components: each oracle routine timed once on the host,
    # labelled baseline only, every rate positive, with its thread count
    sys.path.insert(0, ROOT)
    import bench
    c = bench.oracle_components()
    assert c["label"] == "baseline only"
    keys = {"gen_uniform_bf16": "GB/s", "gen_normal_f32": "GB/s", "gemm_f64_4096": "GFLOP/s",
            "gemm_f64_1024_one_thread": "GFLOP/s", "softmax_f64_8192": "rows/s", "check_f32_4096": "GB/s"}
    for k, unit in keys.items():
        assert c[k][unit] > 0 and c[k]["threads"] >= 1, (k, c[k])
    assert c["gemm_f64_1024_one_thread"]["threads"] == 1


@pytest.mark.gpu
def test_our_arm_line():
    d = _bench("--steps", "3", "--warmup", "3", "--no-kernels", "--no-configs", "--workload", "gemm_bf16_4096")
    assert BASE_KEYS <= set(d) and {"roofline", "gpu_launches", "clocks", "timing_spread"} <= set(d)
    assert d["n_gpus"] == 1 and d["steps"] == 3 and d["warmup"] == 3 and d["value"] > 0
    assert abs(d["value"] - 3 / (d["ms_per_step"] * 3 / 1e3)) < 1e-6 * d["value"]
    # at 4096^3 the candidate GEMM is the dominant kernel (103 launches of ~0.09 ms
    # against one reference of ~2.5 ms)
    r = d["roofline"]
    assert r["bound"] == "tensor" and r["unit"] == "TFLOP/s" and 0 < r["frac"] < 1.2
    assert abs(r["frac"] - r["achieved"] / r["peak"]) < 1e-9
    rr = d["roofline_other_gemm"]
    assert rr["bound"] == "alu" and rr["kernel"] == "gemm_ref_whole" and 0 < rr["frac"] < 1.05
    assert r["device_ms_per_command"] > rr["device_ms_per_command"]
    e = d["e2e"]
    assert e["value"] > 0 and e["h2d_bytes_per_step"] == 2 * 4096 * 4096 * 2
    assert e["d2h_bytes_per_step"] >= 4096 * 4096 * 2
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["value"] > 0
    # launches per command: 2 fills, reference, candidate, check, entry flush, (flush + GEMM) per warm-up and
    # timed iteration of the region
    per_cmd = 2 + 1 + 1 + 1 + 1 + 2 * (3 + 100)
    assert d["gpu_launches"] == 3 * per_cmd
    assert d["clocks"]["samples"] >= 1
