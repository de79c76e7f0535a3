"""GPU: one whole benchmarking command through krex_command_run — inputs,
reference, candidate, check, timed loop — on small and full workloads, with
device-generated and host-supplied inputs."""
import ctypes
import time

import numpy as np
import pytest
import torch

import paper_2609_30057_gb300 as krex
from gpu_util import bits16
from paper_2609_30057_gb300.command import WORKLOADS, Workspace, scaled
from oracle import gen, ref

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    krex.build()


def test_gemm_256_command_matches_oracle():
    w = WORKLOADS["gemm_bf16_256"]
    ws = Workspace(w)
    res = ws.run()
    assert res.passed == 1 and res.check.n_violations == 0
    assert res.n_iters == w.iters and res.p50_ms > 0 and res.p95_ms >= res.p50_ms
    d = list(ws.durations)
    assert res.p50_ms == ref.percentile_linear(d, 0.5)
    # launches: 2 gen + ref + candidate + check + entry flush + warmup*2 + iters*2
    assert res.launches == 2 + 1 + 1 + 1 + 1 + 2 * w.warmup + 2 * w.iters
    want = ref.gemm_f64(gen.uniform_bf16(w.seed, 0, w.M, w.K), gen.uniform_bf16(w.seed, 1, w.K, w.N))
    got = gen.bf16_to_f32(bits16(ws.out)).astype(np.float64)
    assert np.all(np.abs(got - want) <= ref.gemm_tolerance(want, w.K))
    # the check's result equals the oracle's check of the same two device outputs
    # recomputed from oracle inputs: C within tolerance of fp64 means ref fp32 too
    assert np.max(np.abs(ws.ref.cpu().numpy() - want)) < 1e-4


def test_command_with_host_buffers_equals_device_generated():
    w = scaled(WORKLOADS["gemm_bf16_256"], M=384, N=512, K=320, iters=5)
    ws = Workspace(w)
    a = gen.uniform_bf16(w.seed, 0, w.M, w.K)
    b = gen.uniform_bf16(w.seed, 1, w.K, w.N)
    ha = torch.from_numpy(a.view(np.int16)).pin_memory()
    hb = torch.from_numpy(b.view(np.int16)).pin_memory()
    hc = torch.empty(w.M, w.N, dtype=torch.int16).pin_memory()
    res = ws.run(host_in=[ha.data_ptr(), hb.data_ptr()], host_out=hc.data_ptr())
    assert res.passed == 1
    dev_out = bits16(ws.out)
    assert np.array_equal(hc.numpy().view(np.uint16), dev_out)
    res2 = ws.run()
    assert res2.passed == 1
    assert np.array_equal(bits16(ws.out), dev_out)      # same inputs either way: same output


def test_softmax_command_small():
    w = scaled(WORKLOADS["softmax_f32_65536x8192"], M=512, iters=5)
    ws = Workspace(w)
    res = ws.run()
    assert res.passed == 1 and res.n_iters == 5
    x = gen.normal_f32(w.seed, 0, w.M, w.N, w.sigma)
    assert np.max(np.abs(ws.out.cpu().numpy() - ref.softmax_rows_f64(x.astype(np.float64)))) <= ref.SOFTMAX_ATOL


def test_failing_check_skips_the_timed_loop():
    w = scaled(WORKLOADS["gemm_bf16_256"], iters=5)
    ws = Workspace(w)
    ws.cmd.atol = -1.0                                   # nothing can pass
    ws.cmd.rtol = 0.0
    res = ws.run()
    assert res.passed == 0 and res.n_iters == 0 and res.check.n_violations == w.M * w.N


def test_f16_gemm_command_matches_oracle():
    w = scaled(WORKLOADS["gemm_f16_4096"], name="gemm_f16_512", M=512, N=768, K=1024, iters=10)
    ws = Workspace(w)
    res = ws.run()
    assert res.passed == 1 and res.check.n_violations == 0
    assert res.n_iters == w.iters and res.p50_ms > 0
    want = ref.gemm_f64(gen.uniform_f16(w.seed, 0, w.M, w.K), gen.uniform_f16(w.seed, 1, w.K, w.N), dtype="f16")
    got = gen.f16_to_f32(bits16(ws.out)).astype(np.float64)
    assert np.all(np.abs(got - want) <= ref.gemm_tolerance(want, w.K, dtype="f16"))
    assert np.array_equal(bits16(ws.inputs[0]), gen.uniform_f16(w.seed, 0, w.M, w.K))



def test_phase_times_are_positive_and_within_the_command():
    # inputs, reference, candidate and check are timed between CUDA events on
    # the command's stream, the timed loop on the host clock: every phase is
    # positive and together they fit inside the command's wall time
    w = WORKLOADS["gemm_bf16_256"]
    ws = Workspace(w)
    ws.run()
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    r = ws.run()
    torch.cuda.synchronize()
    wall_ms = (time.perf_counter() - t0) * 1e3
    ph = list(r.phase_ms)
    assert all(p > 0 for p in ph), ph
    assert sum(ph) <= wall_ms * 1.02 + 0.02, (ph, wall_ms)
