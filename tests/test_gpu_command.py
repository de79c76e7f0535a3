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
    # the device reference is within the fp32 summation bound of fp64
    assert np.max(np.abs(ws.ref.cpu().numpy() - want)) < 1e-4
    # the command's verdict is the oracle's check of the two downloaded
    # outputs, bit for bit (count and max error)
    mx, nv = ref.check_f32(got.astype(np.float32), ws.ref.cpu().numpy(), w.atol, w.rtol)
    assert int(res.check.n_violations) == nv == 0
    assert ref.check_bits(res.check.max_abs_err) == ref.check_bits(mx)


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


@pytest.mark.parametrize("route", ["pinned", "pinned_strided_device_rows", "pageable", "pinned_misaligned"])
def test_command_host_inputs_by_each_copy_route(route):
    # host inputs reach the device by SM loads when the device reads the
    # buffer directly (page-locked, registered over the whole copy, 16-byte
    # words): one copy kernel per operand in place of its fill; else by the
    # copy engine (no launch).  Every route gives the device-generated output.
    w = scaled(WORKLOADS["gemm_bf16_256"], M=384, N=512, K=320, iters=3)
    ws0 = Workspace(w)
    r0 = ws0.run()
    assert r0.passed == 1
    want = bits16(ws0.out)
    a = gen.uniform_bf16(w.seed, 0, w.M, w.K).view(np.int16)
    b = gen.uniform_bf16(w.seed, 1, w.K, w.N).view(np.int16)
    inputs = pads = None
    if route == "pinned_strided_device_rows":
        pads = (torch.zeros(w.M, w.K + 8, dtype=torch.bfloat16, device="cuda"),
                torch.zeros(w.K, w.N + 8, dtype=torch.bfloat16, device="cuda"))
        inputs = [pads[0][:, :w.K], pads[1][:, :w.N]]
    ws = Workspace(w, inputs=inputs)
    if route == "pageable":
        hosts = [torch.from_numpy(a.copy()), torch.from_numpy(b.copy())]
        assert not any(h.is_pinned() for h in hosts)
    elif route == "pinned_misaligned":
        # 2 bytes past a 16-byte boundary: no 16-byte words, so the copy engine
        hosts = []
        for x in (a, b):
            big = torch.empty(x.size + 8, dtype=torch.int16).pin_memory()
            v = big[1:1 + x.size].view(x.shape)
            v.copy_(torch.from_numpy(x))
            assert v.data_ptr() % 16 == 2
            hosts.append(v)
    else:
        hosts = [torch.from_numpy(a).pin_memory(), torch.from_numpy(b).pin_memory()]
    hc = torch.empty(w.M, w.N, dtype=torch.int16).pin_memory()
    res = ws.run(host_in=[h.data_ptr() for h in hosts], host_out=hc.data_ptr())
    assert res.passed == 1
    assert np.array_equal(bits16(ws.out), want)
    assert np.array_equal(hc.numpy().view(np.uint16), want)
    by_kernel = route in ("pinned", "pinned_strided_device_rows")
    assert res.launches == r0.launches - (0 if by_kernel else 2)
    if pads is not None:   # the padding columns of the strided rows are untouched
        assert not pads[0].view(torch.int16)[:, w.K:].any()
        assert not pads[1].view(torch.int16)[:, w.N:].any()


def test_command_8192_host_inputs_by_copy_kernel_equal_generated():
    # 2 x 128 MiB of page-locked inputs read by the copy kernel (2^23 16-byte
    # words per operand): the candidate's output and the verdict equal those of
    # the same command with device-generated inputs, bit for bit
    w = scaled(WORKLOADS["gemm_bf16_8192"], iters=3)
    ws = Workspace(w)
    r0 = ws.run()
    assert r0.passed == 1
    want = bits16(ws.out)
    hosts = [t.cpu().pin_memory() for t in ws.inputs]
    ws.out.zero_()
    hc = torch.empty(w.M, w.N, dtype=torch.bfloat16).pin_memory()
    r = ws.run(host_in=[h.data_ptr() for h in hosts], host_out=hc.data_ptr())
    assert r.passed == 1 and r.launches == r0.launches   # two copy kernels in place of the two fills
    assert np.array_equal(bits16(ws.out), want)
    assert np.array_equal(hc.view(torch.int16).numpy().view(np.uint16), want)
    assert r.check.n_violations == r0.check.n_violations == 0
    assert ref.check_bits(r.check.max_abs_err) == ref.check_bits(r0.check.max_abs_err)


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


def test_failing_command_verdict_equals_the_oracle_check():
    # a tolerance that part of the output fails: the device verdict (count and
    # max error) equals the oracle's check of the downloaded buffers exactly
    w = scaled(WORKLOADS["gemm_bf16_256"], M=384, N=640, K=512, iters=3)
    ws = Workspace(w)
    ws.cmd.atol = 2.0 ** -9
    ws.cmd.rtol = 2.0 ** -9
    res = ws.run()
    out = gen.bf16_to_f32(bits16(ws.out))
    r32 = ws.ref.cpu().numpy()
    mx, nv = ref.check_f32(out, r32, 2.0 ** -9, 2.0 ** -9)
    assert 0 < nv < w.M * w.N
    assert int(res.check.n_violations) == nv and res.passed == 0 and res.n_iters == 0
    assert ref.check_bits(res.check.max_abs_err) == ref.check_bits(mx)


def test_gemm_16384_command_against_the_oracle():
    # the 16384^3 command (its own seed, flush and tolerance; two timed
    # iterations instead of twenty to keep the test short): inputs on oracle
    # samples, the candidate and the reference on 4096 oracle-sampled outputs,
    # and the verdict equal to the oracle's check of the downloaded buffers
    w = scaled(WORKLOADS["gemm_bf16_16384"], iters=2)
    ws = Workspace(w)
    res = ws.run()
    assert res.passed == 1 and res.n_iters == 2 and krex.krex_device_status() == 0
    n = w.M
    i, j = ref.sample_indices(w.seed, 2, 4096, n, n)
    want = ref.gemm_sampled_f64(w.seed, n, n, n, i, j)
    ti, tj = torch.from_numpy(i).cuda(), torch.from_numpy(j).cuda()
    got = gen.bf16_to_f32(bits16(ws.out[ti, tj])).astype(np.float64)
    assert np.all(np.abs(got - want) <= ref.gemm_tolerance(want, n))
    # the device reference: within the fp32 recursive-summation bound
    # K 2^-24 sum_k |a_ik b_kj| of fp64 (first 512 samples)
    r = ws.ref[ti, tj].cpu().numpy().astype(np.float64)
    kk = np.arange(n, dtype=np.int64)
    for s_ in range(512):
        ra = np.abs(gen.widen("bf16", gen.uniform_at("bf16", w.seed, 0, i[s_] * n + kk)).astype(np.float64))
        cb = np.abs(gen.widen("bf16", gen.uniform_at("bf16", w.seed, 1, kk * n + j[s_])).astype(np.float64))
        assert abs(r[s_] - want[s_]) <= n * 2.0 ** -24 * float(ra @ cb), s_
    # inputs: sampled elements of A and B are the oracle's draws, bit for bit
    k = torch.from_numpy((i * 7 + 3) % n).cuda()
    assert np.array_equal(bits16(ws.inputs[0][ti, k]), gen.uniform_at("bf16", w.seed, 0, i * n + (i * 7 + 3) % n))
    assert np.array_equal(bits16(ws.inputs[1][k, tj]), gen.uniform_at("bf16", w.seed, 1, ((i * 7 + 3) % n) * n + j))
    # the verdict over all 2^28 outputs: the oracle's check of the downloaded buffers
    mx, nv = ref.check_f32(gen.bf16_to_f32(bits16(ws.out)), ws.ref.cpu().numpy(), w.atol, w.rtol)
    assert nv == 0 == int(res.check.n_violations)
    assert ref.check_bits(res.check.max_abs_err) == ref.check_bits(mx)


def test_command_with_library_host_buffers():
    # inputs and output in krex_host_alloc buffers (page-locked, huge-page
    # backed): the same output as device-generated inputs, twice in a row
    w = scaled(WORKLOADS["gemm_bf16_256"], M=512, N=384, K=640, iters=3)
    ws = Workspace(w)
    res = ws.run()
    assert res.passed == 1
    want = bits16(ws.out)
    hin = [krex.host_buffer(t.shape, t.dtype) for t in ws.inputs]
    for h, t in zip(hin, ws.inputs):
        h.copy_(t)
    hout = krex.host_buffer(ws.out.shape, ws.out.dtype)
    assert all(h.is_pinned() for h in hin) and hout.is_pinned()
    for _ in range(2):
        hout.zero_()
        r = ws.run(host_in=[h.data_ptr() for h in hin], host_out=hout.data_ptr())
        assert r.passed == 1
        assert np.array_equal(hout.view(torch.int16).numpy().view(np.uint16), want)


@pytest.mark.parametrize("nbytes", [1, 4096, (2 << 20) + 3, (96 << 20) + 12345])
def test_host_buffer_sizes_round_trip(nbytes):
    # krex_host_alloc buffers of any size (the mapping is rounded up to whole
    # huge pages): page-locked, and a copy to the device and back is exact
    h = krex.host_buffer((nbytes,), torch.uint8)
    assert h.is_pinned() and h.numel() == nbytes
    g = np.random.default_rng(nbytes).integers(0, 256, nbytes, dtype=np.uint8)
    h.copy_(torch.from_numpy(g))
    d = h.to("cuda", non_blocking=True)
    back = krex.host_buffer((nbytes,), torch.uint8)
    back.copy_(d, non_blocking=True)
    torch.cuda.synchronize()
    assert np.array_equal(back.numpy(), g)


def test_softmax_65536x8192_command_against_the_oracle():
    # the softmax workload's command at its full size (two timed iterations
    # instead of a hundred): its input on sampled rows bit for bit, the
    # candidate and the reference on 4096 oracle-sampled rows, and the verdict
    # over all 2^29 outputs equal to the oracle's check of the downloaded buffers
    w = scaled(WORKLOADS["softmax_f32_65536x8192"], iters=2)
    ws = Workspace(w)
    res = ws.run()
    assert res.passed == 1 and res.n_iters == 2 and krex.krex_device_status() == 0
    rows, cols = w.M, w.N
    sample, _ = ref.sample_indices(w.seed, 3, 4096, rows, 1)
    sample = np.unique(sample)
    xs = np.stack([gen.normal_f32_at(w.seed, 0, np.arange(i * cols, (i + 1) * cols), w.sigma) for i in sample])
    st = torch.from_numpy(sample).cuda()
    assert np.array_equal(ws.inputs[0][st].cpu().numpy().view(np.uint32), xs.view(np.uint32))
    want = ref.softmax_rows_f64(xs.astype(np.float64))
    assert np.max(np.abs(ws.out[st].cpu().numpy() - want)) <= ref.SOFTMAX_ATOL
    assert np.max(np.abs(ws.ref[st].cpu().numpy() - want)) <= ref.SOFTMAX_ATOL
    mx, nv = ref.check_f32(ws.out.cpu().numpy(), ws.ref.cpu().numpy(), w.atol, w.rtol)
    assert nv == 0 == int(res.check.n_violations)
    assert ref.check_bits(res.check.max_abs_err) == ref.check_bits(mx)


def test_gemm_8192_command_against_the_oracle():
    # the 8192^3 command (wide pair tiles by the launch code's rule; two timed
    # iterations instead of fifty): 4096 oracle-sampled outputs of the
    # candidate and of the reference, and the verdict over all 2^26 outputs
    # equal to the oracle's check of the downloaded buffers
    w = scaled(WORKLOADS["gemm_bf16_8192"], iters=2)
    ws = Workspace(w)
    res = ws.run()
    assert res.passed == 1 and res.n_iters == 2 and krex.krex_device_status() == 0
    n = w.M
    i, j = ref.sample_indices(w.seed, 2, 4096, n, n)
    want = ref.gemm_sampled_f64(w.seed, n, n, n, i, j)
    ti, tj = torch.from_numpy(i).cuda(), torch.from_numpy(j).cuda()
    got = gen.bf16_to_f32(bits16(ws.out[ti, tj])).astype(np.float64)
    assert np.all(np.abs(got - want) <= ref.gemm_tolerance(want, n))
    r = ws.ref[ti, tj].cpu().numpy().astype(np.float64)
    kk = np.arange(n, dtype=np.int64)
    for s_ in range(256):
        ra = np.abs(gen.widen("bf16", gen.uniform_at("bf16", w.seed, 0, i[s_] * n + kk)).astype(np.float64))
        cb = np.abs(gen.widen("bf16", gen.uniform_at("bf16", w.seed, 1, kk * n + j[s_])).astype(np.float64))
        assert abs(r[s_] - want[s_]) <= n * 2.0 ** -24 * float(ra @ cb), s_
    mx, nv = ref.check_f32(gen.bf16_to_f32(bits16(ws.out)), ws.ref.cpu().numpy(), w.atol, w.rtol)
    assert nv == 0 == int(res.check.n_violations)
    assert ref.check_bits(res.check.max_abs_err) == ref.check_bits(mx)


@pytest.mark.parametrize("name", ["gemm_bf16_4096", "gemm_f16_4096"])
def test_gemm_4096_command_full_output_against_the_oracle(name):
    # the 4096^3 commands (bf16 and binary16; five timed iterations instead of
    # a hundred): the inputs bit for bit, every output of the candidate within
    # the tolerance of the oracle's fp64 product, the reference within the
    # fp32 summation bound, and the verdict equal to the oracle's check
    w = scaled(WORKLOADS[name], iters=5)
    ws = Workspace(w)
    res = ws.run()
    assert res.passed == 1 and res.n_iters == 5 and krex.krex_device_status() == 0
    ah, bh = gen.uniform(w.dtype, w.seed, 0, w.M, w.K), gen.uniform(w.dtype, w.seed, 1, w.K, w.N)
    assert np.array_equal(bits16(ws.inputs[0]), ah) and np.array_equal(bits16(ws.inputs[1]), bh)
    want = ref.gemm_f64(ah, bh, dtype=w.dtype)
    out = gen.widen(w.dtype, bits16(ws.out))
    assert np.all(np.abs(out.astype(np.float64) - want) <= ref.gemm_tolerance(want, w.K, dtype=w.dtype))
    r32 = ws.ref.cpu().numpy()
    fa, fb = gen.widen(w.dtype, ah).astype(np.float64), gen.widen(w.dtype, bh).astype(np.float64)
    assert np.all(np.abs(r32 - want) <= w.K * 2.0 ** -24 * (np.abs(fa) @ np.abs(fb)))
    mx, nv = ref.check_f32(out, r32, w.atol, w.rtol)
    assert nv == 0 == int(res.check.n_violations)
    assert ref.check_bits(res.check.max_abs_err) == ref.check_bits(mx)
