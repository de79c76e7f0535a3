"""GPU: the critical region and the native timing loop — durations, their
p50/p95 against the oracle's percentile, misuse errors, and the drain timeout
(driven from the host: a host callback holds the stream; no GPU wait)."""
import ctypes
import math
import threading
import time

import pytest
import torch

import paper_2609_30057_gb300 as krex
from oracle import ref

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    krex.build()


def _gemm_bufs(n=512):
    a = torch.empty(n, n, dtype=torch.bfloat16, device="cuda")
    b = torch.empty(n, n, dtype=torch.bfloat16, device="cuda")
    krex.krex_gen_inputs(1, 0, 0, 0.0, a)
    krex.krex_gen_inputs(1, 1, 0, 0.0, b)
    return a, b, torch.empty(n, n, dtype=torch.bfloat16, device="cuda")


def test_region_context_manager_times_iterations():
    a, b, c = _gemm_bufs()
    flush = torch.empty(64 << 20, dtype=torch.uint8, device="cuda")
    s = torch.cuda.current_stream()
    with krex.region(s, max_iters=20, flush_scratch=flush, flush_bytes=flush.numel()) as r:
        for _ in range(3):
            krex.krex_run_candidate(0, [a, b], c)
        for _ in range(20):
            krex.krex_flush_l2(flush)
            with r.iteration():
                krex.krex_run_candidate(0, [a, b], c)
    assert len(r.durations_ms) == 20 and all(d > 0 for d in r.durations_ms)
    assert r.p50_ms == ref.percentile_linear(r.durations_ms, 0.5)
    assert r.p95_ms == ref.percentile_linear(r.durations_ms, 0.95)


def test_bench_candidate_native_loop():
    a, b, c = _gemm_bufs()
    flush = torch.empty(32 << 20, dtype=torch.uint8, device="cuda")
    d, p50, p95 = krex.krex_bench_candidate(0, [a, b], c, warmup=3, iters=15, flush_scratch=flush,
                                            flush_bytes=flush.numel(), pin_cpu=True)
    assert len(d) == 15 and min(d) > 0
    assert p50 == ref.percentile_linear(d, 0.5) and p95 == ref.percentile_linear(d, 0.95)
    assert p50 <= p95


def test_region_misuse():
    s = torch.cuda.current_stream()
    h = krex.krex_region_begin(s, max_iters=2)
    with pytest.raises(krex.KrexError, match="STATE"):
        krex.krex_region_begin(s, max_iters=2)          # one region per stream
    with pytest.raises(krex.KrexError, match="STATE"):
        krex.krex_iter_end(h)                           # end without begin
    krex.krex_iter_begin(h)
    with pytest.raises(krex.KrexError, match="STATE"):
        krex.krex_iter_begin(h)                         # begin twice
    krex.krex_iter_end(h)
    krex.krex_iter_begin(h)
    krex.krex_iter_end(h)
    with pytest.raises(krex.KrexError, match="INVALID"):
        krex.krex_iter_begin(h)                         # past max_iters
    d, p50, p95 = krex.krex_region_end(h)
    assert len(d) == 2
    # region released: a new one can open
    krex.krex_region_abort(krex.krex_region_begin(s, max_iters=1))


def test_region_with_no_iterations_reports_nan():
    h = krex.krex_region_begin(torch.cuda.current_stream(), max_iters=4)
    d, p50, p95 = krex.krex_region_end(h)
    assert d == [] and math.isnan(p50) and math.isnan(p95)


def test_drain_timeout_then_recovery():
    s = torch.cuda.Stream()
    gate = ctypes.c_int32(0)
    krex.krex_debug_hold_stream(gate, 5000, stream=s)   # stream busy on the host side
    t0 = time.time()
    with pytest.raises(krex.KrexError, match="TIMEOUT"):
        krex.krex_region_begin(s, max_iters=4, drain_timeout_us=200_000)
    assert 0.15 < time.time() - t0 < 3.0
    gate.value = 1                                      # release the stream
    s.synchronize()
    h = krex.krex_region_begin(s, max_iters=4, drain_timeout_us=2_000_000)
    krex.krex_region_end(h)


def test_drain_waits_for_queued_work():
    s = torch.cuda.Stream()
    gate = ctypes.c_int32(0)
    krex.krex_debug_hold_stream(gate, 5000, stream=s)
    threading.Timer(0.2, lambda: setattr(gate, "value", 1)).start()
    t0 = time.time()
    h = krex.krex_region_begin(s, max_iters=1, drain_timeout_us=3_000_000)
    assert time.time() - t0 >= 0.15                     # entry waited for the drain
    assert s.query()
    krex.krex_region_end(h)
