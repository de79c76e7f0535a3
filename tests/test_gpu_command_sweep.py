"""GPU parity of whole benchmarking commands over seeded random settings: the
operation (bf16 GEMM, binary16 GEMM, softmax), shape, seed, warm-up and timed
iteration counts and flush size (none, ragged, several MiB) are drawn from a
seeded generator.  For each command: the candidate's output within the
oracle's tolerance, the reference within its bound, the verdict equal bit for
bit to the oracle's check of the two downloaded outputs, the percentiles
equal to the oracle's linear interpolation of the durations, and the launch
count equal to the command's definition (generation, candidate, reference,
check, one flush on entry and one per iteration when flushing, one candidate
per iteration)."""
import numpy as np
import pytest
import torch

import paper_2609_30057_gb300 as krex
from gpu_util import bits16
from paper_2609_30057_gb300.command import Workload, Workspace
from oracle import gen, ref

pytestmark = pytest.mark.gpu

MiB = 1 << 20


@pytest.fixture(scope="module", autouse=True)
def built():
    krex.build()


def _workload(rng, case):
    kind = rng.random()
    iters = int(rng.integers(1, 13))
    warmup = int(rng.integers(0, 5))
    flush = int(rng.choice([0, 3, 4096 + 5, MiB + 3, 8 * MiB]))
    seed = int(rng.integers(1, 1 << 40))
    if kind < 0.3:
        M, N = int(rng.integers(1, 301)), int(rng.integers(1, 3001))
        return Workload(f"softmax_{case}", krex.KREX_OP_SOFTMAX_F32, M, N, 0, seed=seed, iters=iters,
                        flush_bytes=flush, warmup=warmup, sigma=float(rng.choice([0.5, 2.0, 8.0])))
    op = krex.KREX_OP_GEMM_F16 if kind < 0.5 else krex.KREX_OP_GEMM_BF16
    M, N, K = (int(rng.integers(1, 81)) * 8 for _ in range(3))
    return Workload(f"gemm_{case}", op, M, N, K, seed=seed, iters=iters, flush_bytes=flush, warmup=warmup)


@pytest.mark.parametrize("block", range(6))
def test_random_commands_match_the_oracle(block):
    rng = np.random.default_rng(41_000 + block)
    for case in range(10):
        w = _workload(rng, case)
        ws = Workspace(w)
        res = ws.run()
        torch.cuda.synchronize()
        where = (w.name, w.M, w.N, w.K, w.seed, w.iters, w.warmup, w.flush_bytes)
        assert krex.krex_device_status() == 0, where
        r32 = ws.ref.cpu().numpy()
        if w.is_gemm:
            ah, bh = gen.uniform(w.dtype, w.seed, 0, w.M, w.K), gen.uniform(w.dtype, w.seed, 1, w.K, w.N)
            assert np.array_equal(bits16(ws.inputs[0]), ah) and np.array_equal(bits16(ws.inputs[1]), bh), where
            want = ref.gemm_f64(ah, bh, dtype=w.dtype)
            out = gen.widen(w.dtype, bits16(ws.out))
            assert np.all(np.abs(out.astype(np.float64) - want) <= ref.gemm_tolerance(want, w.K, dtype=w.dtype)), where
            fa = gen.widen(w.dtype, ah).astype(np.float64)
            fb = gen.widen(w.dtype, bh).astype(np.float64)
            assert np.all(np.abs(r32 - want) <= (w.K + 2) * 2.0 ** -24 * (np.abs(fa) @ np.abs(fb)) + 1e-30), where
            n_gen = 2
        else:
            x = gen.normal_f32(w.seed, 0, w.M, w.N, w.sigma)
            assert np.array_equal(ws.inputs[0].cpu().numpy().view(np.uint32), x.view(np.uint32)), where
            want = ref.softmax_rows_f64(x.astype(np.float64))
            out = ws.out.cpu().numpy()
            assert np.max(np.abs(out - want)) <= ref.SOFTMAX_ATOL, where
            assert np.max(np.abs(r32 - want)) <= ref.SOFTMAX_ATOL, where
            n_gen = 1
        # the verdict is the oracle's check of the downloaded outputs, bit for bit
        mx, nv = ref.check_f32(out.astype(np.float32), r32, w.atol, w.rtol)
        assert int(res.check.n_violations) == nv, where
        assert ref.check_bits(res.check.max_abs_err) == ref.check_bits(mx), where
        assert res.passed == (1 if nv == 0 else 0), where
        if not res.passed:
            assert res.n_iters == 0, where
            continue
        assert res.n_iters == w.iters, where
        d = [float(v) for v in ws.durations[:w.iters]]
        assert all(v > 0 for v in d), where
        assert res.p50_ms == ref.percentile_linear(d, 0.5), where
        assert res.p95_ms == ref.percentile_linear(d, 0.95), where
        f = 1 if w.flush_bytes > 0 else 0
        assert res.launches == n_gen + 3 + f + (w.warmup + w.iters) * (1 + f), where
