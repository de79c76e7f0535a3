"""GPU parity over the launch-configuration space: seeded random GEMM shapes
(tiny, ragged, long K, many tiles), row strides of A, B and C (C rows off 16
bytes too), bf16 and binary16, with and without the split-K workspace, each
under a random tuning record (pair-tile width, stage depth, ring depth, raster
group, tail split, K halves, K alternation).  Every candidate output is within
the GEMM tolerance of the oracle's fp64 product with canaries intact and a
clean device status; every reference tiling gives the same bits, within the
fp32 summation bound of fp64."""
import numpy as np
import pytest
import torch

import paper_2609_30057_gb300 as krex
from gpu_util import Guarded, bits16
from oracle import gen, ref

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    krex.build()
    yield
    krex.krex_set_tuning()


def _shape(rng):
    kind = rng.random()
    if kind < 0.2:
        M, N, K = (int(rng.integers(1, 9)) * 8 for _ in range(3))
    elif kind < 0.55:
        M, N, K = (int(rng.integers(1, 320)) * 8 for _ in range(3))
    elif kind < 0.8:
        M, N = int(rng.integers(1, 129)) * 8, int(rng.integers(1, 129)) * 8
        K = int(rng.integers(256, 1025)) * 8
    else:
        M, N = int(rng.integers(64, 385)) * 8, int(rng.integers(64, 385)) * 8
        K = int(rng.integers(1, 65)) * 8
    while M * N * K > 3_000_000_000:
        K = max(8, (K // 2) // 8 * 8)
    return M, N, K


def _tuning(rng):
    sk = int(rng.choice([0, 64, 128]))
    return dict(gemm_pair_tile_n=int(rng.choice([0, 128, 192, 256, 512])), gemm_stage_k=sk,
                gemm_ring_stages=int(rng.choice([0] + list(range(2, (6 if sk == 64 else 3) + 1)))),
                gemm_raster_group=int(rng.choice([0, 1, 2, 3, 4, 8, 16, 64])),
                gemm_tail_split=int(rng.choice([-1, 0, 1])), gemm_split_k=int(rng.choice([-1, 0, 1])),
                gemm_k_alternate=int(rng.choice([-1, 0, 1])))


def _operands(rng, seed, M, N, K, f16):
    dt = torch.float16 if f16 else torch.bfloat16
    pa, pb = int(rng.choice([0, 8, 16, 64])), int(rng.choice([0, 8, 24]))
    a = torch.empty(M, K + pa, dtype=dt, device="cuda")[:, :K]
    b = torch.empty(K, N + pb, dtype=dt, device="cuda")[:, :N]
    if f16:
        ah, bh = gen.uniform_f16(seed, 0, M, K), gen.uniform_f16(seed, 1, K, N)
        a.copy_(torch.from_numpy(ah.view(np.int16)).view(torch.float16))
        b.copy_(torch.from_numpy(bh.view(np.int16)).view(torch.float16))
    else:
        krex.krex_gen_inputs(seed, 0, krex.KREX_DIST_UNIFORM_PM1, 0.0, a)
        krex.krex_gen_inputs(seed, 1, krex.KREX_DIST_UNIFORM_PM1, 0.0, b)
        ah, bh = gen.uniform_bf16(seed, 0, M, K), gen.uniform_bf16(seed, 1, K, N)
    return a, b, ah, bh


@pytest.mark.parametrize("block", range(8))
def test_candidate_over_random_tunings(block):
    rng = np.random.default_rng(31_000 + block)
    ws = krex.gemm_workspace()
    for case in range(60):
        M, N, K = _shape(rng)
        f16 = bool(rng.random() < 0.25)
        tun = _tuning(rng)
        seed = 200_000 + 1000 * block + case
        a, b, ah, bh = _operands(rng, seed, M, N, K, f16)
        dt = torch.float16 if f16 else torch.bfloat16
        c = Guarded(M, N, dt, ld=N + int(rng.choice([0, 0, 8, 3, 1])))
        op = krex.KREX_OP_GEMM_F16 if f16 else krex.KREX_OP_GEMM_BF16
        krex.krex_set_tuning(**tun)
        if rng.random() < 0.5:
            krex.krex_run_candidate_ws(op, [a, b], c.view, ws)
        else:
            krex.krex_run_candidate(op, [a, b], c.view)
        torch.cuda.synchronize()
        krex.krex_set_tuning()
        where = (M, N, K, f16, tun)
        assert krex.krex_device_status() == 0, where
        assert c.canaries_intact(), where
        dtype = "f16" if f16 else "bf16"
        want = ref.gemm_f64(ah, bh, dtype=dtype)
        gb = bits16(c.view)
        got = (gen.f16_to_f32(gb) if f16 else gen.bf16_to_f32(gb)).astype(np.float64)
        assert np.all(np.abs(got - want) <= ref.gemm_tolerance(want, K, dtype=dtype)), where


def test_reference_tilings_agree_over_random_shapes():
    rng = np.random.default_rng(32_000)
    for case in range(40):
        M, N, K = _shape(rng)
        K = min(K, 2048)
        if case % 3 == 0:  # whole 128 x 128 tiles: the whole-tile kernel where strides allow
            M, N, K = -(-M // 128) * 128, -(-N // 128) * 128, -(-K // 16) * 16
            while M * N * K > 3_000_000_000:
                K = max(16, (K // 2) // 16 * 16)
        f16 = bool(rng.random() < 0.25)
        seed = 300_000 + case
        a, b, ah, bh = _operands(rng, seed, M, N, K, f16)
        op = krex.KREX_OP_GEMM_F16 if f16 else krex.KREX_OP_GEMM_BF16
        outs = []
        for tiling in (-1, int(rng.integers(0, 6))):
            r = Guarded(M, N, torch.float32, ld=N + (0 if case % 3 == 0 else int(rng.choice([0, 4, 1]))))
            krex.krex_set_tuning(reference_tiling=tiling)
            krex.krex_run_reference(op, [a, b], r.view)
            torch.cuda.synchronize()
            krex.krex_set_tuning()
            assert r.canaries_intact(), (M, N, K, tiling)
            outs.append(r.view.cpu().numpy())
        assert np.array_equal(outs[0].view(np.uint32), outs[1].view(np.uint32)), (M, N, K, f16)
        wide = gen.f16_to_f32 if f16 else gen.bf16_to_f32
        fa, fb = wide(ah).astype(np.float64), wide(bh).astype(np.float64)
        want = fa @ fb
        bound = (K + 2) * 2.0 ** -24 * (np.abs(fa) @ np.abs(fb)) + 1e-30
        assert np.all(np.abs(outs[0] - want) <= bound), (M, N, K, f16)
