"""GPU: buffers of more than 2^32 elements, where every element index needs 64
bits.  The fills must stay bit-exact past element 2^32 (seeded samples and the
elements around 2^32 against the oracle's gather form), and the check must
count violations planted past 2^32 exactly.  Buffers of 8 to 24 GiB."""
import numpy as np
import pytest
import torch

import paper_2609_30057_gb300 as krex
from oracle import gen, ref

pytestmark = pytest.mark.gpu

ROWS, COLS = (1 << 16) + 1, 1 << 16     # 2^32 + 2^16 elements
N = ROWS * COLS
BEYOND = 1 << 32


@pytest.fixture(scope="module", autouse=True)
def built():
    krex.build()
    yield
    torch.cuda.empty_cache()


def _indices(seed):
    i, _ = ref.sample_indices(seed, 5, 1 << 16, N, 1)
    around = np.arange(BEYOND - 4096, BEYOND + 4096)
    tail = np.arange(N - 4096, N)
    return np.unique(np.concatenate([i, around, tail]))


def _gather(t, idx):
    return t.view(-1)[torch.from_numpy(idx).cuda()].cpu()


def test_uniform_fill_beyond_2_32_elements():
    t = torch.empty(ROWS, COLS, dtype=torch.bfloat16, device="cuda")
    krex.krex_gen_inputs(11, 3, krex.KREX_DIST_UNIFORM_PM1, 0.0, t)
    torch.cuda.synchronize()
    idx = _indices(11)
    got = _gather(t, idx).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(got, gen.uniform_bf16_at(11, 3, idx))
    del t
    torch.cuda.empty_cache()


def test_normal_fill_beyond_2_32_elements():
    t = torch.empty(ROWS, COLS, dtype=torch.float32, device="cuda")
    krex.krex_gen_inputs(12, 0, krex.KREX_DIST_NORMAL, 2.0, t)
    torch.cuda.synchronize()
    idx = _indices(12)
    got = _gather(t, idx).numpy()
    assert np.array_equal(got.view(np.uint32), gen.normal_f32_at(12, 0, idx, 2.0).view(np.uint32))
    del t
    torch.cuda.empty_cache()


def test_check_counts_exactly_beyond_2_32_elements():
    scratch = torch.zeros(krex.krex_check_scratch_bytes(), dtype=torch.uint8, device="cuda")
    r = torch.zeros(ROWS, COLS, dtype=torch.float32, device="cuda")
    o = torch.zeros(ROWS, COLS, dtype=torch.bfloat16, device="cuda")
    planted = torch.tensor([5, BEYOND - 1, BEYOND, BEYOND + 12345, N - 1], device="cuda")
    o.view(-1)[planted] = torch.tensor([0.5, 0.25, 2.0, 1.0, 0.125], dtype=torch.bfloat16, device="cuda")
    mx, nv = krex.krex_check(o, r, 0.1, 0.0, scratch)
    assert nv == 5 and mx == 2.0
    o.view(-1)[BEYOND] = 0.0625          # now within atol: one fewer, and a new maximum
    mx, nv = krex.krex_check(o, r, 0.1, 0.0, scratch)
    assert nv == 4 and mx == 1.0
    del r, o
    torch.cuda.empty_cache()


def test_gemm_output_beyond_2_32_elements():
    # C of (65536 + 200) x (65536 + 136) bf16 (8.6 GiB) from K = 64: ragged
    # pair tiles in both directions, outputs past element 2^32 sampled against
    # the oracle's regenerated rows and columns
    M, N, K, seed = (1 << 16) + 200, (1 << 16) + 136, 64, 13
    a = torch.empty(M, K, dtype=torch.bfloat16, device="cuda")
    b = torch.empty(K, N, dtype=torch.bfloat16, device="cuda")
    krex.krex_gen_inputs(seed, 0, krex.KREX_DIST_UNIFORM_PM1, 0.0, a)
    krex.krex_gen_inputs(seed, 1, krex.KREX_DIST_UNIFORM_PM1, 0.0, b)
    c = torch.full((M, N), float("nan"), dtype=torch.bfloat16, device="cuda")
    krex.krex_run_candidate(krex.KREX_OP_GEMM_BF16, [a, b], c)
    torch.cuda.synchronize()
    assert krex.krex_device_status() == 0
    i, j = ref.sample_indices(seed, 2, 2048, M, N)
    flat = np.concatenate([i * N + j, np.arange(BEYOND - 64, BEYOND + 64), np.arange(M * N - 64, M * N)])
    flat = np.unique(flat)
    ii, jj = flat // N, flat % N
    got = gen.bf16_to_f32(_gather(c, flat).view(torch.int16).numpy().view(np.uint16)).astype(np.float64)
    want = ref.gemm_sampled_f64(seed, M, N, K, ii, jj)
    assert np.all(np.abs(got - want) <= ref.gemm_tolerance(want, K))
    assert torch.isfinite(c[-256:].float()).all().item()   # the last (ragged) pair-tile row written
    del a, b, c
    torch.cuda.empty_cache()
