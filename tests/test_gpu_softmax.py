"""GPU parity: the single-pass softmax candidate and the three-pass reference
agree with the oracle's fp64 softmax within 1e-6 absolute, element by element,
on ragged widths (every kernel path) and on sampled rows of the full workload."""
import numpy as np
import pytest
import torch

import paper_2609_30057_gb300 as krex
from gpu_util import Guarded
from oracle import gen, ref

pytestmark = pytest.mark.gpu
ATOL = ref.SOFTMAX_ATOL


@pytest.fixture(scope="module", autouse=True)
def built():
    krex.build()


def _softmax_both(x_np, ld=None):
    rows, cols = x_np.shape
    x = Guarded(rows, cols, torch.float32, ld=ld)
    x.view.copy_(torch.from_numpy(x_np))
    y = Guarded(rows, cols, torch.float32, ld=ld)
    r = Guarded(rows, cols, torch.float32, ld=ld)
    krex.krex_run_candidate(krex.KREX_OP_SOFTMAX_F32, [x.view], y.view)
    krex.krex_run_reference(krex.KREX_OP_SOFTMAX_F32, [x.view], r.view)
    torch.cuda.synchronize()
    assert y.canaries_intact() and r.canaries_intact()
    return y.view.cpu().numpy(), r.view.cpu().numpy()


# widths hitting every register-tile size, the online fallback and ragged tails
@pytest.mark.parametrize("rows,cols", [(1, 1), (3, 3), (5, 4), (7, 1000), (4, 1024), (3, 2048), (2, 4096),
                                       (9, 8192), (2, 16384), (2, 8193), (3, 20000), (300, 512)])
def test_softmax_matches_oracle(rows, cols):
    x = gen.normal_f32(3, 0, rows, cols, 2.0)
    y, r = _softmax_both(x)
    want = ref.softmax_rows_f64(x.astype(np.float64))
    assert np.max(np.abs(y - want)) <= ATOL
    assert np.max(np.abs(r - want)) <= ATOL


def test_softmax_strided():
    x = gen.normal_f32(4, 0, 6, 100, 2.0)
    y, r = _softmax_both(x, ld=108)
    want = ref.softmax_rows_f64(x.astype(np.float64))
    assert np.max(np.abs(y - want)) <= ATOL and np.max(np.abs(r - want)) <= ATOL


def test_softmax_degenerate_rows():
    x = np.zeros((4, 8192), dtype=np.float32)
    x[1] = -3.5                      # constant row -> 2^-13 everywhere
    x[2, 17] = 1000.0                # one-hot limit
    x[3] = np.linspace(-80, 80, 8192, dtype=np.float32)
    y, r = _softmax_both(x)
    want = ref.softmax_rows_f64(x.astype(np.float64))
    assert np.max(np.abs(y - want)) <= ATOL and np.max(np.abs(r - want)) <= ATOL
    assert np.all(y[1] == np.float32(2.0 ** -13))
    assert y[2, 17] == 1.0


def test_softmax_full_workload_sampled_rows():
    rows, cols = 65536, 8192
    x = torch.empty(rows, cols, dtype=torch.float32, device="cuda")
    krex.krex_gen_inputs(3, 0, krex.KREX_DIST_NORMAL, 2.0, x)
    y = torch.empty_like(x)
    r = torch.empty_like(x)
    krex.krex_run_candidate(krex.KREX_OP_SOFTMAX_F32, [x], y)
    krex.krex_run_reference(krex.KREX_OP_SOFTMAX_F32, [x], r)
    torch.cuda.synchronize()
    sample, _ = ref.sample_indices(3, 3, 4096, rows, 1)
    sample = np.unique(sample)
    xs = np.stack([gen.normal_f32_at(3, 0, np.arange(i * cols, (i + 1) * cols), 2.0) for i in sample])
    want = ref.softmax_rows_f64(xs.astype(np.float64))
    st = torch.from_numpy(sample).cuda()
    assert np.max(np.abs(y[st].cpu().numpy() - want)) <= ATOL
    assert np.max(np.abs(r[st].cpu().numpy() - want)) <= ATOL
    # property at any size: every row sums to 1 within fp32 rounding
    assert torch.max(torch.abs(y.double().sum(dim=1) - 1.0)).item() < 1e-4


# one width either side of each register-tile limit (16-byte aligned rows: the
# vector kernels) and past the largest tile (the online kernel)
@pytest.mark.parametrize("cols", [1020, 1028, 2044, 2052, 4092, 4100, 8188, 8196, 16380, 16388])
def test_softmax_either_side_of_each_tile_limit(cols):
    x = gen.normal_f32(6, cols, 3, cols, 2.0)
    y, r = _softmax_both(x)
    want = ref.softmax_rows_f64(x.astype(np.float64))
    assert np.max(np.abs(y - want)) <= ATOL and np.max(np.abs(r - want)) <= ATOL


@pytest.mark.parametrize("pad,ld", [(65, None), (64, 1026), (67, 1027)])
def test_softmax_unaligned_layouts(pad, ld):
    # a row base off a 16-byte boundary or an odd leading dimension rules out
    # the vector loads; the result must not depend on which kernel ran
    rows, cols = 5, 1024
    x_np = gen.normal_f32(7, pad, rows, cols, 2.0)
    x = Guarded(rows, cols, torch.float32, ld=ld, pad_elems=pad)
    x.view.copy_(torch.from_numpy(x_np))
    y = Guarded(rows, cols, torch.float32, ld=ld, pad_elems=pad)
    r = Guarded(rows, cols, torch.float32, ld=ld, pad_elems=pad)
    krex.krex_run_candidate(krex.KREX_OP_SOFTMAX_F32, [x.view], y.view)
    krex.krex_run_reference(krex.KREX_OP_SOFTMAX_F32, [x.view], r.view)
    torch.cuda.synchronize()
    assert y.canaries_intact() and r.canaries_intact()
    want = ref.softmax_rows_f64(x_np.astype(np.float64))
    assert np.max(np.abs(y.view.cpu().numpy() - want)) <= ATOL
    assert np.max(np.abs(r.view.cpu().numpy() - want)) <= ATOL


@pytest.mark.parametrize("cols", [4096, 4097, 20000])
def test_softmax_masked_entries_and_float32_extremes(cols):
    # -inf entries (masked logits) get exactly 0, including threads whose
    # every element is masked; +-FLT_MAX entries split the mass evenly
    x = gen.normal_f32(8, cols, 4, cols, 2.0)
    x[0, :-100] = -np.inf
    x[1, 1:] = -np.inf
    x[2, ::3] = -np.inf
    big = np.finfo(np.float32).max
    x[3, ::7] = big
    x[3, 3::7] = -big
    y, r = _softmax_both(x)
    want = ref.softmax_rows_f64(x.astype(np.float64))
    masked = np.isneginf(x)
    for got in (y, r):
        assert np.max(np.abs(got - want)) <= ATOL
        assert np.all(got[masked] == 0.0)
    assert y[1, 0] == 1.0


@pytest.mark.parametrize("rows,cols", [(0, 16), (4, 0), (0, 0)])
def test_softmax_empty_is_noop(rows, cols):
    x = Guarded(rows, cols, torch.float32, ld=max(cols, 8))
    y = Guarded(rows, cols, torch.float32, ld=max(cols, 8))
    krex.krex_run_candidate(krex.KREX_OP_SOFTMAX_F32, [x.view], y.view)
    krex.krex_run_reference(krex.KREX_OP_SOFTMAX_F32, [x.view], y.view)
    torch.cuda.synchronize()
    assert x.canaries_intact() and y.canaries_intact()


def test_softmax_seeded_random_shapes():
    # ten shapes from a seeded generator (widths from 1 to 20000, across every
    # register-tile size and the online fallback), both kernels within 1e-6
    rng = np.random.default_rng(20261204)
    for t in range(10):
        rows, cols = int(rng.integers(1, 40)), int(rng.integers(1, 20000))
        x = gen.normal_f32(700 + t, 0, rows, cols, 2.0)
        y, r = _softmax_both(x)
        want = ref.softmax_rows_f64(x.astype(np.float64))
        assert np.max(np.abs(y - want)) <= ATOL, (rows, cols)
        assert np.max(np.abs(r - want)) <= ATOL, (rows, cols)
