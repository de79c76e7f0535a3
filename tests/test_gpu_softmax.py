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
