"""GPU parity: the compare-and-reduce check returns exactly the oracle's
{max_abs_err, n_violations} on the same (host-generated) inputs, for every
dtype pair, layout, edge case and at the full output sizes."""
import math

import numpy as np
import pytest
import torch

import paper_2609_30057_gb300 as krex
import inputs
from gpu_util import Guarded, to_bf16_tensor, to_f16_tensor
from oracle import gen, ref

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def scratch():
    krex.build()
    return torch.zeros(krex.krex_check_scratch_bytes(), dtype=torch.uint8, device="cuda")


class F16Bits(np.ndarray):
    """uint16 binary16 bit patterns (plain uint16 arrays are bf16)."""


def _f16(bits):
    return np.asarray(bits, dtype=np.uint16).view(F16Bits)


def _f32_of(bits_or_f32):
    a = bits_or_f32
    if isinstance(a, F16Bits):
        return gen.f16_to_f32(np.asarray(a).view(np.ndarray))
    a = np.asarray(a)
    return gen.bf16_to_f32(a) if a.dtype == np.uint16 else a.astype(np.float32)


def _dev(a):
    if isinstance(a, F16Bits):
        return to_f16_tensor(np.asarray(a).view(np.ndarray))
    a = np.asarray(a)
    return to_bf16_tensor(a) if a.dtype == np.uint16 else torch.from_numpy(np.ascontiguousarray(a)).cuda()


def _run(out_h, ref_h, atol, rtol, scratch):
    got = krex.krex_check(_dev(out_h), _dev(ref_h), atol, rtol, scratch)
    want = ref.check_f32(_f32_of(out_h), _f32_of(ref_h), atol, rtol)
    assert got[1] == want[1]
    assert ref.check_bits(got[0]) == ref.check_bits(want[0])
    return got


@pytest.mark.parametrize("n", [1, 7, 8, 9, 1000, 4097, 100003])
@pytest.mark.parametrize("pair", ["bf16_f32", "f32_f32", "bf16_bf16", "f32_bf16"])
def test_check_matches_oracle(n, pair, scratch):
    r32 = inputs.normal_f32(n, (1, n))
    o32 = inputs.perturbed(r32, n + 1, 0.3, 0.05)
    o = inputs.bf16_bits_from_f32(o32) if pair.startswith("bf16") else o32
    r = inputs.bf16_bits_from_f32(r32) if pair.endswith("bf16") else r32
    for atol, rtol in ((1e-2, 1e-2), (2.0 ** -12 * 64, 2.0 ** -7), (0.0, 0.0), (1.0, 0.0)):
        _run(o, r, atol, rtol, scratch)


def test_check_strided_layout(scratch):
    rows, cols, ld = 37, 50, 64
    r32 = inputs.normal_f32(1, (rows, cols))
    o32 = inputs.perturbed(r32, 2, 0.2, 0.1)
    go = Guarded(rows, cols, torch.float32, ld=ld)
    go.view.copy_(torch.from_numpy(o32))
    gr = Guarded(rows, cols, torch.float32, ld=ld + 8)
    gr.view.copy_(torch.from_numpy(r32))
    got = krex.krex_check(go.view, gr.view, 1e-2, 1e-2, scratch)
    want = ref.check_f32(o32, r32, 1e-2, 1e-2)
    assert got[1] == want[1] and ref.check_bits(got[0]) == ref.check_bits(want[0])


def test_check_edges(scratch):
    # exact threshold passes, one ulp above fails; NaN counts and dominates; signed zeros
    r = np.array([1.0, 1.0, 2.0, 0.0, 3.0, 5.0], dtype=np.float32)
    o = np.array([1.5, np.nextafter(np.float32(1.5), np.float32(2)), np.nan, -0.0, 3.0, np.inf], dtype=np.float32)
    mx, nv = _run(o, r, 0.5, 0.0, scratch)
    assert nv == 3 and math.isnan(mx)
    _run(r, r, 0.0, 0.0, scratch)
    # empty inputs
    e = torch.empty(0, 4, dtype=torch.float32, device="cuda")
    assert krex.krex_check(e, e, 0.0, 0.0, scratch) == (0.0, 0)


def test_check_launch_then_fetch_equals_check(scratch):
    r32 = inputs.normal_f32(7, (300, 700))
    o32 = inputs.perturbed(r32, 8, 0.2, 1e-3)
    a, b = _dev(o32), _dev(r32)
    krex.krex_check_launch(a, b, 1e-4, 1e-3, scratch)
    got = krex.krex_check_fetch(scratch)
    want = ref.check_f32(o32, r32, 1e-4, 1e-3)
    assert got[1] == want[1] and ref.check_bits(got[0]) == ref.check_bits(want[0])


def test_check_twice_is_deterministic(scratch):
    r32 = inputs.normal_f32(5, (512, 512))
    o32 = inputs.perturbed(r32, 6, 0.5, 1e-3)
    a, b = _dev(o32), _dev(r32)
    first = krex.krex_check(a, b, 1e-4, 1e-3, scratch)
    second = krex.krex_check(a, b, 1e-4, 1e-3, scratch)
    assert first[1] == second[1] and ref.check_bits(first[0]) == ref.check_bits(second[0])


@pytest.mark.parametrize("shape,pair", [((4096, 4096), "bf16_f32"), ((16384, 16384), "bf16_f32"),
                                         ((65536, 8192), "f32_f32")])
def test_check_full_size(shape, pair, scratch):
    # full output sizes of the workloads, planted violations at seeded positions
    r32 = inputs.normal_f32(17, shape, 4.0)
    o32 = r32.copy()
    g = inputs.rng(18)
    idx = g.integers(0, r32.size, 5000)
    o32.ravel()[idx] += g.standard_normal(idx.size).astype(np.float32) * 0.5
    o = inputs.bf16_bits_from_f32(o32) if pair == "bf16_f32" else o32
    atol, rtol = (2.0 ** -12 * math.sqrt(shape[0]), 2.0 ** -7) if pair == "bf16_f32" else (1e-6, 0.0)
    _run(o, r32, atol, rtol, scratch)


@pytest.mark.parametrize("n", [1, 9, 4097, 100003])
@pytest.mark.parametrize("pair", ["f16_f32", "f16_f16", "f32_f16", "f16_bf16"])
def test_check_f16_pairs_match_oracle(n, pair, scratch):
    r32 = inputs.normal_f32(n + 5, (1, n))
    o32 = inputs.perturbed(r32, n + 6, 0.3, 0.05)
    conv = {"f16": lambda x: _f16(gen.f32_to_f16(x.ravel()).reshape(x.shape)),
            "bf16": inputs.bf16_bits_from_f32, "f32": lambda x: x}
    po, pr = pair.split("_")
    o, r = conv[po](o32), conv[pr](r32)
    for atol, rtol in ((1e-2, 1e-2), (2.0 ** -12 * 64, 2.0 ** -10), (0.0, 0.0)):
        _run(o, r, atol, rtol, scratch)



@pytest.mark.parametrize("fill", [0xFF, 0x01])
def test_scratch_that_was_never_zeroed_is_reported_then_initialised(fill):
    # A scratch whose header was not zeroed (ticket 0xFFFFFFFF: no block sees
    # itself last; ticket 0x01010101: a block would see itself last too early
    # or never) gives STATE, never a result; after krex_check_scratch_init the
    # same buffer gives the oracle's result, and keeps doing so call after call.
    o = inputs.normal_f32(51, (300, 517))
    r = inputs.perturbed(o, 52, 0.2, 1e-3)
    bad = torch.full((krex.krex_check_scratch_bytes(),), fill, dtype=torch.uint8, device="cuda")
    with pytest.raises(RuntimeError, match="not ready"):
        krex.krex_check(_dev(o), _dev(r), 1e-4, 0.0, bad)
    krex.krex_check_scratch_init(bad)
    for _ in range(3):
        _run(o, r, 1e-4, 0.0, bad)


def test_scratch_init_rejects_small_or_unaligned_buffers():
    lib = krex.lib()
    buf = torch.zeros(krex.krex_check_scratch_bytes() + 16, dtype=torch.uint8, device="cuda")
    assert lib.krex_check_scratch_init(buf.data_ptr(), 16, None) == krex.KREX_ERR_INVALID
    assert lib.krex_check_scratch_init(buf.data_ptr() + 8, krex.krex_check_scratch_bytes(),
                                       None) == krex.KREX_ERR_UNSUPPORTED
    assert lib.krex_check_scratch_init(None, krex.krex_check_scratch_bytes(), None) == krex.KREX_ERR_INVALID


def test_consecutive_checks_alternate_slots_and_stay_exact():
    # each call uses the result slot of its parity and readies the other: seven
    # calls in a row on one scratch, interleaved with calls on a second scratch,
    # with inputs whose results all differ, each equal to the oracle's check
    s1 = torch.zeros(krex.krex_check_scratch_bytes(), dtype=torch.uint8, device="cuda")
    s2 = torch.zeros(krex.krex_check_scratch_bytes(), dtype=torch.uint8, device="cuda")
    for i in range(7):
        o = inputs.normal_f32(100 + i, (257, 1000 + 37 * i))
        r = inputs.perturbed(o, 200 + i, 0.05 * (i + 1), 10.0 ** -(i % 4 + 2))
        for sc in (s1, s2) if i % 2 else (s1,):
            _run(o, r, 1e-4, 1e-3, sc)


def test_check_seeded_random_shapes(scratch):
    # ten 2-D shapes from a seeded generator (rows x cols up to ~1.5 M
    # elements, odd widths), random tolerances and planted violations: count
    # and max bits equal the oracle's, for the bf16/fp32 and fp32/fp32 pairs
    rng = np.random.default_rng(20261203)
    for t in range(10):
        rows, cols = int(rng.integers(1, 700)), int(rng.integers(1, 2200))
        n = rows * cols
        r32 = inputs.normal_f32(500 + t, (rows, cols))
        o32 = inputs.perturbed(r32, 600 + t, float(rng.uniform(0.01, 0.5)), float(rng.uniform(0.0, 0.2)))
        atol, rtol = float(rng.choice([0.0, 2.0 ** -8, 1e-3, 0.05])), float(rng.choice([0.0, 2.0 ** -7, 0.01]))
        for pair in ("bf16_f32", "f32_f32"):
            o = inputs.bf16_bits_from_f32(o32) if pair.startswith("bf16") else o32
            _run(o, r32, atol, rtol, scratch)
