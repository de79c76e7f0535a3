"""Pins for the oracle's GEMM, softmax, check and statistics (CPU only).

Pins are closed forms, invariants, hand-worked fixtures (tests/golden) and
brute force (Python Fractions, exact int64, per-element fp32 rounding through
fp64) — never a retyped copy of the function under test.
"""
import math
import struct
from fractions import Fraction

import numpy as np
import pytest

from conftest import read_golden
from oracle import gen, ref


def _bf16(x):
    """bf16 bit patterns of values exactly representable in bf16."""
    b = gen.f32_to_bf16(np.asarray(x, dtype=np.float32))
    assert np.array_equal(gen.bf16_to_f32(b), np.asarray(x, dtype=np.float32))
    return b


# ------------------------------------------------------------------ GEMM ----

def test_gemm_hand_worked_fixture():
    lines = read_golden("gemm_small.txt")
    it = iter(lines)

    def mat():
        _, r, c = next(it).split()
        return np.array([[float(v) for v in next(it).split()] for _ in range(int(r))]).reshape(int(r), int(c))

    a, b, c = mat(), mat(), mat()
    got = ref.gemm_f64(_bf16(a), _bf16(b))
    assert np.array_equal(got, c)
    # a transposed-B mistake would not match (B^T is 2x3, so use the square
    # parts): guard that the fixture distinguishes operand order
    assert not np.array_equal(ref.gemm_f64(_bf16(a[:, :2]), _bf16(b[:2, :])),
                              ref.gemm_f64(_bf16(a[:, :2]), _bf16(b[:2, :].T)))


def test_gemm_identity_and_permutation_exact():
    a = gen.uniform_bf16(1, 0, 64, 96)
    eye = _bf16(np.eye(96))
    assert np.array_equal(ref.gemm_f64(a, eye), gen.bf16_to_f32(a).astype(np.float64))
    perm = np.random.default_rng(3).permutation(96)
    p = np.zeros((96, 96))
    p[perm, np.arange(96)] = 1.0                  # (A P)[:, j] = A[:, perm[j]]
    got = ref.gemm_f64(a, _bf16(p))
    assert np.array_equal(got, gen.bf16_to_f32(a).astype(np.float64)[:, perm])


def test_gemm_rank1_closed_form():
    # A = x 1^T, B = 1 y^T  =>  C = K x y^T  (small integers: exact)
    M, N, K = 8, 16, 32
    x = np.arange(1, M + 1, dtype=np.float64) - 4
    y = np.arange(N, dtype=np.float64) - 7
    a = _bf16(np.outer(x, np.ones(K)))
    b = _bf16(np.outer(np.ones(K), y))
    assert np.array_equal(ref.gemm_f64(a, b), K * np.outer(x, y))


def test_gemm_exact_int64_matches_fraction_brute_force():
    a = gen.uniform_bf16(5, 0, 5, 7)
    b = gen.uniform_bf16(5, 1, 7, 3)
    s = ref.gemm_exact_scaled(a, b)
    af = gen.bf16_to_f32(a).astype(np.float64)
    bf = gen.bf16_to_f32(b).astype(np.float64)
    for i in range(5):
        for j in range(3):
            exact = sum(Fraction(af[i, k]) * Fraction(bf[k, j]) for k in range(7))
            assert ref.exact_fraction(s[i, j]) == exact


def test_gemm_f64_within_rounding_bound_of_exact():
    M, N, K = 16, 24, 512
    a = gen.uniform_bf16(6, 0, M, K)
    b = gen.uniform_bf16(6, 1, K, N)
    exact = ref.gemm_exact_scaled(a, b).astype(np.float64) * 2.0 ** -46   # rounds once
    c64 = ref.gemm_f64(a, b)
    absab = np.abs(gen.bf16_to_f32(a).astype(np.float64)) @ np.abs(gen.bf16_to_f32(b).astype(np.float64))
    assert np.all(np.abs(c64 - exact) <= (K + 1) * 2.0 ** -53 * absab + 2.0 ** -60)


def test_gemm_sampled_matches_full():
    seed, M, N, K = 8, 64, 48, 80
    a = gen.uniform_bf16(seed, 0, M, K)
    b = gen.uniform_bf16(seed, 1, K, N)
    full = ref.gemm_f64(a, b)
    i, j = ref.sample_indices(seed, 2, 200, M, N)
    got = ref.gemm_sampled_f64(seed, M, N, K, i, j)
    assert np.allclose(got, full[i, j], rtol=1e-13, atol=1e-13)


def test_sample_indices_in_range_and_seeded():
    i, j = ref.sample_indices(4, 2, 4096, 8192, 8192)
    assert i.min() >= 0 and i.max() < 8192 and j.min() >= 0 and j.max() < 8192
    i2, j2 = ref.sample_indices(4, 2, 4096, 8192, 8192)
    assert np.array_equal(i, i2) and np.array_equal(j, j2)
    assert len(set(zip(i.tolist(), j.tolist()))) > 4000


def test_sample_indices_hand_worked_from_published_draws():
    # (key, s, z_s, M, N, i, j) read off the published SplitMix64 outputs by hand
    rows = [ln.split() for ln in read_golden("sample_indices.txt")]
    for key, s, z_hex, M, N, i_want, j_want in rows:
        key, s, M, N = int(key), int(s), int(M), int(N)
        z = gen.draws(key, s, 1)
        assert int(z[0]) == int(z_hex, 16)
        i, j = ref.sample_indices_from_key(key, s + 1, M, N)
        assert (int(i[s]), int(j[s])) == (int(i_want), int(j_want)), (key, s, M, N)


def test_sample_indices_use_the_stream_of_seed_and_tensor():
    # the seeded form is the key form on key(seed, tensor): the published
    # vector's entry t is stream_key(1234567, t), whose stream starts with
    # draw(stream_key(1234567, t), 0)
    for seed, tid in ((4, 2), (5, 2), (3, 3)):
        key = int(gen.stream_key(seed, tid))
        a = ref.sample_indices(seed, tid, 64, 16384, 16384)
        b = ref.sample_indices_from_key(key, 64, 16384, 16384)
        assert all(np.array_equal(x, y) for x, y in zip(a, b))
        z = gen.draws(key, 0, 1)
        assert int(a[0][0]) == int(z[0]) % 16384 and int(a[1][0]) == (int(z[0]) >> 32) % 16384


def test_gemm_tolerance_hand_worked_fixture():
    # bound = rtol |c| + 2^-12 sqrt(K), worked by hand for the workloads' K
    for dtype, K, c, atol, rtol, bound in (ln.split() for ln in read_golden("gemm_tolerance.txt")):
        K, c, bound = int(K), float(c), float(bound)
        got = ref.gemm_tolerance(np.array([c]), K, dtype=dtype)
        assert got.shape == (1,) and float(got[0]) == bound, (dtype, K, c)
        assert ref.GEMM_RTOL[dtype] == float(rtol)
        assert float(ref.gemm_tolerance(np.array([0.0]), K, dtype=dtype)[0]) == float(atol)


def test_workload_tolerances_are_the_oracle_bound():
    # the product's per-workload atol / rtol (passed to the device check) are
    # the same bound the oracle accepts with: exactly for the K of the fixture,
    # and atol^2 = 2^-24 K for every other K
    from paper_2609_30057_gb300.command import WORKLOADS
    fixture = {(d, int(K)): (float(a), float(r)) for d, K, _, a, r, _ in
               (ln.split() for ln in read_golden("gemm_tolerance.txt"))}
    seen = 0
    for w in WORKLOADS.values():
        if not w.is_gemm:
            assert (w.atol, w.rtol) == (ref.SOFTMAX_ATOL, 0.0)
            continue
        assert w.rtol == ref.GEMM_RTOL[w.dtype]
        if (w.dtype, w.K) in fixture:
            assert (w.atol, w.rtol) == fixture[(w.dtype, w.K)]
            seen += 1
        assert math.isclose((w.atol * 2 ** 12) ** 2, w.K, rel_tol=1e-15)
        assert w.atol == float(ref.gemm_tolerance(np.array([0.0]), w.K, dtype=w.dtype)[0])
    assert seen >= 4


# --------------------------------------------------------------- softmax ----

def test_softmax_hand_worked_fixture():
    env = {"log": math.log}
    for line in read_golden("softmax_small.txt"):
        lhs, rhs = line[len("row"):].split("|")
        x = [eval(v, env) for v in lhs.split(";")]
        y = [float(Fraction(v.strip())) for v in rhs.split(";")]
        got = ref.softmax_rows_f64(np.array(x))[0]
        assert np.allclose(got, y, rtol=0, atol=1e-15)


def test_softmax_rows_sum_to_one_and_shift_invariant():
    x = gen.normal_f32(3, 0, 64, 8192).astype(np.float64)
    y = ref.softmax_rows_f64(x)
    assert np.max(np.abs(y.sum(axis=1) - 1.0)) <= 1e-12
    y2 = ref.softmax_rows_f64(x + 37.25)
    assert np.max(np.abs(y - y2)) <= 1e-15
    assert np.all(y > 0)


def test_softmax_constant_row_and_one_hot():
    y = ref.softmax_rows_f64(np.full((1, 8192), -3.5))
    assert np.all(y == 2.0 ** -13)
    x = np.zeros((1, 10))
    x[0, 4] = 1000.0
    y = ref.softmax_rows_f64(x)
    assert y[0, 4] == 1.0 and np.all(np.delete(y[0], 4) == 0.0)


def test_softmax_brute_force_tiny_rows():
    rng = np.random.default_rng(1)
    for n in (1, 2, 3, 7):
        x = rng.normal(0, 2, size=n)
        m = max(x)
        ex = [math.exp(v - m) for v in x]
        want = [v / math.fsum(ex) for v in ex]
        assert np.allclose(ref.softmax_rows_f64(x)[0], want, rtol=1e-15, atol=0)


def test_softmax_masked_entries_are_zero_and_the_rest_renormalise():
    # an entry of -inf (a masked logit) gets exactly 0, and the others are the
    # softmax of the unmasked entries alone; extremes of the float32 range too
    rng = np.random.default_rng(2)
    x = rng.normal(0, 2, size=(3, 50))
    keep = rng.random((3, 50)) < 0.3
    keep[:, 0] = True
    x[~keep] = -np.inf
    y = ref.softmax_rows_f64(x)
    assert np.all(y[~keep] == 0.0)
    for r in range(3):
        sub = x[r, keep[r]]
        ex = [math.exp(v - max(sub)) for v in sub]
        assert np.allclose(y[r, keep[r]], [v / math.fsum(ex) for v in ex], rtol=1e-15, atol=0)
    big = np.float64(np.finfo(np.float32).max)
    y = ref.softmax_rows_f64(np.array([[big, -big, big, 0.0]]))
    assert np.array_equal(y[0], [0.5, 0.0, 0.5, 0.0])


# ----------------------------------------------------------------- check ----

def _f32(v):
    return struct.unpack("f", struct.pack("f", v))[0]


def _check_brute(out, ref_, atol, rtol):
    """Element by element: each fp32 operation done exactly in Python floats
    (fp64) and rounded once to fp32 with struct — equal to IEEE fp32 ops for
    these magnitudes."""
    mx_bits, nv = 0, 0
    for o, r in zip(out.tolist(), ref_.tolist()):
        d = abs(_f32(o - r))
        thr = _f32(_f32(atol) + _f32(_f32(rtol) * abs(r)))
        if not (d <= thr):
            nv += 1
        bits = 0x7FC00000 if d != d else struct.unpack("I", struct.pack("f", d))[0]
        mx_bits = max(mx_bits, bits)
    return mx_bits, nv


def test_check_zero_difference():
    r = gen.normal_f32(1, 0, 1, 1000)[0]
    mx, nv = ref.check_f32(r, r, 0.0, 0.0)
    assert mx == 0.0 and nv == 0


def test_check_threshold_edge_is_inclusive():
    atol, rtol = np.float32(0.5), np.float32(0.0)
    ref_ = np.array([1.0, 1.0, 1.0], dtype=np.float32)
    out = np.array([1.5, np.nextafter(np.float32(1.5), np.float32(2)), 0.5], dtype=np.float32)
    mx, nv = ref.check_f32(out, ref_, atol, rtol)
    assert nv == 1                                   # exactly at thr passes, one ulp above fails
    assert mx == np.nextafter(np.float32(1.5), np.float32(2)) - np.float32(1.0)


def test_check_nan_counts_and_dominates():
    ref_ = np.array([1.0, 2.0, 3.0], dtype=np.float32)
    out = np.array([1.0, np.nan, 3.0], dtype=np.float32)
    mx, nv = ref.check_f32(out, ref_, 1.0, 1.0)
    assert nv == 1 and np.isnan(mx)
    # any NaN payload, either sign, is reported as the canonical quiet NaN
    odd_nan = np.array([0xFFC01234], dtype=np.uint32).view(np.float32)
    mx, nv = ref.check_f32(np.concatenate([out, odd_nan]), np.append(ref_, 1.0), 1.0, 1.0)
    assert nv == 2 and ref.check_bits(mx) == 0x7FC00000
    mx, nv = ref.check_f32(np.array([np.inf], np.float32), np.array([np.inf], np.float32), 1.0, 0.0)
    assert nv == 1 and np.isnan(mx)                  # inf - inf = NaN


def test_check_signed_zeros_and_empty():
    mx, nv = ref.check_f32(np.array([-0.0], np.float32), np.array([0.0], np.float32), 0.0, 0.0)
    assert nv == 0 and ref.check_bits(mx) == 0
    mx, nv = ref.check_f32(np.zeros(0, np.float32), np.zeros(0, np.float32), 0.0, 0.0)
    assert nv == 0 and mx == 0.0


def test_check_matches_brute_force():
    rng = np.random.default_rng(11)
    r = rng.normal(0, 1, 3000).astype(np.float32)
    o = (r + rng.normal(0, 1e-3, 3000) * (rng.random(3000) < 0.3)).astype(np.float32)
    for atol, rtol in ((1e-3, 1e-2), (2.0 ** -12 * 64, 2.0 ** -7), (0.0, 0.0)):
        mx, nv = ref.check_f32(o, r, atol, rtol)
        bits, nv2 = _check_brute(o, r, atol, rtol)
        assert nv == nv2 and ref.check_bits(mx) == bits


# ------------------------------------------------------------ statistics ----

def test_percentiles_hand_worked_fixture():
    for line in read_golden("percentiles.txt"):
        parts = line[len("data"):].split("|")
        data = [float(v) for v in parts[0].split()]
        for qv in parts[1:]:
            q, want = (float(v) for v in qv.split())
            assert math.isclose(ref.percentile_linear(data, q), want, rel_tol=0, abs_tol=1e-12)


def test_percentiles_match_numpy_linear():
    rng = np.random.default_rng(2)
    for n in (1, 2, 3, 10, 100, 101):
        x = rng.exponential(1.0, n)
        for q in (0.0, 0.05, 0.5, 0.95, 1.0):
            assert math.isclose(ref.percentile_linear(x, q), float(np.percentile(x, 100 * q)),
                                rel_tol=1e-12, abs_tol=1e-15)


def test_timing_inflation_closed_form():
    native = [1.0, 2.0, 3.0, 4.0]
    assert math.isclose(ref.timing_inflation_p95([1.1 * t for t in native], native), 0.1, rel_tol=1e-12)
    assert ref.timing_inflation_p95(native, native) == 0.0


def test_pairwise_gap_paper_example():
    a, b, want = (float(v) for v in read_golden("pairwise_gap.txt")[0].split())
    assert math.isclose(ref.pairwise_gap(a, b), want, rel_tol=1e-12)
    assert math.isclose(ref.pairwise_gap(b, a), want, rel_tol=1e-12)


def test_kendall_tau_b_against_scipy():
    stats = pytest.importorskip("scipy.stats")
    rng = np.random.default_rng(5)
    x = rng.integers(0, 6, 30).tolist()
    y = (np.array(x) + rng.integers(-2, 3, 30)).tolist()
    assert math.isclose(ref.kendall_tau_b(x, y), stats.kendalltau(x, y).statistic, rel_tol=1e-12)
    assert ref.kendall_tau_b([1, 2, 3], [1, 2, 3]) == 1.0
    assert ref.kendall_tau_b([1, 2, 3], [3, 2, 1]) == -1.0


def test_gemm_f16_exact_int64_matches_fraction_brute_force():
    a = gen.uniform_f16(5, 0, 5, 7)
    b = gen.uniform_f16(5, 1, 7, 3)
    s = ref.gemm_exact_scaled(a, b, dtype="f16")
    af = gen.f16_to_f32(a).astype(np.float64)
    bf = gen.f16_to_f32(b).astype(np.float64)
    for i in range(5):
        for j in range(3):
            exact = sum(Fraction(af[i, k]) * Fraction(bf[k, j]) for k in range(7))
            assert Fraction(int(s[i, j]), 2 ** 48) == exact


def test_gemm_f16_f64_within_rounding_bound_of_exact():
    M, N, K = 16, 24, 512
    a = gen.uniform_f16(6, 0, M, K)
    b = gen.uniform_f16(6, 1, K, N)
    exact = ref.gemm_exact_scaled(a, b, dtype="f16").astype(np.float64) * 2.0 ** -48
    c64 = ref.gemm_f64(a, b, dtype="f16")
    absab = np.abs(gen.f16_to_f32(a).astype(np.float64)) @ np.abs(gen.f16_to_f32(b).astype(np.float64))
    assert np.all(np.abs(c64 - exact) <= (K + 1) * 2.0 ** -53 * absab + 2.0 ** -60)


def test_gemm_f16_sampled_matches_full():
    seed, M, N, K = 9, 64, 48, 80
    a = gen.uniform_f16(seed, 0, M, K)
    b = gen.uniform_f16(seed, 1, K, N)
    full = ref.gemm_f64(a, b, dtype="f16")
    i, j = ref.sample_indices(seed, 2, 200, M, N)
    got = ref.gemm_sampled_f64(seed, M, N, K, i, j, dtype="f16")
    assert np.allclose(got, full[i, j], rtol=1e-13, atol=1e-13)
    # the f16 operands are not the bf16 ones: the products differ
    assert not np.array_equal(full, ref.gemm_f64(gen.uniform_bf16(seed, 0, M, K), gen.uniform_bf16(seed, 1, K, N)))
