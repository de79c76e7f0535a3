"""Pins for the oracle's seeded input generator (CPU only).

Each test checks the oracle against something other than itself: a published
test vector, the inverse of the hash, exhaustive comparison of the fp32
routines with fp64 library math, fp64 restatements of Box–Muller from the raw
64-bit draws, exact sympy values of the series coefficients, independent bf16
rounding (torch), and distribution tests.
"""
import math

import numpy as np
import pytest

from conftest import read_golden
from oracle import gen

MASK = (1 << 64) - 1
C1 = 0xBF58476D1CE4E5B9
C2 = 0x94D049BB133111EB


def _unxorshift(z, s):
    """Inverse of z ^= z >> s on 64 bits."""
    x = z
    for _ in range(64 // s + 1):
        x = z ^ (x >> s)
    return x & MASK


def _unmix64(z):
    z = _unxorshift(z, 31)
    z = (z * pow(C2, -1, 1 << 64)) & MASK
    z = _unxorshift(z, 27)
    z = (z * pow(C1, -1, 1 << 64)) & MASK
    return _unxorshift(z, 30)


def test_mix64_zero_is_fixed_point():
    assert gen.mix64(0) == 0


def test_mix64_is_inverted_by_its_algebraic_inverse():
    rng = np.random.default_rng(7)
    for z in rng.integers(0, 2 ** 63, size=200, dtype=np.int64).tolist() + [1, MASK, 2 ** 63]:
        z = int(z) & MASK
        assert _unmix64(gen.mix64(z)) == z


def test_splitmix64_published_vector():
    lines = read_golden("splitmix64_seed1234567.txt")
    seed = int(lines[0].split()[1])
    want = [int(v) for v in lines[1:]]
    got = [gen.stream_key(seed, t) for t in range(len(want))]
    assert got == want


def test_draws_are_splitmix64_outputs_of_the_key():
    # draw(key, j) must be output j of SplitMix64 seeded with key, i.e. the
    # stream keyed by key continues exactly like the published generator.
    key = 1234567
    want = [int(v) for v in read_golden("splitmix64_seed1234567.txt")[1:]]
    assert [gen.draw(key, j) for j in range(5)] == want
    assert gen.draws(key, 0, 5).tolist() == want


def test_stream_keys_differ_per_tensor_and_seed():
    keys = {gen.stream_key(s, t) for s in range(1, 6) for t in range(4)}
    assert len(keys) == 20


# --------------------------------------------------------------- uniform ----

def _bf16_rne_torch(x64):
    torch = pytest.importorskip("torch")
    t = torch.tensor(np.asarray(x64, dtype=np.float32))
    return t.to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)


def test_uniform_matches_fp64_restatement_and_torch_rounding():
    seed, tid, n = 11, 0, 4096
    key = gen.stream_key(seed, tid)
    z = gen.draws(key, 0, n // 2)
    b = np.empty(n, dtype=np.int64)
    b[0::2] = (z >> np.uint64(40)).astype(np.int64)
    b[1::2] = ((z >> np.uint64(8)) & np.uint64(0xFFFFFF)).astype(np.int64)
    x = (b - 2 ** 23).astype(np.float64) / 2.0 ** 23     # exact in fp64 and fp32
    want = _bf16_rne_torch(x)
    got = gen.uniform_bf16(seed, tid, 64, 64).ravel()
    assert np.array_equal(got, want)


def test_uniform_rounding_exhaustive_over_all_24bit_values():
    # Every 24-bit value b, mapped to (b - 2^23) 2^-23 and rounded to bf16,
    # against torch's independent fp32 -> bf16 RNE conversion.
    b = np.arange(1 << 24, dtype=np.int64)
    x = ((b - 2 ** 23).astype(np.float64) / 2.0 ** 23).astype(np.float32)
    want = _bf16_rne_torch(x)
    got = gen.f32_to_bf16(x)
    assert np.array_equal(got, want)


def test_uniform_values_are_multiples_of_2m23_in_closed_unit_interval():
    v = gen.bf16_to_f32(gen.uniform_bf16(1, 0, 256, 256)).astype(np.float64)
    assert v.min() >= -1.0 and v.max() <= 1.0
    s = v * 2.0 ** 23
    assert np.array_equal(s, np.round(s))


def test_uniform_moments():
    v = gen.bf16_to_f32(gen.uniform_bf16(2, 0, 1024, 1024)).astype(np.float64)
    n = v.size
    assert abs(v.mean()) < 5 * math.sqrt(1 / 3 / n)
    assert abs(v.var() - 1 / 3) < 5e-3
    # both halves of a draw are used: even and odd elements are uncorrelated
    e, o = v.ravel()[0::2], v.ravel()[1::2]
    assert abs(np.corrcoef(e, o)[0, 1]) < 5 / math.sqrt(e.size)


def test_uniform_tensors_with_different_ids_are_uncorrelated():
    a = gen.bf16_to_f32(gen.uniform_bf16(4, 0, 512, 512)).astype(np.float64).ravel()
    b = gen.bf16_to_f32(gen.uniform_bf16(4, 1, 512, 512)).astype(np.float64).ravel()
    assert abs(np.corrcoef(a, b)[0, 1]) < 5 / math.sqrt(a.size)


# ------------------------------------------------------ fp32 ln, sincos ----

def _ulp32(x):
    x = np.abs(np.asarray(x, dtype=np.float64))
    e = np.floor(np.log2(np.maximum(x, 2.0 ** -126)))
    return 2.0 ** (e - 23)


def test_ln_exhaustive_within_two_ulp():
    n1 = np.arange(1, (1 << 24) + 1, dtype=np.uint32)
    got = gen.ln_u1(n1).astype(np.float64)
    want = np.log(n1.astype(np.float64)) - 24 * math.log(2.0)
    err = np.abs(got - want)
    ok = want != 0
    assert np.max(err[ok] / _ulp32(want[ok])) <= 2.0
    assert got[-1] == 0.0                       # u1 = 1 -> ln 1 = 0 exactly
    assert np.all(got <= 0.0)


def test_sincos_exhaustive_within_2m23():
    b2 = np.arange(1 << 24, dtype=np.uint32)
    sn, cs = gen.sincos_turns(b2)
    ang = 2.0 * math.pi * b2.astype(np.float64) / 2.0 ** 24
    assert np.max(np.abs(sn - np.sin(ang))) <= 2.0 ** -23
    assert np.max(np.abs(cs - np.cos(ang))) <= 2.0 ** -23
    # exact values at the quadrant points
    q = np.array([0, 1 << 22, 1 << 23, 3 << 22], dtype=np.uint32)
    s4, c4 = gen.sincos_turns(q)
    assert np.array_equal(np.abs(s4), [0, 1, 0, 1]) and np.array_equal(np.abs(c4), [1, 0, 1, 0])


def test_series_coefficients_are_fp32_roundings_of_closed_forms():
    sympy = pytest.importorskip("sympy")
    c = gen.coefficients()

    def rn32(expr):
        return np.float32(float(sympy.N(expr, 50)))

    for k, v in enumerate(c["atanh"]):
        assert v == rn32(sympy.Rational(1, 2 * k + 3))
    for k, v in enumerate(c["sin"]):
        n = 2 * k + 1
        assert v == rn32((-1) ** k * (sympy.pi / 2) ** n / sympy.factorial(n))
    for k, v in enumerate(c["cos"], start=1):
        n = 2 * k
        assert v == rn32((-1) ** k * (sympy.pi / 2) ** n / sympy.factorial(n))
    assert c["ln2"] == rn32(sympy.log(2))
    assert c["sqrt2"] == rn32(sympy.sqrt(2))


# ---------------------------------------------------------------- normal ----

def test_normal_matches_fp64_box_muller_from_raw_draws():
    seed, tid, sigma, npairs = 3, 0, 2.0, 20000
    key = gen.stream_key(seed, tid)
    z = gen.draws(key, 0, npairs)
    u1 = ((z >> np.uint64(40)).astype(np.float64) + 1.0) / 2.0 ** 24
    u2 = ((z >> np.uint64(8)) & np.uint64(0xFFFFFF)).astype(np.float64) / 2.0 ** 24
    r = np.sqrt(-2.0 * np.log(u1))
    want = np.empty(2 * npairs)
    want[0::2] = sigma * r * np.cos(2 * math.pi * u2)
    want[1::2] = sigma * r * np.sin(2 * math.pi * u2)
    got = gen.normal_f32(seed, tid, 1, 2 * npairs, sigma).ravel().astype(np.float64)
    # fp32 error budget: ln and sincos a few ulp, sqrt and products 0.5 ulp each
    assert np.max(np.abs(got - want)) <= 1e-5 * 12
    assert np.max(np.abs(got - want) / np.maximum(np.abs(want), 1e-3)) < 2e-5


def test_normal_moments_and_bound():
    sigma = 2.0
    x = gen.normal_f32(3, 0, 2048, 2048, sigma).astype(np.float64).ravel()
    n = x.size
    assert abs(x.mean()) < 5 * sigma / math.sqrt(n)
    assert abs(x.var() - sigma ** 2) < 5 * sigma ** 2 * math.sqrt(2 / n)
    kurt = np.mean(((x - x.mean()) / x.std()) ** 4)
    assert abs(kurt - 3.0) < 0.02
    # u1 >= 2^-24, so |y| <= sigma sqrt(2 * 24 ln 2)
    assert np.abs(x).max() <= sigma * math.sqrt(2 * 24 * math.log(2)) * (1 + 1e-6)


def test_normal_ks_against_gaussian_cdf():
    stats = pytest.importorskip("scipy.stats")
    x = gen.normal_f32(5, 0, 1000, 1000, 2.0).astype(np.float64).ravel()
    assert stats.kstest(x / 2.0, "norm").pvalue > 1e-3
    # the two members of a pair are independent
    assert abs(np.corrcoef(x[0::2], x[1::2])[0, 1]) < 5 / math.sqrt(x.size / 2)


def test_gather_matches_bulk():
    a = gen.uniform_bf16(9, 1, 33, 47)
    idx = np.array([0, 1, 2, 46, 47, 33 * 47 - 1, 100, 101])
    assert np.array_equal(gen.uniform_bf16_at(9, 1, idx), a.ravel()[idx])
    x = gen.normal_f32(9, 0, 7, 13)
    idx = np.array([0, 1, 12, 13, 90])
    assert np.array_equal(gen.normal_f32_at(9, 0, idx), x.ravel()[idx])


# ------------------------------------------------------------------ fp16 ----

def _f16_numpy(x):
    """numpy's independent fp32 -> binary16 conversion (round to nearest even,
    subnormals included), as bit patterns."""
    with np.errstate(over="ignore"):
        return np.asarray(x, dtype=np.float32).astype(np.float16).view(np.uint16)


def test_f16_rounding_matches_numpy_on_edges_and_random_values():
    edges = [0.0, -0.0, 2.0 ** -24, 2.0 ** -25, 1.5 * 2.0 ** -25, 2.0 ** -26, 3 * 2.0 ** -26,
             2.0 ** -14, 2.0 ** -14 - 2.0 ** -25, 2.0 ** -14 - 2.0 ** -26, 2.0 ** -15 + 2.0 ** -25,
             1.0, 1.0 + 2.0 ** -11, 1.0 + 3 * 2.0 ** -11, 1.0 - 2.0 ** -12, 65504.0, 65519.0,
             65520.0, 1e6, 1e-30, float(np.finfo(np.float32).tiny), 0.333333]
    x = np.array(edges + [-v for v in edges], dtype=np.float32)
    assert np.array_equal(gen.f32_to_f16(x), _f16_numpy(x))
    rng = np.random.default_rng(5)
    # random fp32 bit patterns with exponents around the binary16 range
    u = (rng.integers(0, 1 << 23, 2_000_000, dtype=np.uint32) |
         (rng.integers(127 - 30, 127 + 17, 2_000_000).astype(np.uint32) << 23) |
         (rng.integers(0, 2, 2_000_000).astype(np.uint32) << 31))
    x = u.view(np.float32)
    assert np.array_equal(gen.f32_to_f16(x), _f16_numpy(x))
    inf_nan = np.array([np.inf, -np.inf, np.nan], dtype=np.float32)
    got = gen.f32_to_f16(inf_nan)
    assert got[0] == 0x7C00 and got[1] == 0xFC00 and (got[2] & 0x7C00) == 0x7C00 and (got[2] & 0x3FF)


def test_uniform_f16_is_the_same_draw_rounded_to_binary16():
    # the fp16 operand generator: the bf16 generator's 24-bit values, rounded
    # to binary16 by numpy's independent conversion
    seed, tid, n = 11, 1, 4096
    key = gen.stream_key(seed, tid)
    z = gen.draws(key, 0, n // 2)
    b = np.empty(n, dtype=np.int64)
    b[0::2] = (z >> np.uint64(40)).astype(np.int64)
    b[1::2] = ((z >> np.uint64(8)) & np.uint64(0xFFFFFF)).astype(np.int64)
    x = ((b - 2 ** 23).astype(np.float64) / 2.0 ** 23).astype(np.float32)   # exact
    assert np.array_equal(gen.uniform_f16(seed, tid, 64, 64).ravel(), _f16_numpy(x))


def test_uniform_f16_exhaustive_over_all_24bit_values():
    b = np.arange(1 << 24, dtype=np.int64)
    x = ((b - 2 ** 23).astype(np.float64) / 2.0 ** 23).astype(np.float32)
    assert np.array_equal(gen.f32_to_f16(x), _f16_numpy(x))


def test_uniform_f16_values_are_multiples_of_2m24_in_closed_unit_interval():
    v = gen.f16_to_f32(gen.uniform_f16(3, 0, 256, 256)).astype(np.float64)
    assert v.min() >= -1.0 and v.max() <= 1.0
    s = v * 2.0 ** 24
    assert np.array_equal(s, np.round(s))
    # and the gather form agrees with the bulk form
    idx = np.arange(0, 256 * 256, 37)
    assert np.array_equal(gen.uniform_f16_at(3, 0, idx), gen.uniform_f16(3, 0, 256, 256).ravel()[idx])
