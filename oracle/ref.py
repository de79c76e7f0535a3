"""Plain CPU definitions of the command's results (oracle — test infrastructure only).

Each function restates a definition; none blocks, fuses or reorders beyond
what the definition says.  fp64 unless the definition fixes fp32.
"""
from __future__ import annotations

import math
from fractions import Fraction

import numpy as np

from . import gen


# ------------------------------------------------------------------ GEMM ----

def gemm_f64(a_bits: np.ndarray, b_bits: np.ndarray, dtype: str = "bf16") -> np.ndarray:
    """C = A·B in fp64 from 16-bit operands (bit patterns of `dtype`, "bf16"
    or "f16").

    The candidate of the paper's GEMM benchmarking command (Section 2.1,
    Figure 1a) computes C[i,j] = Σ_k A[i,k]·B[k,j]; a single fp64 matmul is
    that sum (each 16-bit product is exact in fp64; only the additions round).
    """
    a = gen.widen(dtype, a_bits).astype(np.float64)
    b = gen.widen(dtype, b_bits).astype(np.float64)
    return a @ b


def gemm_exact_scaled(a_bits: np.ndarray, b_bits: np.ndarray, dtype: str = "bf16") -> np.ndarray:
    """Exact C·2^(2s) as int64, for operands that are multiples of 2^-s in
    [-1, 1] (s = 23 for bf16, 24 for fp16).

    Every generated bf16 value x satisfies x·2²³ ∈ ℤ (binary16 values in
    [-1, 1]: x·2²⁴ ∈ ℤ, the subnormal step) and |x·2^s| ≤ 2^s, so each
    product is an integer ≤ 2^(2s) and a K ≤ 2¹⁴ sum stays below 2⁶²: int64
    arithmetic is exact.  Plain loop over k for clarity (tiny shapes).
    """
    sc = 24 if dtype == "f16" else 23
    a = gen.widen(dtype, a_bits).astype(np.float64) * 2.0 ** sc
    b = gen.widen(dtype, b_bits).astype(np.float64) * 2.0 ** sc
    ai = a.astype(np.int64)
    bi = b.astype(np.int64)
    if not (np.array_equal(ai, a) and np.array_equal(bi, b)):
        raise ValueError(f"operands are not multiples of 2^-{sc}")
    if np.abs(ai).max(initial=0) > 2 ** sc or np.abs(bi).max(initial=0) > 2 ** sc:
        raise ValueError("operands exceed |x| <= 1")
    m, k = ai.shape
    n = bi.shape[1]
    if k > 2 ** 14:
        raise ValueError("K > 2^14 could overflow int64")
    c = np.zeros((m, n), dtype=np.int64)
    for kk in range(k):
        c += np.outer(ai[:, kk], bi[kk, :])
    return c


def gemm_sampled_f64(seed: int, M: int, N: int, K: int, rows, cols,
                     tid_a: int = 0, tid_b: int = 1, dtype: str = "bf16") -> np.ndarray:
    """C[rows[s], cols[s]] in fp64, regenerating only the needed row of A and
    column of B from the counter-based generator (no GPU data involved)."""
    rows = np.asarray(rows, dtype=np.int64)
    cols = np.asarray(cols, dtype=np.int64)
    out = np.empty(rows.size, dtype=np.float64)
    kk = np.arange(K, dtype=np.int64)
    cache_a: dict = {}
    cache_b: dict = {}
    for s, (i, j) in enumerate(zip(rows.tolist(), cols.tolist())):
        if i not in cache_a:
            cache_a[i] = gen.widen(dtype, gen.uniform_at(dtype, seed, tid_a, i * K + kk)).astype(np.float64)
        if j not in cache_b:
            cache_b[j] = gen.widen(dtype, gen.uniform_at(dtype, seed, tid_b, kk * N + j)).astype(np.float64)
        out[s] = float(np.dot(cache_a[i], cache_b[j]))
    return out


GEMM_RTOL = {"bf16": 2.0 ** -7, "f16": 2.0 ** -10}


def gemm_tolerance(c_ref: np.ndarray, K: int, dtype: str = "bf16") -> np.ndarray:
    """|C_gpu − C_ref| ≤ rtol·|C_ref| + 2⁻¹²·√K with rtol = 2⁻⁷ for bf16 output
    (workload definition: bf16 rounding ≤ 2⁻⁸ relative, fp32 accumulation-order
    error ≪ 2⁻¹²·√K) and, by the same reasoning, 2⁻¹⁰ for binary16 output
    (rounding ≤ 2⁻¹¹ relative in the normal range; the absolute term covers
    the subnormal range, whose step 2⁻²⁴ is far below it)."""
    return GEMM_RTOL[dtype] * np.abs(c_ref) + 2.0 ** -12 * math.sqrt(K)


# --------------------------------------------------------------- softmax ----

def softmax_rows_f64(x: np.ndarray) -> np.ndarray:
    """Numerically stable row softmax, fp64: m = max_j x_j, y = e^(x−m) / Σ e^(x−m)."""
    x = np.asarray(x, dtype=np.float64)
    if x.ndim == 1:
        x = x[None, :]
    m = x.max(axis=1, keepdims=True)
    e = np.exp(x - m)
    s = e.sum(axis=1, keepdims=True)
    return e / s


SOFTMAX_ATOL = 1e-6


# ----------------------------------------------------------------- check ----

def check_f32(out_f32: np.ndarray, ref_f32: np.ndarray, atol: float, rtol: float):
    """The correctness check of a benchmarking command (Section 2.1: the
    command checks its result against a reference and returns a verdict).

    Element-wise in IEEE fp32 (round-to-nearest, no fused multiply-add):
      d   = |out − ref|
      thr = atol + rtol·|ref|
      violation iff not (d ≤ thr)      (a NaN anywhere counts)
    max_abs_err = maximum of d ordered by bit pattern as unsigned, so any NaN
    dominates, and a NaN maximum is reported as the canonical quiet NaN
    0x7FC00000 (IEEE 754 leaves NaN payloads unspecified, and x86, Arm and the
    GPU produce different ones); 0 for no elements.
    Returns (max_abs_err as float32, n_violations).
    """
    o = np.asarray(out_f32, dtype=np.float32).ravel()
    r = np.asarray(ref_f32, dtype=np.float32).ravel()
    if o.size == 0:
        return np.float32(0.0), 0
    with np.errstate(invalid="ignore", over="ignore"):
        d = np.abs(o - r)
        thr = np.float32(atol) + np.float32(rtol) * np.abs(r)
        viol = ~(d <= thr)
    bits = np.where(np.isnan(d), np.uint32(0x7FC00000), d.view(np.uint32))
    mx = bits.max()
    return np.array([mx], dtype=np.uint32).view(np.float32)[0], int(viol.sum())


def check_bits(max_abs_err) -> int:
    return int(np.array([max_abs_err], dtype=np.float32).view(np.uint32)[0])


# ------------------------------------------------------------ statistics ----

def percentile_linear(x, q: float) -> float:
    """Linear interpolation between order statistics (numpy's default method):
    h = (n−1)·q, v = x₍⌊h⌋₎ + (h − ⌊h⌋)·(x₍⌊h⌋+1₎ − x₍⌊h⌋₎).  The paper reports
    medians and p95 without defining the method (Section 2.1; Eq. 1)."""
    xs = sorted(float(v) for v in x)
    n = len(xs)
    if n == 0:
        raise ValueError("empty")
    h = (n - 1) * q
    lo = int(math.floor(h))
    if lo >= n - 1:
        return xs[n - 1]
    return xs[lo] + (h - lo) * (xs[lo + 1] - xs[lo])


def timing_inflation_p95(t_measured, t_native) -> float:
    """Eq. 1 (Section 6.4): P = p95(r) − 1, r = t_measured / t_native per command."""
    r = [float(a) / float(b) for a, b in zip(t_measured, t_native)]
    return percentile_linear(r, 0.95) - 1.0


def pairwise_gap(t_a: float, t_b: float) -> float:
    """Section 6.4: a pair's native duration gap is |t_a − t_b| divided by the smaller."""
    return abs(t_a - t_b) / min(t_a, t_b)


def kendall_tau_b(x, y) -> float:
    """Kendall's τ_b (with ties), by its O(n²) definition over all pairs."""
    n = len(x)
    conc = disc = tx = ty = 0
    for i in range(n):
        for j in range(i + 1, n):
            dx = (x[i] > x[j]) - (x[i] < x[j])
            dy = (y[i] > y[j]) - (y[i] < y[j])
            if dx == 0 and dy == 0:
                continue
            if dx == 0:
                tx += 1
            elif dy == 0:
                ty += 1
            elif dx == dy:
                conc += 1
            else:
                disc += 1
    denom = math.sqrt((conc + disc + tx) * (conc + disc + ty))
    return (conc - disc) / denom if denom else float("nan")


# --------------------------------------------------------------- samples ----

def sample_indices(seed: int, tensor_id: int, n_samples: int, M: int, N: int = 1):
    """Seeded output sample (reading R12 of the workloads: which elements of a
    large output the oracle recomputes): the draws of the stream keyed by
    key(seed, tensor_id), each mapped to a position by sample_indices_from_key."""
    return sample_indices_from_key(gen.stream_key(seed, tensor_id), n_samples, M, N)


def sample_indices_from_key(key: int, n_samples: int, M: int, N: int = 1):
    """Sample s of an M x N output: z_s = draw(key, s);
    i = z_s mod M, j = (z_s >> 32) mod N (duplicates allowed)."""
    z = gen.draws(key, 0, n_samples)
    i = (z % np.uint64(M)).astype(np.int64)
    j = ((z >> np.uint64(32)) % np.uint64(N)).astype(np.int64)
    return i, j


def exact_fraction(s_scaled: int) -> Fraction:
    """Exact value of an int64 C·2⁴⁶ entry."""
    return Fraction(int(s_scaled), 2 ** 46)
