"""Seeded synthetic inputs shared by the oracle side and the CUDA side of the
tests.  This module holds no arithmetic of the method: it only draws numbers
(numpy PCG64) and builds special matrices.  The method's own seeded inputs
(SplitMix64 / Box-Muller) are generated independently by each side."""
import numpy as np


def rng(seed: int) -> np.random.Generator:
    return np.random.default_rng(seed)


def normal_f32(seed: int, shape, scale: float = 1.0) -> np.ndarray:
    return (rng(seed).standard_normal(shape) * scale).astype(np.float32)


def perturbed(ref: np.ndarray, seed: int, frac: float, scale: float) -> np.ndarray:
    """ref plus N(0, scale^2) noise on a random `frac` of the elements (fp32)."""
    g = rng(seed)
    noise = g.standard_normal(ref.shape) * scale * (g.random(ref.shape) < frac)
    return (ref.astype(np.float64) + noise).astype(np.float32)


def bf16_bits_from_f32(x: np.ndarray) -> np.ndarray:
    """Truncate fp32 to bf16 bit patterns (a data source only: values are then
    exactly representable on both sides)."""
    return (np.asarray(x, dtype=np.float32).view(np.uint32) >> 16).astype(np.uint16)


def identity(n: int) -> np.ndarray:
    return np.eye(n, dtype=np.float32)


def permutation_matrix(n: int, seed: int) -> tuple[np.ndarray, np.ndarray]:
    perm = rng(seed).permutation(n)
    p = np.zeros((n, n), dtype=np.float32)
    p[perm, np.arange(n)] = 1.0
    return p, perm
