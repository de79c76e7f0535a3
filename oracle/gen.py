"""ctypes front end for ``oracle/gen.c`` (oracle — test infrastructure only).

The C file is compiled on first use with gcc (``-O2 -ffp-contract=off``, no
fast-math), so the fp32 Box–Muller steps are IEEE single-precision operations
in the stated order on both x86-64 and AArch64.

Generator definition (workload definition: SplitMix64(seed, index) → U[-1,1]
rounded to bf16; N(0, 4) via Box–Muller; the paper's benchmarking command
generates seeded inputs, Section 2.1):

* ``key(seed, t)   = mix64(seed + (t+1)·γ)`` — one stream per tensor id t
* ``draw(key, j)   = mix64(key + (j+1)·γ)`` — SplitMix64's j-th output
* uniform element e: draw e>>1, bits 63..40 (e even) or 31..8 (e odd),
  ``x = (b − 2²³)·2⁻²³``, bf16 = RNE(x) (binary16 = RNE(x) for fp16 operands)
* normal pair j: ``u1 = (hi24+1)·2⁻²⁴``, ``u2 = lo24·2⁻²⁴``,
  ``y = σ·(sqrt(−2 ln u1)·(cos, sin)(2π u2))``
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "gen.c")
_LIB = os.path.join(_HERE, "liboracle_gen.so")
_lock = threading.Lock()
_lib = None

GAMMA = 0x9E3779B97F4A7C15
MASK64 = (1 << 64) - 1


def build(force: bool = False) -> str:
    """Compile gen.c into liboracle_gen.so next to it (if stale)."""
    with _lock:
        if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
            tmp = _LIB + ".tmp.%d" % os.getpid()
            cmd = ["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math",
                   "-fPIC", "-shared", "-o", tmp, _SRC, "-lm"]
            subprocess.run(cmd, check=True)
            os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    if _lib is None:
        build()
        lib = ctypes.CDLL(_LIB)
        u64, u32, i64, f32 = ctypes.c_uint64, ctypes.c_uint32, ctypes.c_int64, ctypes.c_float
        vp = ctypes.c_void_p
        sig = {
            "oracle_mix64": (u64, [u64]),
            "oracle_stream_key": (u64, [u64, u32]),
            "oracle_draw": (u64, [u64, u64]),
            "oracle_f32_to_bf16_rne": (ctypes.c_uint16, [f32]),
            "oracle_uniform_bf16_at": (ctypes.c_uint16, [u64, u64]),
            "oracle_ln_u1": (f32, [u32]),
            "oracle_coefficients": (None, [vp]),
            "oracle_fill_uniform_bf16": (None, [u64, u32, i64, i64, i64, vp]),
            "oracle_fill_uniform_f16": (None, [u64, u32, i64, i64, i64, vp]),
            "oracle_gather_uniform_f16": (None, [u64, u32, vp, i64, vp]),
            "oracle_uniform_f16_at": (ctypes.c_uint16, [u64, u64]),
            "oracle_f32_to_f16_many": (None, [vp, i64, vp]),
            "oracle_fill_normal_f32": (None, [u64, u32, f32, i64, i64, i64, vp]),
            "oracle_gather_uniform_bf16": (None, [u64, u32, vp, i64, vp]),
            "oracle_gather_normal_f32": (None, [u64, u32, f32, vp, i64, vp]),
            "oracle_ln_u1_many": (None, [vp, i64, vp]),
            "oracle_sincos_turns_many": (None, [vp, i64, vp, vp]),
            "oracle_draw_many": (None, [u64, u64, i64, vp]),
        }
        for name, (res, args) in sig.items():
            fn = getattr(lib, name)
            fn.restype = res
            fn.argtypes = args
        _lib = lib
    return _lib


def _ptr(a: np.ndarray):
    assert a.flags["C_CONTIGUOUS"]
    return a.ctypes.data_as(ctypes.c_void_p)


# ---------------------------------------------------------------- hash ----

def mix64(z: int) -> int:
    return int(_load().oracle_mix64(z & MASK64))


def stream_key(seed: int, tensor_id: int) -> int:
    return int(_load().oracle_stream_key(seed & MASK64, tensor_id))


def draw(key: int, j: int) -> int:
    return int(_load().oracle_draw(key & MASK64, j & MASK64))


def draws(key: int, j0: int, n: int) -> np.ndarray:
    out = np.empty(n, dtype=np.uint64)
    _load().oracle_draw_many(key & MASK64, j0 & MASK64, n, _ptr(out))
    return out


# ------------------------------------------------------------- tensors ----

def uniform_bf16(seed: int, tensor_id: int, rows: int, cols: int) -> np.ndarray:
    """Row-major rows×cols bf16 tensor as uint16 bit patterns."""
    out = np.empty((rows, cols), dtype=np.uint16)
    if out.size:
        _load().oracle_fill_uniform_bf16(seed & MASK64, tensor_id, rows, cols, cols, _ptr(out))
    return out


def uniform_f16(seed: int, tensor_id: int, rows: int, cols: int) -> np.ndarray:
    """Row-major rows×cols binary16 tensor as uint16 bit patterns (the same
    24-bit values as uniform_bf16, rounded to binary16)."""
    out = np.empty((rows, cols), dtype=np.uint16)
    if out.size:
        _load().oracle_fill_uniform_f16(seed & MASK64, tensor_id, rows, cols, cols, _ptr(out))
    return out


def uniform_f16_at(seed: int, tensor_id: int, idx) -> np.ndarray:
    idx = np.ascontiguousarray(np.asarray(idx, dtype=np.int64).ravel())
    out = np.empty(idx.size, dtype=np.uint16)
    if idx.size:
        _load().oracle_gather_uniform_f16(seed & MASK64, tensor_id, _ptr(idx), idx.size, _ptr(out))
    return out


def uniform_at(dtype: str, seed: int, tensor_id: int, idx) -> np.ndarray:
    return (uniform_f16_at if dtype == "f16" else uniform_bf16_at)(seed, tensor_id, idx)


def uniform(dtype: str, seed: int, tensor_id: int, rows: int, cols: int) -> np.ndarray:
    return (uniform_f16 if dtype == "f16" else uniform_bf16)(seed, tensor_id, rows, cols)


def normal_f32(seed: int, tensor_id: int, rows: int, cols: int, sigma: float = 2.0) -> np.ndarray:
    out = np.empty((rows, cols), dtype=np.float32)
    if out.size:
        _load().oracle_fill_normal_f32(seed & MASK64, tensor_id, sigma, rows, cols, cols, _ptr(out))
    return out


def uniform_bf16_at(seed: int, tensor_id: int, idx) -> np.ndarray:
    idx = np.ascontiguousarray(np.asarray(idx, dtype=np.int64).ravel())
    out = np.empty(idx.size, dtype=np.uint16)
    if idx.size:
        _load().oracle_gather_uniform_bf16(seed & MASK64, tensor_id, _ptr(idx), idx.size, _ptr(out))
    return out


def normal_f32_at(seed: int, tensor_id: int, idx, sigma: float = 2.0) -> np.ndarray:
    idx = np.ascontiguousarray(np.asarray(idx, dtype=np.int64).ravel())
    out = np.empty(idx.size, dtype=np.float32)
    if idx.size:
        _load().oracle_gather_normal_f32(seed & MASK64, tensor_id, sigma, _ptr(idx), idx.size, _ptr(out))
    return out


def bf16_to_f32(h: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns (uint16) to fp32."""
    return (np.asarray(h, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


def f16_to_f32(h: np.ndarray) -> np.ndarray:
    """Exact widening of binary16 bit patterns (uint16) to fp32."""
    return np.asarray(h, dtype=np.uint16).view(np.float16).astype(np.float32)


def f32_to_f16(x: np.ndarray) -> np.ndarray:
    """RNE narrowing fp32 → binary16 bit patterns (gen.c's routine)."""
    x = np.ascontiguousarray(np.asarray(x, dtype=np.float32).ravel())
    out = np.empty(x.size, dtype=np.uint16)
    if x.size:
        _load().oracle_f32_to_f16_many(_ptr(x), x.size, _ptr(out))
    return out


def widen(dtype: str, h: np.ndarray) -> np.ndarray:
    """Exact fp32 values of 16-bit patterns of `dtype` ("bf16" or "f16")."""
    return f16_to_f32(h) if dtype == "f16" else bf16_to_f32(h)


def f32_to_bf16(x: np.ndarray) -> np.ndarray:
    """RNE narrowing fp32 → bf16 bit patterns (finite values)."""
    u = np.asarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    u = u + 0x7FFF + ((u >> 16) & 1)
    return (u >> 16).astype(np.uint16)


# ----------------------------------------------------- fp32 routines ------

def ln_u1(n1) -> np.ndarray:
    n1 = np.ascontiguousarray(np.asarray(n1, dtype=np.uint32).ravel())
    out = np.empty(n1.size, dtype=np.float32)
    _load().oracle_ln_u1_many(_ptr(n1), n1.size, _ptr(out))
    return out


def sincos_turns(b2):
    b2 = np.ascontiguousarray(np.asarray(b2, dtype=np.uint32).ravel())
    sn = np.empty(b2.size, dtype=np.float32)
    cs = np.empty(b2.size, dtype=np.float32)
    _load().oracle_sincos_turns_many(_ptr(b2), b2.size, _ptr(sn), _ptr(cs))
    return sn, cs


def coefficients() -> dict:
    out = np.empty(16, dtype=np.float32)
    _load().oracle_coefficients(_ptr(out))
    return {"atanh": out[0:4].copy(), "sin": out[4:9].copy(), "cos": out[9:14].copy(),
            "ln2": out[14], "sqrt2": out[15]}
