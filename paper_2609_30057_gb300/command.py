"""Benchmarking-command workloads and a device workspace for them.

A workload is one benchmarking command of the paper's Section 2.1 (generate
seeded inputs, run the candidate once and the reference, check it, then time
it in a flushed warm-up + timed loop).  The workloads below are named by
what they are; sizes, seeds and iteration counts are part of the workload
(the last one is a smaller softmax for full ncu captures).

PyTorch only allocates the buffers; ``run`` is a single ``krex_command_run``
call into the library.
"""
from __future__ import annotations

import ctypes
import math
from dataclasses import dataclass, replace

from . import (KREX_BF16, KREX_F32, KREX_OP_GEMM_BF16, KREX_OP_GEMM_F16, KREX_OP_SOFTMAX_F32, buf,
               krex_check_scratch_bytes,
               krex_command, krex_command_bufs, krex_command_run, krex_gemm_workspace_bytes)

MiB = 1 << 20


@dataclass(frozen=True)
class Workload:
    name: str
    op: int
    M: int
    N: int
    K: int
    seed: int
    iters: int
    flush_bytes: int
    warmup: int = 3
    sigma: float = 2.0
    oracle_samples: int | None = None   # None: the oracle checks the full output
    repeat: int = 1                     # commands per measurement

    @property
    def is_gemm(self) -> bool:
        return self.op in (KREX_OP_GEMM_BF16, KREX_OP_GEMM_F16)

    @property
    def dtype(self) -> str:
        """Operand dtype: "bf16", "f16" (GEMMs) or "f32" (softmax)."""
        return {KREX_OP_GEMM_BF16: "bf16", KREX_OP_GEMM_F16: "f16"}.get(self.op, "f32")

    @property
    def atol(self) -> float:
        # GEMM: 2^-12 sqrt(K) (fp32 accumulation order); softmax: 1e-6 absolute
        return 2.0 ** -12 * math.sqrt(self.K) if self.is_gemm else 1e-6

    @property
    def rtol(self) -> float:
        # GEMM: 2^-7 for bf16 output (rounding <= 2^-8 relative), 2^-10 for
        # binary16 output (<= 2^-11); softmax: 0
        return {KREX_OP_GEMM_BF16: 2.0 ** -7, KREX_OP_GEMM_F16: 2.0 ** -10}.get(self.op, 0.0)

    @property
    def flops(self) -> int:
        return 2 * self.M * self.N * self.K if self.is_gemm else 0

    @property
    def candidate_bytes(self) -> int:
        """Algorithmic HBM bytes of one candidate launch."""
        if self.is_gemm:
            return 2 * (self.M * self.K + self.K * self.N + self.M * self.N)
        return 8 * self.M * self.N


WORKLOADS = {
    "gemm_bf16_256": Workload("gemm_bf16_256", KREX_OP_GEMM_BF16, 256, 256, 256, seed=1, iters=10,
                              flush_bytes=32 * MiB),
    "gemm_bf16_4096": Workload("gemm_bf16_4096", KREX_OP_GEMM_BF16, 4096, 4096, 4096, seed=2, iters=100,
                               flush_bytes=256 * MiB),
    "softmax_f32_65536x8192": Workload("softmax_f32_65536x8192", KREX_OP_SOFTMAX_F32, 65536, 8192, 0, seed=3,
                                       iters=100, flush_bytes=256 * MiB, oracle_samples=4096),
    "gemm_bf16_8192": Workload("gemm_bf16_8192", KREX_OP_GEMM_BF16, 8192, 8192, 8192, seed=4, iters=50,
                               flush_bytes=256 * MiB, oracle_samples=4096),
    "gemm_f16_4096": Workload("gemm_f16_4096", KREX_OP_GEMM_F16, 4096, 4096, 4096, seed=2, iters=100,
                              flush_bytes=256 * MiB),
    "gemm_bf16_16384": Workload("gemm_bf16_16384", KREX_OP_GEMM_BF16, 16384, 16384, 16384, seed=5, iters=20,
                                flush_bytes=256 * MiB, oracle_samples=4096, repeat=32),
    # a quarter of the softmax workload's rows (512 MiB in, 512 MiB out, still
    # four times L2): the size at which its kernels are profiled in full
    "softmax_f32_16384x8192": Workload("softmax_f32_16384x8192", KREX_OP_SOFTMAX_F32, 16384, 8192, 0, seed=3,
                                       iters=100, flush_bytes=256 * MiB, oracle_samples=4096),
}


def scaled(w: Workload, **kw) -> Workload:
    return replace(w, **kw)


class Workspace:
    """Caller-owned device buffers of one workload (allocated with torch)."""

    def __init__(self, w: Workload, device="cuda", inputs=None):
        """``inputs``: the caller's own device tensors for the operands (any
        row stride), instead of contiguous new ones."""
        import torch
        self.w = w
        f32 = torch.float32
        if w.is_gemm:
            t16 = torch.float16 if w.op == KREX_OP_GEMM_F16 else torch.bfloat16
            self.inputs = [torch.empty(w.M, w.K, dtype=t16, device=device),
                           torch.empty(w.K, w.N, dtype=t16, device=device)]
            self.out = torch.empty(w.M, w.N, dtype=t16, device=device)
        else:
            self.inputs = [torch.empty(w.M, w.N, dtype=f32, device=device)]
            self.out = torch.empty(w.M, w.N, dtype=f32, device=device)
        if inputs is not None:
            if len(inputs) != len(self.inputs) or any(
                    a.shape != b.shape or a.dtype != b.dtype for a, b in zip(inputs, self.inputs)):
                raise ValueError("inputs must match the workload's operand shapes and dtypes")
            self.inputs = list(inputs)
        self.ref = torch.empty(w.M, w.N, dtype=f32, device=device)
        self.flush = torch.empty(max(w.flush_bytes, 16), dtype=torch.uint8, device=device)
        self.check_scratch = torch.zeros(krex_check_scratch_bytes(), dtype=torch.uint8, device=device)
        # the GEMM's split-K meeting place: zero-filled once, left ready by every call
        self.gemm_ws = (torch.zeros(krex_gemm_workspace_bytes(), dtype=torch.uint8, device=device)
                        if w.is_gemm else None)
        self.durations = (ctypes.c_float * w.iters)()
        self.cmd = krex_command(w.op, w.warmup, w.iters, 0, w.M, w.N, w.K, w.seed, w.sigma, w.atol, w.rtol, 0, 0,
                                w.flush_bytes)
        ins = [buf(t) for t in self.inputs] + [buf(self.inputs[0])] * (2 - len(self.inputs))
        self.bufs = krex_command_bufs((type(ins[0]) * 2)(*ins), buf(self.out), buf(self.ref), self.flush.data_ptr(),
                                      self.check_scratch.data_ptr(), krex_check_scratch_bytes(),
                                      None if self.gemm_ws is None else self.gemm_ws.data_ptr(),
                                      0 if self.gemm_ws is None else self.gemm_ws.numel())

    def run(self, host_in=None, host_out=None, stream=None):
        """One benchmarking command; returns the krex_command_result."""
        return krex_command_run(self.cmd, self.bufs, host_in, host_out, self.durations, stream)

    @property
    def elem_bytes_in(self) -> list[int]:
        return [t.numel() * t.element_size() for t in self.inputs]
