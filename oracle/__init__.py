"""CPU oracle for the benchmarking-command data path — TEST INFRASTRUCTURE ONLY.

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py`` (its
``cpu_baseline`` leg and its ``--impl reference`` arm) may import this package.
The product path (``paper_2609_30057_gb300``) never imports it and shares no
code, header, table or constant with it.

Contents (each function cites the passage it follows):

* ``gen``     — seeded input generation (SplitMix64 → U[-1,1] bf16 and
  Box–Muller N(0, σ²) fp32), plain C in ``gen.c`` loaded with ctypes.
* ``ref``     — the definitions the candidate and the check must reproduce:
  fp64 GEMM, exact int64 GEMM, fp64 row softmax, the fp32 check predicate,
  linear-interpolated percentiles, p95 timing inflation, pairwise gaps.

Everything here is deliberately plain: loops or single library primitives
(a matmul, an exp), in the order the definitions state, in fp64 unless the
definition fixes fp32 (the generator and the check predicate).

Parity status: every function has at least one pin in ``tests/test_oracle_*``
(closed forms, invariants, exhaustive sweeps, brute force).  Nothing is
"parity unpinned" except measured timings themselves, which are a property
of the hardware.
"""
from . import gen, ref  # noqa: F401
