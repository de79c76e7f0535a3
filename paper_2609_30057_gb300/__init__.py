"""Python binding of libkrex.so — the GB300 benchmarking-command data path.

Argument marshalling only: every step runs in the library's CUDA kernels.
PyTorch supplies device memory (tensors) and streams; nothing here computes.
Functions keep the C names of ``include/krex.h``.  If the library is not built
the first call raises: there is no CPU fallback.

    from paper_2609_30057_gb300 import krex_gen_inputs, krex_run_candidate, region
"""
from __future__ import annotations

import contextlib
import ctypes
import math
import os

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libkrex.so")

KREX_OK, KREX_ERR_INVALID, KREX_ERR_UNSUPPORTED, KREX_ERR_CUDA, KREX_ERR_STATE, KREX_ERR_TIMEOUT, \
    KREX_ERR_DEVICE = range(7)
KREX_BF16, KREX_F32, KREX_F16 = 1, 2, 3
KREX_DIST_UNIFORM_PM1, KREX_DIST_NORMAL = 0, 1
KREX_OP_GEMM_BF16, KREX_OP_SOFTMAX_F32, KREX_OP_GEMM_F16 = 0, 1, 2
KREX_MAX_ITERS = 100000


class krex_buf(ctypes.Structure):
    _fields_ = [("ptr", ctypes.c_void_p), ("dtype", ctypes.c_int32), ("reserved", ctypes.c_int32),
                ("rows", ctypes.c_int64), ("cols", ctypes.c_int64), ("ld", ctypes.c_int64)]


class krex_check_result(ctypes.Structure):
    _fields_ = [("max_abs_err", ctypes.c_float), ("reserved", ctypes.c_uint32),
                ("n_violations", ctypes.c_uint64)]


class krex_region_opts(ctypes.Structure):
    _fields_ = [("max_iters", ctypes.c_int32), ("flush_on_entry", ctypes.c_int32),
                ("pin_cpu", ctypes.c_int32), ("reserved", ctypes.c_int32),
                ("drain_timeout_us", ctypes.c_int64), ("flush_scratch", ctypes.c_void_p),
                ("flush_bytes", ctypes.c_size_t), ("gate", ctypes.c_void_p), ("tenant", ctypes.c_int32),
                ("reserved2", ctypes.c_int32)]


class krex_tuning(ctypes.Structure):
    _fields_ = [("gemm_pair_tile_n", ctypes.c_int32), ("gemm_stage_k", ctypes.c_int32),
                ("gemm_ring_stages", ctypes.c_int32), ("gemm_raster_group", ctypes.c_int32),
                ("gemm_tail_split", ctypes.c_int32), ("gemm_split_k", ctypes.c_int32),
                ("gemm_k_alternate", ctypes.c_int32), ("reference_tiling", ctypes.c_int32),
                ("wait_timeout_ms", ctypes.c_int32)]


class krex_command(ctypes.Structure):
    _fields_ = [("op", ctypes.c_int32), ("warmup", ctypes.c_int32), ("iters", ctypes.c_int32),
                ("pin_cpu", ctypes.c_int32), ("M", ctypes.c_int64), ("N", ctypes.c_int64),
                ("K", ctypes.c_int64), ("seed", ctypes.c_uint64), ("sigma", ctypes.c_float),
                ("atol", ctypes.c_float), ("rtol", ctypes.c_float), ("reserved", ctypes.c_int32),
                ("drain_timeout_us", ctypes.c_int64), ("flush_bytes", ctypes.c_size_t)]


class krex_command_bufs(ctypes.Structure):
    _fields_ = [("in_", krex_buf * 2), ("out", krex_buf), ("ref", krex_buf),
                ("flush_scratch", ctypes.c_void_p), ("check_scratch", ctypes.c_void_p),
                ("check_scratch_bytes", ctypes.c_size_t), ("gemm_workspace", ctypes.c_void_p),
                ("gemm_workspace_bytes", ctypes.c_size_t)]


class krex_command_result(ctypes.Structure):
    _fields_ = [("check", krex_check_result), ("passed", ctypes.c_int32), ("n_iters", ctypes.c_int32),
                ("p50_ms", ctypes.c_double), ("p95_ms", ctypes.c_double), ("launches", ctypes.c_int32),
                ("reserved", ctypes.c_int32), ("phase_ms", ctypes.c_double * 5)]


_P = ctypes.POINTER
_vp, _i32, _u32, _i64, _u64, _f32, _f64, _sz = (ctypes.c_void_p, ctypes.c_int32, ctypes.c_uint32,
                                                ctypes.c_int64, ctypes.c_uint64, ctypes.c_float,
                                                ctypes.c_double, ctypes.c_size_t)

# name -> (restype, argtypes); every symbol include/krex.h declares
SIGNATURES = {
    "krex_gen_inputs": (_i32, [_u64, _u32, _i32, _f32, krex_buf, _vp]),
    "krex_run_candidate": (_i32, [_i32, _P(krex_buf), _i32, krex_buf, _vp]),
    "krex_gemm_workspace_bytes": (_sz, []),
    "krex_run_candidate_ws": (_i32, [_i32, _P(krex_buf), _i32, krex_buf, _vp, _sz, _vp]),
    "krex_run_reference": (_i32, [_i32, _P(krex_buf), _i32, krex_buf, _vp]),
    "krex_flush_l2": (_i32, [_vp, _sz, _vp]),
    "krex_l2_bytes": (_i32, [_P(_sz)]),
    "krex_check_scratch_bytes": (_sz, []),
    "krex_check_scratch_init": (_i32, [_vp, _sz, _vp]),
    "krex_check": (_i32, [krex_buf, krex_buf, _f32, _f32, _vp, _sz, _P(krex_check_result), _vp]),
    "krex_check_launch": (_i32, [krex_buf, krex_buf, _f32, _f32, _vp, _sz, _vp]),
    "krex_check_fetch": (_i32, [_vp, _P(krex_check_result), _vp]),
    "krex_check_noalloc": (_i32, [krex_buf, krex_buf, _f32, _f32, _P(krex_check_result), _vp]),
    "krex_region_begin": (_i32, [_P(_vp), _vp, _P(krex_region_opts)]),
    "krex_iter_begin": (_i32, [_vp]),
    "krex_iter_end": (_i32, [_vp]),
    "krex_region_end": (_i32, [_vp, _P(_f32), _i32, _P(_i32), _P(_f64), _P(_f64)]),
    "krex_region_abort": (_i32, [_vp]),
    "krex_bench_candidate": (_i32, [_i32, _P(krex_buf), _i32, krex_buf, _P(krex_region_opts), _i32, _i32,
                                    _P(_f32), _P(_f64), _P(_f64), _vp, _sz, _vp]),
    "krex_command_run": (_i32, [_P(krex_command), _P(krex_command_bufs), _P(_vp), _vp, _P(_f32),
                                _P(krex_command_result), _vp]),
    "krex_percentile": (_i32, [_P(_f32), _i32, _f64, _P(_f64)]),
    "krex_device_status": (_i32, [_P(_u32)]),
    "krex_device_status_detail": (_i32, [_P(_u64)]),
    "krex_launch_count": (_u64, []),
    "krex_status_string": (ctypes.c_char_p, [_i32]),
    "krex_last_error_string": (ctypes.c_char_p, []),
    "krex_version": (_i32, []),
    "krex_debug_hold_stream": (_i32, [_vp, _P(_i32), _i32]),
    "krex_tuning_defaults": (None, [_P(krex_tuning)]),
    "krex_set_tuning": (_i32, [_P(krex_tuning)]),
    "krex_get_tuning": (_i32, [_P(krex_tuning)]),
    "krex_debug_stall_handover": (_i32, [_i32]),
    "krex_probe_generator": (_i32, [_i32, _u64, _i32, _f32, _vp, _vp]),
    "krex_probe_fma": (_i32, [_i32, _i32, _vp, _vp]),
    "krex_host_alloc": (_i32, [_sz, _P(_vp)]),
    "krex_host_free": (_i32, [_vp, _sz]),
    "krex_gate_shared_bytes": (_sz, [_i32]),
    "krex_gate_shared_init": (_i32, [_vp, _sz, _i32]),
    "krex_gate_shared_attach": (_i32, [_vp, _sz, _P(_vp)]),
    "krex_gate_recover": (_i32, [_vp, _i32, _u64]),
    "krex_ring_bytes": (_sz, [_u32, _u32]),
    "krex_ring_init": (_i32, [_vp, _sz, _u32, _u32]),
    "krex_ring_push": (_i32, [_vp, _vp, _i64]),
    "krex_ring_pop": (_i32, [_vp, _vp, _i64]),
    "krex_ring_count": (_i32, [_vp, _P(_u64)]),
    "krex_ring_set_spin": (_i32, [_vp, _i64]),
    "krex_ring_stats": (_i32, [_vp, _P(_u64)]),
    "krex_gate_create": (_i32, [_P(_vp), _i32]),
    "krex_gate_destroy": (_i32, [_vp]),
    "krex_gate_register": (_i32, [_vp, _vp, _i64, _P(_i32)]),
    "krex_gate_unregister": (_i32, [_vp, _i32]),
    "krex_gate_submit_begin": (_i32, [_vp, _i32, _i64]),
    "krex_gate_submit_end": (_i32, [_vp, _i32]),
    "krex_gate_enter": (_i32, [_vp, _i32, _i64, _P(_u64)]),
    "krex_gate_exit": (_i32, [_vp, _i32, _u64]),
    "krex_gate_state": (_i32, [_vp, _P(_i32), _P(_u64), _P(_i32)]),
}

_lib = None


def build(force: bool = False) -> str:
    """Compile libkrex.so in-tree (nvcc, sm_103a)."""
    from . import _build
    return _build.build(force=force)


def lib() -> ctypes.CDLL:
    """The loaded library; raises if it has not been built."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is not built: run paper_2609_30057_gb300.build() "
                               "(the CUDA path has no fallback)")
        l = ctypes.CDLL(LIB_PATH)
        for name, (res, args) in SIGNATURES.items():
            fn = getattr(l, name)
            fn.restype = res
            fn.argtypes = args
        _lib = l
    return _lib


class KrexError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        l = lib()
        msg = l.krex_last_error_string().decode(errors="replace")
        name = l.krex_status_string(status).decode()
        super().__init__(f"{where}: {name}: {msg}")


def _ok(status: int, where: str):
    if status != KREX_OK:
        raise KrexError(status, where)


# ------------------------------------------------------------- marshalling --

def buf(t, rows: int | None = None, cols: int | None = None) -> krex_buf:
    """krex_buf view of a 2-D (or 1-D = one row) torch tensor with unit column stride."""
    import torch
    if t.dim() == 1:
        t = t.view(1, -1)
    if t.dim() != 2 or (t.size(1) > 1 and t.stride(1) != 1):
        raise ValueError("need a 2-D tensor with unit column stride")
    dt = {torch.bfloat16: KREX_BF16, torch.float32: KREX_F32, torch.float16: KREX_F16}.get(t.dtype)
    if dt is None:
        raise ValueError(f"unsupported dtype {t.dtype}")
    r = t.size(0) if rows is None else rows
    c = t.size(1) if cols is None else cols
    return krex_buf(t.data_ptr(), dt, 0, r, c, t.stride(0) if t.size(0) > 1 else max(c, t.stride(0)))


def _stream(stream) -> int | None:
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    return int(stream.cuda_stream) if hasattr(stream, "cuda_stream") else stream


def _bufs(ts):
    arr = (krex_buf * len(ts))(*[t if isinstance(t, krex_buf) else buf(t) for t in ts])
    return arr, len(ts)


# ------------------------------------------------------------- entry points --

def krex_gen_inputs(seed: int, tensor_id: int, dist: int, sigma: float, out, stream=None):
    b = out if isinstance(out, krex_buf) else buf(out)
    _ok(lib().krex_gen_inputs(seed & (2 ** 64 - 1), tensor_id, dist, sigma, b, _stream(stream)),
        "krex_gen_inputs")


def krex_run_candidate(op: int, inputs, out, stream=None):
    arr, n = _bufs(inputs)
    b = out if isinstance(out, krex_buf) else buf(out)
    _ok(lib().krex_run_candidate(op, arr, n, b, _stream(stream)), "krex_run_candidate")


def krex_gemm_workspace_bytes() -> int:
    return lib().krex_gemm_workspace_bytes()


def gemm_workspace(device="cuda"):
    """A zero-filled GEMM workspace (a uint8 tensor) for krex_run_candidate_ws."""
    import torch
    return torch.zeros(krex_gemm_workspace_bytes(), dtype=torch.uint8, device=device)


def _ptr_bytes(workspace):
    if workspace is None:
        return None, 0
    if isinstance(workspace, int):
        return workspace, krex_gemm_workspace_bytes()
    return workspace.data_ptr(), workspace.numel() * workspace.element_size()


def krex_run_candidate_ws(op: int, inputs, out, workspace, stream=None):
    arr, n = _bufs(inputs)
    b = out if isinstance(out, krex_buf) else buf(out)
    p, nb = _ptr_bytes(workspace)
    _ok(lib().krex_run_candidate_ws(op, arr, n, b, p, nb, _stream(stream)), "krex_run_candidate_ws")


def krex_run_reference(op: int, inputs, ref, stream=None):
    arr, n = _bufs(inputs)
    b = ref if isinstance(ref, krex_buf) else buf(ref)
    _ok(lib().krex_run_reference(op, arr, n, b, _stream(stream)), "krex_run_reference")


def krex_flush_l2(scratch, nbytes: int | None = None, stream=None):
    if nbytes is None:
        nbytes = scratch.numel() * scratch.element_size()
    ptr = scratch if isinstance(scratch, int) else scratch.data_ptr()
    _ok(lib().krex_flush_l2(ptr, nbytes, _stream(stream)), "krex_flush_l2")


def krex_l2_bytes() -> int:
    v = _sz(0)
    _ok(lib().krex_l2_bytes(ctypes.byref(v)), "krex_l2_bytes")
    return v.value


def krex_check_scratch_bytes() -> int:
    return int(lib().krex_check_scratch_bytes())


def krex_check_scratch_init(scratch, stream=None):
    """Zero a check scratch's header once before its first check."""
    ptr = scratch if isinstance(scratch, int) else scratch.data_ptr()
    nbytes = krex_check_scratch_bytes() if isinstance(scratch, int) else scratch.numel() * scratch.element_size()
    _ok(lib().krex_check_scratch_init(ptr, nbytes, _stream(stream)), "krex_check_scratch_init")


def check_scratch(device="cuda"):
    """A check scratch buffer ready for use (zero-filled, torch-allocated)."""
    import torch
    return torch.zeros(krex_check_scratch_bytes(), dtype=torch.uint8, device=device)


def krex_check(out, ref, atol: float, rtol: float, scratch, stream=None):
    """Returns (max_abs_err, n_violations); synchronises the stream."""
    res = krex_check_result()
    ptr = scratch if isinstance(scratch, int) else scratch.data_ptr()
    nbytes = krex_check_scratch_bytes() if isinstance(scratch, int) else scratch.numel() * scratch.element_size()
    bo = out if isinstance(out, krex_buf) else buf(out)
    br = ref if isinstance(ref, krex_buf) else buf(ref)
    _ok(lib().krex_check(bo, br, atol, rtol, ptr, nbytes, ctypes.byref(res), _stream(stream)), "krex_check")
    return res.max_abs_err, int(res.n_violations)


def krex_check_launch(out, ref, atol: float, rtol: float, scratch, stream=None):
    """Asynchronous check kernel; the result stays in `scratch` (see krex_check_fetch)."""
    ptr = scratch if isinstance(scratch, int) else scratch.data_ptr()
    nbytes = krex_check_scratch_bytes() if isinstance(scratch, int) else scratch.numel() * scratch.element_size()
    bo = out if isinstance(out, krex_buf) else buf(out)
    br = ref if isinstance(ref, krex_buf) else buf(ref)
    _ok(lib().krex_check_launch(bo, br, atol, rtol, ptr, nbytes, _stream(stream)), "krex_check_launch")


def krex_check_fetch(scratch, stream=None):
    """(max_abs_err, n_violations) left by krex_check_launch; synchronises the stream."""
    res = krex_check_result()
    ptr = scratch if isinstance(scratch, int) else scratch.data_ptr()
    _ok(lib().krex_check_fetch(ptr, ctypes.byref(res), _stream(stream)), "krex_check_fetch")
    return res.max_abs_err, int(res.n_violations)


def krex_check_noalloc(out, ref, atol: float, rtol: float, stream=None):
    """krex_check with the library's static scratch (no device allocation);
    returns (max_abs_err, n_violations); synchronises the stream."""
    res = krex_check_result()
    bo = out if isinstance(out, krex_buf) else buf(out)
    br = ref if isinstance(ref, krex_buf) else buf(ref)
    _ok(lib().krex_check_noalloc(bo, br, atol, rtol, ctypes.byref(res), _stream(stream)), "krex_check_noalloc")
    return res.max_abs_err, int(res.n_violations)


def krex_region_begin(stream=None, max_iters: int = 100, flush_scratch=None, flush_bytes: int = 0,
                      flush_on_entry: bool = True, pin_cpu: bool = False, drain_timeout_us: int = 0,
                      gate=None, tenant: int = 0) -> int:
    o = krex_region_opts(max_iters, int(bool(flush_on_entry and flush_bytes)), int(pin_cpu), 0, drain_timeout_us,
                         None if flush_scratch is None else
                         (flush_scratch if isinstance(flush_scratch, int) else flush_scratch.data_ptr()),
                         flush_bytes, None if gate is None else gate.handle, tenant, 0)
    h = _vp()
    _ok(lib().krex_region_begin(ctypes.byref(h), _stream(stream), ctypes.byref(o)), "krex_region_begin")
    return h.value


def krex_iter_begin(r: int):
    _ok(lib().krex_iter_begin(r), "krex_iter_begin")


def krex_iter_end(r: int):
    _ok(lib().krex_iter_end(r), "krex_iter_end")


def krex_region_end(r: int, cap: int = KREX_MAX_ITERS):
    """Returns (durations_ms list, p50_ms, p95_ms)."""
    n = _i32(0)
    p50, p95 = _f64(math.nan), _f64(math.nan)
    d = (_f32 * cap)()
    _ok(lib().krex_region_end(r, d, cap, ctypes.byref(n), ctypes.byref(p50), ctypes.byref(p95)), "krex_region_end")
    return list(d[: min(n.value, cap)]), p50.value, p95.value


def krex_region_abort(r: int):
    _ok(lib().krex_region_abort(r), "krex_region_abort")


class Region:
    """Result holder of a ``region`` block."""
    durations_ms: list
    p50_ms: float
    p95_ms: float

    def __init__(self, handle: int):
        self.handle = handle

    @contextlib.contextmanager
    def iteration(self):
        krex_iter_begin(self.handle)
        yield
        krex_iter_end(self.handle)


@contextlib.contextmanager
def region(stream=None, max_iters: int = 100, flush_scratch=None, flush_bytes: int = 0, pin_cpu: bool = False,
           drain_timeout_us: int = 0, gate=None, tenant: int = 0):
    """Critical region (the paper's ``region.critical()``, Section 4.1): enters the
    gate if one is given (sibling tenants blocked and drained), drains the stream,
    flushes L2, optionally pins the thread; ``r.iteration()`` brackets a timed
    iteration; after the block ``r.durations_ms``, ``r.p50_ms``, ``r.p95_ms``."""
    h = krex_region_begin(stream, max_iters, flush_scratch, flush_bytes, True, pin_cpu, drain_timeout_us, gate,
                          tenant)
    r = Region(h)
    try:
        yield r
    except BaseException:
        krex_region_abort(h)
        raise
    r.durations_ms, r.p50_ms, r.p95_ms = krex_region_end(h, max_iters)


def krex_bench_candidate(op: int, inputs, out, warmup: int, iters: int, flush_scratch=None, flush_bytes: int = 0,
                         pin_cpu: bool = False, drain_timeout_us: int = 0, stream=None, gate=None, tenant: int = 0,
                         workspace=None):
    """Native timing loop (optionally gated); returns (durations_ms, p50_ms, p95_ms)."""
    arr, n = _bufs(inputs)
    bo = out if isinstance(out, krex_buf) else buf(out)
    fs = None if flush_scratch is None else (flush_scratch if isinstance(flush_scratch, int) else flush_scratch.data_ptr())
    o = krex_region_opts(max(iters, 1), int(flush_bytes > 0), int(pin_cpu), 0, drain_timeout_us, fs, flush_bytes,
                         None if gate is None else gate.handle, tenant, 0)
    d = (_f32 * max(iters, 1))()
    p50, p95 = _f64(math.nan), _f64(math.nan)
    wp, wn = _ptr_bytes(workspace)
    _ok(lib().krex_bench_candidate(op, arr, n, bo, ctypes.byref(o), warmup, iters, d, ctypes.byref(p50),
                                   ctypes.byref(p95), wp, wn, _stream(stream)), "krex_bench_candidate")
    return list(d[:iters]), p50.value, p95.value


def krex_command_run(cmd: krex_command, bufs: krex_command_bufs, host_in=None, host_out=None, durations=None,
                     stream=None) -> krex_command_result:
    """One benchmarking command.  host_in: list of host data pointers (or None);
    host_out: host data pointer (or None); durations: ctypes float array or None."""
    res = krex_command_result()
    hin = None
    if host_in is not None:
        hin = (_vp * 2)(*[p if p is None else int(p) for p in list(host_in) + [None] * (2 - len(host_in))])
    _ok(lib().krex_command_run(ctypes.byref(cmd), ctypes.byref(bufs), hin, host_out, durations, ctypes.byref(res),
                               _stream(stream)), "krex_command_run")
    return res


def krex_percentile(x, q: float) -> float:
    arr = (_f32 * len(x))(*x)
    out = _f64(0.0)
    _ok(lib().krex_percentile(arr, len(x), q, ctypes.byref(out)), "krex_percentile")
    return out.value


def krex_device_status() -> int:
    """Reads and clears the kernels' device status word; raises KrexError if set."""
    code = _u32(0)
    _ok(lib().krex_device_status(ctypes.byref(code)), "krex_device_status")
    return code.value


def krex_device_status_detail() -> dict:
    """Where the first time-out happened (all zero if none); does not clear."""
    w = (_u64 * 8)()
    _ok(lib().krex_device_status_detail(w), "krex_device_status_detail")
    m = (1 << 21) - 1
    lo, hi = (lambda x: x & 0xFFFFFFFF), (lambda x: x >> 32)
    return {"code": lo(w[0]), "parity": hi(w[0]), "cta": lo(w[1]), "grid": hi(w[1]), "sm": lo(w[2]),
            "cluster_rank": hi(w[2]), "waited_ns": w[3], "producer": (lo(w[4]), hi(w[4])),
            "mma": (lo(w[5]), hi(w[5])), "epilogue": (lo(w[6]), hi(w[6])),
            "MNK": (w[7] & m, (w[7] >> 21) & m, (w[7] >> 42) & m)}


def krex_get_tuning() -> dict:
    t = krex_tuning()
    _ok(lib().krex_get_tuning(ctypes.byref(t)), "krex_get_tuning")
    return {name: getattr(t, name) for name, _ in krex_tuning._fields_}


def krex_set_tuning(**fields) -> None:
    """Set the process-wide tuning: the defaults with `fields` replaced
    (krex_set_tuning() alone restores the defaults)."""
    t = krex_tuning()
    lib().krex_tuning_defaults(ctypes.byref(t))
    for k, v in fields.items():
        if k not in dict(krex_tuning._fields_):
            raise KeyError(k)
        setattr(t, k, int(v))
    _ok(lib().krex_set_tuning(ctypes.byref(t)), "krex_set_tuning")


class tuning:
    """Context manager: the given tuning fields while inside, the previous
    tuning restored on exit (process-wide: use where no other thread of the
    process launches kernels whose configuration matters meanwhile)."""

    def __init__(self, **fields):
        self.fields = fields
        self.saved = None

    def __enter__(self):
        self.saved = krex_get_tuning()
        krex_set_tuning(**{**self.saved, **self.fields})
        return self

    def __exit__(self, *exc):
        krex_set_tuning(**self.saved)


def krex_probe_generator(dist: int, n_elements: int, blocks: int, sink, sigma: float = 2.0, stream=None):
    """Launch the generator probe (asynchronous): the fill of `dist` over
    n_elements with folds instead of stores; sink: a device tensor of at
    least blocks * 256 * 4 bytes."""
    _ok(lib().krex_probe_generator(dist, n_elements, blocks, sigma, sink.data_ptr(), _stream(stream)),
        "krex_probe_generator")


def krex_probe_fma(iters: int, blocks: int, sink, stream=None):
    """Launch the FP32 FMA-rate probe (asynchronous); sink: a device tensor of
    at least blocks * 256 * 4 bytes."""
    _ok(lib().krex_probe_fma(iters, blocks, sink.data_ptr(), _stream(stream)), "krex_probe_fma")


def host_buffer(shape, dtype):
    """A CPU tensor over page-locked, huge-page-backed host memory from
    krex_host_alloc (for a command's host_in / host_out); the memory is freed
    with the tensor."""
    import weakref

    import torch
    shape = tuple(int(x) for x in shape)
    nbytes = max(1, math.prod(shape) * torch.empty((), dtype=dtype).element_size())
    p = ctypes.c_void_p()
    _ok(lib().krex_host_alloc(nbytes, ctypes.byref(p)), "krex_host_alloc")
    raw = (ctypes.c_uint8 * nbytes).from_address(p.value)
    t = torch.frombuffer(raw, dtype=torch.uint8, count=nbytes)
    out = t[:math.prod(shape) * torch.empty((), dtype=dtype).element_size()].view(dtype).view(shape)
    addr = p.value
    weakref.finalize(raw, lambda: lib().krex_host_free(addr, nbytes))
    out._krex_host_owner = raw   # keeps the mapping alive as long as the tensor
    return out


def krex_debug_stall_handover(on: bool) -> None:
    _ok(lib().krex_debug_stall_handover(1 if on else 0), "krex_debug_stall_handover")


def krex_launch_count() -> int:
    return int(lib().krex_launch_count())


def krex_debug_hold_stream(gate, hold_ms: int, stream=None):
    """Test hook: block `stream` on the host until gate.value != 0 (or hold_ms)."""
    _ok(lib().krex_debug_hold_stream(_stream(stream), ctypes.byref(gate), hold_ms), "krex_debug_hold_stream")


# ------------------------------------------------------------------ gate --

class Gate:
    """The in-region gate (paper Section 4.2): tenants bracket submissions
    with ``submission(t)``; a holder's ``enter``/``exit`` (or a
    ``region(..., gate=g, tenant=t)``) blocks and drains sibling tenants.
    ``Gate(n)`` is the in-process form; ``Gate.attach(addr, nbytes)`` joins a
    gate formatted in shared memory by ``gate_shared_init`` (cross-process)."""

    def __init__(self, max_tenants: int = 64, _handle=None):
        if _handle is not None:
            self.handle = _handle
            return
        h = _vp()
        _ok(lib().krex_gate_create(ctypes.byref(h), max_tenants), "krex_gate_create")
        self.handle = h.value

    @classmethod
    def attach(cls, addr: int, nbytes: int) -> "Gate":
        h = _vp()
        _ok(lib().krex_gate_shared_attach(addr, nbytes, ctypes.byref(h)), "krex_gate_shared_attach")
        return cls(_handle=h.value)

    def recover(self, holder: int, epoch: int):
        _ok(lib().krex_gate_recover(self.handle, holder, epoch), "krex_gate_recover")

    def close(self):
        if self.handle:
            _ok(lib().krex_gate_destroy(self.handle), "krex_gate_destroy")
            self.handle = None

    def register(self, stream=None, timeout_us: int = 0) -> int:
        t = _i32(-1)
        s = None if stream is None else _stream(stream)
        _ok(lib().krex_gate_register(self.handle, s, timeout_us, ctypes.byref(t)), "krex_gate_register")
        return t.value

    def unregister(self, tenant: int):
        _ok(lib().krex_gate_unregister(self.handle, tenant), "krex_gate_unregister")

    def submit_begin(self, tenant: int, timeout_us: int = 0):
        _ok(lib().krex_gate_submit_begin(self.handle, tenant, timeout_us), "krex_gate_submit_begin")

    def submit_end(self, tenant: int):
        _ok(lib().krex_gate_submit_end(self.handle, tenant), "krex_gate_submit_end")

    @contextlib.contextmanager
    def submission(self, tenant: int, timeout_us: int = 0):
        self.submit_begin(tenant, timeout_us)
        try:
            yield
        finally:
            self.submit_end(tenant)

    def enter(self, holder: int, timeout_us: int = 0) -> int:
        e = _u64(0)
        _ok(lib().krex_gate_enter(self.handle, holder, timeout_us, ctypes.byref(e)), "krex_gate_enter")
        return e.value

    def exit(self, holder: int, epoch: int):
        _ok(lib().krex_gate_exit(self.handle, holder, epoch), "krex_gate_exit")

    def state(self):
        h, e, p = _i32(0), _u64(0), _i32(0)
        _ok(lib().krex_gate_state(self.handle, ctypes.byref(h), ctypes.byref(e), ctypes.byref(p)), "krex_gate_state")
        return h.value, e.value, p.value


def gate_shared_bytes(max_tenants: int) -> int:
    return int(lib().krex_gate_shared_bytes(max_tenants))


def gate_shared_init(addr: int, nbytes: int, max_tenants: int):
    _ok(lib().krex_gate_shared_init(addr, nbytes, max_tenants), "krex_gate_shared_init")


class Ring:
    """View of a single-producer single-consumer ring in shared memory
    (paper Section 4.3); ``Ring.init`` formats the memory first."""

    def __init__(self, addr: int):
        self.addr = addr
        n = _u64(0)
        _ok(lib().krex_ring_count(addr, ctypes.byref(n)), "krex_ring_count")  # validates the header

    @staticmethod
    def nbytes(capacity: int, entry_bytes: int) -> int:
        return int(lib().krex_ring_bytes(capacity, entry_bytes))

    @classmethod
    def init(cls, addr: int, nbytes: int, capacity: int, entry_bytes: int) -> "Ring":
        _ok(lib().krex_ring_init(addr, nbytes, capacity, entry_bytes), "krex_ring_init")
        return cls(addr)

    def push(self, entry, timeout_us: int = 0):
        """entry: a ctypes object or a bytes-like object of the ring's entry size."""
        if isinstance(entry, (bytes, bytearray, memoryview)):
            entry = ctypes.create_string_buffer(bytes(entry), len(entry))
        _ok(lib().krex_ring_push(self.addr, ctypes.byref(entry), timeout_us), "krex_ring_push")

    def pop_into(self, entry, timeout_us: int = 0):
        _ok(lib().krex_ring_pop(self.addr, ctypes.byref(entry), timeout_us), "krex_ring_pop")
        return entry

    def count(self) -> int:
        n = _u64(0)
        _ok(lib().krex_ring_count(self.addr, ctypes.byref(n)), "krex_ring_count")
        return n.value

    def set_spin(self, spin_us: int):
        _ok(lib().krex_ring_set_spin(self.addr, spin_us), "krex_ring_set_spin")

    def stats(self) -> dict:
        o = (_u64 * 5)()
        _ok(lib().krex_ring_stats(self.addr, o), "krex_ring_stats")
        return dict(zip(("pushes", "pops", "consumer_parks", "producer_parks", "wakes"), list(o)))


class SharedMap:
    """A file mapped MAP_SHARED (e.g. under /dev/shm): memory every process can
    map for a shared gate or ring.  ``addr`` is this process's address of it."""

    def __init__(self, path: str, nbytes: int, create: bool = False):
        import mmap
        import os
        self.path, self.nbytes = path, nbytes
        flags = os.O_RDWR | (os.O_CREAT if create else 0)
        fd = os.open(path, flags, 0o600)
        try:
            if create:
                os.ftruncate(fd, nbytes)
            self.mm = mmap.mmap(fd, nbytes, mmap.MAP_SHARED, mmap.PROT_READ | mmap.PROT_WRITE)
        finally:
            os.close(fd)
        self._anchor = ctypes.c_char.from_buffer(self.mm)
        self.addr = ctypes.addressof(self._anchor)

