"""The C-ABI library builds, loads without a GPU, exports every symbol that
include/krex.h declares, and its host-only logic behaves (CPU only: no call
here reaches a kernel)."""
import ctypes
import math
import os
import re

import numpy as np
import pytest

import paper_2609_30057_gb300 as krex
from conftest import ROOT
from oracle import ref as oref


@pytest.fixture(scope="module")
def lib():
    krex.build()
    return krex.lib()


def _header_functions():
    with open(os.path.join(ROOT, "include", "krex.h")) as f:
        text = f.read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"^[A-Za-z_][\w\s\*]*?\b(krex_\w+)\s*\(", text, flags=re.M)))


def test_header_declares_the_boundary():
    names = _header_functions()
    for required in ("krex_gen_inputs", "krex_run_candidate", "krex_flush_l2", "krex_check",
                     "krex_region_begin", "krex_region_end"):
        assert required in names


def test_library_exports_every_declared_symbol(lib):
    for name in _header_functions():
        assert hasattr(lib, name), name


def test_binding_covers_every_declared_symbol():
    assert set(_header_functions()) == set(krex.SIGNATURES)


def test_struct_layouts_match_the_header():
    assert ctypes.sizeof(krex.krex_buf) == 40
    assert ctypes.sizeof(krex.krex_check_result) == 16
    assert ctypes.sizeof(krex.krex_region_opts) == 56
    assert ctypes.sizeof(krex.krex_command) == 80
    assert ctypes.sizeof(krex.krex_command_result) == 88
    assert ctypes.sizeof(krex.krex_command_bufs) == 200


def test_status_strings_and_version(lib):
    assert lib.krex_status_string(0) == b"KREX_OK"
    assert lib.krex_status_string(5) == b"KREX_ERR_TIMEOUT"
    assert lib.krex_version() >= 10000
    assert lib.krex_check_scratch_bytes() >= 16


def test_percentile_matches_oracle_bit_for_bit(lib):
    rng = np.random.default_rng(3)
    for n in (1, 2, 5, 10, 100, 101):
        x = rng.exponential(0.2, n).astype(np.float32)
        for q in (0.0, 0.5, 0.95, 1.0):
            assert krex.krex_percentile(x.tolist(), q) == oref.percentile_linear(x.astype(np.float64), q)


def test_percentile_rejects_bad_arguments(lib):
    out = ctypes.c_double()
    assert lib.krex_percentile(None, 3, 0.5, ctypes.byref(out)) == krex.KREX_ERR_INVALID
    arr = (ctypes.c_float * 2)(1, 2)
    assert lib.krex_percentile(arr, 0, 0.5, ctypes.byref(out)) == krex.KREX_ERR_INVALID
    assert lib.krex_percentile(arr, 2, 1.5, ctypes.byref(out)) == krex.KREX_ERR_INVALID


def _b(ptr, dtype, rows, cols, ld=None):
    return krex.krex_buf(ptr, dtype, 0, rows, cols, cols if ld is None else ld)


def test_invalid_arguments_fail_before_any_cuda_call(lib):
    BF, F = krex.KREX_BF16, krex.KREX_F32
    # null pointer with a nonzero shape
    assert lib.krex_gen_inputs(1, 0, 0, 0.0, _b(None, BF, 4, 4), None) == krex.KREX_ERR_INVALID
    # dtype / distribution mismatch
    assert lib.krex_gen_inputs(1, 0, 0, 0.0, _b(16, F, 4, 4), None) == krex.KREX_ERR_INVALID
    assert lib.krex_gen_inputs(1, 0, 1, math.inf, _b(16, F, 4, 4), None) == krex.KREX_ERR_INVALID
    # ld < cols, bad dtype
    assert lib.krex_gen_inputs(1, 0, 0, 0.0, _b(16, BF, 4, 8, 4), None) == krex.KREX_ERR_INVALID
    assert lib.krex_gen_inputs(1, 0, 0, 0.0, _b(16, 7, 4, 4), None) == krex.KREX_ERR_INVALID
    # empty output is a no-op
    assert lib.krex_gen_inputs(1, 0, 0, 0.0, _b(None, BF, 0, 4), None) == krex.KREX_OK
    # GEMM shape mismatch and wrong input count
    ins = (krex.krex_buf * 2)(_b(16, BF, 8, 16), _b(16, BF, 8, 8))
    assert lib.krex_run_candidate(0, ins, 2, _b(16, BF, 8, 8), None) == krex.KREX_ERR_INVALID
    assert lib.krex_run_candidate(0, ins, 1, _b(16, BF, 8, 8), None) == krex.KREX_ERR_INVALID
    assert lib.krex_run_candidate(9, ins, 2, _b(16, BF, 8, 8), None) == krex.KREX_ERR_INVALID
    # an optional GEMM workspace must be large enough and 16-byte aligned
    # (checked before anything reaches the GPU)
    ok_ins = (krex.krex_buf * 2)(_b(16, BF, 8, 8), _b(16, BF, 8, 8))
    nws = lib.krex_gemm_workspace_bytes()
    assert nws >= 16 << 20
    assert lib.krex_run_candidate_ws(0, ok_ins, 2, _b(16, BF, 8, 8), 4096, nws - 16, None) == krex.KREX_ERR_INVALID
    assert lib.krex_run_candidate_ws(0, ok_ins, 2, _b(16, BF, 8, 8), 4104, nws, None) == krex.KREX_ERR_UNSUPPORTED
    # the reference writes fp32
    ins = (krex.krex_buf * 2)(_b(16, BF, 8, 8), _b(16, BF, 8, 8))
    assert lib.krex_run_reference(0, ins, 2, _b(16, BF, 8, 8), None) == krex.KREX_ERR_INVALID
    # softmax dtypes
    one = (krex.krex_buf * 1)(_b(16, BF, 8, 8))
    assert lib.krex_run_candidate(1, one, 1, _b(16, F, 8, 8), None) == krex.KREX_ERR_INVALID
    # check: shape mismatch, small scratch, null result
    res = krex.krex_check_result()
    assert lib.krex_check(_b(16, BF, 4, 4), _b(16, F, 4, 5), 0, 0, 16, 1 << 20, ctypes.byref(res), None) \
        == krex.KREX_ERR_INVALID
    assert lib.krex_check(_b(16, BF, 4, 4), _b(16, F, 4, 4), 0, 0, 16, 8, ctypes.byref(res), None) \
        == krex.KREX_ERR_INVALID
    assert lib.krex_check(_b(16, BF, 4, 4), _b(16, F, 4, 4), 0, 0, 16, 1 << 20, None, None) \
        == krex.KREX_ERR_INVALID
    # region misuse
    h = ctypes.c_void_p()
    o = krex.krex_region_opts(0, 0, 0, 0, 0, None, 0, None, 0, 0)
    assert lib.krex_region_begin(ctypes.byref(h), None, ctypes.byref(o)) == krex.KREX_ERR_INVALID
    o = krex.krex_region_opts(krex.KREX_MAX_ITERS + 1, 0, 0, 0, 0, None, 0, None, 0, 0)
    assert lib.krex_region_begin(ctypes.byref(h), None, ctypes.byref(o)) == krex.KREX_ERR_INVALID
    o = krex.krex_region_opts(10, 1, 0, 0, 0, None, 1 << 20, None, 0, 0)
    assert lib.krex_region_begin(ctypes.byref(h), None, ctypes.byref(o)) == krex.KREX_ERR_INVALID
    assert lib.krex_iter_begin(None) == krex.KREX_ERR_INVALID
    assert lib.krex_iter_end(None) == krex.KREX_ERR_INVALID
    assert lib.krex_region_end(None, None, 0, None, None, None) == krex.KREX_ERR_INVALID
    assert lib.krex_region_abort(None) == krex.KREX_ERR_INVALID
    assert b"null" in lib.krex_last_error_string() or lib.krex_last_error_string()
    # flush needs aligned scratch
    assert lib.krex_flush_l2(None, 1024, None) == krex.KREX_ERR_INVALID
    assert lib.krex_flush_l2(3, 1024, None) == krex.KREX_ERR_UNSUPPORTED
    assert lib.krex_flush_l2(None, 0, None) == krex.KREX_OK
    assert lib.krex_launch_count() == 0


def test_command_argument_validation(lib):
    cmd = krex.krex_command(0, 3, 0, 0, 8, 8, 8, 1, 2.0, 1e-3, 1e-2, 0, 0, 0)
    bufs = krex.krex_command_bufs()
    res = krex.krex_command_result()
    assert lib.krex_command_run(ctypes.byref(cmd), ctypes.byref(bufs), None, None, None, ctypes.byref(res), None) \
        == krex.KREX_ERR_INVALID
    assert lib.krex_command_run(None, ctypes.byref(bufs), None, None, None, ctypes.byref(res), None) \
        == krex.KREX_ERR_INVALID


def test_tuning_defaults_roundtrip_and_range_checks():
    # the library's launch configuration is an explicit record, never its
    # environment: defaults, a set/get round trip, rejection of out-of-range
    # fields (which leaves the record unchanged), NULL restoring the defaults
    import paper_2609_30057_gb300 as krex
    lib = krex.lib()
    d = krex.krex_tuning()
    lib.krex_tuning_defaults(ctypes.byref(d))
    assert (d.gemm_pair_tile_n, d.gemm_stage_k, d.gemm_ring_stages, d.gemm_raster_group, d.gemm_tail_split,
            d.gemm_split_k, d.gemm_k_alternate, d.reference_tiling, d.wait_timeout_ms) == (0, 0, 0, 0, -1, -1, -1, -1, 0)
    try:
        krex.krex_set_tuning(gemm_pair_tile_n=192, gemm_stage_k=64, gemm_ring_stages=5, gemm_raster_group=3,
                             gemm_tail_split=0, gemm_split_k=1, gemm_k_alternate=0, reference_tiling=2,
                             wait_timeout_ms=500)
        got = krex.krex_get_tuning()
        assert got == {"gemm_pair_tile_n": 192, "gemm_stage_k": 64, "gemm_ring_stages": 5, "gemm_raster_group": 3,
                       "gemm_tail_split": 0, "gemm_split_k": 1, "gemm_k_alternate": 0, "reference_tiling": 2,
                       "wait_timeout_ms": 500}
        bad = [{"gemm_pair_tile_n": 100}, {"gemm_stage_k": 32}, {"gemm_ring_stages": 4},  # 4 > 3 stages of K 128
               {"gemm_ring_stages": 1}, {"gemm_raster_group": 65}, {"gemm_tail_split": 2}, {"gemm_split_k": -2},
               {"gemm_k_alternate": 2},
               {"reference_tiling": 6}, {"wait_timeout_ms": -1}]
        for b in bad:
            with pytest.raises(krex.KrexError, match="INVALID"):
                krex.krex_set_tuning(**b)
            assert krex.krex_get_tuning() == got
        with krex.tuning(gemm_raster_group=9):
            assert krex.krex_get_tuning()["gemm_raster_group"] == 9
        assert krex.krex_get_tuning() == got
    finally:
        assert lib.krex_set_tuning(None) == krex.KREX_OK
    assert krex.krex_get_tuning()["reference_tiling"] == -1


def test_library_reads_no_environment_variables():
    # configuration is explicit (krex_tuning): no translation unit calls getenv
    import glob
    for f in glob.glob(os.path.join(ROOT, "paper_2609_30057_gb300", "csrc", "*")):
        with open(f) as fh:
            assert "getenv" not in fh.read(), f


def test_generator_probe_rejects_bad_arguments_before_any_launch():
    import paper_2609_30057_gb300 as krex
    lib = krex.lib()
    assert lib.krex_probe_generator(7, 64, 1, 2.0, 16, None) == krex.KREX_ERR_INVALID      # bad distribution
    assert lib.krex_probe_generator(0, 64, 1, 2.0, None, None) == krex.KREX_ERR_INVALID    # no sink
    assert lib.krex_probe_generator(0, 60, 1, 2.0, 16, None) == krex.KREX_ERR_INVALID      # not a multiple of 8
    assert lib.krex_probe_generator(1, 0, 1, 2.0, 16, None) == krex.KREX_ERR_INVALID       # no draws
    assert lib.krex_probe_generator(1, 64, 0, 2.0, 16, None) == krex.KREX_ERR_INVALID      # no blocks


def test_host_alloc_rejects_bad_arguments():
    import paper_2609_30057_gb300 as krex
    lib = krex.lib()
    p = ctypes.c_void_p()
    assert lib.krex_host_alloc(0, ctypes.byref(p)) == krex.KREX_ERR_INVALID
    assert lib.krex_host_alloc(4096, None) == krex.KREX_ERR_INVALID
    assert lib.krex_host_free(None, 4096) == krex.KREX_ERR_INVALID


def test_fma_probe_rejects_bad_arguments():
    import paper_2609_30057_gb300 as krex
    lib = krex.lib()
    assert lib.krex_probe_fma(16, 1, None, None) == krex.KREX_ERR_INVALID
    assert lib.krex_probe_fma(0, 1, 16, None) == krex.KREX_ERR_INVALID
    assert lib.krex_probe_fma(16, 0, 16, None) == krex.KREX_ERR_INVALID


def test_missing_library_fails_loudly(tmp_path):
    # without libkrex.so every entry point raises: the binding has no CPU or
    # PyTorch fallback for any step of the path
    import subprocess
    import sys
    code = (
        "import paper_2609_30057_gb300 as k, torch\n"
        f"k.LIB_PATH = {str(tmp_path / 'absent' / 'libkrex.so')!r}\n"
        "k._lib = None\n"
        "calls = [lambda: k.krex_gen_inputs(1, 0, 0, 0.0, torch.empty(8, 8, dtype=torch.bfloat16)),\n"
        "         lambda: k.krex_check_scratch_bytes(), lambda: k.krex_set_tuning()]\n"
        "for c in calls:\n"
        "    try:\n"
        "        c()\n"
        "    except RuntimeError as e:\n"
        "        assert 'no fallback' in str(e), e\n"
        "    else:\n"
        "        raise SystemExit('a call ran without the library')\n"
        "print('raised')\n")
    r = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, cwd=ROOT, timeout=300)
    assert r.returncode == 0 and r.stdout.strip().endswith("raised"), r.stdout + r.stderr
