"""The allocation-free check entry point, called through the C ABI.

krex_check_noalloc serves callers that cannot allocate device memory (their
memory belongs to another allocator, or a cudaMalloc/cudaFree could
synchronise the device in the middle of a measurement).  It must give exactly
the result of krex_check with caller scratch, and keep doing so on repeated
calls that share its one static scratch array.  This file is collected last
on purpose and passes both alone in a fresh process and after the other tests.
"""
import ctypes

import numpy as np
import pytest
import torch

import paper_2609_30057_gb300 as krex
import inputs
from gpu_util import to_bf16_tensor
from oracle import ref

pytestmark = pytest.mark.gpu


def _cases():
    r32 = inputs.normal_f32(31, (2048, 2048), 4.0)
    o32 = inputs.perturbed(r32, 32, 0.01, 0.5)
    yield "bf16_out_f32_ref", to_bf16_tensor(inputs.bf16_bits_from_f32(o32)), torch.from_numpy(r32).cuda(), \
        2.0 ** -12 * 64, 2.0 ** -7
    s32 = inputs.normal_f32(33, (300, 1000))
    t32 = inputs.perturbed(s32, 34, 0.3, 1e-5)
    t32[7, 11] = np.nan
    yield "f32_with_nan", torch.from_numpy(t32).cuda(), torch.from_numpy(s32).cuda(), 1e-6, 0.0
    w32 = inputs.normal_f32(35, (64, 136))
    wide = torch.from_numpy(w32).cuda()
    wide2 = torch.from_numpy(inputs.perturbed(w32, 36, 0.5, 1e-3)).cuda()
    yield "f32_strided", wide[:, :128], wide2[:, :128], 1e-4, 1e-3     # row stride 136


def _call_noalloc(lib, out, ref_t, atol, rtol):
    res = krex.krex_check_result()
    st = lib.krex_check_noalloc(krex.buf(out), krex.buf(ref_t), atol, rtol, ctypes.byref(res),
                                torch.cuda.current_stream().cuda_stream)
    assert st == krex.KREX_OK, lib.krex_last_error_string()
    return res.max_abs_err, int(res.n_violations)


def test_noalloc_check_matches_scratch_check_on_two_calls_in_a_row():
    krex.build()
    lib = krex.lib()
    scratch = torch.zeros(krex.krex_check_scratch_bytes(), dtype=torch.uint8, device="cuda")
    for name, out, ref_t, atol, rtol in _cases():
        want = krex.krex_check(out, ref_t, atol, rtol, scratch)
        first = _call_noalloc(lib, out, ref_t, atol, rtol)
        second = _call_noalloc(lib, out, ref_t, atol, rtol)
        # and the oracle's check of the same two buffers, bit for bit
        o32 = out.float().cpu().numpy() if out.dtype == torch.bfloat16 else out.cpu().numpy()
        oracle = ref.check_f32(o32, ref_t.cpu().numpy(), atol, rtol)
        for got in (first, second):
            assert got[1] == want[1] == oracle[1], name
            assert ref.check_bits(got[0]) == ref.check_bits(want[0]) == ref.check_bits(oracle[0]), name
        assert want[1] > 0, name        # every case has violations to count


def test_noalloc_check_takes_no_device_memory():
    # after a first call (the set-up), a call leaves the device's free memory
    # exactly as it was: nothing is allocated, not even by the driver
    lib = krex.lib()
    o = torch.from_numpy(inputs.normal_f32(37, (1024, 1024))).cuda().half()
    r = torch.from_numpy(inputs.normal_f32(38, (1024, 1024))).cuda()
    _call_noalloc(lib, o, r, 1e-3, 1e-3)
    torch.cuda.synchronize()
    free0, _ = torch.cuda.mem_get_info()
    got = _call_noalloc(lib, o, r, 1e-3, 1e-3)
    torch.cuda.synchronize()
    free1, _ = torch.cuda.mem_get_info()
    assert free1 == free0
    want = ref.check_f32(o.float().cpu().numpy(), r.cpu().numpy(), 1e-3, 1e-3)
    assert got[1] == want[1] and ref.check_bits(got[0]) == ref.check_bits(want[0])


def test_noalloc_check_rejects_bad_arguments():
    lib = krex.lib()
    res = krex.krex_check_result()
    a = krex.krex_buf(16, krex.KREX_F32, 0, 4, 4, 4)
    b = krex.krex_buf(16, krex.KREX_F32, 0, 4, 5, 5)
    assert lib.krex_check_noalloc(a, b, 0.0, 0.0, ctypes.byref(res), None) == krex.KREX_ERR_INVALID
    assert lib.krex_check_noalloc(a, a, 0.0, 0.0, None, None) == krex.KREX_ERR_INVALID
    # a row stride past 2^40 elements is rejected, as krex_check rejects it
    huge = krex.krex_buf(16, krex.KREX_F32, 0, 4, 4, (1 << 40) + 8)
    assert lib.krex_check_noalloc(huge, huge, 0.0, 0.0, ctypes.byref(res), None) == krex.KREX_ERR_INVALID
    scratch = torch.zeros(krex.krex_check_scratch_bytes(), dtype=torch.uint8, device="cuda")
    assert lib.krex_check(huge, huge, 0.0, 0.0, scratch.data_ptr(), scratch.numel(), ctypes.byref(res),
                          None) == krex.KREX_ERR_INVALID
