"""GPU: failure detection without a fault.  A bounded wait inside the GEMM is
made to run out (the second K half of a split tile waits for a tag that no
launch publishes, switched on by the krex_debug_stall_handover test hook);
the kernel must report it through the status word and its detail record,
return, and leave the context usable: the same GEMM right after is correct.
Runs in a child process so that the shortened wait bound (the tuning's
wait_timeout_ms) and the hook touch no other test."""
import json
import os
import subprocess
import sys

import pytest

from conftest import ROOT

pytestmark = pytest.mark.gpu

CHILD = r'''
import json, os, sys, time
import numpy as np
import torch
sys.path.insert(0, ROOT)
import paper_2609_30057_gb300 as krex
from oracle import gen, ref
krex.build()
M, N, K = 1024, 2048, 512            # one partial wave: K halves through the workspace
# K halves (at this K only when asked for) and a 300 ms bound on every wait
krex.krex_set_tuning(gemm_split_k=1, wait_timeout_ms=300)
a = torch.empty(M, K, dtype=torch.bfloat16, device="cuda")
b = torch.empty(K, N, dtype=torch.bfloat16, device="cuda")
krex.krex_gen_inputs(31, 0, 0, 0.0, a)
krex.krex_gen_inputs(31, 1, 0, 0.0, b)
c = torch.empty(M, N, dtype=torch.bfloat16, device="cuda")
ws = krex.gemm_workspace()
out = {}
krex.krex_debug_stall_handover(True)
t0 = time.monotonic()
krex.krex_run_candidate_ws(krex.KREX_OP_GEMM_BF16, [a, b], c, ws)
torch.cuda.synchronize()
out["stalled_s"] = time.monotonic() - t0
out["detail"] = krex.krex_device_status_detail()
try:
    out["status"] = krex.krex_device_status()
except krex.KrexError as e:
    out["status"] = int(str(e).split("status 0x")[1].rstrip(")"), 16)
krex.krex_debug_stall_handover(False)
ws.zero_()
krex.krex_run_candidate_ws(krex.KREX_OP_GEMM_BF16, [a, b], c, ws)
torch.cuda.synchronize()
out["status_after"] = krex.krex_device_status()
want = ref.gemm_f64(gen.uniform_bf16(31, 0, M, K), gen.uniform_bf16(31, 1, K, N))
got = gen.bf16_to_f32(c.view(torch.int16).cpu().numpy().view(np.uint16)).astype(np.float64)
out["correct_after"] = bool(np.all(np.abs(got - want) <= ref.gemm_tolerance(want, K)))
print("RESULT " + json.dumps(out))
'''


def test_bounded_wait_runs_out_and_the_context_stays_usable():
    r = subprocess.run([sys.executable, "-c", "ROOT = %r\n" % ROOT + CHILD], capture_output=True,
                       text=True, timeout=300)
    assert r.returncode == 0, r.stdout[-2000:] + r.stderr[-2000:]
    line = [l for l in r.stdout.splitlines() if l.startswith("RESULT ")][-1]
    out = json.loads(line[len("RESULT "):])
    assert out["status"] == 0x1052, out                    # the hand-over wait ran out
    assert out["detail"]["code"] == 0x1052 and out["detail"]["waited_ns"] >= 300_000_000
    assert out["detail"]["MNK"] == [1024, 2048, 512]
    assert 0.25 < out["stalled_s"] < 30.0                  # bounded: the kernel returned
    assert out["status_after"] == 0 and out["correct_after"]
