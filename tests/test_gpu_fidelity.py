"""GPU: the fidelity experiment in small.  Background tenants inflate the
measured candidate durations when ungated; with the in-region gate the
measurement matches the native one (the paper's Section 6.4 in one process)."""
import json

import pytest

from paper_2609_30057_gb300 import fidelity

pytestmark = pytest.mark.gpu


def test_gate_restores_native_timings():
    res = fidelity.run(tenants=2, iters=10, quick=True)
    assert res["device_status"] == {"native": 0, "ungated": 0, "gated": 0}, json.dumps(res["device_status_detail"])
    c = res["conditions"]
    assert c["ungated"]["background_launches"] > 0 and c["gated"]["background_launches"] > 0
    assert c["ungated"]["median_ratio"] > 1.2           # contention inflates every candidate
    assert 0.95 < c["gated"]["median_ratio"] < 1.05     # gated: as if alone
    assert c["gated"]["P_p95_inflation"] < 0.10
    assert c["gated"]["P_p95_inflation"] < c["ungated"]["P_p95_inflation"]
