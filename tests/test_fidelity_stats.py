"""The fidelity experiment's statistics (product code) against the oracle's
definitions: Eq. 1 (P = p95(r) - 1), percentiles, Kendall's tau_b and the
pairwise-gap grouping of Section 6.4 (CPU only)."""
import math

import numpy as np

from conftest import read_golden
from oracle import ref
from paper_2609_30057_gb300 import fidelity


def test_percentile_and_inflation_match_oracle():
    rng = np.random.default_rng(9)
    for n in (1, 2, 7, 40):
        nat = rng.uniform(0.01, 10, n).tolist()
        meas = [t * rng.uniform(0.9, 1.6) for t in nat]
        for q in (0.0, 0.5, 0.95, 1.0):
            assert fidelity.percentile(meas, q) == ref.percentile_linear(meas, q)
        assert fidelity.inflation_p95(meas, nat) == ref.timing_inflation_p95(meas, nat)


def test_kendall_matches_oracle():
    rng = np.random.default_rng(10)
    x = rng.integers(0, 5, 25).tolist()
    y = (np.array(x) + rng.integers(-1, 2, 25)).tolist()
    assert fidelity.kendall_tau_b(x, y) == ref.kendall_tau_b(x, y)


def test_flip_groups_follow_the_paper_gap_definition():
    # the paper's worked example (1.0 vs 1.1 ms) is a 10% gap: the top group
    a, b, gap = (float(v) for v in read_golden("pairwise_gap.txt")[0].split())
    assert math.isclose(ref.pairwise_gap(a, b), gap)
    f = fidelity.flip_rates([1.2, 1.0], [a, b])          # order reversed
    assert f["0.10-inf"] == {"pairs": 1, "flip_rate": 1.0}
    f = fidelity.flip_rates([1.0, 1.01], [1.0, 1.01])     # 1% gap, kept
    assert f["0.00-0.02"] == {"pairs": 1, "flip_rate": 0.0}


def test_summary_of_identical_runs():
    nat = [0.1, 0.2, 0.3]
    s = fidelity.summarize(nat, nat)
    assert s["P_p95_inflation"] == 0.0 and s["median_ratio"] == 1.0 and s["within_5pct"] == 1.0
    assert s["kendall_tau_b"] == 1.0
