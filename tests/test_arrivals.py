"""Arrival generators of the online stream: Poisson (Sec. 5) and MMPP-2 (the
appendix on correlated arrivals), checked against the paper's rate table and
the processes' long-run statistics."""
import json
import os

import numpy as np
import pytest

from paper_2607_18253_gb300 import workloads as W

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "mmpp2_rates.json")


def test_mmpp2_rates_reproduce_the_printed_table():
    g = json.load(open(GOLDEN))
    assert g["z_lh"] / (g["z_lh"] + g["z_hl"]) == pytest.approx(g["p_high"])
    for mean, r, low, high in g["rows"]:
        lo, hi = W.mmpp2_rates(mean, r, g["p_high"])
        assert round(lo, 2) == pytest.approx(low) and round(hi, 2) == pytest.approx(high)
        assert (1 - g["p_high"]) * lo + g["p_high"] * hi == pytest.approx(mean)


@pytest.mark.parametrize("ratio", [3.0, 6.0])
def test_mmpp2_long_run_rate_and_burstiness(ratio):
    mean = 7.0
    a = W.mmpp2_arrivals(400_000, mean, ratio, seed=1)
    assert np.all(np.diff(a) >= 0) and a.shape == (400_000,)
    assert a.shape[0] / a[-1] == pytest.approx(mean, rel=0.04)
    # counts in 1 s windows: over-dispersed (index of dispersion well above 1), and
    # the busiest windows near the high-state rate
    counts = np.bincount(a.astype(np.int64))[:-1]
    assert counts.var() / counts.mean() > 1.5
    lo, hi = W.mmpp2_rates(mean, ratio)
    assert np.quantile(counts, 0.99) > 0.8 * hi


def test_poisson_arrivals_are_poisson():
    a = W.poisson_arrivals(400_000, 131.0, seed=3)
    gaps = np.diff(a)
    assert gaps.mean() == pytest.approx(1 / 131.0, rel=0.01)
    assert gaps.std() / gaps.mean() == pytest.approx(1.0, rel=0.02)   # exponential gaps
    counts = np.bincount(a.astype(np.int64))[:-1]
    assert counts.var() / counts.mean() == pytest.approx(1.0, rel=0.1)


def test_arrivals_are_seeded():
    np.testing.assert_array_equal(W.mmpp2_arrivals(1000, 6.0, 3.0, 5), W.mmpp2_arrivals(1000, 6.0, 3.0, 5))
    assert not np.array_equal(W.mmpp2_arrivals(1000, 6.0, 3.0, 5), W.mmpp2_arrivals(1000, 6.0, 3.0, 6))
