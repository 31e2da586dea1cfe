"""Pins of the oracle's average-case TTFT estimators (Sec. 4, App. E).

The limited-processor-sharing wait is checked against the series it is derived
from, against a seeded simulation of the queue, against the Pollaczek-Khinchine
mean wait of M/G/1 (the G/G/k form at k = 1 with Poisson arrivals), and in its
limits; the throughput-based wait against the prefill tokens the serving
simulation itself consumes.
"""
import math
from collections import deque
from fractions import Fraction

import numpy as np
import pytest

import oracle
from paper_2607_18253_gb300 import workloads as W


@pytest.mark.parametrize("alpha,mu,k", [(0.5, 1.0, 1), (7.0, 10.0, 3), (24.0, 25.0, 25), (0.9, 1.0, 8)])
def test_lps_wait_equals_the_series(alpha, mu, k):
    # sum over the state n an arrival sees: (1 - rho) rho^n * (n - k + 1) / mu for n >= k
    rho = alpha / mu
    terms, n = [], k
    while True:
        term = (1.0 - rho) * rho ** n * (n - k + 1) / mu
        terms.append(term)
        if term < 1e-20 * max(terms) and n > k + 10:
            break
        n += 1
    assert oracle.lps_wait(alpha, mu, k) == pytest.approx(math.fsum(terms), rel=1e-11)


def _simulate_lps(alpha, mu, k, n_arrivals, seed):
    # continuous-time chain of the resident count: arrivals at alpha, completions at mu
    # whenever someone is active; FIFO entry into the k active slots
    rng = np.random.default_rng(seed)
    t, n, waits, fifo = 0.0, 0, [], deque()
    arrivals = 0
    while arrivals < n_arrivals:
        rate = alpha + (mu if n > 0 else 0.0)
        t += rng.exponential(1.0 / rate)
        if rng.random() < alpha / rate:
            arrivals += 1
            n += 1
            if n <= k:
                waits.append(0.0)
            else:
                fifo.append(t)
        else:
            n -= 1
            if fifo:
                waits.append(t - fifo.popleft())
    return float(np.mean(waits))


@pytest.mark.parametrize("k", [1, 3])
def test_lps_wait_matches_a_simulated_queue(k):
    alpha, mu = 0.7, 1.0
    sim = _simulate_lps(alpha, mu, k, 300_000, seed=11 + k)
    assert sim == pytest.approx(oracle.lps_wait(alpha, mu, k), rel=0.06)


@pytest.mark.parametrize("cs2", [0.0, 0.5, 1.0, 2.0])
def test_gg1_is_pollaczek_khinchine(cs2):
    # M/G/1 mean wait: alpha E[S^2] / (2 (1 - rho)) with E[S] = 1/mu, E[S^2] = (1 + cs2) / mu^2
    alpha, mu = 3.0, 5.0
    es2 = (1.0 + cs2) / mu ** 2
    pk = alpha * es2 / (2.0 * (1.0 - alpha / mu))
    assert oracle.lps_wait(alpha, mu, 1, 1.0, cs2) == pytest.approx(pk, rel=1e-14)


def test_lps_limits():
    assert oracle.lps_wait(0.8, 1.0, 400) < 1e-35            # processor sharing: no wait
    assert oracle.lps_wait(0.8, 1.0, 5, 0.0, 0.0) == 0.0        # no variability, no wait
    assert oracle.lps_wait(2.0, 3.0, 4, 1.0, 1.0) == oracle.lps_wait(2.0, 3.0, 4)
    assert oracle.lps_wait(0.0, 3.0, 2) == 0.0
    # the wait only grows with load and shrinks with parallelism
    w = [oracle.lps_wait(a, 1.0, 4) for a in (0.2, 0.5, 0.8, 0.95)]
    assert all(x < y for x, y in zip(w, w[1:]))
    assert all(oracle.lps_wait(0.9, 1.0, k + 1) < oracle.lps_wait(0.9, 1.0, k) for k in range(1, 12))
    for bad in ((1.0, 1.0, 2), (2.0, 1.0, 1), (0.5, 0.0, 1), (0.5, 1.0, 0), (-0.1, 1.0, 1)):
        assert math.isnan(oracle.lps_wait(*bad))


def test_pow_int_is_the_exact_power_to_rounding():
    cases = [(x, k) for x in (0.3, 0.97, 1.7) for k in (0, 1, 2, 3, 7, 25, 64, 300)]
    cases += [(1.0 - 1e-9, 1 << 17), (0.9999, 5000)]
    for x, k in cases:
        exact = Fraction(x) ** k
        got = oracle.pow_int(x, k)
        assert abs(Fraction(got) - exact) <= exact * Fraction(1, 10 ** 12), (x, k)
    assert oracle.pow_int(0.5, 10) == 2.0 ** -10


def test_throughput_wait_counts_the_prefill_the_simulation_serves():
    # the residents' prefill tokens equal what the SFS run serves before q's own prompt
    for seed in range(30):
        wl = W.small_workload(seed, num_instances=5, num_queries=3)
        theta = 1000.0 + 37.0 * seed
        tw = oracle.throughput_wait(wl, theta)
        for j in range(wl.num_instances):
            run = [(int(wl.run_ctx[j, r]), int(wl.run_pre[j, r]), int(wl.run_dec[j, r])) for r in range(wl.n_run[j])]
            wait = [(int(wl.wait_pre[j, w]), int(wl.wait_dec[j, w])) for w in range(wl.n_wait[j])]
            p = int(wl.prompt_len[0])
            F, _, _ = oracle.simulate(run, wait, int(wl.max_batched_tokens[j]), int(wl.max_seqs[j]), p, 1)
            assert tw[j] * theta == pytest.approx(float(F[1] - p), rel=1e-15)


def test_avgcase_matrix_rounding():
    wl = W.make_workload("pool64", num_queries=300)
    rng = np.random.default_rng(5)
    I = wl.num_instances
    Wj = rng.uniform(0.0, 2.0, I)
    theta = rng.uniform(2e3, 3e4, I)
    tdec = rng.uniform(0.005, 0.05, I)
    t32, t64 = oracle.avgcase_matrix(wl, Wj, theta, tdec)
    rel = np.abs(t32.astype(np.float64) - t64) / t64
    assert rel.max() < 3e-7
    np.testing.assert_allclose(t64, Wj[None, :] + wl.prompt_len[:, None] / theta[None, :] + tdec[None, :], rtol=1e-15)
    # powers of two: every step is exact
    wl1 = W.make_workload("tiny")
    wl1.prompt_len[:] = 100
    t32, t64 = oracle.avgcase_matrix(wl1, 0.25, 1024.0, 1.0 / 64)
    assert np.all(t32 == np.float32(0.25 + 100 / 1024 + 1 / 64)) and np.all(t64 == 0.25 + 100 / 1024 + 1 / 64)
    with pytest.raises(ValueError):
        oracle.avgcase_matrix(wl1, 0.25, 0.0, 0.01)
