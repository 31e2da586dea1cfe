"""Pins of the oracle's baseline policies and stream metrics (Sec. 6 baselines, Eq. 4).

Each function is checked against something other than itself: a hand-worked case,
an independent definition (Shortest Queue as the k-th smallest (level, index) slot),
the special case that reduces to another policy, or another oracle path.
"""
import numpy as np
import pytest

import oracle
from paper_2607_18253_gb300 import workloads as W


def test_round_robin_hand_case_and_balance():
    # start 4 on 3 instances: 4 mod 3 = 1, then 2, 0, 1, 2
    np.testing.assert_array_equal(oracle.round_robin(5, 3, 4), [1, 2, 0, 1, 2])
    a = oracle.round_robin(1000, 7, 123)
    counts = np.bincount(a, minlength=7)
    assert counts.max() - counts.min() <= 1


def test_shortest_queue_hand_case():
    # resident (2, 0, 1): the empty instance 1 takes two queries (levels 0 and 1,
    # instance 1 wins the tie at level 1), then instance 2 and instance 0 at level 2
    np.testing.assert_array_equal(oracle.shortest_queue([2, 0, 1], 4), [1, 1, 2, 0])


def test_shortest_queue_equal_queues_is_round_robin():
    for I in (1, 3, 8):
        np.testing.assert_array_equal(oracle.shortest_queue(np.full(I, 5), 29), oracle.round_robin(29, I, 0))


@pytest.mark.parametrize("seed", range(6))
def test_shortest_queue_is_the_kth_smallest_slot(seed):
    # Query k takes the k-th smallest slot (level, instance) over the slots that
    # instance j offers at levels c_j, c_j + 1, ... -- a definition without a loop
    # over queries
    rng = np.random.default_rng(seed)
    I = int(rng.integers(1, 12))
    c = rng.integers(0, 9, I)
    Q = int(rng.integers(1, 60))
    slots = sorted((lvl, j) for j in range(I) for lvl in range(int(c[j]), int(c.max()) + Q + 1))
    expect = [j for _, j in slots[:Q]]
    np.testing.assert_array_equal(oracle.shortest_queue(c, Q), expect)


def test_latency_agnostic_is_lagrangian_with_zero_delta():
    wl = W.small_workload(3, num_instances=9, num_models=3, num_queries=40)
    _, _, t32, _ = oracle.estimate_matrix(wl)
    lam = float(wl.lam[0])
    a, u, t = oracle.baseline_route(wl, oracle.POLICY_LATENCY_AGNOSTIC, lam, ttft32=t32)
    ra, ru, rt = oracle.route(wl, t32, lam=np.array([lam], np.float32), mu=np.zeros(1, np.float32))
    np.testing.assert_array_equal(a, ra[0])
    np.testing.assert_array_equal(u.view(np.uint32), ru[0].view(np.uint32))
    np.testing.assert_array_equal(t.view(np.uint32), rt[0].view(np.uint32))


def test_baseline_ttft_is_the_chosen_candidates_estimate():
    wl = W.small_workload(4, num_instances=6, num_models=2, num_queries=25)
    _, _, t32, _ = oracle.estimate_matrix(wl)
    for pol in (oracle.POLICY_ROUND_ROBIN, oracle.POLICY_SHORTEST_QUEUE):
        a, u, t = oracle.baseline_route(wl, pol, 0.5, rr_start=3)
        np.testing.assert_array_equal(t.view(np.uint32), t32[np.arange(25), a].view(np.uint32))


def test_on_time_utility_hand_case():
    # on time: queries 0 (1 <= 2) and 2 (0.5 <= 1); query 1 is late (3 > 2)
    otu, slo = oracle.on_time_utility([0.5, 0.8, -0.1], [1.0, 3.0, 0.5], [2.0, 2.0, 1.0])
    assert otu == pytest.approx((0.5 + float(np.float32(-0.1))) / 3, rel=1e-15)  # fp64 sum of fp32 values
    assert slo == pytest.approx(2 / 3, rel=1e-15)


def test_on_time_utility_delay_nan_and_boundary():
    util = np.array([1.0, 1.0, 1.0, 1.0], np.float32)
    ttft = np.array([1.0, np.nan, 2.0, 0.25], np.float32)
    tau = np.array([1.0, 5.0, 2.0, 0.5], np.float32)
    # no delay: 1 <= 1 on time (boundary), NaN late, 2 <= 2 on time, 0.25 on time
    assert oracle.on_time_utility(util, ttft, tau) == (0.75, 0.75)
    # a delay of 0.5 s makes queries 0 and 2 late; 0.25 + 0.25 = 0.5 <= 0.5 stays on time
    delay = np.array([0.5, 0.0, 0.5, 0.25], np.float32)
    assert oracle.on_time_utility(util, ttft, tau, delay) == (0.25, 0.25)
