"""Pins of the CPU oracle against what the paper and plain arithmetic fix.

Each test pins a different part of the oracle so that a dropped term, a wrong
sign, a swapped operand or a wrong index in it fails at least one of them:
hand-traced batch sequences (Sec. 4.1, Eq. 7-9), closed forms for the empty
and the decode-only instance, the telescoping prefill-attention identity,
token conservation, monotonicity, and the routing rules of Eq. 2, 3 and 5 in
cases with an exact answer.
"""
import json
import math
import os

import numpy as np
import pytest

import oracle
from paper_2607_18253_gb300 import workloads as W

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "hand_traces.json")


def _traces():
    with open(GOLDEN) as f:
        return json.load(f)["traces"]


@pytest.mark.parametrize("trace", _traces(), ids=lambda t: t["name"].split()[0])
@pytest.mark.parametrize("mode", [0, 1])
def test_hand_traces(trace, mode):
    F, la, lt = oracle.simulate(trace["running"], trace["waiting"], trace["B"], trace["S"], trace["p"],
                                trace["d"], mode)
    exp = trace[f"mode{mode}"]
    assert F.tolist() == exp["F"]
    assert la == exp["admit"]
    assert lt == exp["ttft"]
    assert F[0] == lt


@pytest.mark.parametrize("B", [1, 7, 64, 2048, 8192])
@pytest.mark.parametrize("p", [1, 2, 63, 64, 65, 5000, 32768])
def test_empty_instance_closed_form(B, p):
    # An idle instance: ceil(p/B) prefill batches, then (mode 0) one decode batch at context p.
    n = -(-p // B)
    F0, _, _ = oracle.simulate([], [], B, 1, p, 3, 0)
    assert F0.tolist() == [n + 1, p, 1, p, p * (p + 1) // 2]
    F1, _, _ = oracle.simulate([], [], B, 1, p, 3, 1)
    assert F1.tolist() == [n, p, 0, 0, p * (p + 1) // 2]


def test_decode_only_closed_form():
    # n < S decoders with total context C and long decodes leave r = B - n tokens per batch.
    rng = np.random.default_rng(11)
    for _ in range(300):
        B = int(rng.integers(2, 300))
        n = int(rng.integers(0, min(B, 40)))
        S = int(rng.integers(n + 1, B + 1))
        p = int(rng.integers(1, 2000))
        ctx = rng.integers(0, 5000, n)
        L = -(-p // (B - n)) + 1
        running = [(int(c), 0, L + 5) for c in ctx]
        F, la, lt = oracle.simulate(running, [], B, S, p, 1, 0)
        C = int(ctx.sum())
        assert F.tolist() == [L, p, n * L + 1, L * C + n * L * (L - 1) // 2 + p, p * (p + 1) // 2]
        assert la == 1 and lt == L


def test_prefill_attention_telescopes():
    # Any chunking of a p-token prompt from context c sums x*c_k + x(x+1)/2 to p*c + p(p+1)/2.
    rng = np.random.default_rng(5)
    for _ in range(200):
        c0 = int(rng.integers(0, 1000))
        p = int(rng.integers(1, 3000))
        B = int(rng.integers(1, 500))
        # the query is alone: its F4 is exactly its own prompt's term
        F, _, _ = oracle.simulate([], [], B, 4, p, 1, 0)
        assert F[4] == p * (p + 1) // 2
        # a running request mid-prefill at context c0 ahead of the query
        pre = int(rng.integers(1, 3000))
        F, _, _ = oracle.simulate([(c0, pre, 1)], [], B, 4, p, 1, 0)
        assert F[4] == pre * c0 + pre * (pre + 1) // 2 + p * (p + 1) // 2


def _rand_state(rng, tail_prefill=True, general=False):
    B = int(rng.integers(2, 80))
    S = int(rng.integers(1, B + 1))
    nr = int(rng.integers(0, S + 1))
    running = []
    for r in range(nr):
        pre = 0
        if general and rng.random() < 0.3:
            pre = int(rng.integers(1, 150))
        running.append((int(rng.integers(0, 400)), pre, int(rng.integers(1, 50))))
    if tail_prefill and nr and rng.random() < 0.5:
        c, _, d = running[-1]
        running[-1] = (c, int(rng.integers(1, 150)), d)
    waiting = [(int(rng.integers(1, 150)), int(rng.integers(1, 50))) for _ in range(int(rng.integers(0, 10)))]
    return B, S, running, waiting


@pytest.mark.parametrize("mode", [0, 1])
def test_all_residents_finish_prefill_before_the_query(mode):
    # FCFS with the query last: every resident's prefill is complete by the query's
    # first token, so F1 and F4 equal the residents' totals plus the query's own.
    rng = np.random.default_rng(7 + mode)
    for _ in range(400):
        B, S, running, waiting = _rand_state(rng, general=True)
        p = int(rng.integers(1, 300))
        F, la, lt = oracle.simulate(running, waiting, B, S, p, 4, mode)
        pre_tot = sum(pre for _, pre, _ in running) + sum(w for w, _ in waiting) + p
        att = sum(pre * c + pre * (pre + 1) // 2 for c, pre, _ in running) + \
            sum(w * (w + 1) // 2 for w, _ in waiting) + p * (p + 1) // 2
        assert F[1] == pre_tot
        assert F[4] == att
        assert F[0] == lt >= la >= 1


@pytest.mark.parametrize("mode", [0, 1])
def test_ttft_monotone_in_prompt_and_queue(mode):
    rng = np.random.default_rng(23 + mode)
    coef = np.array([3e-3, 1e-4, 2e-4, 1e-7, 1e-8], np.float32)
    for _ in range(150):
        B, S, running, waiting = _rand_state(rng)
        p = int(rng.integers(1, 200))
        base, _, _ = oracle.simulate(running, waiting, B, S, p, 4, mode)
        longer, _, _ = oracle.simulate(running, waiting, B, S, p + int(rng.integers(1, 100)), 4, mode)
        assert oracle.ttft_f64(coef, longer) >= oracle.ttft_f64(coef, base)
        assert longer[0] >= base[0]
        # one more waiting request ahead of the query: every feature can only grow
        more, _, _ = oracle.simulate(running, waiting + [(int(rng.integers(1, 150)), 3)], B, S, p, 4, mode)
        assert np.all(more >= base)
        # a longer waiting prompt ahead of the query
        if waiting:
            k = int(rng.integers(0, len(waiting)))
            grown = list(waiting)
            grown[k] = (grown[k][0] + int(rng.integers(1, 100)), grown[k][1])
            g, _, _ = oracle.simulate(running, grown, B, S, p, 4, mode)
            assert oracle.ttft_f64(coef, g) >= oracle.ttft_f64(coef, base)


def test_query_decode_length_does_not_change_ttft():
    # TTFT stops at the query's first output token; its own decode length never enters.
    rng = np.random.default_rng(3)
    for _ in range(100):
        B, S, running, waiting = _rand_state(rng)
        p = int(rng.integers(1, 200))
        for mode in (0, 1):
            a, _, _ = oracle.simulate(running, waiting, B, S, p, 1, mode)
            b, _, _ = oracle.simulate(running, waiting, B, S, p, 977, mode)
            assert a.tolist() == b.tolist()


def test_ttft_weights_each_feature_once():
    # Coefficients and features chosen so every product and sum is exact in fp32.
    coef = np.array([1.0, 10.0, 100.0, 1000.0, 10000.0], np.float32)
    F = np.array([1, 2, 3, 4, 5], np.int64)
    assert float(oracle.ttft_f32(coef, F)) == 54321.0
    assert oracle.ttft_f64(coef, F) == 54321.0
    # each coefficient alone picks out its own feature
    for k in range(5):
        c = np.zeros(5, np.float32)
        c[k] = 1.0
        assert float(oracle.ttft_f32(c, F)) == float(F[k])


def test_ttft_fp32_within_rounding_of_fp64():
    rng = np.random.default_rng(9)
    for _ in range(2000):
        coef = rng.uniform(1e-9, 1e-2, 5).astype(np.float32)
        F = rng.integers(0, 1 << 40, 5).astype(np.int64)
        t32 = float(oracle.ttft_f32(coef, F))
        t64 = oracle.ttft_f64(coef, F)
        # 5 conversions + 1 product + 4 fmas, all terms positive: well under 1e-6 relative
        assert abs(t32 - t64) <= 1e-6 * t64


def test_utility_exact_case():
    # cost = 1024 * 2^-20 + 256 * 2^-18 = 2^-9; U = 0.5 - 2 * 2^-9 (all exact in fp32)
    u = oracle.utility(0.5, 2.0, 1024, 256, 2.0 ** -20, 2.0 ** -18)
    assert float(u) == 0.5 - 2.0 * 2.0 ** -9
    # the prompt is priced with price_in, the response with price_out
    u2 = oracle.utility(0.5, 1.0, 2, 1, 0.125, 0.0)
    assert float(u2) == 0.25
    u3 = oracle.utility(0.5, 1.0, 1, 2, 0.0, 0.125)
    assert float(u3) == 0.25


def _tiny_route_case(seed=0, Q=40, I=7, M=3):
    wl = W.small_workload(seed, num_instances=I, num_models=M, num_queries=Q)
    rng = np.random.default_rng(seed)
    ttft = rng.uniform(0.05, 2.0, (Q, I)).astype(np.float32)
    return wl, ttft


def test_route_latency_agnostic_picks_best_accuracy_model():
    # lambda = mu = 0: J = acc, so the lowest-index instance of the most accurate model wins (Eq. 5, delta = 0).
    wl, ttft = _tiny_route_case()
    assign, util, tch = oracle.route(wl, ttft, lam=[0.0], mu=[0.0])
    for i in range(wl.num_queries):
        best_m = int(np.argmax(wl.acc[i]))
        inst = np.flatnonzero(wl.model_of_instance == best_m)
        if inst.size == 0:
            continue
        assert assign[0, i] == inst.min()
        assert util[0, i] == wl.acc[i, best_m]
        assert tch[0, i] == ttft[i, assign[0, i]]


def test_route_pure_latency_picks_fastest():
    # equal accuracy, no price: J = -mu * TTFT, so the argmin TTFT wins, ties to the lowest index.
    wl, ttft = _tiny_route_case(1)
    wl.acc[:] = 0.5
    ttft[:, 3] = ttft[:, 5] = ttft.min(axis=1) * 0.5   # a tie between instances 3 and 5
    assign, _, _ = oracle.route(wl, ttft, lam=[0.0], mu=[1.0])
    assert np.all(assign[0] == 3)


def test_route_constrained_limits():
    wl, ttft = _tiny_route_case(2)
    inf = np.full(wl.num_queries, np.inf, np.float32)
    a_inf, u_inf, _ = oracle.route(wl, ttft, lam=[0.7], tau=inf)
    a_lag, u_lag, _ = oracle.route(wl, ttft, lam=[0.7], mu=[0.0])
    assert np.array_equal(a_inf, a_lag) and np.array_equal(u_inf, u_lag)
    # nothing feasible: the least estimated latency (Eq. 3, empty feasible set)
    neg = np.full(wl.num_queries, -1.0, np.float32)
    a_neg, _, t_neg = oracle.route(wl, ttft, lam=[0.7], tau=neg)
    assert np.array_equal(a_neg[0], np.argmin(ttft, axis=1))
    assert np.array_equal(t_neg[0], ttft.min(axis=1))
    # exactly one feasible instance per query
    only = np.random.default_rng(0).integers(0, wl.num_instances, wl.num_queries)
    t2 = ttft + 10.0
    t2[np.arange(wl.num_queries), only] = 0.01
    a_one, _, _ = oracle.route(wl, t2, lam=[0.7], tau=np.full(wl.num_queries, 0.02, np.float32))
    assert np.array_equal(a_one[0], only)


def test_frontier_means():
    wl, ttft = _tiny_route_case(3, Q=4)
    assign = np.array([[0, 1, 2, 3]], np.int32)
    tch = np.array([[0.5, 1.0, 1.5, 2.0]], np.float32)
    out = oracle.frontier(wl, assign, tch)
    accs, costs = [], []
    for i, j in enumerate(assign[0]):
        m = wl.model_of_instance[j]
        accs.append(float(wl.acc[i, m]))
        costs.append(int(wl.prompt_len[i]) * float(wl.price_in[m]) + int(wl.dec_hat[i, m]) * float(wl.price_out[m]))
    assert out[0, 0] == pytest.approx(sum(accs) / 4, rel=1e-12)
    assert out[0, 1] == pytest.approx(sum(costs) / 4, rel=1e-6)
    assert out[0, 2] == pytest.approx(1.25, rel=1e-12)


def test_ttft_target_generator_mean():
    # App. B.2: E[tau] is about 158 + 3.5e-3 p ms where the clip is inactive.
    rng = np.random.default_rng(0)
    for p in (500, 10000, 100000):
        t = W.ttft_targets(rng, np.full(200000, p, np.int32)).astype(np.float64) * 1e3
        expect = min(1120.0, max(150.0, 158.0 + 3.5e-3 * p))
        assert abs(t.mean() - expect) < 0.01 * expect
        assert t.min() >= 150.0 - 1e-3 and t.max() <= 1120.0 + 1e-3


def test_coefficient_row_follows_the_instance_model():
    # Each instance's estimate uses its own model's Eq. 9 coefficients.  Two idle
    # instances, instance 0 serving
    # model 1 and instance 1 serving model 0; power-of-two coefficients make every
    # product and partial sum exact in fp32, so the expected times are exact rationals.
    import dataclasses
    from fractions import Fraction as Fr
    base = W.small_workload(0, num_instances=2, num_models=2, num_queries=3)
    z = np.zeros(2, np.int32)
    coef = np.array([[2.0 ** -8, 2.0 ** -12, 2.0 ** -10, 2.0 ** -16, 2.0 ** -20],
                     [2.0 ** -6, 2.0 ** -11, 2.0 ** -9, 2.0 ** -15, 2.0 ** -19]], np.float32)
    wl = dataclasses.replace(base, model_of_instance=np.array([1, 0], np.int32), coef=coef,
                             max_batched_tokens=np.array([2048, 2048], np.int32), max_seqs=np.array([8, 8], np.int32),
                             n_run=z, n_wait=z.copy(), prompt_len=np.array([100, 3000, 1], np.int32),
                             dec_hat=np.array([[5, 7], [1, 2], [3, 4]], np.int32), first_token_mode=0)
    F, lt, t32, t64 = oracle.estimate_matrix(wl)
    for i, p in enumerate((100, 3000, 1)):
        # idle instance, paper mode: ceil(p/B) prefill batches then one decode batch at context p
        Fx = [-(-p // 2048) + 1, p, 1, p, p * (p + 1) // 2]
        for j in range(2):
            assert F[i, j].tolist() == Fx
            m = 1 - j
            exact = sum(Fr(float(coef[m, k])) * Fx[k] for k in range(5))
            assert Fr(float(t32[i, j])) == exact, (i, j)
            assert Fr(t64[i, j]) == exact, (i, j)
    # the two instances differ (a shared or swapped row would make them equal or exchange them)
    assert t32[0, 0] == np.float32(2.0 ** -6 * 2 + 100 * 2.0 ** -11 + 2.0 ** -9 + 100 * 2.0 ** -15 + 5050 * 2.0 ** -19)
    assert t32[0, 1] == np.float32(2.0 ** -8 * 2 + 100 * 2.0 ** -12 + 2.0 ** -10 + 100 * 2.0 ** -16 + 5050 * 2.0 ** -20)


def test_candidate_slices_on_several_threads_change_nothing():
    # the candidate loop split over host threads gives the single-thread result bit for bit
    wl = W.make_workload("pool64", num_queries=70)
    Q, I = wl.num_queries, wl.num_instances
    qq, jj = np.meshgrid(np.arange(Q), np.arange(I), indexing="ij")
    one = oracle.estimate_candidates(wl, qq.ravel(), jj.ravel(), threads=1)
    many = oracle.estimate_candidates(wl, qq.ravel(), jj.ravel(), threads=5)
    for a, b in zip(one, many):
        np.testing.assert_array_equal(a.view(np.uint8), b.view(np.uint8))
    lim = W.kv_limits(wl, 3)
    one = oracle.estimate_matrix_kv(wl, *lim, threads=1)
    many = oracle.estimate_matrix_kv(wl, *lim, threads=3)
    for a, b in zip(one, many):
        np.testing.assert_array_equal(np.ascontiguousarray(a).view(np.uint8), np.ascontiguousarray(b).view(np.uint8))
