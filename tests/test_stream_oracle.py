"""Pins of the oracle's online stream step (append + advance to t_now).

The advance executes the same scheduler step as the estimator and times each
batch with Eq. 9 for its own composition, so it must agree with the SFS
estimate of Eq. 8: a query routed to an instance emits its first token exactly
when the summed batch times reach its estimate.
"""
import numpy as np
import pytest

import oracle
from paper_2607_18253_gb300 import workloads as W


def _one_instance(running, waiting, B, S, coef, cap=64):
    wl = W.small_workload(0, num_instances=1, num_models=1, num_queries=1, cap_running=cap, cap_waiting=cap)
    wl.max_batched_tokens[:] = B
    wl.max_seqs[:] = S
    wl.coef[:] = coef
    wl.model_of_instance[:] = 0
    for a in (wl.run_ctx, wl.run_pre, wl.run_dec, wl.wait_pre, wl.wait_dec):
        a[:] = 0
    wl.n_run[:] = len(running)
    wl.n_wait[:] = len(waiting)
    for r, (c, p, d) in enumerate(running):
        wl.run_ctx[0, r], wl.run_pre[0, r], wl.run_dec[0, r] = c, p, d
    for w, (p, d) in enumerate(waiting):
        wl.wait_pre[0, w], wl.wait_dec[0, w] = p, d
    return wl


# powers of two: every product and sum below is exact in fp32 and fp64
COEF = np.array([0.25, 2.0 ** -4, 2.0 ** -3, 2.0 ** -10, 2.0 ** -12], np.float32)
NONE = np.zeros(0, np.int32)


def test_idle_instance_jumps_to_now():
    wl = _one_instance([], [], 16, 4, COEF)
    w2, clk = oracle.advance(wl, [3.0], NONE, NONE, NONE, 7.5)
    assert clk[0] == 7.5 and w2.n_run[0] == 0 and w2.n_wait[0] == 0
    w3, clk3 = oracle.advance(wl, [9.0], NONE, NONE, NONE, 7.5)
    assert clk3[0] == 9.0  # a clock never runs backwards


def test_hand_trace_batch_times():
    # B = 4, S = 2; running A (ctx 10, dec 2); waiting W1 (prompt 5, dec 1) -- trace T1 of the estimator
    # batch 1: A decodes at ctx 10, W1 chunk 3:   F = (1, 3, 1, 10, 6)
    # batch 2: A decodes at ctx 11, W1 chunk 2:   F = (1, 2, 1, 11, 9)  -> A finishes
    # batch 3: W1 decodes at ctx 5:               F = (1, 0, 1, 5, 0)   -> W1 finishes
    wl = _one_instance([(10, 0, 2)], [(5, 1)], 4, 2, COEF)
    c0, c1, c2, c3, c4 = (float(x) for x in COEF)
    T = [c0 + c2 + c1 * 3 + c3 * 10 + c4 * 6, c0 + c2 + c1 * 2 + c3 * 11 + c4 * 9, c0 + c2 + c3 * 5]
    w2, clk = oracle.advance(wl, [0.0], NONE, NONE, NONE, T[0] + T[1] + 0.5 * T[2])
    assert clk[0] == T[0] + T[1]
    assert w2.n_run[0] == 1 and w2.n_wait[0] == 0
    assert (w2.run_ctx[0, 0], w2.run_pre[0, 0], w2.run_dec[0, 0]) == (5, 0, 1)
    w3, clk3 = oracle.advance(wl, [0.0], NONE, NONE, NONE, 100.0)
    assert clk3[0] == 100.0 and w3.n_run[0] == 0


@pytest.mark.parametrize("mode", [0, 1])
def test_first_token_when_the_estimate_says(mode):
    # Route one query and advance: its first output token appears exactly after the
    # batches whose times sum to the SFS estimate of Eq. 8 (fp32 feature sum vs fp64
    # sum of per-batch times differ only by rounding, far below the 1e-4 margins).
    for trial in range(40):
        wl = W.small_workload(100 + trial, num_instances=1, num_models=1, num_queries=1, cap_running=64,
                              cap_waiting=64, first_token_mode=mode, budget_range=(8, 40), wait_max=40)
        p, d = int(wl.prompt_len[0]), 7
        F, la, lt = oracle.simulate(
            [(int(wl.run_ctx[0, r]), int(wl.run_pre[0, r]), int(wl.run_dec[0, r])) for r in range(wl.n_run[0])],
            [(int(wl.wait_pre[0, w]), int(wl.wait_dec[0, w])) for w in range(wl.n_wait[0])],
            int(wl.max_batched_tokens[0]), int(wl.max_seqs[0]), p, d, mode)
        t64 = oracle.ttft_f64(wl.coef[0], F)
        for frac, emitted in ((1 - 1e-4, False), (1 + 1e-4, True)):
            w2, clk = oracle.advance(wl, [0.0], np.zeros(1, np.int32), np.array([p], np.int32),
                                     np.array([d], np.int32), t64 * frac)
            nw = int(w2.n_wait[0])
            if nw and int(w2.wait_pre[0, nw - 1]) == p and int(w2.wait_dec[0, nw - 1]) == d:
                dec_left = d  # still waiting
            else:
                nr = int(w2.n_run[0])
                dec_left = int(w2.run_dec[0, nr - 1]) if nr else 0  # the query is the last admitted
            assert (dec_left < d) == emitted, (trial, frac, dec_left)


def test_advance_conserves_requests():
    rng = np.random.default_rng(1)
    wl = W.make_workload("pool64", num_queries=300, cap_running=64, cap_waiting=256)
    clk = np.zeros(wl.num_instances)
    a = rng.integers(-1, wl.num_instances, 300).astype(np.int32)
    w2, c2 = oracle.advance(wl, clk, a, wl.prompt_len, wl.dec_hat[:, 0], 0.05)
    before = wl.n_run + wl.n_wait + np.bincount(a[a >= 0], minlength=wl.num_instances)
    after = w2.n_run + w2.n_wait
    assert np.all(after <= before)
    assert np.all(c2 <= 0.05) and np.all(c2 >= 0)
    # a later time never leaves more work than an earlier one
    w3, c3 = oracle.advance(w2, c2, NONE, NONE, NONE, 0.5)
    assert np.all(w3.n_run + w3.n_wait <= after)
    assert np.all(c3 >= c2)


# ---------------------------------------------------------------------------
# The realized first output token (Sec. 4.1; Eq. 4 scores the realized TTFT)

HAND = np.array([1.0, 2.0 ** -2, 2.0 ** -3, 2.0 ** -5, 2.0 ** -6], np.float32)


@pytest.mark.parametrize("mode", [0, 1])
def test_first_token_time_hand_trace(mode):
    # an idle instance (B = 4, S = 2) gets one tracked query (prompt 6, 3 output tokens) at t = 0:
    # batch 1: prefill 4 at ctx 0:  T = 1 + 4/4 + (0 + 10)/64          = 2.15625
    # batch 2: prefill 2 at ctx 4:  T = 1 + 2/4 + (2*4 + 3)/64         = 1.671875
    # batch 3: decode at ctx 6:     T = 1 + 1/8 + 6/32                 = 1.3125
    # first token: end of batch 3 (its own decode batch), or of batch 2 (with the last chunk)
    wl = _one_instance([], [], 4, 2, HAND).with_mode(mode)
    tr = oracle.new_track(wl, 3)
    a = np.array([0], np.int32)
    w2, clk, tr2 = oracle.advance(wl, [0.0], a, np.array([6], np.int32), np.array([3], np.int32), 100.0,
                                  track=tr, id_base=1)
    exp = 2.15625 + 1.671875 + (1.3125 if mode == 0 else 0.0)
    assert tr2["first_token_time"][1] == exp
    assert np.isnan(tr2["first_token_time"][0]) and np.isnan(tr2["first_token_time"][2])
    # the same total is the SFS estimate of that query on the idle instance (Eq. 8)
    q = w2.with_queries(np.array([0]))
    q = q.__class__(**{**q.__dict__, "prompt_len": np.array([6], np.int32)})
    F, _, _ = oracle.simulate([], [], 4, 2, 6, 3, mode)
    assert oracle.ttft_f64(HAND, F) == exp
    # a batch that would end after t_now is not executed: the time is not recorded yet
    _, _, tr3 = oracle.advance(wl, [0.0], a, np.array([6], np.int32), np.array([3], np.int32), exp - 0.25,
                               track=tr, id_base=1)
    assert np.isnan(tr3["first_token_time"][1])
    assert tr3["wait_id"][0, 0] == 1 or tr3["run_id"][0, 0] == 1  # still tracked


def test_untracked_requests_and_plain_advance_agree():
    # tracking changes no state or clock; residents of a loaded snapshot stay untracked
    wl = W.small_workload(3, num_instances=6, num_models=2, num_queries=40, cap_running=64, cap_waiting=160,
                          wait_max=24, budget_range=(8, 64), min_gap=8)
    rng = np.random.default_rng(5)
    a = rng.integers(-1, 6, 40).astype(np.int32)
    p = rng.integers(1, 120, 40).astype(np.int32)
    d = rng.integers(1, 20, 40).astype(np.int32)
    w1, c1 = oracle.advance(wl, np.zeros(6), a, p, d, 30.0)
    w2, c2, tr = oracle.advance(wl, np.zeros(6), a, p, d, 30.0, track=oracle.new_track(wl, 40), id_base=0)
    for k in ("n_run", "run_ctx", "run_pre", "run_dec", "n_wait", "wait_pre", "wait_dec"):
        np.testing.assert_array_equal(getattr(w1, k), getattr(w2, k))
    np.testing.assert_array_equal(c1.view(np.uint64), c2.view(np.uint64))
    got = np.isfinite(tr["first_token_time"])
    # a query that got its first token holds no id any more; the others still do
    ids = set(tr["run_id"][tr["run_id"] >= 0].tolist()) | set(tr["wait_id"][tr["wait_id"] >= 0].tolist())
    for i in range(40):
        if a[i] < 0:
            assert not got[i] and i not in ids
        else:
            assert got[i] != (i in ids)


@pytest.mark.parametrize("mode", [0, 1])
def test_first_token_time_against_snapshot_clock_plus_estimate(mode):
    # Routed one at a time, a query waits behind everything already queued, and what is
    # routed later never changes its token allocation (FCFS): its first token comes after
    # exactly the batches the estimate simulated from the decision's snapshot.  Those
    # batches can only grow longer when later queries share them (Eq. 9 has no negative
    # term), so the realized first-token time is at least the snapshot's clock plus the SFS
    # estimate, and equal to it (up to rounding: the executed batches are timed one by one
    # in fp32 and summed in fp64) when no later query reached the instance first.
    wl = W.make_workload("pool64", num_queries=400, first_token_mode=mode, cap_waiting=512)
    I = wl.num_instances
    tr = oracle.new_track(wl, wl.num_queries)
    rate = 0.8 * float(oracle.pool_capacity(wl).sum())
    arr = W.poisson_arrivals(wl.num_queries, rate, 9)
    st, clk = wl, np.zeros(I)
    none = np.zeros(0, np.int32)
    expect = np.zeros(wl.num_queries)
    inst = np.zeros(wl.num_queries, np.int64)
    for i in range(wl.num_queries):
        if i == 0:
            st, clk, tr = oracle.advance(st, clk, none, none, none, float(arr[0]), track=tr)
        else:
            st, clk, tr = oracle.advance(st, clk, prev_a, prev_p, prev_d, float(arr[i]), track=tr, id_base=i - 1)
        q = st.with_queries(np.array([i]))
        _, _, t32, t64 = oracle.estimate_matrix(q)
        a, _, _ = oracle.route(q, t32, lam=wl.lam, mu=wl.mu)
        j = int(a[0, 0])
        inst[i] = j
        expect[i] = clk[j] + t64[0, j]
        prev_a = a[0].astype(np.int32)
        prev_p = wl.prompt_len[i:i + 1]
        prev_d = np.ascontiguousarray(wl.dec_hat[i:i + 1, wl.model_of_instance[j]])
    st, clk, tr = oracle.advance(st, clk, prev_a, prev_p, prev_d, 1e9, track=tr, id_base=wl.num_queries - 1)
    ftt = tr["first_token_time"]
    assert np.all(np.isfinite(ftt)) and np.all(ftt >= arr)
    tol = 1e-6 * np.max(expect)
    assert np.all(ftt >= expect - tol)
    alone = np.array([not np.any((inst[i + 1:] == inst[i]) & (arr[i + 1:] < ftt[i])) for i in range(len(ftt))])
    assert alone.sum() >= 10 and (~alone).sum() >= 10  # both cases occur on this trace
    assert np.max(np.abs(ftt[alone] - expect[alone])) <= tol
    # some queries that shared their batches with later ones did come later than estimated
    assert np.max(ftt[~alone] - expect[~alone]) > 1e3 * tol
