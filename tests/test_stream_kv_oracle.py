"""Pins of the oracle's stream step under KV-cache limits (orc_advance_kv).

Each executed batch follows the KV step rule of App. F's reading (blocks found in
running order, preemption of the last running request, admission only with the
first chunk's blocks, the context limit ending a request).  Pinned against:
- the hand-worked KV traces (tests/golden/kv_hand_trace_residents*.json) replayed
  as an executed stream: t_now set to the exact sum of the batches' Eq. 9 times
  (power-of-two coefficients, so every time is exact), the state after each batch
  read off the trace by hand, and the query's first token at the trace's batch;
- the plain stream step (an independent loop) when the limits cannot bind;
- a context limit that acts as a shorter response.
"""
import json
import os
from fractions import Fraction

import numpy as np
import pytest

import oracle
from paper_2607_18253_gb300 import workloads as W

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
# b0, prefill-token, decode-request, context-sum and attention-pair coefficients of Eq. 9;
# powers of two, so every batch time and every partial sum below is exact
COEF = (Fraction(1, 4), Fraction(1, 16), Fraction(1, 8), Fraction(1, 1024), Fraction(1, 4096))
STATE = ("n_run", "run_ctx", "run_pre", "run_dec", "n_wait", "wait_pre", "wait_dec")


def _one_instance(running, waiting, B, S, mode, cap=16):
    wl = W.small_workload(0, num_instances=1, num_models=1, num_queries=1, cap_running=cap, cap_waiting=cap,
                          first_token_mode=mode)
    wl.max_batched_tokens[:] = B
    wl.max_seqs[:] = S
    wl.coef[:] = np.array([float(c) for c in COEF], np.float32)
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


def _batch_time(F):
    """Eq. 9 for one batch with features F = (1, F1, F2, F3, F4), exactly."""
    return sum(c * int(f) for c, f in zip(COEF, F))


def _state(wl):
    nr, nw = int(wl.n_run[0]), int(wl.n_wait[0])
    run = [(int(wl.run_ctx[0, r]), int(wl.run_pre[0, r]), int(wl.run_dec[0, r])) for r in range(nr)]
    wait = [(int(wl.wait_pre[0, w]), int(wl.wait_dec[0, w])) for w in range(nw)]
    return run, wait


# The state after batch l of each hand trace, read off its batch-by-batch notes (R1, R2
# the residents, W the waiting resident, q the query routed at the start): running list
# (context, prefill left, decode left) in order, waiting queue (prefill, decode) in order.
# Batch l's features are the trace's residents_per_batch row plus the query's share: in
# the separate-decode trace q is admitted with 2 tokens in batch 10 (F1 += 2, F4 += 3) and
# decodes at context 2 in batch 11; with the last chunk it is admitted in batch 8.
HAND = {
    "kv_hand_trace_residents.json": {
        "query_rows": {10: (0, 2, 0, 0, 3), 11: (0, 0, 1, 2, 0)},
        "first_token_batch": 11,
        "after": {
            1: ([(4, 0, 4), (5, 0, 4)], [(3, 2), (2, 1)]),
            2: ([(5, 0, 3), (6, 0, 3)], [(3, 2), (2, 1)]),
            3: ([(6, 0, 2), (6, 0, 3)], [(3, 2), (2, 1)]),
            4: ([(7, 0, 1)], [(6, 3), (3, 2), (2, 1)]),
            5: ([], [(6, 3), (3, 2), (2, 1)]),
            6: ([(6, 0, 3), (2, 1, 2)], [(2, 1)]),
            7: ([(7, 0, 2), (3, 0, 2)], [(2, 1)]),
            8: ([(8, 0, 1), (4, 0, 1)], [(2, 1)]),
            9: ([], [(4, 1), (2, 1)]),
            10: ([(4, 0, 1), (2, 0, 1)], []),
            11: ([], []),
        },
    },
    "kv_hand_trace_residents_mode1.json": {
        "query_rows": {8: (0, 2, 0, 0, 3)},
        "first_token_batch": 8,
        "after": {
            1: ([(4, 0, 4), (5, 0, 4)], [(3, 2), (2, 1)]),
            2: ([(5, 0, 3), (6, 0, 3)], [(3, 2), (2, 1)]),
            3: ([(6, 0, 2), (6, 0, 2)], [(3, 2), (2, 1)]),
            4: ([(7, 0, 1)], [(6, 2), (3, 2), (2, 1)]),
            5: ([], [(6, 2), (3, 2), (2, 1)]),
            6: ([(6, 0, 1), (2, 1, 2)], [(2, 1)]),
            7: ([(3, 0, 1)], [(2, 1)]),
            8: ([], []),
        },
    },
}


def _hand_batches(fixture):
    g = json.load(open(os.path.join(GOLDEN, fixture)))
    h = HAND[fixture]
    rows = [np.asarray(r, np.int64) for r in g["residents_per_batch"]]
    for l, q in h["query_rows"].items():
        rows[l - 1] = rows[l - 1] + np.asarray(q, np.int64)
    # the whole batches add up to the trace's totals (the query's F included)
    np.testing.assert_array_equal(np.sum(rows, axis=0), g["F"])
    ends = np.cumsum([_batch_time(r) for r in rows])  # exact: Fractions
    return g, h, ends


@pytest.mark.parametrize("fixture", sorted(HAND))
def test_hand_traces_replayed_as_an_executed_stream(fixture):
    g, h, ends = _hand_batches(fixture)
    wl = _one_instance(g["running"], g["waiting"], g["B"], g["S"], g["mode"])
    kv = (g["block_size"], g["num_blocks"], g["max_ctx"])
    p, d = g["query"]
    one = lambda x: np.asarray([x], np.int32)
    for l, (run, wait) in h["after"].items():
        t_end = ends[l - 1]
        # t_now at batch l's end runs exactly l batches ...
        w2, clk, tr = oracle.advance(wl, [0.0], one(0), one(p), one(d), float(t_end), track=oracle.new_track(wl, 1),
                                     id_base=0, kv=kv)
        assert _state(w2) == (run, wait), l
        assert clk[0] == float(t_end)
        ft = tr["first_token_time"][0]
        if l >= h["first_token_batch"]:
            assert ft == float(ends[h["first_token_batch"] - 1])
        else:
            assert np.isnan(ft)
        # ... and a hair before it, l - 1 (batch l would still be running)
        before = float(t_end - Fraction(1, 1 << 20))
        w3, clk3 = oracle.advance(wl, [0.0], one(0), one(p), one(d), before, kv=kv)
        prev = h["after"].get(l - 1, ([tuple(r) for r in g["running"]],
                                      [tuple(w) for w in g["waiting"]] + [(p, d)]))
        assert _state(w3) == prev, l
        assert clk3[0] == (float(ends[l - 2]) if l > 1 else 0.0)


def _stream(wl, steps, seed, kv, dt=0.05):
    """A few stream steps (append + advance) with first-token tracking; returns every
    snapshot, clocks and the tracking state."""
    rng = np.random.default_rng(seed)
    I = wl.num_instances
    tr = oracle.new_track(wl, 4 * steps)
    st, clk, out = wl, np.zeros(I), []
    for s in range(steps):
        a = rng.integers(-1, I, 4).astype(np.int32)
        p = rng.integers(1, 120, 4).astype(np.int32)
        d = rng.integers(1, 30, 4).astype(np.int32)
        st, clk, tr = oracle.advance(st, clk, a, p, d, dt * (s + 1), track=tr, id_base=4 * s, kv=kv)
        out.append((st, clk.copy()))
    return out, tr


@pytest.mark.parametrize("mode", [0, 1])
def test_limits_that_cannot_bind_give_the_plain_stream(mode):
    # the KV loop with unlimited blocks and context is the plain stream step, an
    # independent loop: every snapshot, clock and first-token time bit for bit
    for seed in range(4):
        wl = W.small_workload(20 + seed, num_instances=5, num_models=2, num_queries=8, cap_running=64,
                              cap_waiting=96, first_token_mode=mode, budget_range=(8, 64), wait_max=12)
        big = (16, 1 << 40, 1 << 40)
        got, tr = _stream(wl, 12, seed, big)
        ref, tr0 = _stream(wl, 12, seed, None)
        for (a, ca), (b, cb) in zip(got, ref):
            for k in STATE:
                np.testing.assert_array_equal(getattr(a, k), getattr(b, k))
            np.testing.assert_array_equal(ca.view(np.uint64), cb.view(np.uint64))
        np.testing.assert_array_equal(tr["first_token_time"].view(np.uint64), tr0["first_token_time"].view(np.uint64))


@pytest.mark.parametrize("mode", [0, 1])
def test_context_limit_is_a_shorter_response(mode):
    # a decoder at context 60 under a limit of 62 ends after two decode batches, exactly
    # as one with two tokens left and no limit; the limit never shortens the one that
    # needs fewer
    kv = (8, 1 << 20, 62)
    wl = _one_instance([(60, 0, 100), (5, 0, 9)], [(20, 4)], 16, 4, mode)
    ref = _one_instance([(60, 0, 2), (5, 0, 9)], [(20, 4)], 16, 4, mode)
    a, p, d = (np.asarray([0], np.int32), np.asarray([30], np.int32), np.asarray([3], np.int32))
    ended = 0
    for t_now in (0.3, 1.5, 3.0, 6.0, 12.0, 30.0):
        w1, c1 = oracle.advance(wl, [0.0], a, p, d, t_now, kv=kv)
        w0, c0 = oracle.advance(ref, [0.0], a, p, d, t_now)
        (r1, q1), (r0, q0) = _state(w1), _state(w0)
        # while it runs, the limited request (the only one past context 14) has 98 more
        # decode tokens on record
        assert [(c, pr, dd - 98 if c >= 60 else dd) for c, pr, dd in r1] == r0 and q1 == q0
        assert c1[0] == c0[0]
        ended += all(c < 60 for c, _, _ in r1)
    assert ended >= 3


def test_a_query_that_could_never_run_is_refused():
    wl = _one_instance([(5, 0, 3)], [], 16, 4, 0)
    a = np.asarray([0], np.int32)
    with pytest.raises(RuntimeError):  # its prompt reaches the context limit
        oracle.advance(wl, [0.0], a, np.asarray([64], np.int32), np.asarray([2], np.int32), 1.0, kv=(8, 100, 64))
    with pytest.raises(RuntimeError):  # its whole context needs more blocks than there are
        oracle.advance(wl, [0.0], a, np.asarray([30], np.int32), np.asarray([20], np.int32), 1.0, kv=(8, 6, 1000))
    # the same query within the limits runs
    oracle.advance(wl, [0.0], a, np.asarray([30], np.int32), np.asarray([10], np.int32), 1.0, kv=(8, 6, 1000))


@pytest.mark.parametrize("mode", [0, 1])
def test_binding_limits_keep_every_snapshot_valid(mode):
    # Under limits that bind, every published snapshot is a valid KV snapshot (what the
    # KV load checks): the running requests' blocks fit, only the last running request
    # is in prefill, no context reaches the limit, every request's whole context fits;
    # and requests are conserved (routed = resident + finished).
    differs = 0
    for seed in range(6):
        wl = W.small_workload(50 + seed, num_instances=4, num_models=2, num_queries=8, cap_running=64,
                              cap_waiting=128, first_token_mode=mode, budget_range=(8, 64), wait_max=10)
        bs, nb, mc = W.kv_limits(wl, seed, block_sizes=(1, 4, 16), tightness=(0.0, 0.3), max_new=30)
        got, tr = _stream(wl, 16, seed, (bs, nb, mc))
        ref, _ = _stream(wl, 16, seed, None)
        for (st, _), (st0, _) in zip(got, ref):
            differs += int(any(not np.array_equal(getattr(st, k), getattr(st0, k)) for k in STATE))
            for j in range(wl.num_instances):
                b = int(bs[j])
                nr, nw = int(st.n_run[j]), int(st.n_wait[j])
                ctx, pre, dec = st.run_ctx[j, :nr], st.run_pre[j, :nr], st.run_dec[j, :nr]
                assert sum((int(c) + b - 1) // b for c in ctx) <= nb[j]
                assert all(int(x) == 0 for x in pre[:-1])
                assert all(int(c) + int(p) < mc[j] for c, p in zip(ctx, pre))
                assert (dec >= 1).all()
                wp, wd = st.wait_pre[j, :nw], st.wait_dec[j, :nw]
                assert all(int(p) < mc[j] for p in wp) and (wd >= 1).all()
                whole = [min(int(c) + int(p) + int(d), int(mc[j])) for c, p, d in zip(ctx, pre, dec)]
                whole += [min(int(p) + int(d), int(mc[j])) for p, d in zip(wp, wd)]
                assert all((x + b - 1) // b <= nb[j] for x in whole)
        # every tracked query that holds no id any more has its first-token time
        ids = set(tr["run_id"][tr["run_id"] >= 0].tolist()) | set(tr["wait_id"][tr["wait_id"] >= 0].tolist())
        got_t = np.isfinite(tr["first_token_time"])
        assert not any(got_t[i] for i in ids)
    assert differs >= 10  # the limits change the stream
