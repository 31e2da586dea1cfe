"""Pins of the oracle's KV-cache step rule (App. F: context limits, KV-cache
allocation, preemption; the reading is stated in oracle/sfs_oracle.c).

The rule is pinned against: the plain step rule when the limits cannot bind (an
independent code path), a hand-worked trace with a preemption of the query
(tests/golden/kv_hand_trace.json), a context limit that reduces to a shorter
response, and the property the GPU design rests on: the residents' batches do not
depend on the appended query, preemptions included.
"""
import json
import os

import numpy as np
import pytest

import oracle

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "kv_hand_trace.json")


def random_pool(rng, max_run=12, max_wait=10):
    S = int(rng.integers(2, 16))
    B = int(rng.integers(S + 4, 200))
    nr = int(rng.integers(0, min(S, max_run) + 1))
    running = [(int(rng.integers(0, 300)), 0, int(rng.integers(1, 40))) for _ in range(nr)]
    if nr and rng.random() < 0.3:  # the last running request still in prefill
        c, _, d = running[-1]
        running[-1] = (c, int(rng.integers(1, 150)), d)
    waiting = [(int(rng.integers(1, 200)), int(rng.integers(1, 40))) for _ in range(int(rng.integers(0, max_wait + 1)))]
    return B, S, running, waiting


@pytest.mark.parametrize("mode", [0, 1])
def test_unbounded_limits_reduce_to_the_plain_rule(mode):
    rng = np.random.default_rng(100 + mode)
    for _ in range(300):
        B, S, running, waiting = random_pool(rng)
        p, d = int(rng.integers(1, 300)), int(rng.integers(1, 30))
        F0, la0, lt0 = oracle.simulate(running, waiting, B, S, p, d, mode=mode)
        F, la, lt, _, _ = oracle.simulate_kv(running, waiting, B, S, p, d, block_size=16, num_blocks=1 << 40,
                                             max_ctx=1 << 40, mode=mode)
        np.testing.assert_array_equal(F, F0)
        assert (la, lt) == (la0, lt0)


def test_hand_trace_with_a_preemption_of_the_query():
    g = json.load(open(GOLDEN))
    F, la, lt, _, used = oracle.simulate_kv(g["running"], g["waiting"], g["B"], g["S"], *g["query"],
                                            block_size=g["block_size"], num_blocks=g["num_blocks"],
                                            max_ctx=g["max_ctx"], mode=g["mode"])
    np.testing.assert_array_equal(F, g["F"])
    assert la == g["admit_batch"] and lt == g["first_token_batch"] and used == g["most_blocks_in_use"]


@pytest.mark.parametrize("fixture", ["kv_hand_trace_residents.json", "kv_hand_trace_residents_mode1.json"])
def test_hand_trace_with_residents_preempting_each_other(fixture):
    # a resident preempting itself and readmitted in the same batch, one preempted
    # by an older one, a partial chunk, and the query admitted once the instance
    # drains (tests/golden/kv_hand_trace_residents*.json, both first-token modes);
    # the residents' own batches are also those of the residents alone
    g = json.load(open(os.path.join(os.path.dirname(__file__), "golden", fixture)))
    args = (g["running"], g["waiting"], g["B"], g["S"])
    kw = dict(block_size=g["block_size"], num_blocks=g["num_blocks"], max_ctx=g["max_ctx"], mode=g["mode"])
    F, la, lt, res, used = oracle.simulate_kv(*args, *g["query"], **kw)
    np.testing.assert_array_equal(F, g["F"])
    assert la == g["admit_batch"] and lt == g["first_token_batch"] and used == g["most_blocks_in_use"]
    np.testing.assert_array_equal(res, g["residents_per_batch"])
    alone = oracle.kv_residents(*args, lt, **kw)
    np.testing.assert_array_equal(alone, g["residents_per_batch"])


def test_context_limit_is_a_shorter_response():
    # a decoder at context 60 under a limit of 62 decodes twice, exactly like one
    # with two tokens left and no limit
    for mode in (0, 1):
        F, la, lt, _, _ = oracle.simulate_kv([(60, 0, 100), (5, 0, 9)], [(20, 4)], 16, 4, 30, 3, block_size=8,
                                             num_blocks=1 << 20, max_ctx=62, mode=mode)
        F0, la0, lt0 = oracle.simulate([(60, 0, 2), (5, 0, 9)], [(20, 4)], 16, 4, 30, 3, mode=mode)
        np.testing.assert_array_equal(F, F0)
        assert (la, lt) == (la0, lt0)


def test_invalid_inputs():
    with pytest.raises(RuntimeError):  # the query's prompt reaches the context limit
        oracle.simulate_kv([], [], 16, 4, 64, 2, block_size=8, num_blocks=100, max_ctx=64)
    with pytest.raises(RuntimeError):  # the query could never hold its whole context
        oracle.simulate_kv([], [], 16, 4, 30, 20, block_size=8, num_blocks=6, max_ctx=1000)
    with pytest.raises(RuntimeError):  # the residents hold more blocks than there are
        oracle.simulate_kv([(40, 0, 3)], [], 16, 4, 5, 2, block_size=8, num_blocks=4, max_ctx=1000)


@pytest.mark.parametrize("mode", [0, 1])
def test_residents_do_not_depend_on_the_query(mode):
    # the residents' batches up to the query's first token are those of the residents
    # alone, also when blocks run out and requests (the query included) are preempted
    rng = np.random.default_rng(7 + mode)
    binding = 0
    n = 400
    for _ in range(n):
        B, S, running, waiting = random_pool(rng)
        bs = int(rng.integers(1, 9))
        p, d = int(rng.integers(1, 250)), int(rng.integers(1, 30))
        held = sum((c + bs - 1) // bs for c, _, _ in running)
        # enough blocks for any one request's whole context, few enough to bind
        whole = [c + pr + dd for c, pr, dd in running] + [pr + dd for pr, dd in waiting] + [p + d]
        nb = max(held + int(rng.integers(1, 40)), max((w + bs - 1) // bs for w in whole))
        max_ctx = 1 << 20
        F, la, lt, res, used = oracle.simulate_kv(running, waiting, B, S, p, d, block_size=bs, num_blocks=nb,
                                                  max_ctx=max_ctx, mode=mode)
        alone = oracle.kv_residents(running, waiting, B, S, lt, block_size=bs, num_blocks=nb, max_ctx=max_ctx,
                                    mode=mode)
        np.testing.assert_array_equal(res, alone)
        assert used <= nb
        F0, _, lt0 = oracle.simulate(running, waiting, B, S, p, d, mode=mode)
        binding += int(lt != lt0 or not np.array_equal(F, F0))
    assert binding >= n // 4  # the limits bind in a good share of the cases


@pytest.mark.parametrize("mode", [0, 1])
def test_candidate_matrix_reduces_to_the_plain_matrix(mode):
    # the batch entry point with limits that cannot bind gives the plain SFS matrix
    # (an independent code path): features, first-token batches and times
    from paper_2607_18253_gb300 import workloads as W
    wl = W.small_workload(40 + mode, num_instances=7, num_queries=20, first_token_mode=mode)
    st, F, lt, t32, t64 = oracle.estimate_matrix_kv(wl, 16, 1 << 40, 1 << 40)
    F0, lt0, t320, t640 = oracle.estimate_matrix(wl)
    assert (st == 0).all()
    np.testing.assert_array_equal(F, F0)
    np.testing.assert_array_equal(lt, lt0)
    np.testing.assert_array_equal(t32.view(np.uint32), t320.view(np.uint32))
    np.testing.assert_array_equal(t64, t640)


@pytest.mark.parametrize("mode", [0, 1])
def test_candidate_matrix_matches_single_candidates(mode):
    # the batch entry point under binding limits: each candidate as the single-candidate
    # simulation gives it with one output token; invalid queries are flagged, not fatal
    from paper_2607_18253_gb300 import workloads as W
    wl = W.small_workload(50 + mode, num_instances=6, num_queries=12, first_token_mode=mode)
    bs, nb, mc = W.kv_limits(wl, 3, block_sizes=(1, 4, 16))
    mc = mc.copy()
    wl.n_run[0] = 0  # an idle instance whose context limit some queries' prompts reach
    wl.n_wait[0] = 0
    mc[0] = int(np.median(wl.prompt_len))
    nb[0] = max(nb[0], int(wl.run_ctx[0].max() + wl.run_pre[0].max() + wl.run_dec[0].max()) + 64)
    st, F, lt, t32, _ = oracle.estimate_matrix_kv(wl, bs, nb, mc)
    changed = 0
    F0, lt0, _, _ = oracle.estimate_matrix(wl)
    for i in range(wl.num_queries):
        for j in range(wl.num_instances):
            n, w = int(wl.n_run[j]), int(wl.n_wait[j])
            running = list(zip(wl.run_ctx[j, :n], wl.run_pre[j, :n], wl.run_dec[j, :n]))
            waiting = list(zip(wl.wait_pre[j, :w], wl.wait_dec[j, :w]))
            p = int(wl.prompt_len[i])
            try:
                Fs, _, lts, _, _ = oracle.simulate_kv(running, waiting, int(wl.max_batched_tokens[j]),
                                                      int(wl.max_seqs[j]), p, 1, block_size=int(bs[j]),
                                                      num_blocks=int(nb[j]), max_ctx=int(mc[j]), mode=mode,
                                                      max_batches=1 << 16)
            except RuntimeError:
                assert st[i, j] != 0 and (F[i, j] == -1).all() and lt[i, j] == -1 and np.isnan(t32[i, j])
                assert j == 0 and p >= mc[0]
                continue
            assert st[i, j] == 0
            np.testing.assert_array_equal(F[i, j], Fs)
            assert lt[i, j] == lts
            changed += int(lts != lt0[i, j] or not np.array_equal(Fs, F0[i, j]))
    assert (st[:, 0] != 0).any() and (st[:, 0] == 0).any()
    assert changed > 0  # the generated limits bind somewhere


def test_route_skips_candidates_without_an_estimate():
    # a NaN time (no estimate) is not eligible: on rows with a finite time the choice
    # equals the choice with NaN read as an infinite time (never preferred under
    # Eq. 5 with mu > 0, never within a target under Eq. 3, never the least); a row
    # with no finite time gets -1 and NaN
    from paper_2607_18253_gb300 import workloads as W
    wl = W.small_workload(80, num_instances=9, num_queries=40)
    rng = np.random.default_rng(2)
    t = rng.uniform(0.05, 2.0, (40, 9)).astype(np.float32)
    t[rng.random(t.shape) < 0.3] = np.nan
    t[:, 0] = np.nan       # the lowest index never has a time
    t[5, :] = np.nan       # nor does any instance of row 5
    inf = np.where(np.isnan(t), np.float32(np.inf), t)
    lam = np.array([0.5], np.float32)
    for mu in (np.array([0.2], np.float32), np.array([3.0], np.float32)):
        a, u, tc = oracle.route(wl, t, lam=lam, mu=mu)
        ai, ui, tci = oracle.route(wl, inf, lam=lam, mu=mu)
        ok = ~np.isnan(t).all(axis=1)
        np.testing.assert_array_equal(a[0, ok], ai[0, ok])
        np.testing.assert_array_equal(u[0, ok], ui[0, ok])
        assert (a[0, ~ok] == -1).all() and np.isnan(u[0, ~ok]).all() and np.isnan(tc[0, ~ok]).all()
        assert not (a[0] == 0).any()
    tau = np.full(40, 0.6, np.float32)
    a, u, tc = oracle.route(wl, t, lam=lam, tau=tau)
    ai, _, _ = oracle.route(wl, inf, lam=lam, tau=tau)
    ok = ~np.isnan(t).all(axis=1)
    np.testing.assert_array_equal(a[0, ok], ai[0, ok])
    assert (a[0, ~ok] == -1).all() and not (a[0] == 0).any()


@pytest.mark.parametrize("name", ["tiny", "pool64", "pool256"])
def test_generated_limits_are_valid_inputs(name):
    # the seeded limits keep every snapshot valid under the KV rule: the running
    # requests' blocks fit, every request's whole context (capped) fits, no context
    # reaches the limit, and the longest prompt's first token fits
    from paper_2607_18253_gb300 import workloads as W
    wl = W.make_workload(name)
    bs, nb, mc = W.kv_limits(wl, 11, block_sizes=(16,))
    ceil = lambda c, b: -(-c // b)  # noqa: E731
    for j in range(wl.num_instances):
        n, w = int(wl.n_run[j]), int(wl.n_wait[j])
        ctx, pre, dec = (a[j, :n].astype(np.int64) for a in (wl.run_ctx, wl.run_pre, wl.run_dec))
        wp, wd = (a[j, :w].astype(np.int64) for a in (wl.wait_pre, wl.wait_dec))
        b = int(bs[j])
        assert ceil(ctx, b).sum() <= nb[j]
        assert ((ctx + pre) < mc[j]).all() and (wp < mc[j]).all() and wl.max_prompt_len < mc[j]
        assert (ceil(np.minimum(ctx + pre + dec, mc[j]), b) <= nb[j]).all()
        assert (ceil(np.minimum(wp + wd, mc[j]), b) <= nb[j]).all()
        assert ceil(wl.max_prompt_len + 1, b) <= nb[j]
    assert (mc < (1 << 40)).any() and (mc == (1 << 40)).any()  # both kinds of instance
