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
