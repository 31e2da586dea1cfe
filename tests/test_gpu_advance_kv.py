"""The online stream step under KV-cache limits (App. F: KV-cache allocation, context
limits, preemption) through the C ABI: CUDA path vs the CPU oracle's orc_advance_kv.

Snapshots (running and waiting lists, counts) match exactly, clocks and first-token
times bit for bit (both sides time every executed batch with the same fp32 Eq. 9
expression and sum into an fp64 clock), and the KV estimate over each advanced
snapshot matches the oracle's KV matrix over the oracle's snapshot.
"""
import dataclasses

import numpy as np
import pytest

torch = pytest.importorskip("torch")

import oracle  # noqa: E402
from paper_2607_18253_gb300 import workloads as W  # noqa: E402

pytestmark = pytest.mark.gpu
STATE = ("n_run", "run_ctx", "run_pre", "run_dec", "n_wait", "wait_pre", "wait_dec")


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def R():
    from paper_2607_18253_gb300 import router
    return router


def bits(a):
    return np.ascontiguousarray(a, np.float32).view(np.uint32)


def dev(a, dtype=torch.int32):
    return torch.from_numpy(np.ascontiguousarray(a)).to("cuda", dtype)


def make(wl, limits, horizon=4096, **kw):
    rt = R().LatencyRouter.from_workload(wl, **kw)
    rt.set_kv_limits(*limits, horizon=horizon)
    rt.load_state(*R().state_tensors(wl))
    return rt


def read(rt):
    st = rt.read_state()
    torch.cuda.synchronize()
    return {k: v.cpu().numpy() for k, v in st.items()}


def check_state(st, wl, clk, msg=""):
    np.testing.assert_array_equal(st["n_run"], wl.n_run, err_msg=msg)
    np.testing.assert_array_equal(st["n_wait"], wl.n_wait, err_msg=msg)
    np.testing.assert_array_equal(st["clock"].view(np.uint64), np.asarray(clk, np.float64).view(np.uint64),
                                  err_msg=msg)
    for j in range(wl.num_instances):
        nr, nw = int(wl.n_run[j]), int(wl.n_wait[j])
        for k in ("run_ctx", "run_pre", "run_dec"):
            np.testing.assert_array_equal(st[k][j, :nr], getattr(wl, k)[j, :nr], err_msg=f"{msg} {k} row {j}")
        for k in ("wait_pre", "wait_dec"):
            np.testing.assert_array_equal(st[k][j, :nw], getattr(wl, k)[j, :nw], err_msg=f"{msg} {k} row {j}")


def check_kv_estimate(rt, wl, limits, msg=""):
    p = dev(wl.prompt_len)
    fb = torch.empty((wl.num_queries, wl.num_instances), dtype=torch.int32, device="cuda")
    t = rt.estimate_ttft(p, first_batch=fb)
    F = rt.estimate_features(p)
    torch.cuda.synchronize()
    st, eF, elt, et, _ = oracle.estimate_matrix_kv(wl, *limits)
    ok = st == 0
    np.testing.assert_array_equal(F.cpu().numpy()[ok], eF[ok], err_msg=msg)
    np.testing.assert_array_equal(fb.cpu().numpy()[ok], elt[ok], err_msg=msg)
    np.testing.assert_array_equal(bits(t.cpu().numpy()[ok]), bits(et[ok]), err_msg=msg)
    assert np.isnan(t.cpu().numpy()[~ok]).all()
    assert rt.status() == (R().LR_OK if ok.all() else R().LR_EINVAL), msg


@pytest.mark.parametrize("mode", [0, 1])
def test_stream_matches_the_oracle(mode):
    # random small pools under binding limits (blocks of 1, 4 or 16 tokens, a context
    # limit on half the instances), four successive advances with tracked appends (one
    # untracked), the last one draining everything
    binding = 0
    for seed in range(8):
        rng = np.random.default_rng(4000 + seed)
        wl = W.small_workload(300 + seed, num_instances=int(3 + seed % 29), num_models=3, num_queries=24,
                              cap_running=64, cap_waiting=200, first_token_mode=mode, wait_max=24,
                              budget_range=(8, 64), min_gap=8)
        limits = W.kv_limits(wl, seed, block_sizes=(1, 4, 16), tightness=(0.0, 0.3), max_new=30)
        rt = make(wl, limits)
        N = 4 * 40
        ftt = torch.full((N,), float("nan"), dtype=torch.float64, device="cuda")
        rt.track_first_tokens(ftt)
        tr = oracle.new_track(wl, N)
        clk = np.zeros(wl.num_instances)
        plain, pclk = wl, clk
        for step, t_now in enumerate((0.05, 0.4, 2.0, 1e7)):
            Q = 40
            a = rng.integers(-1, wl.num_instances, Q).astype(np.int32)
            p = rng.integers(1, 160, Q).astype(np.int32)
            d = rng.integers(1, 30, Q).astype(np.int32)
            base = None if step == 2 else 40 * step
            rt.advance(dev(a), dev(p), dev(d), t_now, id_base=base)
            torch.cuda.synchronize()
            msg = f"seed {seed} step {step}"
            assert rt.status() == R().LR_OK, msg
            wl, clk, tr = oracle.advance(wl, clk, a, p, d, t_now, track=tr, id_base=-1 if base is None else base,
                                         kv=limits)
            plain, pclk = oracle.advance(plain, pclk, a, p, d, t_now)
            binding += int(any(not np.array_equal(getattr(wl, k), getattr(plain, k)) for k in STATE))
            check_state(read(rt), wl, clk, msg)
            got, exp = ftt.cpu().numpy(), tr["first_token_time"]
            np.testing.assert_array_equal(np.isnan(got), np.isnan(exp), err_msg=msg)
            np.testing.assert_array_equal(got[~np.isnan(exp)].view(np.uint64), exp[~np.isnan(exp)].view(np.uint64))
            if step < 3:
                check_kv_estimate(rt, wl, limits, msg)
        assert np.isnan(got[80:120]).all()
        assert np.isfinite(got[:80]).sum() > 0
        rt.close()
    assert binding >= 6  # the limits change the stream


def test_hand_trace_pools_step_by_step():
    # the pools of the hand-worked KV traces (a resident preempting itself and admitted
    # again in the same batch, one preempted by an older one, a partial chunk), advanced
    # in 40 small steps: the state after every step as the oracle's
    running, waiting = [(3, 0, 5), (4, 0, 5)], [(3, 2)]
    for mode in (0, 1):
        wl = W.small_workload(0, num_instances=1, num_models=1, num_queries=1, cap_running=16, cap_waiting=16,
                              first_token_mode=mode)
        wl.max_batched_tokens[:] = 8
        wl.max_seqs[:] = 4
        wl.coef[:] = np.array([0.25, 2.0 ** -4, 2.0 ** -3, 2.0 ** -10, 2.0 ** -12], np.float32)
        wl.model_of_instance[:] = 0
        for arr in (wl.run_ctx, wl.run_pre, wl.run_dec, wl.wait_pre, wl.wait_dec):
            arr[:] = 0
        wl.n_run[:] = len(running)
        wl.n_wait[:] = len(waiting)
        for r, (c, pr, d) in enumerate(running):
            wl.run_ctx[0, r], wl.run_pre[0, r], wl.run_dec[0, r] = c, pr, d
        for w, (pr, d) in enumerate(waiting):
            wl.wait_pre[0, w], wl.wait_dec[0, w] = pr, d
        wl.prompt_len[:] = 2
        limits = (np.array([2], np.int32), np.array([6], np.int64), np.array([1 << 20], np.int64))
        rt = make(wl, limits)
        ftt = torch.full((1,), float("nan"), dtype=torch.float64, device="cuda")
        rt.track_first_tokens(ftt)
        tr = oracle.new_track(wl, 1)
        clk = np.zeros(1)
        for s in range(40):
            t_now = 0.2 * (s + 1)
            a = np.zeros(1 if s == 0 else 0, np.int32)
            p = np.full(a.shape, 2, np.int32)
            d = np.ones(a.shape, np.int32)
            rt.advance(dev(a), dev(p), dev(d), t_now, id_base=0 if s == 0 else None)
            torch.cuda.synchronize()
            assert rt.status() == R().LR_OK
            wl, clk, tr = oracle.advance(wl, clk, a, p, d, t_now, track=tr, id_base=0 if s == 0 else -1, kv=limits)
            check_state(read(rt), wl, clk, f"mode {mode} step {s}")
        assert np.isfinite(tr["first_token_time"][0])
        np.testing.assert_array_equal(ftt.cpu().numpy().view(np.uint64), tr["first_token_time"].view(np.uint64))
        rt.close()


@pytest.mark.parametrize("mode", [0, 1])
def test_route_advance_loop_under_limits(mode):
    # the online loop of Sec. 5 under KV limits: route a micro-batch on the live
    # snapshot (the KV estimate), append it to the chosen instances, advance the pool;
    # assignments, utilities and states stay identical to the oracle's
    per, steps = 25, 6
    full, limits = _pool(80 + mode, mode, per * steps)
    rt = make(full, limits, max_queries=per)
    wl, clk = full, np.zeros(full.num_instances)
    lam, mu = full.lam[:1], full.mu[:1]
    for s in range(steps):
        sl = slice(s * per, (s + 1) * per)
        q = dataclasses.replace(wl, prompt_len=full.prompt_len[sl], dec_hat=full.dec_hat[sl], acc=full.acc[sl],
                                tau=full.tau[sl])
        out = rt.route(dev(q.prompt_len), dev(q.dec_hat), dev(q.acc, torch.float32), lam, mu)
        torch.cuda.synchronize()
        _, _, _, et, _ = oracle.estimate_matrix_kv(q, *limits)
        a, u, _ = oracle.route(q, et, lam=lam, mu=mu)
        np.testing.assert_array_equal(out["assign"].cpu().numpy(), a)
        np.testing.assert_array_equal(bits(out["util"].cpu().numpy()), bits(u))
        a0 = a[0]
        d = np.where(a0 >= 0, q.dec_hat[np.arange(per), q.model_of_instance[np.maximum(a0, 0)]], 1)
        t_now = 0.03 * (s + 1)
        rt.advance(dev(a0), dev(q.prompt_len), dev(d), t_now)
        torch.cuda.synchronize()
        assert rt.status() == R().LR_OK
        wl, clk = oracle.advance(q, clk, a0, q.prompt_len, d, t_now, kv=limits)
        check_state(read(rt), wl, clk, f"step {s}")
    rt.close()


def _pool(seed, mode, nq):
    wl = W.small_workload(seed, num_instances=24, num_models=3, num_queries=nq, first_token_mode=mode,
                          cap_running=64, cap_waiting=256, budget_range=(8, 96), min_gap=8)
    return wl, W.kv_limits(wl, seed, block_sizes=(1, 4, 16), tightness=(0.0, 0.4), max_new=50)


def test_a_query_that_could_never_run_keeps_the_live_snapshot():
    wl, limits = _pool(90, 0, 8)
    bs, nb, mc = limits
    rt = make(wl, limits)
    before = read(rt)
    j = int(np.argmin(mc))
    assert mc[j] < (1 << 24)  # an instance with a context limit
    a = np.array([j], np.int32)
    # its prompt reaches the instance's context limit
    rt.advance(dev(a), dev(np.array([int(mc[j])])), dev(np.array([2])), 0.5)
    assert rt.status() == R().LR_EINVAL
    # its whole context needs more blocks than an instance without a context limit has
    # (under a limit the context stops there, and the limits leave room for that)
    u = int(np.argmax(mc))
    assert mc[u] >= (1 << 24)
    big = int(nb[u]) * int(bs[u]) + 1
    rt.advance(dev(np.array([u], np.int32)), dev(np.array([1])), dev(np.array([big])), 0.5)
    assert rt.status() == R().LR_EINVAL
    with pytest.raises(RuntimeError):  # the oracle refuses it too
        oracle.advance(wl, np.zeros(wl.num_instances), [u], [1], [big], 0.5, kv=limits)
    after = read(rt)
    for k in STATE + ("clock",):
        np.testing.assert_array_equal(after[k], before[k], err_msg=k)
    # a valid advance afterwards matches the oracle
    rt.advance(dev(np.zeros(0, np.int32)), dev(np.zeros(0)), dev(np.zeros(0)), 0.5)
    assert rt.status() == R().LR_OK
    w2, c2 = oracle.advance(wl, np.zeros(wl.num_instances), [], [], [], 0.5, kv=limits)
    check_state(read(rt), w2, c2)
    rt.close()
