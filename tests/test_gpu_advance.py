"""Online stream step on the GPU (append routed queries, advance to t_now) vs the oracle.

Every state array and every fp64 clock must match the oracle exactly: both
sides execute the same scheduler steps and add the same fp32 batch times
(Eq. 9 per batch) into an fp64 clock in the same order.  The estimates made
from an advanced snapshot must then match the oracle's estimates on the
oracle's advanced state, bit for bit as for a loaded snapshot.
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


def make_router(wl, **kw):
    rt = R().LatencyRouter.from_workload(wl, **kw)
    rt.load_state(*R().state_tensors(wl))
    return rt


def dev(a, dtype=torch.int32):
    return torch.from_numpy(np.ascontiguousarray(a)).to("cuda", dtype)


def read(rt):
    st = rt.read_state()
    torch.cuda.synchronize()
    return {k: v.cpu().numpy() for k, v in st.items()}


def check_state(st, wl, clk):
    np.testing.assert_array_equal(st["n_run"], wl.n_run)
    np.testing.assert_array_equal(st["n_wait"], wl.n_wait)
    np.testing.assert_array_equal(st["clock"].view(np.uint64), np.asarray(clk, np.float64).view(np.uint64))
    for j in range(wl.num_instances):
        nr, nw = int(wl.n_run[j]), int(wl.n_wait[j])
        for k in ("run_ctx", "run_pre", "run_dec"):
            np.testing.assert_array_equal(st[k][j, :nr], getattr(wl, k)[j, :nr], err_msg=f"{k} row {j}")
        for k in ("wait_pre", "wait_dec"):
            np.testing.assert_array_equal(st[k][j, :nw], getattr(wl, k)[j, :nw], err_msg=f"{k} row {j}")


def check_estimates(rt, wl):
    p = dev(wl.prompt_len)
    t = rt.estimate_ttft(p)
    F = rt.estimate_features(p)
    torch.cuda.synchronize()
    assert rt.status() == R().LR_OK
    Q, I = wl.num_queries, wl.num_instances
    qq, jj = np.meshgrid(np.arange(Q), np.arange(I), indexing="ij")
    Fo, _, t32, _ = oracle.estimate_candidates(wl, qq.ravel(), jj.ravel())
    np.testing.assert_array_equal(F.cpu().numpy().reshape(-1, 5), Fo)
    np.testing.assert_array_equal(bits(t.cpu().numpy().ravel()), bits(t32))


@pytest.mark.parametrize("mode", [0, 1])
def test_advance_small_pools(mode):
    # random small pools (seat caps that bind, a prefill at the running tail,
    # instance counts off the warp and CTA sizes), three successive advances,
    # the last one long enough to drain every instance
    for seed in range(12):
        rng = np.random.default_rng(1000 + seed)
        wl = W.small_workload(seed, num_instances=int(3 + seed % 37), num_models=3, num_queries=48,
                              cap_running=64, cap_waiting=160, first_token_mode=mode, wait_max=24,
                              budget_range=(8, 64), min_gap=8)
        rt = make_router(wl)
        clk = np.zeros(wl.num_instances)
        for step, t_now in enumerate((6.0, 25.0, 1e7)):
            Q = 48
            a = rng.integers(-1, wl.num_instances, Q).astype(np.int32)
            p = rng.integers(1, 160, Q).astype(np.int32)
            d = rng.integers(1, 30, Q).astype(np.int32)
            rt.advance(dev(a), dev(p), dev(d), t_now)
            torch.cuda.synchronize()
            assert rt.status() == R().LR_OK, (seed, step)
            wl, clk = oracle.advance(wl, clk, a, p, d, t_now)
            check_state(read(rt), wl, clk)
            if step < 2:
                check_estimates(rt, wl)
        assert np.all(wl.n_run == 0) and np.all(wl.n_wait == 0) and np.all(clk == 1e7)


@pytest.mark.parametrize("mode", [0, 1])
def test_route_advance_loop_pool64(mode):
    # the online loop of Sec. 5: route a micro-batch on the live snapshot, append it
    # to the chosen instances, advance the pool; assignments and states stay identical
    per, steps = 128, 5
    full = W.make_workload("pool64", num_queries=per * steps, first_token_mode=mode, cap_waiting=64 + per * steps)
    rt = make_router(full, max_queries=per)
    wl, clk = full, np.zeros(full.num_instances)
    lam, mu = full.lam[:1], full.mu[:1]
    for s in range(steps):
        sl = slice(s * per, (s + 1) * per)
        q = dataclasses.replace(wl, prompt_len=full.prompt_len[sl], dec_hat=full.dec_hat[sl], acc=full.acc[sl],
                                tau=full.tau[sl])
        out = rt.route(dev(q.prompt_len), dev(q.dec_hat), dev(q.acc, torch.float32), lam, mu)
        torch.cuda.synchronize()
        assert rt.status() == R().LR_OK
        _, _, t32, _ = oracle.estimate_matrix(q)
        a, u, _ = oracle.route(q, t32, lam=lam, mu=mu)
        np.testing.assert_array_equal(out["assign"].cpu().numpy(), a)
        np.testing.assert_array_equal(bits(out["util"].cpu().numpy()), bits(u))
        a0 = a[0]
        d = q.dec_hat[np.arange(per), q.model_of_instance[a0]]  # the chosen model's predicted length
        t_now = 0.02 * (s + 1)
        # the advance reads that column itself from the [Q, M] matrix on even steps
        rt.advance(dev(a0), dev(q.prompt_len), dev(q.dec_hat if s % 2 == 0 else d), t_now)
        torch.cuda.synchronize()
        assert rt.status() == R().LR_OK
        wl, clk = oracle.advance(q, clk, a0, q.prompt_len, d, t_now)
        check_state(read(rt), wl, clk)


def test_waiting_overflow_keeps_previous_snapshot():
    wl = W.make_workload("tiny", cap_running=64)
    rt = make_router(wl)
    before = read(rt)
    Q = wl.cap_waiting + 1
    a = np.zeros(Q, np.int32)
    rt.advance(dev(a), dev(np.full(Q, 8)), dev(np.full(Q, 2)), 0.5)
    assert rt.status() == R().LR_ECAPACITY
    after = read(rt)
    for k in STATE + ("clock",):
        np.testing.assert_array_equal(after[k], before[k], err_msg=k)
    # an out-of-range length is flagged the same way
    rt.advance(dev(np.array([1], np.int32)), dev(np.array([0])), dev(np.array([3])), 0.5)
    assert rt.status() == R().LR_EINVAL
    np.testing.assert_array_equal(read(rt)["n_wait"], before["n_wait"])
    # and a valid advance afterwards still matches the oracle
    rt.advance(dev(np.zeros(0, np.int32)), dev(np.zeros(0)), dev(np.zeros(0)), 0.5)
    assert rt.status() == R().LR_OK
    w2, c2 = oracle.advance(wl, np.zeros(wl.num_instances), [], [], [], 0.5)
    check_state(read(rt), w2, c2)


def test_clock_never_runs_backwards_and_idle_jump():
    wl = W.make_workload("tiny", cap_running=64)
    wl.n_run[::2] = 0
    wl.n_wait[::2] = 0
    rt = make_router(wl)
    z = dev(np.zeros(0, np.int32))
    rt.advance(z, z, z, 0.25)
    w1, c1 = oracle.advance(wl, np.zeros(wl.num_instances), [], [], [], 0.25)
    check_state(read(rt), w1, c1)
    assert np.all(c1[::2] == 0.25)
    rt.advance(z, z, z, 0.1)
    assert rt.status() == R().LR_OK
    w2, c2 = oracle.advance(w1, c1, [], [], [], 0.1)
    st = read(rt)
    check_state(st, w2, c2)
    np.testing.assert_array_equal(st["clock"], c1)


def test_advance_host_side_errors():
    wl = W.make_workload("tiny")  # cap_running 32 < max_seqs 64: the advance cannot hold a full batch
    rt = make_router(wl)
    z = dev(np.zeros(0, np.int32))
    with pytest.raises(R().LRError) as e:
        rt.advance(z, z, z, 1.0)
    assert e.value.code == R().LR_ECAPACITY
    wl2 = W.make_workload("tiny", cap_running=64)
    rt2 = make_router(wl2)
    with pytest.raises(R().LRError) as e:
        rt2.advance(z, z, z, float("nan"))
    assert e.value.code == R().LR_EINVAL
    one = dev(np.zeros(1, np.int32))
    with pytest.raises(R().LRError) as e:  # dec must have 1 or num_models columns
        rt2.advance(one, dev(np.ones(1)), dev(np.ones((1, wl2.num_models + 1))), 1.0)
    assert e.value.code == R().LR_EINVAL
    rt3 = R().LatencyRouter.from_workload(wl2)
    rt3.advance(z, z, z, 1.0)
    assert rt3.status() == R().LR_ENOSTATE


def test_advance_beyond_max_iters_keeps_previous_snapshot():
    wl = W.make_workload("tiny", cap_running=64)
    wl.n_wait[:] = 0  # the load needs few steps; draining the decoders needs thousands
    rt = make_router(wl, max_iters=200)
    torch.cuda.synchronize()
    assert rt.status() == R().LR_OK
    before = read(rt)
    z = dev(np.zeros(0, np.int32))
    rt.advance(z, z, z, 1e9)
    assert rt.status() == R().LR_ETRAJ
    after = read(rt)
    for k in STATE + ("clock",):
        np.testing.assert_array_equal(after[k], before[k], err_msg=k)
    # a short advance within the limit still matches the oracle
    rt.advance(z, z, z, 0.05)
    assert rt.status() == R().LR_OK
    w2, c2 = oracle.advance(wl, np.zeros(wl.num_instances), [], [], [], 0.05)
    check_state(read(rt), w2, c2)


@pytest.mark.parametrize("mode", [0, 1])
def test_first_token_times_match_the_oracle(mode):
    # random small pools, four successive advances with tracked appends (one of them
    # untracked), the last one draining everything: every first-token time equal to the
    # oracle's, bit for bit, and the same queries without one until then
    for seed in range(8):
        rng = np.random.default_rng(2000 + seed)
        wl = W.small_workload(seed, num_instances=int(3 + seed % 29), num_models=3, num_queries=48,
                              cap_running=64, cap_waiting=200, first_token_mode=mode, wait_max=24,
                              budget_range=(8, 64), min_gap=8)
        rt = make_router(wl)
        N = 4 * 40
        ftt = torch.full((N,), float("nan"), dtype=torch.float64, device="cuda")
        rt.track_first_tokens(ftt)
        tr = oracle.new_track(wl, N)
        clk = np.zeros(wl.num_instances)
        for step, t_now in enumerate((4.0, 9.0, 15.0, 1e7)):
            Q = 40
            a = rng.integers(-1, wl.num_instances, Q).astype(np.int32)
            p = rng.integers(1, 160, Q).astype(np.int32)
            d = rng.integers(1, 30, Q).astype(np.int32)
            base = None if step == 2 else 40 * step
            rt.advance(dev(a), dev(p), dev(d), t_now, id_base=base)
            torch.cuda.synchronize()
            assert rt.status() == R().LR_OK, (seed, step)
            wl, clk, tr = oracle.advance(wl, clk, a, p, d, t_now, track=tr, id_base=-1 if base is None else base)
            check_state(read(rt), wl, clk)
            got, exp = ftt.cpu().numpy(), tr["first_token_time"]
            np.testing.assert_array_equal(np.isnan(got), np.isnan(exp), err_msg=f"seed {seed} step {step}")
            np.testing.assert_array_equal(got[~np.isnan(exp)].view(np.uint64), exp[~np.isnan(exp)].view(np.uint64))
        # everything drained; the untracked step's ids were never given out
        assert np.isnan(got[80:120]).all()
        assert np.isfinite(got[:80]).sum() > 0
        rt.close()


def test_tracking_errors_and_reload():
    wl = W.make_workload("tiny", cap_running=64)
    rt = make_router(wl)
    a = dev(np.zeros(4, np.int32))
    p = dev(np.full(4, 10, np.int32))
    d = dev(np.full(4, 3, np.int32))
    with pytest.raises(R().LRError) as e:  # ids without tracking
        rt.advance(a, p, d, 1.0, id_base=0)
    assert e.value.code == R().LR_EINVAL
    ftt = torch.full((6,), float("nan"), dtype=torch.float64, device="cuda")
    rt.track_first_tokens(ftt)
    with pytest.raises(R().LRError) as e:  # ids 3 .. 6 beyond the capacity of 6
        rt.advance(a, p, d, 1.0, id_base=3)
    assert e.value.code == R().LR_ECAPACITY
    rt.advance(a, p, d, 1.0, id_base=2)
    # a reload makes every request untracked: draining it records nothing more
    rt.load_state(*R().state_tensors(wl))
    before = ftt.cpu().numpy().copy()
    rt.advance(a[:0], p[:0], d[:0], 1e7)
    torch.cuda.synchronize()
    assert rt.status() == R().LR_OK
    after = ftt.cpu().numpy()
    np.testing.assert_array_equal(np.isnan(after), np.isnan(before))
    rt.track_first_tokens(None)
    rt.close()
