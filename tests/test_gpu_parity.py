"""CUDA path vs the CPU oracle, through the C ABI.

Tolerances: the integer batch features F, the first-token batch index and
the assignments must match exactly; fp32 TTFT and utility must equal the
oracle's canonical fp32 evaluation bit for bit (both sides evaluate the same
fixed sequence of IEEE operations), which in turn is within 1e-5 relative of
the oracle's fp64 value.
"""
import dataclasses

import numpy as np
import pytest

torch = pytest.importorskip("torch")

import oracle  # noqa: E402
from paper_2607_18253_gb300 import workloads as W  # noqa: E402

pytestmark = pytest.mark.gpu

REL_TOL = 1e-5


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def R():
    from paper_2607_18253_gb300 import router
    return router


def make_router(wl, **kw):
    rt = R().LatencyRouter.from_workload(wl, **kw)
    rt.load_state(*R().state_tensors(wl))
    return rt


def bits(a):
    return np.ascontiguousarray(a, np.float32).view(np.uint32)


def check_candidates(wl, F_gpu, t_gpu, lt_gpu, cq, cj):
    F, lt, t32, t64 = oracle.estimate_candidates(wl, cq, cj)
    np.testing.assert_array_equal(F_gpu, F)
    np.testing.assert_array_equal(lt_gpu, lt)
    np.testing.assert_array_equal(bits(t_gpu), bits(t32))
    rel = np.abs(t_gpu.astype(np.float64) - t64) / t64
    assert rel.max() <= REL_TOL, rel.max()


def full_estimate(rt, wl):
    p, _, _, _ = R().query_tensors(wl)
    fb = torch.empty((wl.num_queries, wl.num_instances), dtype=torch.int32, device="cuda")
    t = rt.estimate_ttft(p, first_batch=fb)
    F = rt.estimate_features(p)
    torch.cuda.synchronize()
    assert rt.status() == R().LR_OK
    return F.cpu().numpy(), t.cpu().numpy(), fb.cpu().numpy()


@pytest.mark.parametrize("mode", [0, 1])
@pytest.mark.parametrize("name,nq", [("tiny", None), ("pool64", 600)])
def test_every_candidate_matches(name, nq, mode):
    wl = W.make_workload(name, num_queries=nq, first_token_mode=mode)
    rt = make_router(wl)
    F, t, fb = full_estimate(rt, wl)
    Q, I = wl.num_queries, wl.num_instances
    qq, jj = np.meshgrid(np.arange(Q), np.arange(I), indexing="ij")
    check_candidates(wl, F.reshape(-1, 5), t.ravel(), fb.ravel(), qq.ravel(), jj.ravel())


@pytest.mark.parametrize("mode", [0, 1])
def test_random_small_pools(mode):
    # many small random pools: seat caps that bind, tiny budgets, a running request in
    # mid-prefill at the tail, one-token responses, instance counts off the warp size
    for seed in range(24):
        wl = W.small_workload(seed, num_instances=int(3 + seed % 37), num_models=3, num_queries=41,
                              first_token_mode=mode, budget_range=(8, 96), min_gap=8)
        rt = make_router(wl)
        F, t, fb = full_estimate(rt, wl)
        Q, I = wl.num_queries, wl.num_instances
        qq, jj = np.meshgrid(np.arange(Q), np.arange(I), indexing="ij")
        check_candidates(wl, F.reshape(-1, 5), t.ravel(), fb.ravel(), qq.ravel(), jj.ravel())
        rt.close()


@pytest.mark.parametrize("mode", [0, 1])
def test_seat_limited_pools(mode):
    # long queues behind nearly full seat caps: most admissions refill the seats freed
    # in the batch before, which the trajectory kernel takes many end batches at a
    # time; prompts close to the budget, short responses and queues that run out in
    # the middle of such a run cut it short
    for seed in range(8):
        wl = W.small_workload(seed, num_instances=32, num_models=3, num_queries=29, cap_running=64,
                              cap_waiting=128, first_token_mode=mode, budget_range=(300, 1200), min_gap=8)
        rt = make_router(wl)
        F, t, fb = full_estimate(rt, wl)
        Q, I = wl.num_queries, wl.num_instances
        qq, jj = np.meshgrid(np.arange(Q), np.arange(I), indexing="ij")
        check_candidates(wl, F.reshape(-1, 5), t.ravel(), fb.ravel(), qq.ravel(), jj.ravel())
        rt.close()


def test_instance_tiles_beyond_one_cta():
    # 300 instances: the estimate kernel splits instances over several CTAs
    wl = W.small_workload(101, num_instances=300, num_models=5, num_queries=37, budget_range=(16, 128), min_gap=16)
    rt = make_router(wl)
    F, t, fb = full_estimate(rt, wl)
    qq, jj = np.meshgrid(np.arange(37), np.arange(300), indexing="ij")
    check_candidates(wl, F.reshape(-1, 5), t.ravel(), fb.ravel(), qq.ravel(), jj.ravel())


@pytest.mark.parametrize("mode", [0, 1])
def test_window_list_overflow(mode):
    # 450 running decoders that all end within the first table rows' batches: more
    # window decoders than the trajectory kernel's compacted list holds
    wl = W.small_workload(11, num_instances=5, num_models=2, num_queries=31, cap_running=512, cap_waiting=32,
                          first_token_mode=mode, budget_range=(2048, 4096), min_gap=1024)
    rng = np.random.default_rng(5)
    I = wl.num_instances
    n_run = np.full(I, 450, np.int32)
    run_ctx = np.zeros((I, 512), np.int32)
    run_dec = np.zeros((I, 512), np.int32)
    run_ctx[:, :450] = rng.integers(1, 400, (I, 450))
    run_dec[:, :450] = rng.integers(1, 12, (I, 450))
    S = np.maximum(wl.max_seqs, 480).astype(np.int32)
    wl = dataclasses.replace(wl, n_run=n_run, run_ctx=run_ctx, run_pre=np.zeros((I, 512), np.int32),
                             run_dec=run_dec, max_seqs=np.minimum(S, wl.max_batched_tokens).astype(np.int32))
    rt = make_router(wl)
    F, t, fb = full_estimate(rt, wl)
    qq, jj = np.meshgrid(np.arange(wl.num_queries), np.arange(I), indexing="ij")
    check_candidates(wl, F.reshape(-1, 5), t.ravel(), fb.ravel(), qq.ravel(), jj.ravel())
    rt.close()


def test_two_instance_tiles():
    # 1100 instances: two instance tiles, whose CTAs claim every query row dynamically
    wl = W.small_workload(7, num_instances=1100, num_models=4, num_queries=53, budget_range=(64, 160), min_gap=64)
    rt = make_router(wl)
    F, t, fb = full_estimate(rt, wl)
    qq, jj = np.meshgrid(np.arange(53), np.arange(1100), indexing="ij")
    check_candidates(wl, F.reshape(-1, 5), t.ravel(), fb.ravel(), qq.ravel(), jj.ravel())
    # a second call starts from counters the first one cleared
    F2, t2, fb2 = full_estimate(rt, wl)
    np.testing.assert_array_equal(bits(t2), bits(t))
    rt.close()


@pytest.mark.parametrize("name,ns", [("pool64", 40000), ("pool256", 60000)])
def test_full_size_sampled(name, ns):
    # full query count, the launch shape the benchmark times; sampled candidates
    wl = W.make_workload(name)
    rt = make_router(wl)
    F, t, fb = full_estimate(rt, wl)
    rng = np.random.default_rng(7)
    cq = rng.integers(0, wl.num_queries, ns)
    cj = rng.integers(0, wl.num_instances, ns)
    # include the first and last rows/columns (ragged edges of the tiles)
    cq[:4] = [0, 0, wl.num_queries - 1, wl.num_queries - 1]
    cj[:4] = [0, wl.num_instances - 1, 0, wl.num_instances - 1]
    check_candidates(wl, F[cq, cj], t[cq, cj], fb[cq, cj], cq, cj)
    # properties at every candidate: positive finite times, first-token batch = F0,
    # and a longer prompt never reaches its first token earlier
    assert np.all(np.isfinite(t)) and np.all(t > 0)
    assert np.all(fb == F[..., 0])
    order = np.argsort(wl.prompt_len, kind="stable")
    assert np.all(np.diff(F[order, :, 0], axis=0) >= 0)
    assert np.all(np.diff(t[order].astype(np.float64), axis=0) >= 0)


def _route_case(wl, rt, P_lam, P_mu, tau=None, ttft_matrix=False):
    p, dh, acc, tau_d = R().query_tensors(wl)
    mat = torch.empty((wl.num_queries, wl.num_instances), dtype=torch.float32, device="cuda") if ttft_matrix else None
    out = rt.route(p, dh, acc, P_lam, None if tau is not None else P_mu, tau=tau_d if tau is not None else None,
                   frontier=True, ttft_matrix=mat)
    torch.cuda.synchronize()
    assert rt.status() == R().LR_OK
    return {k: v.cpu().numpy() for k, v in out.items()}


@pytest.mark.parametrize("mode", [0, 1])
@pytest.mark.parametrize("name,nq", [("tiny", None), ("pool64", 700)])
def test_route_lagrangian_and_constrained(name, nq, mode):
    wl = W.make_workload(name, num_queries=nq, first_token_mode=mode)
    rt = make_router(wl)
    _, _, t32, _ = oracle.estimate_matrix(wl)
    lam, mu = wl.lam, wl.mu
    o = _route_case(wl, rt, lam, mu, ttft_matrix=True)
    np.testing.assert_array_equal(bits(o["ttft_matrix"]), bits(t32))
    a, u, tc = oracle.route(wl, t32, lam=lam, mu=mu)
    np.testing.assert_array_equal(o["assign"], a)
    np.testing.assert_array_equal(bits(o["util"]), bits(u))
    np.testing.assert_array_equal(bits(o["ttft_chosen"]), bits(tc))
    fr = oracle.frontier(wl, a, tc)
    np.testing.assert_allclose(o["frontier"], fr, rtol=1e-12)
    # constrained objective with the App. B.2 targets
    oc = _route_case(wl, rt, lam, None, tau=wl.tau)
    ac, uc, tcc = oracle.route(wl, t32, lam=lam, tau=wl.tau)
    np.testing.assert_array_equal(oc["assign"], ac)
    np.testing.assert_array_equal(bits(oc["util"]), bits(uc))
    np.testing.assert_array_equal(bits(oc["ttft_chosen"]), bits(tcc))


def test_route_sweep_32_pairs():
    lam, mu = W.sweep_pairs()
    wl = W.make_workload("pool64", num_queries=512, lam=lam, mu=mu)
    rt = make_router(wl)
    _, _, t32, _ = oracle.estimate_matrix(wl)
    o = _route_case(wl, rt, lam, mu)
    a, u, tc = oracle.route(wl, t32, lam=lam, mu=mu)
    np.testing.assert_array_equal(o["assign"], a)
    np.testing.assert_array_equal(bits(o["util"]), bits(u))
    np.testing.assert_allclose(o["frontier"], oracle.frontier(wl, a, tc), rtol=1e-12)
    # more latency weight never raises the mean chosen TTFT for a fixed lambda
    tmean = o["frontier"][:, 2].reshape(4, 8)
    assert np.all(np.diff(tmean, axis=1) <= 1e-6 * tmean[:, 1:])


def test_route_full_size_against_gpu_matrix():
    # pool256 at full size: the oracle's brute-force argmax over the GPU's own TTFT rows
    wl = W.make_workload("pool256")
    rt = make_router(wl)
    o = _route_case(wl, rt, wl.lam, wl.mu, ttft_matrix=True)
    a, u, tc = oracle.route(wl, o["ttft_matrix"], lam=wl.lam, mu=wl.mu)
    np.testing.assert_array_equal(o["assign"], a)
    np.testing.assert_array_equal(bits(o["util"]), bits(u))
    rng = np.random.default_rng(3)
    cq = rng.integers(0, wl.num_queries, 20000)
    cj = rng.integers(0, wl.num_instances, 20000)
    _, _, t32, _ = oracle.estimate_candidates(wl, cq, cj)
    np.testing.assert_array_equal(bits(o["ttft_matrix"][cq, cj]), bits(t32))


def test_route_on_a_second_stream_full_size():
    # the bench's step configuration: pool256 routed on a stream other than the
    # load's, so that its rows are claimed dynamically, first alone and then beside a
    # concurrent reload of the same snapshot; 256 sampled queries against the
    # oracle's route over their full oracle rows
    wl = W.make_workload("pool256")
    rt = make_router(wl)
    state = R().state_tensors(wl)
    p, dh, acc, _ = R().query_tensors(wl)
    main = torch.cuda.current_stream()
    side = torch.cuda.Stream()
    results = []
    for reload in (False, True):
        side.wait_stream(main)
        if reload:
            rt.load_state(*state)  # on the main stream, while the side stream routes
        with torch.cuda.stream(side):
            o = rt.route(p, dh, acc, wl.lam, wl.mu, stream=side)
        torch.cuda.synchronize()
        assert rt.status() == R().LR_OK
        results.append({k: o[k].cpu().numpy() for k in ("assign", "util", "ttft_chosen")})
    for k in ("assign", "util", "ttft_chosen"):
        np.testing.assert_array_equal(results[0][k].view(np.uint32), results[1][k].view(np.uint32))
    qs = np.sort(np.random.default_rng(11).choice(wl.num_queries, 256, replace=False))
    sub = wl.with_queries(qs)
    _, _, t32, _ = oracle.estimate_matrix(sub)
    ea, eu, et = oracle.route(sub, t32, lam=wl.lam, mu=wl.mu)
    np.testing.assert_array_equal(results[0]["assign"][0][qs], ea[0])
    np.testing.assert_array_equal(bits(results[0]["util"][0][qs]), bits(eu[0]))
    np.testing.assert_array_equal(bits(results[0]["ttft_chosen"][0][qs]), bits(et[0]))


def test_edge_prompts_and_ragged_rows():
    wl = W.make_workload("pool64", num_queries=1001)
    wl.prompt_len[:6] = [1, 2, wl.max_prompt_len, wl.max_prompt_len - 1, 4095, 4097]
    rt = make_router(wl)
    F, t, fb = full_estimate(rt, wl)
    qq, jj = np.meshgrid(np.arange(1001), np.arange(64), indexing="ij")
    check_candidates(wl, F.reshape(-1, 5), t.ravel(), fb.ravel(), qq.ravel(), jj.ravel())


def test_empty_instances_and_zero_queries():
    wl = W.make_workload("tiny")
    wl.n_run[:] = 0
    wl.n_wait[:] = 0
    rt = make_router(wl)
    F, t, fb = full_estimate(rt, wl)
    p = wl.prompt_len.astype(np.int64)
    B = wl.max_batched_tokens[0]
    exp0 = -(-p // B) + 1
    assert np.all(F[..., 0] == exp0[:, None])
    assert np.all(F[..., 4] == (p * (p + 1) // 2)[:, None])
    z = torch.empty(0, dtype=torch.int32, device="cuda")
    assert rt.estimate_ttft(z).numel() == 0


def test_invalid_prompt_is_flagged():
    wl = W.make_workload("tiny")
    rt = make_router(wl)
    p, _, _, _ = R().query_tensors(wl)
    p[3] = 0
    p[5] = wl.max_prompt_len + 1
    t = rt.estimate_ttft(p).cpu().numpy()
    assert rt.status() == R().LR_EINVAL
    assert np.all(np.isnan(t[[3, 5]]))
    assert np.all(np.isfinite(np.delete(t, [3, 5], axis=0)))
    assert rt.status() == R().LR_OK  # cleared


def test_no_snapshot_yet():
    wl = W.make_workload("tiny")
    rt = R().LatencyRouter.from_workload(wl)
    p, _, _, _ = R().query_tensors(wl)
    t = rt.estimate_ttft(p).cpu().numpy()
    assert rt.status() == R().LR_ENOSTATE
    assert np.all(np.isnan(t))


def test_invalid_snapshot_keeps_previous():
    wl = W.make_workload("tiny")
    rt = make_router(wl)
    p, _, _, _ = R().query_tensors(wl)
    before = rt.estimate_ttft(p).cpu().numpy()
    assert rt.status() == R().LR_OK
    bad = R().state_tensors(wl)
    j = int(np.flatnonzero(wl.n_run >= 2)[0])
    bad[2].view(wl.num_instances, wl.cap_running)[j, 0] = 5  # prefill ahead of a decoder
    rt.load_state(*bad)
    assert rt.status() == R().LR_ESTATE
    after = rt.estimate_ttft(p).cpu().numpy()
    np.testing.assert_array_equal(bits(after), bits(before))
    # a snapshot that exceeds max_iters also leaves the previous one live
    rt2 = R().LatencyRouter.from_workload(wl, max_iters=2)
    rt2.load_state(*R().state_tensors(wl))
    assert rt2.status() == R().LR_ETRAJ


def test_host_side_errors():
    wl = W.make_workload("tiny")
    rt = make_router(wl, max_queries=16, max_pairs=2)
    p = torch.ones(17, dtype=torch.int32, device="cuda")
    with pytest.raises(R().LRError) as e:
        rt.estimate_ttft(p)
    assert e.value.code == R().LR_ECAPACITY
    p16, dh, acc, _ = R().query_tensors(wl)
    with pytest.raises(R().LRError) as e:
        rt.route(p16, dh, acc, [1.0, 1.0, 1.0], [0.1, 0.1, 0.1])
    assert e.value.code == R().LR_ECAPACITY
    with pytest.raises(R().LRError) as e:
        rt.route(p16, dh, acc, [-1.0], [0.1])
    assert e.value.code == R().LR_EINVAL
    with pytest.raises(R().LRError) as e:  # the constrained objective takes one lambda
        rt.route(p16, dh, acc, [1.0, 2.0], None, tau=torch.ones(16, dtype=torch.float32, device="cuda"))
    assert e.value.code == R().LR_EINVAL
    with pytest.raises(R().LRError):
        R().LatencyRouter(model_of_instance=[0], coef=np.ones((1, 5)), price_in=[0], price_out=[0],
                          max_batched_tokens=[8], max_seqs=[9], cap_running=4, cap_waiting=4, max_queries=4,
                          max_prompt_len=16)


def test_load_overlapping_estimates_sees_whole_snapshots():
    # A snapshot load on one stream overlapping estimates on another: every query row
    # must be exactly the oracle's row under the previous or under the new snapshot.
    old = W.make_workload("pool64", num_queries=2048)
    new = W.make_workload("pool64", num_queries=2048, seed=7)
    rt = make_router(old)
    p = R().query_tensors(old)[0]
    _, _, t_old, _ = oracle.estimate_matrix(old)
    _, _, t_new, _ = oracle.estimate_matrix(dataclasses.replace(new, prompt_len=old.prompt_len))
    s_load, s_est = torch.cuda.Stream(), torch.cuda.Stream()
    new_state = R().state_tensors(new)
    outs = [torch.empty((2048, 64), dtype=torch.float32, device="cuda") for _ in range(6)]
    torch.cuda.synchronize()
    with torch.cuda.stream(s_est):
        for o in outs[:3]:
            rt.estimate_ttft(p, out=o, stream=s_est)
    rt.load_state(*new_state, stream=s_load)
    with torch.cuda.stream(s_est):
        for o in outs[3:]:
            rt.estimate_ttft(p, out=o, stream=s_est)
    torch.cuda.synchronize()
    assert rt.status() == R().LR_OK
    b_old, b_new = bits(t_old), bits(t_new)
    for o in outs:
        got = bits(o.cpu().numpy())
        is_old = np.all(got == b_old, axis=1)
        is_new = np.all(got == b_new, axis=1)
        assert np.all(is_old | is_new)
    # after both streams finished, the new snapshot is live everywhere
    np.testing.assert_array_equal(bits(rt.estimate_ttft(p).cpu().numpy()), b_new)
