"""KV-cache block limits, context limits and preemption in the SFS estimate (App. F):
CUDA path vs the CPU oracle, through the C ABI.

Features and first-token batches match exactly and times bit for bit (both sides
take the canonical fp32 sum of the same integer features).  Candidates the oracle
rejects (a prompt at the context limit, a first token that cannot fit) are NaN with
features -1 and the status word reads LR_EINVAL; queries that need more batches than
the recorded horizon are NaN with LR_ETRAJ.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

import oracle  # noqa: E402
from paper_2607_18253_gb300 import workloads as W  # noqa: E402

pytestmark = pytest.mark.gpu


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


def make(wl, limits, horizon=4096, load=True, **kw):
    rt = R().LatencyRouter.from_workload(wl, **kw)
    rt.set_kv_limits(*limits, horizon=horizon)
    if load:
        rt.load_state(*R().state_tensors(wl))
    return rt


def gpu_estimate(rt, wl):
    p = torch.from_numpy(np.ascontiguousarray(wl.prompt_len, np.int32)).cuda()
    fb = torch.empty((wl.num_queries, wl.num_instances), dtype=torch.int32, device="cuda")
    t = rt.estimate_ttft(p, first_batch=fb)
    F = rt.estimate_features(p)
    torch.cuda.synchronize()
    return t.cpu().numpy(), fb.cpu().numpy(), F.cpu().numpy()


def compare(got, want, ok):
    t, fb, F = got
    eF, elt, et = want
    np.testing.assert_array_equal(F[ok], eF[ok])
    np.testing.assert_array_equal(fb[ok], elt[ok])
    np.testing.assert_array_equal(bits(t[ok]), bits(et[ok]))


def check(wl, limits, horizon=4096):
    rt = make(wl, limits, horizon)
    got = gpu_estimate(rt, wl)
    st, eF, elt, et, _ = oracle.estimate_matrix_kv(wl, *limits)
    ok = st == 0
    compare(got, (eF, elt, et), ok)
    t, fb, F = got
    assert np.isnan(t[~ok]).all() and (fb[~ok] == -1).all() and (F[~ok] == -1).all()
    assert rt.status() == (R().LR_OK if ok.all() else R().LR_EINVAL)
    rt.close()
    return st, eF


@pytest.mark.parametrize("mode", [0, 1])
def test_small_pools(mode):
    binding = 0
    for seed in range(8):
        I = (1, 3, 6, 17, 33, 64, 5, 100)[seed]
        wl = W.small_workload(seed, num_instances=I, num_models=3, num_queries=45, first_token_mode=mode,
                              budget_range=(8, 96), min_gap=8)
        limits = W.kv_limits(wl, 100 + seed, block_sizes=(1, 4, 16))
        st, eF = check(wl, limits)
        F0 = oracle.estimate_matrix(wl)[0]
        binding += int((eF != F0).any(axis=-1).sum())
    assert binding > 0


@pytest.mark.parametrize("mode", [0, 1])
def test_tight_blocks_and_context_limits(mode):
    # every instance near its least block count, most with a context limit that
    # decoding runs into: preemptions and limit-ended responses throughout
    for seed in range(4):
        wl = W.small_workload(20 + seed, num_instances=24, num_models=2, num_queries=40, first_token_mode=mode,
                              cap_running=16, cap_waiting=24, budget_range=(16, 128), min_gap=8)
        limits = W.kv_limits(wl, 200 + seed, block_sizes=(1, 2, 8), tightness=(0.0, 0.2), ctx_limited=0.8,
                             ctx_slack=(1, 12))
        check(wl, limits)


@pytest.mark.parametrize("mode", [0, 1])
def test_unbounded_limits_give_the_plain_estimate(mode):
    wl = W.small_workload(31 + mode, num_instances=40, num_models=3, num_queries=64, first_token_mode=mode,
                          budget_range=(8, 96), min_gap=8)
    I = wl.num_instances
    limits = (np.full(I, 16, np.int32), np.full(I, 1 << 40, np.int64), np.full(I, 1 << 40, np.int64))
    rt = make(wl, limits)
    got = gpu_estimate(rt, wl)
    assert rt.status() == R().LR_OK
    rt.close()
    plain = R().LatencyRouter.from_workload(wl)
    plain.load_state(*R().state_tensors(wl))
    ref = gpu_estimate(plain, wl)
    plain.close()
    for a, b in zip(got, ref):
        np.testing.assert_array_equal(np.asarray(a).view(np.uint8), np.asarray(b).view(np.uint8))
    F0, lt0, t0, _ = oracle.estimate_matrix(wl)
    compare(got, (F0, lt0, t0), np.ones(lt0.shape, bool))


def test_invalid_queries_are_nan():
    # an idle instance whose context limit some prompts reach, and one whose blocks
    # cannot hold some prompts' first token
    wl = W.small_workload(61, num_instances=5, num_models=2, num_queries=50, budget_range=(8, 96), min_gap=8)
    bs, nb, mc = W.kv_limits(wl, 7, block_sizes=(4,))
    for j in (0, 1):
        wl.n_run[j] = 0
        wl.n_wait[j] = 0
    med = int(np.median(wl.prompt_len))
    mc[0] = med
    nb[1] = med // 4
    st, _ = check(wl, (bs, nb, mc))
    assert (st[:, 0] != 0).any() and (st[:, 1] != 0).any() and (st[:, 2:] == 0).all()


def test_horizon_exceeded():
    wl = W.small_workload(62, num_instances=12, num_models=2, num_queries=30, budget_range=(8, 48), min_gap=8)
    limits = W.kv_limits(wl, 8, block_sizes=(4,))
    rt = make(wl, limits, horizon=2)
    t, fb, F = gpu_estimate(rt, wl)
    st, eF, elt, et, _ = oracle.estimate_matrix_kv(wl, *limits)
    assert (st == 0).all()
    cut = np.isnan(t)
    assert cut.any() and (~cut).any()
    compare((t, fb, F), (eF, elt, et), ~cut)
    assert (fb[cut] == -1).all() and (F[cut] == -1).all()
    assert rt.status() == R().LR_ETRAJ
    rt.close()


def test_long_walks_across_record_tiles():
    # pool256 under the bench's limits: a candidate whose first token comes more than
    # 84 batches after the earliest one on its instance walked past the 52 staged
    # leading records and through two or more of the warp's 32-record tiles; those
    # candidates match the oracle exactly.  With a horizon of 40 records (below the
    # staged count) a walk past an unfinished instance's records is cut (NaN, LR_ETRAJ)
    # and the others still match.
    wl = W.make_workload("pool256")
    limits = W.kv_limits(wl, 11, block_sizes=(16,))
    rng = np.random.default_rng(9)
    for horizon in (4096, 40):
        rt = make(wl, limits, horizon=horizon)
        t, fb, F = gpu_estimate(rt, wl)
        status = rt.status()
        rt.close()
        cut = np.isnan(t)
        assert (fb[cut] == -1).all() and (F[cut] == -1).all()
        assert status == (R().LR_ETRAJ if cut.any() else R().LR_OK)
        fbm = np.where(cut, np.iinfo(np.int32).max, fb)
        far = np.where(cut, -1, fb - fbm.min(axis=0, keepdims=True))
        # one query per (prompt length, instance): the other queries' rows are copies
        _, first = np.unique(wl.prompt_len, return_index=True)
        sub = far[first]
        qi, cj = np.nonzero(sub > 84)
        if horizon == 4096:
            assert len(qi) > 50
        else:
            qi, cj = np.nonzero(~cut[first])
            assert cut.any() and len(qi) > 0
        pick = rng.choice(len(qi), min(len(qi), 1500), replace=False)
        cq, cj = first[qi[pick]], cj[pick]
        st, eF, elt, et, _ = oracle.estimate_matrix_kv(wl, *limits, cand_q=cq, cand_j=cj)
        assert (st == 0).all()
        np.testing.assert_array_equal(F[cq, cj], eF)
        np.testing.assert_array_equal(fb[cq, cj], elt)
        np.testing.assert_array_equal(bits(t[cq, cj]), bits(et))


def test_invalid_snapshot_keeps_the_live_one():
    wl = W.small_workload(63, num_instances=9, num_models=2, num_queries=20, budget_range=(8, 96), min_gap=8)
    bs, nb, mc = W.kv_limits(wl, 9, block_sizes=(4,))
    j = int(np.argmax(wl.n_run))
    assert wl.n_run[j] > 0 and wl.run_ctx[j, :wl.n_run[j]].sum() > 8
    # before any load: no snapshot
    rt = make(wl, (bs, nb, mc), load=False)
    t, _, _ = gpu_estimate(rt, wl)
    assert np.isnan(t).all() and rt.status() == R().LR_ENOSTATE
    rt.load_state(*R().state_tensors(wl))
    good = gpu_estimate(rt, wl)
    assert rt.status() == R().LR_OK
    # the same snapshot with one request's context past the instance's blocks
    bad = [a.clone() for a in R().state_tensors(wl)]
    bad[1][j, 0] = int(nb[j] * bs[j] + 1)
    rt.load_state(*bad)
    again = gpu_estimate(rt, wl)
    assert rt.status() == R().LR_ESTATE
    for a, b in zip(good, again):
        np.testing.assert_array_equal(np.asarray(a).view(np.uint8), np.asarray(b).view(np.uint8))
    rt.close()


def _route_pool(seed, mode, nq=200):
    wl = W.small_workload(seed, num_instances=24, num_models=3, num_queries=nq, first_token_mode=mode,
                          budget_range=(8, 96), min_gap=8)
    bs, nb, mc = W.kv_limits(wl, seed, block_sizes=(1, 4, 16))
    # an idle instance whose context limit a third of the prompts reach: rows mixing
    # candidates with and without an estimate
    wl.n_run[0] = 0
    wl.n_wait[0] = 0
    mc[0] = int(np.percentile(wl.prompt_len, 66))
    return wl, (bs, nb, mc)


@pytest.mark.parametrize("mode", [0, 1])
def test_route_under_limits(mode):
    # Eq. 5 and Eq. 3 over the KV estimate matrix: assignments exact, utility and
    # chosen time bit for bit against the oracle's argmax over its own KV matrix, a
    # candidate without an estimate never chosen
    wl, limits = _route_pool(70 + mode, mode)
    rt = make(wl, limits, max_pairs=32)
    p, dh, acc, tau = R().query_tensors(wl)
    st, _, _, et, _ = oracle.estimate_matrix_kv(wl, *limits)
    assert (st[:, 0] != 0).any() and (st[:, 0] == 0).any()
    mat = torch.empty((wl.num_queries, wl.num_instances), dtype=torch.float32, device="cuda")
    lam, mu = [float(wl.lam[0])], [float(wl.mu[0])]
    o = rt.route(p, dh, acc, lam, mu, ttft_matrix=mat)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(bits(mat.cpu().numpy()), bits(et))
    a, u, tc = oracle.route(wl, et, lam=np.array(lam, np.float32), mu=np.array(mu, np.float32))
    np.testing.assert_array_equal(o["assign"].cpu().numpy(), a)
    np.testing.assert_array_equal(bits(o["util"].cpu().numpy()), bits(u))
    np.testing.assert_array_equal(bits(o["ttft_chosen"].cpu().numpy()), bits(tc))
    assert (a[0] != 0).all() or np.isfinite(et[a[0] == 0, 0]).all()
    # the constrained objective, without a matrix output (library memory)
    oc = rt.route(p, dh, acc, lam, None, tau=tau)
    torch.cuda.synchronize()
    ac, uc, tcc = oracle.route(wl, et, lam=np.array(lam, np.float32), tau=wl.tau)
    np.testing.assert_array_equal(oc["assign"].cpu().numpy(), ac)
    np.testing.assert_array_equal(bits(oc["util"].cpu().numpy()), bits(uc))
    np.testing.assert_array_equal(bits(oc["ttft_chosen"].cpu().numpy()), bits(tcc))
    # a 32-pair sweep
    lam_s, mu_s = W.sweep_pairs()
    os_ = rt.route(p, dh, acc, lam_s, mu_s)
    torch.cuda.synchronize()
    asw, usw, _ = oracle.route(wl, et, lam=lam_s, mu=mu_s)
    np.testing.assert_array_equal(os_["assign"].cpu().numpy(), asw)
    np.testing.assert_array_equal(bits(os_["util"].cpu().numpy()), bits(usw))
    assert rt.status() == R().LR_EINVAL  # the candidates without an estimate
    rt.close()


def test_route_under_limits_no_eligible_instance():
    # a row whose every candidate lacks an estimate gets -1 and NaN
    wl = W.small_workload(72, num_instances=4, num_models=2, num_queries=30, budget_range=(8, 96), min_gap=8)
    bs, nb, mc = W.kv_limits(wl, 15, block_sizes=(4,))
    wl.n_run[:] = 0
    wl.n_wait[:] = 0
    mc[:] = int(np.median(wl.prompt_len))
    rt = make(wl, (bs, nb, mc))
    p, dh, acc, tau = R().query_tensors(wl)
    o = rt.route(p, dh, acc, [1.0], [0.1])
    torch.cuda.synchronize()
    st, _, _, et, _ = oracle.estimate_matrix_kv(wl, bs, nb, mc)
    a, u, tc = oracle.route(wl, et, lam=np.array([1.0], np.float32), mu=np.array([0.1], np.float32))
    none = (st != 0).all(axis=1)
    assert none.any() and (~none).any()
    np.testing.assert_array_equal(o["assign"].cpu().numpy(), a)
    assert (a[0, none] == -1).all() and np.isnan(u[0, none]).all()
    np.testing.assert_array_equal(bits(o["util"].cpu().numpy()), bits(u))
    np.testing.assert_array_equal(bits(o["ttft_chosen"].cpu().numpy()), bits(tc))
    rt.close()


def test_calls_closed_with_limits_and_turning_them_off():
    wl = W.small_workload(64, num_instances=8, num_models=2, num_queries=16, budget_range=(8, 96), min_gap=8)
    limits = W.kv_limits(wl, 10)
    rt = make(wl, limits)
    p, dh, acc, tau = R().query_tensors(wl)
    with pytest.raises(R().LRError) as e:
        rt.set_ttft_source(R().LR_TTFT_THROUGHPUT)
    assert e.value.code == R().LR_EINVAL
    # the baselines: their choices, with the chosen instance's KV-limited time
    _, _, _, et, _ = oracle.estimate_matrix_kv(wl, *limits)
    for pol in (R().LR_POLICY_ROUND_ROBIN, R().LR_POLICY_SHORTEST_QUEUE, R().LR_POLICY_LATENCY_AGNOSTIC):
        o = rt.route_baseline(pol, p, dh, acc, 1.0, 3)
        torch.cuda.synchronize()
        ea, eu, _ = oracle.baseline_route(wl, pol, 1.0, 3)
        got = o["assign"].cpu().numpy()
        np.testing.assert_array_equal(got, ea)
        np.testing.assert_array_equal(bits(o["util"].cpu().numpy()), bits(eu))
        np.testing.assert_array_equal(bits(o["ttft_chosen"].cpu().numpy()), bits(et[np.arange(len(got)), got]))
    # turning the limits off drops the snapshot; a new load gives the plain estimate
    rt.set_kv_limits()
    t, _, _ = gpu_estimate(rt, wl)
    assert np.isnan(t).all() and rt.status() == R().LR_ENOSTATE
    rt.load_state(*R().state_tensors(wl))
    got = gpu_estimate(rt, wl)
    F0, lt0, t0, _ = oracle.estimate_matrix(wl)
    compare(got, (F0, lt0, t0), np.ones(lt0.shape, bool))
    assert rt.status() == R().LR_OK
    rt.close()


@pytest.mark.parametrize("name", ["pool64", "pool256"])
def test_full_size_sampled(name):
    # the full query set and pool in one call; the oracle checks sampled candidates
    wl = W.make_workload(name)
    limits = W.kv_limits(wl, 11, block_sizes=(16,))
    rt = make(wl, limits)
    t, fb, F = gpu_estimate(rt, wl)
    assert rt.status() == R().LR_OK
    rt.close()
    rng = np.random.default_rng(5)
    n = 4000
    cq = rng.integers(0, wl.num_queries, n)
    cj = rng.integers(0, wl.num_instances, n)
    st, eF, elt, et, _ = oracle.estimate_matrix_kv(wl, *limits, cand_q=cq, cand_j=cj)
    assert (st == 0).all()
    np.testing.assert_array_equal(F[cq, cj], eF)
    np.testing.assert_array_equal(fb[cq, cj], elt)
    np.testing.assert_array_equal(bits(t[cq, cj]), bits(et))
    assert not np.isnan(t).any()


def test_prompt_bound_beyond_exact_buckets():
    # a prompt bound above 2^16 - 2: the sort buckets group several lengths, so
    # every query is estimated (in sorted order) instead of one per length
    wl = W.small_workload(65, num_instances=10, num_models=2, num_queries=60, max_prompt_len=150_000,
                          budget_range=(6000, 8192), min_gap=4096)
    p = wl.prompt_len.copy()
    p[:6] = (1, 1, 150_000, 150_000, 65_535, 65_536)  # duplicates and bucket edges
    wl.prompt_len = p
    limits = W.kv_limits(wl, 12, block_sizes=(16, 64))
    check(wl, limits)


def test_many_duplicate_lengths():
    # 2,000 queries over 40 distinct prompt lengths: most rows are copies of the
    # row of the first query with the same length
    wl = W.small_workload(66, num_instances=12, num_models=2, num_queries=2000, budget_range=(8, 96), min_gap=8)
    rng = np.random.default_rng(0)
    wl.prompt_len = rng.choice(np.arange(1, 161, 4, dtype=np.int32), 2000)
    limits = W.kv_limits(wl, 13, block_sizes=(4,))
    rt = make(wl, limits)
    p = torch.from_numpy(np.ascontiguousarray(wl.prompt_len, np.int32)).cuda()
    t_only = rt.estimate_ttft(p).cpu().numpy()  # times alone, then with first batches
    got = gpu_estimate(rt, wl)
    assert rt.status() == R().LR_OK
    rt.close()
    np.testing.assert_array_equal(bits(t_only), bits(got[0]))
    st, eF, elt, et, _ = oracle.estimate_matrix_kv(wl, *limits)
    compare(got, (eF, elt, et), st == 0)


def test_hand_trace_with_residents_preempting_each_other():
    # the worked trace of tests/golden/kv_hand_trace_residents.json on the GPU: one
    # instance, the query of the trace twice (one walk, a copied row) and a longer one
    import json
    import os
    g = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "kv_hand_trace_residents.json")))
    wl = W.small_workload(90, num_instances=1, num_models=1, num_queries=3, cap_running=8, cap_waiting=8,
                          first_token_mode=g["mode"])
    wl.max_batched_tokens[:] = g["B"]
    wl.max_seqs[:] = g["S"]
    wl.n_run[:] = len(g["running"])
    wl.run_ctx[:] = 0
    wl.run_pre[:] = 0
    wl.run_dec[:] = 0
    for r, (c_, p_, d_) in enumerate(g["running"]):
        wl.run_ctx[0, r], wl.run_pre[0, r], wl.run_dec[0, r] = c_, p_, d_
    wl.n_wait[:] = len(g["waiting"])
    wl.wait_pre[:] = 0
    wl.wait_dec[:] = 0
    for r, (p_, d_) in enumerate(g["waiting"]):
        wl.wait_pre[0, r], wl.wait_dec[0, r] = p_, d_
    wl.prompt_len = np.array([g["query"][0], g["query"][0], 3], np.int32)
    limits = (np.array([g["block_size"]], np.int32), np.array([g["num_blocks"]], np.int64),
              np.array([g["max_ctx"]], np.int64))
    rt = make(wl, limits)
    t, fb, F = gpu_estimate(rt, wl)
    assert rt.status() == R().LR_OK
    rt.close()
    for row in (0, 1):
        assert F[row, 0].tolist() == g["F"] and fb[row, 0] == g["first_token_batch"]
    st, eF, elt, et, _ = oracle.estimate_matrix_kv(wl, *limits)
    assert (st == 0).all()
    compare((t, fb, F), (eF, elt, et), np.ones(st.shape, bool))
