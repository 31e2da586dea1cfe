"""Baseline routing policies (Sec. 6) and OnTimeUtility / SLO attainment (Eq. 4):
CUDA path vs the CPU oracle, through the C ABI.

Assignments match exactly; utility and TTFT of the chosen instance bit for bit
(the same fp32 operations); the SLO count exactly; OnTimeUtility within 1e-12 of
the mean |U| (fp64 sums in another fixed order).
"""
import dataclasses

import numpy as np
import pytest

torch = pytest.importorskip("torch")

import oracle  # noqa: E402
from paper_2607_18253_gb300 import workloads as W  # noqa: E402

pytestmark = pytest.mark.gpu

POLICIES = (0, 1, 2)


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


def run_policy(rt, wl, policy, lam, rr_start=0):
    p, dh, acc, _ = R().query_tensors(wl)
    o = rt.route_baseline(policy, p, dh, acc, lam, rr_start)
    torch.cuda.synchronize()
    return o["assign"].cpu().numpy(), o["util"].cpu().numpy(), o["ttft_chosen"].cpu().numpy()


def check(wl, rt, policy, lam, rr_start=0):
    a, u, t = run_policy(rt, wl, policy, lam, rr_start)
    ea, eu, et = oracle.baseline_route(wl, policy, lam, rr_start)
    np.testing.assert_array_equal(a, ea)
    np.testing.assert_array_equal(bits(u), bits(eu))
    np.testing.assert_array_equal(bits(t), bits(et))
    assert rt.status() == R().LR_OK


@pytest.mark.parametrize("mode", [0, 1])
@pytest.mark.parametrize("policy", POLICIES)
def test_small_pools(policy, mode):
    for seed in range(8):
        I = (1, 3, 6, 17, 33, 64, 5, 100)[seed]
        wl = W.small_workload(seed, num_instances=I, num_models=3, num_queries=45, first_token_mode=mode,
                              budget_range=(8, 96), min_gap=8)
        rt = make_router(wl)
        check(wl, rt, policy, float(wl.lam[0]), rr_start=seed * 7)
        rt.close()


def test_shortest_queue_many_levels():
    # many more queries than instances: the water level rises through several counts
    wl = W.small_workload(21, num_instances=6, num_models=2, num_queries=500, budget_range=(8, 96), min_gap=8)
    rt = make_router(wl)
    check(wl, rt, 1, 0.25)
    rt.close()


def test_three_hundred_instances():
    wl = W.small_workload(101, num_instances=300, num_models=5, num_queries=37, budget_range=(16, 128), min_gap=16)
    rt = make_router(wl)
    for policy in POLICIES:
        check(wl, rt, policy, 0.1, rr_start=299)
    rt.close()


def test_pool256_sampled():
    # the benchmark pool, 4096 of its queries
    wl = W.make_workload("pool256", num_queries=4096)
    rt = make_router(wl)
    for policy in POLICIES:
        check(wl, rt, policy, float(wl.lam[0]), rr_start=5)
    rt.close()


def test_invalid_prompts_and_no_snapshot():
    wl = W.small_workload(2, num_instances=5, num_models=2, num_queries=12)
    pl = wl.prompt_len.copy()
    pl[3], pl[7] = 0, wl.max_prompt_len + 1
    wl2 = dataclasses.replace(wl, prompt_len=pl)
    rt = make_router(wl2)
    a, u, t = run_policy(rt, wl2, 0, 0.5)
    assert a[3] == -1 and a[7] == -1 and np.isnan(u[[3, 7]]).all() and np.isnan(t[[3, 7]]).all()
    assert rt.status() == R().LR_EINVAL
    ok = np.ones(12, bool)
    ok[[3, 7]] = False
    ea, eu, et = oracle.baseline_route(wl2, 0, 0.5)
    np.testing.assert_array_equal(a, ea)
    np.testing.assert_array_equal(bits(u[ok]), bits(eu[ok]))
    rt.close()
    rt = R().LatencyRouter.from_workload(wl)  # no snapshot loaded
    a, u, t = run_policy(rt, wl, 1, 0.5)
    assert (a == -1).all() and np.isnan(u).all()
    assert rt.status() == R().LR_ENOSTATE
    rt.close()


def test_host_side_errors():
    wl = W.small_workload(2, num_instances=5, num_models=2, num_queries=12)
    rt = make_router(wl)
    p, dh, acc, _ = R().query_tensors(wl)
    for kw in ({"policy": 3}, {"policy": -1}, {"policy": 0, "rr_start": -1}, {"policy": 0, "lam": float("nan")}):
        with pytest.raises(R().LRError) as e:
            rt.route_baseline(kw.get("policy"), p, dh, acc, kw.get("lam", 0.5), kw.get("rr_start", 0))
        assert e.value.code == R().LR_EINVAL
    rt.close()


@pytest.mark.parametrize("Q", [1, 7, 3000, 250000])
def test_on_time_utility(Q):
    rng = np.random.default_rng(Q)
    util = rng.normal(0.3, 0.4, Q).astype(np.float32)
    ttft = rng.exponential(1.0, Q).astype(np.float32)
    ttft[rng.random(Q) < 0.05] = np.nan
    tau = rng.exponential(1.2, Q).astype(np.float32)
    delay = rng.exponential(0.1, Q).astype(np.float32)
    wl = W.small_workload(0, num_instances=3, num_models=2, num_queries=Q)
    rt = R().LatencyRouter.from_workload(wl)
    dev = torch.device("cuda")
    tt = [torch.from_numpy(x).to(dev) for x in (util, ttft, tau, delay)]
    for d in (None, tt[3]):
        got = rt.on_time_utility(tt[0], tt[1], tt[2], d).cpu().numpy()
        again = rt.on_time_utility(tt[0], tt[1], tt[2], d).cpu().numpy()
        otu, slo = oracle.on_time_utility(util, ttft, tau, None if d is None else delay)
        assert got[1] == slo
        assert abs(got[0] - otu) <= 1e-12 * max(float(np.mean(np.abs(util))), 1e-30)
        np.testing.assert_array_equal(got.view(np.uint64), again.view(np.uint64))
    rt.close()
