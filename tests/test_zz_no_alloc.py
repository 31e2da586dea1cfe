"""The allocation-free route + frontier entry point against lr_route.

lr_route_frontier_static runs the same kernels as lr_route with a frontier,
keeping the chosen-TTFT intermediate in the library's static device memory;
its outputs must equal lr_route's (assignments and utilities bit for bit, the
fp64 frontier within 1e-12 relative) on every call, including back-to-back
calls that reuse the static array, with and without KV-cache limits; and the
device's free memory must not change across the calls (nothing is allocated).
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from paper_2607_18253_gb300 import workloads as W  # noqa: E402

pytestmark = pytest.mark.gpu

FRONTIER_RTOL = 1e-12


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


def check_same(o, ref):
    np.testing.assert_array_equal(o["assign"].cpu().numpy(), ref["assign"].cpu().numpy())
    np.testing.assert_array_equal(bits(o["util"].cpu().numpy()), bits(ref["util"].cpu().numpy()))
    np.testing.assert_allclose(o["frontier"].cpu().numpy(), ref["frontier"].cpu().numpy(), rtol=FRONTIER_RTOL)


@pytest.mark.parametrize("mode", [0, 1])
def test_static_route_matches_lr_route(mode):
    lam, mu = W.sweep_pairs()
    wl = W.make_workload("pool64", num_queries=2000, lam=lam, mu=mu, first_token_mode=mode)
    rt = make_router(wl)
    p, dh, acc, tau = R().query_tensors(wl)
    ref = rt.route(p, dh, acc, lam, mu, ttft_chosen=False, frontier=True)
    P, Q = len(lam), wl.num_queries
    out = {"assign": torch.empty((P, Q), dtype=torch.int32, device="cuda"),
           "util": torch.empty((P, Q), dtype=torch.float32, device="cuda"),
           "frontier": torch.empty((P, 3), dtype=torch.float64, device="cuda")}
    torch.cuda.synchronize()
    free0 = torch.cuda.mem_get_info()[0]
    for _ in range(2):  # two calls in a row reuse the static array
        o = rt.route_frontier_static(p, dh, acc, lam, mu, out=out)
        torch.cuda.synchronize()
        assert rt.status() == R().LR_OK
        check_same(o, ref)
    assert torch.cuda.mem_get_info()[0] == free0
    # constrained objective (Eq. 3, one lambda) with the per-query targets
    refc = rt.route(p, dh, acc, lam[:1], None, tau=tau, ttft_chosen=False, frontier=True)
    for _ in range(2):
        oc = rt.route_frontier_static(p, dh, acc, lam[:1], None, tau=tau)
        torch.cuda.synchronize()
        assert rt.status() == R().LR_OK
        check_same(oc, refc)


def test_static_route_capacity_is_checked_before_launch():
    wl = W.make_workload("tiny")
    rt = make_router(wl, max_queries=4097, max_pairs=64)
    Q, M = 4097, wl.num_models
    p = torch.full((Q,), 100, dtype=torch.int32, device="cuda")
    dh = torch.full((Q, M), 10, dtype=torch.int32, device="cuda")
    acc = torch.full((Q, M), 0.5, dtype=torch.float32, device="cuda")
    lam = np.ones(64, np.float32)
    with pytest.raises(R().LRError) as e:  # 64 * 4097 > 2^18 entries
        rt.route_frontier_static(p, dh, acc, lam, lam)
    assert e.value.code == R().LR_ECAPACITY
    # at the limit it runs and matches lr_route
    o = rt.route_frontier_static(p[:4096], dh[:4096], acc[:4096], lam, lam)
    ref = rt.route(p[:4096], dh[:4096], acc[:4096], lam, lam, ttft_chosen=False, frontier=True)
    torch.cuda.synchronize()
    assert rt.status() == R().LR_OK
    check_same(o, ref)


def test_static_route_under_kv_limits():
    # with KV-cache limits the route scores the KV-limited estimate matrix, which the
    # library keeps in memory taken by lr_set_kv_limits: still nothing allocated per call
    wl = W.make_workload("tiny")
    rt = make_router(wl, max_pairs=32)
    rt.set_kv_limits(*W.kv_limits(wl, 1, block_sizes=(16,)), horizon=1024)
    rt.load_state(*R().state_tensors(wl))
    p, dh, acc, _ = R().query_tensors(wl)
    lam, mu = W.sweep_pairs()
    ref = rt.route(p, dh, acc, lam, mu, ttft_chosen=False, frontier=True)
    P, Q = len(lam), wl.num_queries
    out = {"assign": torch.empty((P, Q), dtype=torch.int32, device="cuda"),
           "util": torch.empty((P, Q), dtype=torch.float32, device="cuda"),
           "frontier": torch.empty((P, 3), dtype=torch.float64, device="cuda")}
    torch.cuda.synchronize()
    assert rt.status() == R().LR_OK
    free0 = torch.cuda.mem_get_info()[0]
    for _ in range(2):
        o = rt.route_frontier_static(p, dh, acc, lam, mu, out=out)
        torch.cuda.synchronize()
        assert rt.status() == R().LR_OK
        check_same(o, ref)
    assert torch.cuda.mem_get_info()[0] == free0
    rt.close()
