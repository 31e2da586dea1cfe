"""Average-case TTFT sources on the GPU (Sec. 4, App. E) vs the oracle, through the C ABI.

The estimate matrix must equal the oracle's canonical fp32 evaluation bit for bit
(W in fp64 with the same operation order, then fmaf(p, fp32(1/theta), fp32(W + Tdec))),
and routing over it must equal the oracle's brute-force argmax over the same matrix.
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


def queue_params(I, seed):
    rng = np.random.default_rng(seed)
    mu = rng.uniform(2.0, 30.0, I)
    alpha = mu * rng.uniform(0.0, 0.97, I)
    alpha[:3] = [0.0, mu[1] * 0.999, mu[2] * 0.5]
    k = rng.integers(1, 64, I).astype(np.int32)
    k[:2] = [1, 1 << 20]
    ca2 = rng.uniform(0.0, 3.0, I)
    cs2 = rng.uniform(0.0, 3.0, I)
    theta = rng.uniform(3e3, 4e4, I)
    tdec = rng.uniform(0.004, 0.06, I)
    return dict(prefill_tput=theta, decode_batch_time=tdec, arrival_rate=alpha, service_rate=mu,
                parallelism=k, arrival_scv=ca2, service_scv=cs2)


def lps_reference(wl, qp):
    Wj = np.array([oracle.lps_wait(a, m, k, c1, c2) for a, m, k, c1, c2 in
                   zip(qp["arrival_rate"], qp["service_rate"], qp["parallelism"], qp["arrival_scv"],
                       qp["service_scv"])])
    return oracle.avgcase_matrix(wl, Wj, qp["prefill_tput"], qp["decode_batch_time"])


def estimate(rt, wl):
    t = rt.estimate_ttft(R().query_tensors(wl)[0])
    torch.cuda.synchronize()
    return t.cpu().numpy()


@pytest.mark.parametrize("name,nq", [("tiny", None), ("pool64", 3000), ("pool256", 65536)])
def test_lps_matrix_matches_without_a_snapshot(name, nq):
    wl = W.make_workload(name, num_queries=nq)
    rt = R().LatencyRouter.from_workload(wl)  # no snapshot: the LPS source needs none
    qp = queue_params(wl.num_instances, 3)
    rt.set_queue_params(**qp)
    rt.set_ttft_source(R().LR_TTFT_LPS)
    t = estimate(rt, wl)
    assert rt.status() == R().LR_OK
    t32, t64 = lps_reference(wl, qp)
    np.testing.assert_array_equal(bits(t), bits(t32))
    assert np.max(np.abs(t - t64) / t64) < 1e-6


@pytest.mark.parametrize("mode", [0, 1])
def test_throughput_matrix_follows_the_live_snapshot(mode):
    wl = W.make_workload("pool64", num_queries=700, first_token_mode=mode, cap_running=64, cap_waiting=160)
    rt = R().LatencyRouter.from_workload(wl)
    qp = queue_params(wl.num_instances, 4)
    rt.set_queue_params(qp["prefill_tput"], qp["decode_batch_time"])  # no rates: throughput source only
    rt.set_ttft_source(R().LR_TTFT_THROUGHPUT)
    t = estimate(rt, wl)  # before any snapshot
    assert rt.status() == R().LR_ENOSTATE and np.all(np.isnan(t))
    rt.load_state(*R().state_tensors(wl))
    t = estimate(rt, wl)
    assert rt.status() == R().LR_OK
    Wj = oracle.throughput_wait(wl, qp["prefill_tput"])
    t32, _ = oracle.avgcase_matrix(wl, Wj, qp["prefill_tput"], qp["decode_batch_time"])
    np.testing.assert_array_equal(bits(t), bits(t32))
    # after the pool advances, the residents' prefill work is the advanced snapshot's
    rng = np.random.default_rng(9)
    a = rng.integers(-1, wl.num_instances, 100).astype(np.int32)
    d = np.full(100, 50, np.int32)
    dev = lambda x: torch.from_numpy(np.ascontiguousarray(x)).cuda()  # noqa: E731
    rt.advance(dev(a), dev(wl.prompt_len[:100]), dev(d), 0.3)
    t = estimate(rt, wl)
    assert rt.status() == R().LR_OK
    w2, _ = oracle.advance(wl, np.zeros(wl.num_instances), a, wl.prompt_len[:100], d, 0.3)
    t32, _ = oracle.avgcase_matrix(w2, oracle.throughput_wait(w2, qp["prefill_tput"]), qp["prefill_tput"],
                                   qp["decode_batch_time"])
    np.testing.assert_array_equal(bits(t), bits(t32))


def test_routing_over_the_lps_source():
    lam, mu = W.sweep_pairs()
    wl = W.make_workload("pool64", num_queries=1500, lam=lam, mu=mu)
    rt = R().LatencyRouter.from_workload(wl)
    qp = queue_params(wl.num_instances, 5)
    rt.set_queue_params(**qp)
    rt.set_ttft_source(R().LR_TTFT_LPS)
    t32, _ = lps_reference(wl, qp)
    p, dh, acc, tau = R().query_tensors(wl)
    # 32-pair Lagrangian sweep with its frontier
    o = rt.route(p, dh, acc, lam, mu, frontier=True)
    torch.cuda.synchronize()
    assert rt.status() == R().LR_OK
    a, u, tc = oracle.route(wl, t32, lam=lam, mu=mu)
    np.testing.assert_array_equal(o["assign"].cpu().numpy(), a)
    np.testing.assert_array_equal(bits(o["util"].cpu().numpy()), bits(u))
    np.testing.assert_array_equal(bits(o["ttft_chosen"].cpu().numpy()), bits(tc))
    np.testing.assert_allclose(o["frontier"].cpu().numpy(), oracle.frontier(wl, a, tc), rtol=1e-12)
    # constrained objective (Eq. 3) with the App. B.2 targets
    oc = rt.route(p, dh, acc, lam[:1], None, tau=tau)
    torch.cuda.synchronize()
    ac, uc, _ = oracle.route(wl, t32, lam=lam[:1], tau=wl.tau)
    np.testing.assert_array_equal(oc["assign"].cpu().numpy(), ac)
    np.testing.assert_array_equal(bits(oc["util"].cpu().numpy()), bits(uc))


def test_switching_sources_and_errors():
    wl = W.make_workload("tiny")
    rt = R().LatencyRouter.from_workload(wl)
    rt.load_state(*R().state_tensors(wl))
    sfs = estimate(rt, wl)
    with pytest.raises(R().LRError) as e:  # no parameters yet
        rt.set_ttft_source(R().LR_TTFT_LPS)
    assert e.value.code == R().LR_EINVAL
    qp = queue_params(wl.num_instances, 6)
    bad = dict(qp, arrival_rate=qp["service_rate"] * 1.0)  # alpha == mu: unstable
    with pytest.raises(R().LRError) as e:
        rt.set_queue_params(**bad)
    assert e.value.code == R().LR_EINVAL
    with pytest.raises(R().LRError):
        rt.set_queue_params(**dict(qp, parallelism=np.zeros(wl.num_instances, np.int32)))
    with pytest.raises(R().LRError):
        rt.set_queue_params(**dict(qp, prefill_tput=np.zeros(wl.num_instances)))
    rt.set_queue_params(qp["prefill_tput"], qp["decode_batch_time"])
    with pytest.raises(R().LRError):  # rates were not given
        rt.set_ttft_source(R().LR_TTFT_LPS)
    rt.set_queue_params(**qp)
    rt.set_ttft_source(R().LR_TTFT_LPS)
    p = R().query_tensors(wl)[0]
    fb = torch.empty((wl.num_queries, wl.num_instances), dtype=torch.int32, device="cuda")
    with pytest.raises(R().LRError) as e:  # the first-token batch is an SFS quantity
        rt.estimate_ttft(p, first_batch=fb)
    assert e.value.code == R().LR_EINVAL
    with pytest.raises(R().LRError):
        rt.set_ttft_source(7)
    rt.set_ttft_source(R().LR_TTFT_SFS)
    np.testing.assert_array_equal(bits(estimate(rt, wl)), bits(sfs))
