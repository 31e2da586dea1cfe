"""Full-size parity: every candidate of the large configurations against the oracle.

* pool256 (256 instances x 65,536 queries): the whole TTFT matrix, its integer
  features and first-token batches, then the Lagrangian and constrained routes
  over the oracle's whole matrix.
* The trade-off sweep on the 64-instance pool: 4,096 queries x 32 (lambda, mu)
  pairs, every assignment, utility and chosen TTFT, and the frontier.
* The online stream: the seeded Poisson trace at 0.8 x pool capacity, routed in
  micro-batches of 1, 16 and 256 queries for 2,000 decisions each; after every
  decision the advanced snapshot (every state array and fp64 clock) and the
  batch's assignments, utilities and chosen TTFTs.

A candidate's estimate depends on its prompt length and its instance only: the
new query's predicted output, accuracy and target do not enter the simulation up
to its first token (Eq. 7-9).  The oracle therefore simulates one query per
distinct prompt length (7,604 of pool256's 65,536) on every instance, on all
host cores; the GPU rows of the other queries must equal their leader's row bit
for bit, which is checked directly, and a random sample of non-leader
candidates also goes through the oracle itself.

Tolerances as in test_gpu_parity: integers and assignments exact, fp32 times and
utilities bit-exact against the oracle's canonical fp32 evaluation, which is
within 1e-5 relative of its fp64 value.
"""
import dataclasses

import numpy as np
import pytest

torch = pytest.importorskip("torch")

import oracle  # noqa: E402
from paper_2607_18253_gb300 import workloads as W  # noqa: E402

pytestmark = pytest.mark.gpu

REL_TOL = 1e-5
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


def oracle_by_length(wl):
    """The oracle on the first query of each distinct prompt length, every instance.

    Returns (leaders, inverse, F, first-token batch, fp32, fp64): row inverse[i] of
    the oracle arrays is query i's."""
    _, first, inv = np.unique(wl.prompt_len, return_index=True, return_inverse=True)
    F, lt, t32, t64 = oracle.estimate_matrix(wl.with_queries(first))
    return first, inv.ravel(), F, lt, t32, t64


@pytest.mark.parametrize("mode", [0, 1])
def test_pool256_every_candidate(mode):
    wl = W.make_workload("pool256", first_token_mode=mode)
    Q, I = wl.num_queries, wl.num_instances
    rt = make_router(wl)
    p, dh, acc, tau = R().query_tensors(wl)
    fb_d = torch.empty((Q, I), dtype=torch.int32, device="cuda")
    t = rt.estimate_ttft(p, first_batch=fb_d).cpu().numpy()
    fb = fb_d.cpu().numpy()
    del fb_d
    F = rt.estimate_features(p).cpu().numpy()
    torch.cuda.synchronize()
    assert rt.status() == R().LR_OK

    first, inv, Fo, lto, t32o, t64o = oracle_by_length(wl)
    # the leaders against the oracle
    np.testing.assert_array_equal(F[first], Fo)
    np.testing.assert_array_equal(fb[first], lto)
    np.testing.assert_array_equal(bits(t[first]), bits(t32o))
    assert (np.abs(t[first].astype(np.float64) - t64o) / t64o).max() <= REL_TOL
    # every other query equals its leader, so every candidate equals the oracle's value
    lead = first[inv]
    np.testing.assert_array_equal(bits(t), bits(t[lead]))
    np.testing.assert_array_equal(fb, fb[lead])
    for f in range(5):
        np.testing.assert_array_equal(F[..., f], F[lead, :, f])
    del F
    # and a sample of non-leader candidates straight through the oracle
    rng = np.random.default_rng(29)
    cq = rng.integers(0, Q, 4000)
    cj = rng.integers(0, I, 4000)
    _, lt_s, t32_s, _ = oracle.estimate_candidates(wl, cq, cj)
    np.testing.assert_array_equal(fb[cq, cj], lt_s)
    np.testing.assert_array_equal(bits(t[cq, cj]), bits(t32_s))

    # routing over the oracle's whole matrix: Lagrangian (Eq. 5) and constrained (Eq. 3)
    t32 = t32o[inv]
    mat = torch.empty((Q, I), dtype=torch.float32, device="cuda")
    o = rt.route(p, dh, acc, wl.lam, wl.mu, ttft_matrix=mat)
    torch.cuda.synchronize()
    assert rt.status() == R().LR_OK
    np.testing.assert_array_equal(bits(mat.cpu().numpy()), bits(t32))
    a, u, tc = oracle.route(wl, t32, lam=wl.lam, mu=wl.mu)
    np.testing.assert_array_equal(o["assign"].cpu().numpy(), a)
    np.testing.assert_array_equal(bits(o["util"].cpu().numpy()), bits(u))
    np.testing.assert_array_equal(bits(o["ttft_chosen"].cpu().numpy()), bits(tc))
    oc = rt.route(p, dh, acc, wl.lam, None, tau=tau)
    torch.cuda.synchronize()
    assert rt.status() == R().LR_OK
    ac, uc, tcc = oracle.route(wl, t32, lam=wl.lam, tau=wl.tau)
    np.testing.assert_array_equal(oc["assign"].cpu().numpy(), ac)
    np.testing.assert_array_equal(bits(oc["util"].cpu().numpy()), bits(uc))
    np.testing.assert_array_equal(bits(oc["ttft_chosen"].cpu().numpy()), bits(tcc))
    rt.close()


def test_sweep_32_pairs_full_size():
    # 4,096 queries x 32 pairs on the 64-instance pool: 32 assignment vectors and the frontier
    lam, mu = W.sweep_pairs()
    wl = W.make_workload("pool64", lam=lam, mu=mu)
    Q, I = wl.num_queries, wl.num_instances
    rt = make_router(wl)
    first, inv, _, _, t32o, _ = oracle_by_length(wl)
    t32 = t32o[inv]
    p, dh, acc, _ = R().query_tensors(wl)
    mat = torch.empty((Q, I), dtype=torch.float32, device="cuda")
    o = rt.route(p, dh, acc, lam, mu, frontier=True, ttft_matrix=mat)
    torch.cuda.synchronize()
    assert rt.status() == R().LR_OK
    np.testing.assert_array_equal(bits(mat.cpu().numpy()), bits(t32))
    a, u, tc = oracle.route(wl, t32, lam=lam, mu=mu)
    np.testing.assert_array_equal(o["assign"].cpu().numpy(), a)
    np.testing.assert_array_equal(bits(o["util"].cpu().numpy()), bits(u))
    np.testing.assert_array_equal(bits(o["ttft_chosen"].cpu().numpy()), bits(tc))
    np.testing.assert_allclose(o["frontier"].cpu().numpy(), oracle.frontier(wl, a, tc), rtol=1e-12)
    # the static-memory variant gives the same frontier
    fs = rt.route_frontier_static(p, dh, acc, lam, mu)
    torch.cuda.synchronize()
    assert rt.status() == R().LR_OK
    np.testing.assert_array_equal(fs["assign"].cpu().numpy(), a)
    np.testing.assert_array_equal(fs["frontier"].cpu().numpy().view(np.uint64),
                                  o["frontier"].cpu().numpy().view(np.uint64))
    rt.close()


# ---------------------------------------------------------------------------
# The online stream (Sec. 5, App. F)

STREAM_QUERIES = 1_000_000
STREAM_SEED = 3
STREAM_DECISIONS = 2000


@pytest.fixture(scope="module")
def stream_trace():
    wl = W.make_workload("pool64", num_queries=STREAM_QUERIES, seed=STREAM_SEED, cap_waiting=512)
    rate = 0.8 * float(oracle.pool_capacity(wl).sum())
    return wl, W.poisson_arrivals(STREAM_QUERIES, rate, STREAM_SEED)


@pytest.mark.parametrize("m", [1, 16, 256])
def test_stream_micro_batches(stream_trace, m):
    # at each decision time (the arrival of the batch's last query) the previous batch
    # joins its instances' queues and the pool advances (K3 + K1), then the batch is
    # routed on the new snapshot (K2, Lagrangian), as the stream benchmark runs it; the
    # GPU keeps every snapshot and result, the oracle then replays the trace on its own
    wl, arr = stream_trace
    nb, I, M = STREAM_DECISIONS, wl.num_instances, wl.num_models
    n = nb * m
    rt = make_router(wl, max_queries=m)
    lib, h = rt._lib, rt._h
    p, dh, acc, _ = R().query_tensors(wl.with_queries(np.arange(n)))
    snaps = {"n_run": torch.empty((nb, I), dtype=torch.int32, device="cuda"),
             "run_ctx": torch.empty((nb, I, wl.cap_running), dtype=torch.int32, device="cuda"),
             "run_pre": torch.empty((nb, I, wl.cap_running), dtype=torch.int32, device="cuda"),
             "run_dec": torch.empty((nb, I, wl.cap_running), dtype=torch.int32, device="cuda"),
             "n_wait": torch.empty((nb, I), dtype=torch.int32, device="cuda"),
             "wait_pre": torch.empty((nb, I, wl.cap_waiting), dtype=torch.int32, device="cuda"),
             "wait_dec": torch.empty((nb, I, wl.cap_waiting), dtype=torch.int32, device="cuda"),
             "clock": torch.empty((nb, I), dtype=torch.float64, device="cuda")}
    assign = torch.empty((nb, m), dtype=torch.int32, device="cuda")
    util = torch.empty((nb, m), dtype=torch.float32, device="cuda")
    tch = torch.empty((nb, m), dtype=torch.float32, device="cuda")
    # every routed query is tracked to its first output token (its id = its trace index)
    ftt = torch.full((n,), float("nan"), dtype=torch.float64, device="cuda")
    rt.track_first_tokens(ftt)
    import ctypes
    V = ctypes.c_void_p
    sp = V(torch.cuda.current_stream().cuda_stream)
    for b in range(nb):
        lo = b * m
        t_now = float(arr[lo + m - 1])
        if b == 0:
            rt.advance(assign[0, :0], p[:0], dh[:0], t_now)
        else:
            rt.advance(assign[b - 1], p[lo - m:lo], dh[lo - m:lo], t_now, id_base=lo - m)
        rc = lib.lr_read_state(h, *(V(snaps[k][b].data_ptr()) for k in STATE + ("clock",)), sp)
        assert rc == 0
        rt.route(p[lo:lo + m], dh[lo:lo + m], acc[lo:lo + m], wl.lam, wl.mu,
                 out={"assign": assign[b:b + 1], "util": util[b:b + 1], "ttft_chosen": tch[b:b + 1]})
    torch.cuda.synchronize()
    assert rt.status() == R().LR_OK
    snaps = {k: v.cpu().numpy() for k, v in snaps.items()}
    assign, util, tch = assign.cpu().numpy(), util.cpu().numpy(), tch.cpu().numpy()
    ftt = ftt.cpu().numpy()
    rt.close()

    st, clk = wl, np.zeros(I)
    tr = oracle.new_track(wl, n)
    none = np.zeros(0, np.int32)
    prev = None
    for b in range(nb):
        lo = b * m
        t_now = float(arr[lo + m - 1])
        if prev is None:
            st, clk, tr = oracle.advance(st, clk, none, none, none, t_now, track=tr)
        else:
            pa, pq = prev
            d = np.ascontiguousarray(pq.dec_hat[np.arange(m), wl.model_of_instance[np.maximum(pa, 0)]])
            st, clk, tr = oracle.advance(st, clk, pa, pq.prompt_len, d, t_now, track=tr, id_base=lo - m)
        np.testing.assert_array_equal(snaps["n_run"][b], st.n_run, err_msg=f"decision {b}")
        np.testing.assert_array_equal(snaps["n_wait"][b], st.n_wait, err_msg=f"decision {b}")
        np.testing.assert_array_equal(snaps["clock"][b].view(np.uint64), clk.view(np.uint64),
                                      err_msg=f"decision {b}")
        for k in ("run_ctx", "run_pre", "run_dec"):
            mask = np.arange(wl.cap_running)[None, :] < st.n_run[:, None]
            np.testing.assert_array_equal(snaps[k][b][mask], getattr(st, k)[mask], err_msg=f"{k} decision {b}")
        for k in ("wait_pre", "wait_dec"):
            mask = np.arange(wl.cap_waiting)[None, :] < st.n_wait[:, None]
            np.testing.assert_array_equal(snaps[k][b][mask], getattr(st, k)[mask], err_msg=f"{k} decision {b}")
        sl = slice(lo, lo + m)
        q = dataclasses.replace(st, prompt_len=wl.prompt_len[sl], dec_hat=wl.dec_hat[sl], acc=wl.acc[sl],
                                tau=wl.tau[sl])
        _, _, t32, _ = oracle.estimate_matrix(q)
        a, u, tc = oracle.route(q, t32, lam=wl.lam, mu=wl.mu)
        np.testing.assert_array_equal(assign[b], a[0], err_msg=f"decision {b}")
        np.testing.assert_array_equal(bits(util[b]), bits(u[0]), err_msg=f"decision {b}")
        np.testing.assert_array_equal(bits(tch[b]), bits(tc[0]), err_msg=f"decision {b}")
        prev = (a[0], q)
    # the trace kept the pool busy: work arrived and queues formed somewhere
    assert st.n_run.sum() > 0
    # the realized first-token times (Eq. 4's realized TTFT): the same queries have one, at
    # the same fp64 times
    ot = tr["first_token_time"]
    np.testing.assert_array_equal(np.isnan(ftt), np.isnan(ot))
    np.testing.assert_array_equal(ftt[~np.isnan(ot)].view(np.uint64), ot[~np.isnan(ot)].view(np.uint64))
    assert (~np.isnan(ot)).sum() > n // 2
