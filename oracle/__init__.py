"""CPU oracle for the latency-aware router -- test infrastructure only.

A ctypes front end to ``sfs_oracle.c``: the literal per-candidate serving
simulation of Sec. 4.1 (Eq. 7-9) and brute-force routing (Eq. 2, 3, 5).

Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this package.  The product path (the CUDA library and
its binding) never does.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from typing import Optional

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "sfs_oracle.c")
_LIBDIR = os.path.join(_HERE, "_lib")
_LIB = os.path.join(_LIBDIR, "libsfs_oracle.so")
_lib = None

FIRST_TOKEN_SEPARATE_DECODE = 0
FIRST_TOKEN_WITH_LAST_CHUNK = 1
DEFAULT_MAX_BATCHES = 1 << 40


def host_threads() -> int:
    """Host threads the candidate loops use by default: every core this process may run on."""
    try:
        return max(1, len(os.sched_getaffinity(0)))
    except (AttributeError, OSError):
        return max(1, os.cpu_count() or 1)


def _in_slices(C: int, threads: Optional[int], call) -> None:
    """Run call(lo, hi) over [0, C) split into contiguous slices, one per thread.

    Every candidate is independent (its own copy of its instance's state), and the
    C loop holds no shared state, so slices may run concurrently; ctypes releases
    the interpreter lock for the duration of each foreign call.  The result does
    not depend on the thread count."""
    n = host_threads() if threads is None else max(1, int(threads))
    n = min(n, max(1, C // 64))
    if n <= 1:
        call(0, C)
        return
    from concurrent.futures import ThreadPoolExecutor
    bounds = [C * k // n for k in range(n + 1)]
    with ThreadPoolExecutor(max_workers=n) as ex:
        for f in [ex.submit(call, bounds[k], bounds[k + 1]) for k in range(n)]:
            f.result()


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (no fp contraction, no fast-math)."""
    os.makedirs(_LIBDIR, exist_ok=True)
    hdr = os.path.join(_HERE, "sfs_oracle.h")
    if (not force and os.path.exists(_LIB)
            and os.path.getmtime(_LIB) >= max(os.path.getmtime(_SRC), os.path.getmtime(hdr))):
        return _LIB
    tmp = _LIB + f".tmp{os.getpid()}"
    cmd = ["gcc", "-std=c11", "-O2", "-ffp-contract=off", "-fno-fast-math", "-fPIC", "-shared",
           "-o", tmp, _SRC, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    if _lib is None:
        build()
        lib = ctypes.CDLL(_LIB)
        P = ctypes.c_void_p
        i32, i64 = ctypes.c_int32, ctypes.c_int64
        lib.orc_sfs_candidate.argtypes = [P, i32, i32, i32, i32, i32, i64, P, P, P]
        lib.orc_sfs_candidate.restype = ctypes.c_int
        lib.orc_ttft_f32.argtypes = [P, P]
        lib.orc_ttft_f32.restype = ctypes.c_float
        lib.orc_ttft_f64.argtypes = [P, P]
        lib.orc_ttft_f64.restype = ctypes.c_double
        lib.orc_estimate_candidates.argtypes = [i32, P, P, P, P, i32, i32, P, P, P, P, P, P, P, i32, P, P,
                                                i32, i64, i64, P, P, P, P, P, P]
        lib.orc_estimate_candidates.restype = ctypes.c_int
        lib.orc_route.argtypes = [i32, i32, i32, P, P, P, P, P, P, P, P, i32, P, P, P, P, P]
        lib.orc_route.restype = ctypes.c_int
        lib.orc_frontier.argtypes = [i32, i32, i32, P, P, P, P, P, P, i32, P, P, P]
        lib.orc_frontier.restype = ctypes.c_int
        lib.orc_advance.argtypes = [i32, P, P, P, P, i32, i32, P, P, P, P, P, P, P, P, i32, P, P, P, i32,
                                    ctypes.c_double, i64]
        lib.orc_advance.restype = ctypes.c_int
        lib.orc_advance_ids.argtypes = [i32, P, P, P, P, i32, i32, P, P, P, P, P, P, P, P, i32, P, P, P, i32,
                                        ctypes.c_double, i64, P, P, i64, P]
        lib.orc_advance_ids.restype = ctypes.c_int
        lib.orc_advance_kv.argtypes = [i32, P, P, P, P, i32, i32, P, P, P, P, P, P, P, P, i32, P, P, P, i32,
                                       ctypes.c_double, i64, P, P, P, P, P, i64, P]
        lib.orc_advance_kv.restype = ctypes.c_int
        lib.orc_utility.argtypes = [ctypes.c_float, ctypes.c_float, i32, i32, ctypes.c_float, ctypes.c_float]
        lib.orc_utility.restype = ctypes.c_float
        lib.orc_pow_int.argtypes = [ctypes.c_double, i32]
        lib.orc_pow_int.restype = ctypes.c_double
        lib.orc_lps_wait.argtypes = [ctypes.c_double, ctypes.c_double, i32, ctypes.c_double, ctypes.c_double]
        lib.orc_lps_wait.restype = ctypes.c_double
        lib.orc_throughput_wait.argtypes = [P, ctypes.c_double]
        lib.orc_throughput_wait.restype = ctypes.c_double
        lib.orc_avgcase_ttft.argtypes = [i32, i32, P, P, P, P, P, P]
        lib.orc_avgcase_ttft.restype = ctypes.c_int
        lib.orc_round_robin.argtypes = [i32, i32, i64, P]
        lib.orc_round_robin.restype = ctypes.c_int
        lib.orc_shortest_queue.argtypes = [i32, i32, P, P]
        lib.orc_shortest_queue.restype = ctypes.c_int
        lib.orc_latency_agnostic.argtypes = [i32, i32, i32, P, P, P, P, P, P, ctypes.c_float, P]
        lib.orc_latency_agnostic.restype = ctypes.c_int
        lib.orc_on_time_utility.argtypes = [i32, P, P, P, P, P]
        lib.orc_on_time_utility.restype = ctypes.c_int
        lib.orc_sfs_candidate_kv.argtypes = [P, i32, i32, i32, P, i32, i32, i64, P, P, P, P, P]
        lib.orc_sfs_candidate_kv.restype = ctypes.c_int
        lib.orc_kv_residents.argtypes = [P, i32, i32, i32, P, i64, P]
        lib.orc_kv_residents.restype = ctypes.c_int
        lib.orc_estimate_candidates_kv.argtypes = [i32, P, P, P, P, i32, i32, P, P, P, P, P, P, P, P, P, P, P,
                                                   i32, i64, i64, P, P, P, P, P, P, P]
        lib.orc_estimate_candidates_kv.restype = ctypes.c_int
        _lib = lib
    return _lib


def _p(a: Optional[np.ndarray]):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _c(a, dtype):
    return np.ascontiguousarray(a, dtype=dtype)


class _Instance(ctypes.Structure):
    _fields_ = [("n_run", ctypes.c_int32), ("run_ctx", ctypes.c_void_p), ("run_pre", ctypes.c_void_p),
                ("run_dec", ctypes.c_void_p), ("n_wait", ctypes.c_int32), ("wait_pre", ctypes.c_void_p),
                ("wait_dec", ctypes.c_void_p)]


def simulate(running, waiting, B: int, S: int, p: int, d: int = 1, mode: int = FIRST_TOKEN_SEPARATE_DECODE,
             max_batches: int = DEFAULT_MAX_BATCHES):
    """One candidate.  running: list of (ctx, pre, dec); waiting: list of (pre, dec).

    Returns (F[5] int64, admit batch, first-token batch)."""
    run = np.asarray(running, dtype=np.int32).reshape(-1, 3)
    wt = np.asarray(waiting, dtype=np.int32).reshape(-1, 2)
    rc_, rp_, rd_ = (_c(run[:, k], np.int32) for k in range(3))
    wp_, wd_ = (_c(wt[:, k], np.int32) for k in range(2))
    inst = _Instance(run.shape[0], _p(rc_), _p(rp_), _p(rd_), wt.shape[0], _p(wp_), _p(wd_))
    F = np.zeros(5, np.int64)
    la = ctypes.c_int64(0)
    lt = ctypes.c_int64(0)
    rc = _load().orc_sfs_candidate(ctypes.byref(inst), B, S, mode, p, d, max_batches, _p(F),
                                   ctypes.byref(la), ctypes.byref(lt))
    if rc != 0:
        raise RuntimeError(f"oracle simulation failed with code {rc}")
    return F, int(la.value), int(lt.value)


def ttft_f32(coef, F) -> np.float32:
    c = _c(coef, np.float32)
    f = _c(F, np.int64)
    return np.float32(_load().orc_ttft_f32(_p(c), _p(f)))


def ttft_f64(coef, F) -> float:
    c = _c(coef, np.float32)
    f = _c(F, np.int64)
    return float(_load().orc_ttft_f64(_p(c), _p(f)))


def utility(acc, lam, p, dec_hat, price_in, price_out) -> np.float32:
    return np.float32(_load().orc_utility(float(np.float32(acc)), float(np.float32(lam)), int(p), int(dec_hat),
                                          float(np.float32(price_in)), float(np.float32(price_out))))


def estimate_candidates(wl, cand_q, cand_j, max_batches: int = DEFAULT_MAX_BATCHES,
                        threads: Optional[int] = None):
    """F[C,5], first-token batch [C], canonical fp32 TTFT [C], fp64 TTFT [C].

    The candidates are split over `threads` host threads (default: every core)."""
    cq = _c(cand_q, np.int32)
    cj = _c(cand_j, np.int32)
    C = cq.shape[0]
    F = np.zeros((C, 5), np.int64)
    lt = np.zeros(C, np.int64)
    t32 = np.zeros(C, np.float32)
    t64 = np.zeros(C, np.float64)
    arrs = [_c(a, np.int32) for a in (wl.model_of_instance, wl.max_batched_tokens, wl.max_seqs, wl.n_run,
                                      wl.run_ctx, wl.run_pre, wl.run_dec, wl.n_wait, wl.wait_pre,
                                      wl.wait_dec, wl.prompt_len, wl.dec_hat)]
    coef = _c(wl.coef, np.float32)
    moi, B, S, n_run, run_ctx, run_pre, run_dec, n_wait, wait_pre, wait_dec, p, dh = arrs
    lib = _load()
    codes = []

    def run(lo, hi):
        rc = lib.orc_estimate_candidates(
            wl.num_instances, _p(moi), _p(coef), _p(B), _p(S), wl.cap_running, wl.cap_waiting, _p(n_run),
            _p(run_ctx), _p(run_pre), _p(run_dec), _p(n_wait), _p(wait_pre), _p(wait_dec), wl.num_models, _p(p),
            _p(dh), wl.first_token_mode, max_batches, hi - lo, _p(cq[lo:]), _p(cj[lo:]), _p(F[lo:]), _p(lt[lo:]),
            _p(t32[lo:]), _p(t64[lo:]))
        codes.append(rc)

    _in_slices(C, threads, run)
    rc = next((r for r in codes if r != 0), 0)
    if rc != 0:
        raise RuntimeError(f"oracle estimate failed with code {rc}")
    return F, lt, t32, t64


def estimate_matrix(wl, max_batches: int = DEFAULT_MAX_BATCHES, threads: Optional[int] = None):
    """Every candidate: F[Q,I,5], first-token batch [Q,I], fp32 [Q,I], fp64 [Q,I]."""
    Q, I = wl.num_queries, wl.num_instances
    qq, jj = np.meshgrid(np.arange(Q), np.arange(I), indexing="ij")
    F, lt, t32, t64 = estimate_candidates(wl, qq.ravel(), jj.ravel(), max_batches, threads)
    return F.reshape(Q, I, 5), lt.reshape(Q, I), t32.reshape(Q, I), t64.reshape(Q, I)


def route(wl, ttft32: np.ndarray, lam=None, mu=None, tau=None):
    """Brute-force routing over full TTFT rows: assign/util/ttft_chosen [P,Q]."""
    lam = _c(wl.lam if lam is None else lam, np.float32)
    P = lam.shape[0]
    mu_a = _c(np.zeros(P, np.float32) if (mu is None and tau is not None) else (wl.mu if mu is None else mu),
              np.float32)
    t = _c(ttft32, np.float32)
    Q, I = t.shape
    tau_a = None if tau is None else _c(tau, np.float32)
    assign = np.zeros((P, Q), np.int32)
    util = np.zeros((P, Q), np.float32)
    tch = np.zeros((P, Q), np.float32)
    moi, p, dh = (_c(a, np.int32) for a in (wl.model_of_instance, wl.prompt_len, wl.dec_hat))
    acc, pin, pout = (_c(a, np.float32) for a in (wl.acc, wl.price_in, wl.price_out))
    rc = _load().orc_route(Q, I, wl.num_models, _p(moi), _p(pin), _p(pout), _p(p), _p(dh), _p(acc), _p(t),
                           _p(tau_a), P, _p(lam), _p(mu_a), _p(assign), _p(util), _p(tch))
    if rc != 0:
        raise RuntimeError(f"oracle route failed with code {rc}")
    return assign, util, tch


def frontier(wl, assign: np.ndarray, ttft_chosen: np.ndarray) -> np.ndarray:
    a = _c(assign, np.int32)
    tch = _c(ttft_chosen, np.float32)
    P, Q = a.shape
    out = np.zeros((P, 3), np.float64)
    moi, p, dh = (_c(x, np.int32) for x in (wl.model_of_instance, wl.prompt_len, wl.dec_hat))
    acc, pin, pout = (_c(x, np.float32) for x in (wl.acc, wl.price_in, wl.price_out))
    rc = _load().orc_frontier(Q, wl.num_instances, wl.num_models, _p(moi), _p(pin), _p(pout), _p(p), _p(dh),
                              _p(acc), P, _p(a), _p(tch), _p(out))
    if rc != 0:
        raise RuntimeError(f"oracle frontier failed with code {rc}")
    return out


def advance(wl, clock, assign, prompt_len, dec, t_now: float, max_batches: int = 1 << 30, track=None,
            id_base: int = -1, kv=None):
    """Online stream step on a copy of the workload's state.

    Returns (new workload with the advanced state, new clocks).  With `track` -- a dict of
    run_id [I, cap_running] int64, wait_id [I, cap_waiting] int64 and first_token_time [N]
    float64 -- the routed query i joins as id id_base + i (id_base >= 0) and every tracked
    request that emits its first output token in an executed batch gets that batch's end
    time; the call then returns (workload, clocks, new track dict).  With `kv` =
    (block_size, num_blocks, max_ctx), scalars or per-instance arrays, every executed
    batch follows the KV step rule (orc_advance_kv)."""
    import dataclasses
    st = {k: np.array(getattr(wl, k), dtype=np.int32, copy=True)
          for k in ("n_run", "run_ctx", "run_pre", "run_dec", "n_wait", "wait_pre", "wait_dec")}
    clk = np.array(clock, dtype=np.float64, copy=True)
    a = _c(assign, np.int32)
    p = _c(prompt_len, np.int32)
    d = _c(dec, np.int32)
    moi, B, S = (_c(x, np.int32) for x in (wl.model_of_instance, wl.max_batched_tokens, wl.max_seqs))
    coef = _c(wl.coef, np.float32)
    tr = None
    if track is not None:
        tr = {k: np.array(track[k], dtype=(np.float64 if k == "first_token_time" else np.int64), copy=True)
              for k in ("run_id", "wait_id", "first_token_time")}
    head = (wl.num_instances, _p(moi), _p(coef), _p(B), _p(S), wl.cap_running, wl.cap_waiting, _p(st["n_run"]),
            _p(st["run_ctx"]), _p(st["run_pre"]), _p(st["run_dec"]), _p(st["n_wait"]), _p(st["wait_pre"]),
            _p(st["wait_dec"]), _p(clk), int(a.shape[0]), _p(a), _p(p), _p(d), wl.first_token_mode,
            float(t_now), int(max_batches))
    ids = (_p(None if tr is None else tr["run_id"]), _p(None if tr is None else tr["wait_id"]), int(id_base),
           _p(None if tr is None else tr["first_token_time"]))
    if kv is None:
        rc = _load().orc_advance_ids(*head, *ids)
    else:
        I = wl.num_instances
        bs = _c(np.broadcast_to(np.asarray(kv[0], np.int32), (I,)), np.int32)
        nb = _c(np.broadcast_to(np.asarray(kv[1], np.int64), (I,)), np.int64)
        mc = _c(np.broadcast_to(np.asarray(kv[2], np.int64), (I,)), np.int64)
        rc = _load().orc_advance_kv(*head, _p(bs), _p(nb), _p(mc), *ids)
    if rc != 0:
        raise RuntimeError(f"oracle advance failed with code {rc}")
    if tr is None:
        return dataclasses.replace(wl, **st), clk
    return dataclasses.replace(wl, **st), clk, tr


def new_track(wl, num_ids: int):
    """Empty first-token tracking state for `advance`: every resident untracked, times NaN."""
    return {"run_id": np.full((wl.num_instances, wl.cap_running), -1, np.int64),
            "wait_id": np.full((wl.num_instances, wl.cap_waiting), -1, np.int64),
            "first_token_time": np.full(num_ids, np.nan)}


def pool_capacity(wl, horizon: float = 300.0, warm: float = 30.0, dt: float = 2.0, depth: int = 256) -> np.ndarray:
    """Completions/s of every instance fed a saturating FCFS stream of the workload's queries.

    The reading of pool capacity for the online stream (App. E defines an
    instance's capacity from its peak throughput): each instance starts empty;
    before every advance of dt seconds (the oracle's stream step) its waiting
    queue is topped up to `depth` with the workload's next queries, each with the
    predicted output length of the instance's model, so the scheduler never runs
    dry; completions are counted from t = warm to t = horizon."""
    import dataclasses
    I = wl.num_instances
    z = np.zeros(I, np.int32)
    st = dataclasses.replace(wl, n_run=z, n_wait=z.copy(), cap_waiting=depth,
                             run_ctx=np.zeros((I, wl.cap_running), np.int32),
                             run_pre=np.zeros((I, wl.cap_running), np.int32),
                             run_dec=np.zeros((I, wl.cap_running), np.int32),
                             wait_pre=np.zeros((I, depth), np.int32), wait_dec=np.zeros((I, depth), np.int32))
    clk = np.zeros(I)
    appended = np.zeros(I, np.int64)
    nxt, t, c_warm = 0, 0.0, None
    while True:
        completed = appended - st.n_run - st.n_wait
        if c_warm is None and t >= warm:
            c_warm = completed.copy()
        if t >= horizon:
            break
        need = depth - st.n_wait
        a = np.repeat(np.arange(I, dtype=np.int32), need)
        idx = (nxt + np.arange(a.shape[0])) % wl.num_queries
        nxt += a.shape[0]
        appended += need
        t += dt
        dec = np.ascontiguousarray(wl.dec_hat[idx, wl.model_of_instance[a]])
        st, clk = advance(st, clk, a, wl.prompt_len[idx], dec, t)
    return (completed - c_warm) / (horizon - warm)


# ---------------------------------------------------------------------------
# Average-case estimators (Sec. 4, average-case TTFT estimation; App. E)

def pow_int(x: float, k: int) -> float:
    """x**k by binary exponentiation in fp64 (the order both sides use)."""
    return float(_load().orc_pow_int(float(x), int(k)))


def lps_wait(alpha: float, mu: float, k: int, ca2: float = 1.0, cs2: float = 1.0) -> float:
    """Expected LPS queueing delay ((ca2 + cs2)/2) * (alpha/mu)^k / (mu - alpha) (App. E)."""
    return float(_load().orc_lps_wait(float(alpha), float(mu), int(k), float(ca2), float(cs2)))


def throughput_wait(wl, theta) -> np.ndarray:
    """Per instance: remaining prefill tokens of the residents / theta (Sec. 4)."""
    th = np.broadcast_to(np.asarray(theta, np.float64), (wl.num_instances,))
    out = np.zeros(wl.num_instances)
    lib = _load()
    for j in range(wl.num_instances):
        rc = _c(wl.run_pre[j], np.int32)
        wp = _c(wl.wait_pre[j], np.int32)
        inst = _Instance(int(wl.n_run[j]), None, _p(rc), None, int(wl.n_wait[j]), _p(wp), None)
        out[j] = lib.orc_throughput_wait(ctypes.byref(inst), float(th[j]))
    return out


def avgcase_matrix(wl, W, theta, tdec):
    """TTFT[Q][I] = W_j + p_i/theta_j + Tdec_j: canonical fp32 and fp64."""
    I, Q = wl.num_instances, wl.num_queries
    Wd, th, td = (np.ascontiguousarray(np.broadcast_to(np.asarray(x, np.float64), (I,))) for x in (W, theta, tdec))
    p = _c(wl.prompt_len, np.int32)
    t32 = np.zeros((Q, I), np.float32)
    t64 = np.zeros((Q, I), np.float64)
    rc = _load().orc_avgcase_ttft(I, Q, _p(Wd), _p(th), _p(td), _p(p), _p(t32), _p(t64))
    if rc != 0:
        raise ValueError(f"oracle average-case estimate failed with code {rc}")
    return t32, t64


# ---------------------------------------------------------------------------
# Calibration of the batch-time model (Sec. 4.1, the token-batch time estimator:
# the coefficients are calibrated from observed batch times)

def calibrate(features, model, time, num_models: int, shared_beta1: bool = True) -> np.ndarray:
    """Least-squares Eq. 9 coefficients per model from per-batch (F, observed time) rows.

    features [N][5] (F0 .. F4 of each executed batch), model [N], time [N] seconds.
    shared_beta1: the paper's four-coefficient form, one beta1 for prefill and
    decode tokens (regressor F1 + F2); otherwise five coefficients.
    Returns [M][5] fp64 (beta0, beta1p, beta1d, beta2, beta3); NaN rows for models
    with fewer rows than unknowns or a rank-deficient design."""
    F = np.asarray(features, np.float64)
    mdl = np.asarray(model, np.int64)
    y = np.asarray(time, np.float64)
    out = np.full((num_models, 5), np.nan)
    for m in range(num_models):
        sel = mdl == m
        X = F[sel]
        if shared_beta1:
            X = np.stack([X[:, 0], X[:, 1] + X[:, 2], X[:, 3], X[:, 4]], axis=1)
        if X.shape[0] < X.shape[1]:
            continue
        beta, _, rank, _ = np.linalg.lstsq(X, y[sel], rcond=None)
        if rank < X.shape[1]:
            continue
        out[m] = [beta[0], beta[1], beta[1], beta[2], beta[3]] if shared_beta1 else beta
    return out


# ---- Baseline routing policies and stream metrics (Sec. 6 baselines; Eq. 4) ----

POLICY_ROUND_ROBIN, POLICY_SHORTEST_QUEUE, POLICY_LATENCY_AGNOSTIC = 0, 1, 2


def round_robin(Q: int, I: int, start: int = 0) -> np.ndarray:
    """Round Robin: query q to instance (start + q) mod I."""
    a = np.zeros(Q, np.int32)
    if _load().orc_round_robin(Q, I, int(start), _p(a)) != 0:
        raise RuntimeError("oracle round robin failed")
    return a


def shortest_queue(counts, Q: int) -> np.ndarray:
    """Shortest Queue: each query in turn to the instance with the fewest resident
    requests, the queries routed before it included (ties to the lowest index)."""
    c = _c(counts, np.int32)
    a = np.zeros(Q, np.int32)
    if _load().orc_shortest_queue(Q, c.shape[0], _p(c), _p(a)) != 0:
        raise RuntimeError("oracle shortest queue failed")
    return a


def baseline_route(wl, policy: int, lam: float, rr_start: int = 0, ttft32: Optional[np.ndarray] = None):
    """A baseline policy's assignment, the chosen instance's utility (Eq. 2) and its
    canonical fp32 SFS TTFT: assign/util/ttft [Q].  Latency-Agnostic is the argmax of
    U over the instances (ties to the lowest index); rows whose prompt is out of range
    get -1 / NaN / NaN."""
    Q, I = wl.num_queries, wl.num_instances
    lam32 = np.float32(lam)
    if policy == POLICY_ROUND_ROBIN:
        assign = round_robin(Q, I, rr_start)
    elif policy == POLICY_SHORTEST_QUEUE:
        assign = shortest_queue(np.asarray(wl.n_run) + np.asarray(wl.n_wait), Q)
    elif policy == POLICY_LATENCY_AGNOSTIC:
        assign = np.zeros(Q, np.int32)
        moi, p, dh = (_c(a, np.int32) for a in (wl.model_of_instance, wl.prompt_len, wl.dec_hat))
        acc, pin, pout = (_c(a, np.float32) for a in (wl.acc, wl.price_in, wl.price_out))
        if _load().orc_latency_agnostic(Q, I, wl.num_models, _p(moi), _p(pin), _p(pout), _p(p), _p(dh), _p(acc),
                                        float(lam32), _p(assign)) != 0:
            raise RuntimeError("oracle latency-agnostic failed")
    else:
        raise ValueError(policy)
    valid = (np.asarray(wl.prompt_len) >= 1) & (np.asarray(wl.prompt_len) <= wl.max_prompt_len)
    util = np.full(Q, np.nan, np.float32)
    ttft = np.full(Q, np.nan, np.float32)
    qs = np.nonzero(valid)[0]
    if qs.size:
        if ttft32 is None:
            _, _, t32, _ = estimate_candidates(wl, qs, assign[qs])
        else:
            t32 = np.asarray(ttft32, np.float32)[qs, assign[qs]]
        ttft[qs] = t32
        for i in qs:
            m = wl.model_of_instance[assign[i]]
            util[i] = utility(wl.acc[i, m], lam32, wl.prompt_len[i], wl.dec_hat[i, m], wl.price_in[m],
                              wl.price_out[m])
    assign = np.where(valid, assign, -1).astype(np.int32)
    return assign, util, ttft


def on_time_utility(util, ttft, tau, delay=None):
    """(OnTimeUtility of Eq. 4, SLO attainment): realized TTFT = fp32 delay + ttft."""
    u, t, ta = (_c(x, np.float32) for x in (util, ttft, tau))
    d = None if delay is None else _c(delay, np.float32)
    out = np.zeros(2, np.float64)
    if _load().orc_on_time_utility(u.shape[0], _p(u), _p(t), _p(ta), _p(d), _p(out)) != 0:
        raise RuntimeError("oracle on-time utility failed")
    return float(out[0]), float(out[1])


# ---- KV-cache limits, context limit and preemption (App. F; rule in sfs_oracle.c) ----

class _KV(ctypes.Structure):
    _fields_ = [("block_size", ctypes.c_int32), ("num_blocks", ctypes.c_int64), ("max_ctx", ctypes.c_int64)]


ORC_ELIMIT = 2


def simulate_kv(running, waiting, B: int, S: int, p: int, d: int, block_size: int, num_blocks: int, max_ctx: int,
                mode: int = FIRST_TOKEN_SEPARATE_DECODE, max_batches: int = 1 << 20):
    """One candidate under KV limits.  running: list of (ctx, pre, dec); waiting: list of (pre, dec).

    Returns (F[5], admit batch, first-token batch, residents' per-batch features [l][5],
    most blocks in use)."""
    run = np.asarray(running, dtype=np.int32).reshape(-1, 3)
    wt = np.asarray(waiting, dtype=np.int32).reshape(-1, 2)
    rc_, rp_, rd_ = (_c(run[:, k], np.int32) for k in range(3))
    wp_, wd_ = (_c(wt[:, k], np.int32) for k in range(2))
    inst = _Instance(run.shape[0], _p(rc_), _p(rp_), _p(rd_), wt.shape[0], _p(wp_), _p(wd_))
    kv = _KV(block_size, num_blocks, max_ctx)
    F = np.zeros(5, np.int64)
    res = np.zeros((max_batches, 5), np.int64)
    la, lt, mu = ctypes.c_int64(0), ctypes.c_int64(0), ctypes.c_int64(0)
    rc = _load().orc_sfs_candidate_kv(ctypes.byref(inst), B, S, mode, ctypes.byref(kv), p, d, max_batches, _p(F),
                                      ctypes.byref(la), ctypes.byref(lt), _p(res), ctypes.byref(mu))
    if rc != 0:
        raise RuntimeError(f"oracle KV simulation failed with code {rc}")
    return F, la.value, lt.value, res[:lt.value].copy(), mu.value


def kv_residents(running, waiting, B: int, S: int, L: int, block_size: int, num_blocks: int, max_ctx: int,
                 mode: int = FIRST_TOKEN_SEPARATE_DECODE):
    """The residents alone for L batches under KV limits: per-batch features [L][5]."""
    run = np.asarray(running, dtype=np.int32).reshape(-1, 3)
    wt = np.asarray(waiting, dtype=np.int32).reshape(-1, 2)
    rc_, rp_, rd_ = (_c(run[:, k], np.int32) for k in range(3))
    wp_, wd_ = (_c(wt[:, k], np.int32) for k in range(2))
    inst = _Instance(run.shape[0], _p(rc_), _p(rp_), _p(rd_), wt.shape[0], _p(wp_), _p(wd_))
    kv = _KV(block_size, num_blocks, max_ctx)
    res = np.zeros((L, 5), np.int64)
    rc = _load().orc_kv_residents(ctypes.byref(inst), B, S, mode, ctypes.byref(kv), L, _p(res))
    if rc != 0:
        raise RuntimeError(f"oracle KV residents failed with code {rc}")
    return res


def estimate_matrix_kv(wl, block_size, num_blocks, max_ctx, max_batches: int = DEFAULT_MAX_BATCHES,
                       cand_q=None, cand_j=None, threads: Optional[int] = None):
    """Every candidate (or the listed ones) under per-instance KV limits, the query taken
    up to its first token.  Returns status, F[...,5], first-token batch, fp32, fp64
    ([Q,I] shapes for the full matrix, [C] for a list); failed candidates carry F = -1,
    batch -1 and NaN times."""
    Q, I = wl.num_queries, wl.num_instances
    full = cand_q is None
    if full:
        qq, jj = np.meshgrid(np.arange(Q), np.arange(I), indexing="ij")
        cand_q, cand_j = qq.ravel(), jj.ravel()
    cq, cj = _c(cand_q, np.int32), _c(cand_j, np.int32)
    C = cq.shape[0]
    st = np.zeros(C, np.int32)
    F = np.zeros((C, 5), np.int64)
    lt = np.zeros(C, np.int64)
    t32 = np.zeros(C, np.float32)
    t64 = np.zeros(C, np.float64)
    arrs = [_c(a, np.int32) for a in (wl.model_of_instance, wl.max_batched_tokens, wl.max_seqs, wl.n_run,
                                      wl.run_ctx, wl.run_pre, wl.run_dec, wl.n_wait, wl.wait_pre,
                                      wl.wait_dec, wl.prompt_len)]
    moi, B, S, n_run, run_ctx, run_pre, run_dec, n_wait, wait_pre, wait_dec, p = arrs
    bs = _c(np.broadcast_to(np.asarray(block_size, np.int32), (I,)), np.int32)
    nb = _c(np.broadcast_to(np.asarray(num_blocks, np.int64), (I,)), np.int64)
    mc = _c(np.broadcast_to(np.asarray(max_ctx, np.int64), (I,)), np.int64)
    coef = _c(wl.coef, np.float32)
    lib = _load()
    codes = []

    def run(lo, hi):
        codes.append(lib.orc_estimate_candidates_kv(
            I, _p(moi), _p(coef), _p(B), _p(S), wl.cap_running, wl.cap_waiting, _p(n_run), _p(run_ctx),
            _p(run_pre), _p(run_dec), _p(n_wait), _p(wait_pre), _p(wait_dec), _p(p), _p(bs), _p(nb), _p(mc),
            wl.first_token_mode, max_batches, hi - lo, _p(cq[lo:]), _p(cj[lo:]), _p(st[lo:]), _p(F[lo:]),
            _p(lt[lo:]), _p(t32[lo:]), _p(t64[lo:])))

    _in_slices(C, threads, run)
    rc = next((r for r in codes if r != 0), 0)
    if rc != 0:
        raise RuntimeError(f"oracle KV estimate failed with code {rc}")
    if full:
        return st.reshape(Q, I), F.reshape(Q, I, 5), lt.reshape(Q, I), t32.reshape(Q, I), t64.reshape(Q, I)
    return st, F, lt, t32, t64
