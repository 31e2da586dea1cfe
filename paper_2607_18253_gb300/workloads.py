"""Seeded synthetic workloads for the latency-aware router.

This module only draws random numbers and lays them out; it holds none of the
estimator's arithmetic (no batch simulation, no utility, no argmax).  Both the
CUDA path and the CPU oracle consume the arrays it returns, so they always see
identical bytes.

Shapes follow the paper's setting: model instances with a running set and an
FCFS waiting queue (Sec. 4 setup), prompts of roughly 10 to 1e4 tokens and
responses of roughly 1e2 to 1e3 tokens (App. B.3), per-token prices
(App. B.1/B.4) and TTFT targets drawn with the recipe of App. B.2.  The paper's
datasets (Alpaca, HotpotQA, GovReport, WritingPrompts) are not available; these
lognormal stand-ins take their length ranges.

Batch-time coefficients use the five-term form of Eq. 9 with separate
prefill/decode token slopes.  A model described by (alpha, beta, gamma) -- a
fixed per-batch cost, a per-token cost and the cost of one decode token at
context 1024 -- maps to

    beta0 = alpha, beta1p = beta1d = beta,
    beta2 = (gamma - beta) / 1024, beta3 = beta2 / 16,

all in seconds.  This mapping is configuration, not part of the method.
"""
from __future__ import annotations

import dataclasses
import math
from typing import Dict, Optional

import numpy as np

FIRST_TOKEN_SEPARATE_DECODE = 0   # first output token takes its own decode batch (Sec. 4.1)
FIRST_TOKEN_WITH_LAST_CHUNK = 1   # first output token sampled in the last prefill batch


@dataclasses.dataclass
class Workload:
    """All inputs of one routing problem, as little-endian numpy arrays."""
    name: str
    # pool
    model_of_instance: np.ndarray     # [I] int32
    coef: np.ndarray                  # [M,5] float32: beta0, beta1p, beta1d, beta2, beta3 (s)
    price_in: np.ndarray              # [M] float32, $ per prompt token
    price_out: np.ndarray             # [M] float32, $ per response token
    max_batched_tokens: np.ndarray    # [I] int32 (token budget B_j)
    max_seqs: np.ndarray              # [I] int32 (sequence cap S_j)
    cap_running: int
    cap_waiting: int
    # instance state snapshot (SoA, row stride = cap)
    n_run: np.ndarray                 # [I] int32
    run_ctx: np.ndarray               # [I,capR] int32 tokens already in the KV cache
    run_pre: np.ndarray               # [I,capR] int32 remaining prefill tokens
    run_dec: np.ndarray               # [I,capR] int32 remaining predicted decode tokens (>=1)
    n_wait: np.ndarray                # [I] int32
    wait_pre: np.ndarray              # [I,capW] int32 prompt tokens
    wait_dec: np.ndarray              # [I,capW] int32 predicted decode tokens (>=1)
    # queries
    prompt_len: np.ndarray            # [Q] int32
    dec_hat: np.ndarray               # [Q,M] int32 predicted output length per model
    acc: np.ndarray                   # [Q,M] float32 predicted accuracy per model
    tau: np.ndarray                   # [Q] float32 TTFT target (s)
    lam: np.ndarray                   # [P] float32 accuracy-cost trade-off
    mu: np.ndarray                    # [P] float32 latency weight (1/s)
    max_prompt_len: int
    first_token_mode: int = FIRST_TOKEN_SEPARATE_DECODE
    seed: int = 0

    @property
    def num_instances(self) -> int:
        return int(self.model_of_instance.shape[0])

    @property
    def num_models(self) -> int:
        return int(self.coef.shape[0])

    @property
    def num_queries(self) -> int:
        return int(self.prompt_len.shape[0])

    @property
    def num_pairs(self) -> int:
        return int(self.lam.shape[0])

    def with_queries(self, idx: np.ndarray) -> "Workload":
        """Same pool and state, a subset of the queries (in the given order)."""
        idx = np.asarray(idx, dtype=np.int64)
        return dataclasses.replace(
            self, prompt_len=np.ascontiguousarray(self.prompt_len[idx]),
            dec_hat=np.ascontiguousarray(self.dec_hat[idx]),
            acc=np.ascontiguousarray(self.acc[idx]),
            tau=np.ascontiguousarray(self.tau[idx]))

    def with_mode(self, mode: int) -> "Workload":
        return dataclasses.replace(self, first_token_mode=int(mode))


def _lognormal_int(rng: np.random.Generator, median: float, cap: int, size, sigma: float = 1.0) -> np.ndarray:
    v = np.rint(median * np.exp(sigma * rng.standard_normal(size)))
    return np.clip(v, 1, cap).astype(np.int32)


def model_pool(num_models: int):
    """Per-model (alpha, beta, gamma) in ms and price in $/Mtok.

    Two models take the small/large values directly; more models place alpha
    linearly in [3, 10] ms and beta, gamma, price geometrically between the
    small and large values.
    """
    if num_models == 2:
        alpha = np.array([4.0, 8.0])
        beta = np.array([0.05, 0.12])
        gamma = np.array([0.2, 0.5])
        price = np.array([0.2, 2.0])
    else:
        x = np.arange(num_models) / (num_models - 1)
        alpha = 3.0 + 7.0 * x
        beta = 0.05 * (0.12 / 0.05) ** x
        gamma = 0.2 * (0.5 / 0.2) ** x
        price = 0.2 * (2.0 / 0.2) ** x
    return alpha, beta, gamma, price


def coefficients(alpha_ms, beta_ms, gamma_ms) -> np.ndarray:
    """(alpha, beta, gamma) in ms -> [M,5] float32 Eq. 9 coefficients in seconds."""
    a = np.asarray(alpha_ms, dtype=np.float64) * 1e-3
    b = np.asarray(beta_ms, dtype=np.float64) * 1e-3
    g = np.asarray(gamma_ms, dtype=np.float64) * 1e-3
    b2 = (g - b) / 1024.0
    b3 = b2 / 16.0
    return np.stack([a, b, b, b2, b3], axis=1).astype(np.float32)


def ttft_targets(rng: np.random.Generator, prompt_len: np.ndarray) -> np.ndarray:
    """TTFT targets of App. B.2: clip(u + (155 + 3.5e-3 p) v, 150, 1120) ms, in seconds."""
    n = prompt_len.shape[0]
    uv = rng.uniform(0.0, 1.0, (n, 2))  # row-wise draws keep a prefix of queries unchanged
    u = 1.0 + 4.0 * uv[:, 0]
    v = 0.98 + 0.04 * uv[:, 1]
    t_ms = np.minimum(1120.0, np.maximum(150.0, u + (155.0 + 3.5e-3 * prompt_len.astype(np.float64)) * v))
    return (t_ms * 1e-3).astype(np.float32)


# name -> recipe.  Instance state: running requests are decoding (no remaining
# prefill), context U[128, 2048], remaining decode lognormal(median 128, cap
# 2048); waiting prompts lognormal with the listed median/cap, decode
# lognormal(median 256, cap 2048).  Query prompts share the waiting recipe.
RECIPES: Dict[str, dict] = {
    "tiny": dict(models=2, replicas=4, queries=16, seed=0, run_max=32, wait_max=16,
                 p_median=512, p_cap=4096, budget=2048, seqs=64, acc="uniform"),
    "pool64": dict(models=4, replicas=16, queries=4096, seed=1, run_max=64, wait_max=64,
                   p_median=1024, p_cap=8192, budget=4096, seqs=64, acc="uniform"),
    "pool256": dict(models=8, replicas=32, queries=65536, seed=2, run_max=256, wait_max=256,
                    p_median=1024, p_cap=32768, budget=8192, seqs=256, acc="beta22"),
    # one instance per model, as in the paper's pool of three models (Sec. 6)
    "paper3": dict(models=3, replicas=1, queries=4096, seed=4, run_max=64, wait_max=64,
                   p_median=1024, p_cap=8192, budget=4096, seqs=64, acc="uniform"),
}


def _round_up(x: int, m: int) -> int:
    return ((x + m - 1) // m) * m


def make_workload(name: str, num_queries: Optional[int] = None, seed: Optional[int] = None,
                  lam: Optional[np.ndarray] = None, mu: Optional[np.ndarray] = None,
                  first_token_mode: int = FIRST_TOKEN_SEPARATE_DECODE, cap_running: Optional[int] = None,
                  cap_waiting: Optional[int] = None) -> Workload:
    """Build one of the named workloads ("tiny", "pool64", "pool256", "paper3").

    The instance state and the queries come from independent child streams of
    the seed, so changing the query count leaves the state unchanged and keeps
    the query prefix unchanged.  Larger capacities (row strides) only pad the
    state arrays; the drawn values do not change.
    """
    r = RECIPES[name]
    seed = r["seed"] if seed is None else seed
    nq = r["queries"] if num_queries is None else int(num_queries)
    M, R = r["models"], r["replicas"]
    I = M * R
    ss = np.random.SeedSequence(seed)
    g_state, g_p, g_d, g_a, g_t = [np.random.default_rng(s) for s in ss.spawn(5)]

    alpha, beta, gamma, price = model_pool(M)
    coef = coefficients(alpha, beta, gamma)
    price_tok = (price * 1e-6).astype(np.float32)

    dR = _round_up(r["run_max"], 32)
    dW = _round_up(r["wait_max"], 32)
    capR = max(dR, int(cap_running or 0))
    capW = max(dW, int(cap_waiting or 0))
    n_run = g_state.integers(0, r["run_max"] + 1, I).astype(np.int32)
    n_wait = g_state.integers(0, r["wait_max"] + 1, I).astype(np.int32)

    def pad(a, cap):
        out = np.zeros((I, cap), np.int32)
        out[:, :a.shape[1]] = a
        return out

    run_ctx = pad(g_state.integers(128, 2048 + 1, (I, dR)).astype(np.int32), capR)
    run_dec = pad(_lognormal_int(g_state, 128, 2048, (I, dR)), capR)
    run_pre = np.zeros((I, capR), np.int32)
    wait_pre = pad(_lognormal_int(g_state, r["p_median"], r["p_cap"], (I, dW)), capW)
    wait_dec = pad(_lognormal_int(g_state, 256, 2048, (I, dW)), capW)
    # zero the padding beyond each row's count
    cols_r = np.arange(capR)[None, :]
    cols_w = np.arange(capW)[None, :]
    run_ctx[cols_r >= n_run[:, None]] = 0
    run_dec[cols_r >= n_run[:, None]] = 0
    wait_pre[cols_w >= n_wait[:, None]] = 0
    wait_dec[cols_w >= n_wait[:, None]] = 0

    p = _lognormal_int(g_p, r["p_median"], r["p_cap"], nq)
    dec_hat = _lognormal_int(g_d, 256, 2048, (nq, M))
    if r["acc"] == "uniform":
        acc = g_a.uniform(0.0, 1.0, (nq, M)).astype(np.float32)
    else:
        acc = g_a.beta(2.0, 2.0, (nq, M)).astype(np.float32)
    tau = ttft_targets(g_t, p)

    lam = np.array([1.0], np.float32) if lam is None else np.asarray(lam, np.float32)
    mu = np.array([0.1], np.float32) if mu is None else np.asarray(mu, np.float32)

    return Workload(
        name=name, model_of_instance=(np.arange(I) // R).astype(np.int32), coef=coef,
        price_in=price_tok.copy(), price_out=price_tok.copy(),
        max_batched_tokens=np.full(I, r["budget"], np.int32), max_seqs=np.full(I, r["seqs"], np.int32),
        cap_running=capR, cap_waiting=capW, n_run=n_run, run_ctx=run_ctx, run_pre=run_pre, run_dec=run_dec,
        n_wait=n_wait, wait_pre=wait_pre, wait_dec=wait_dec, prompt_len=p, dec_hat=dec_hat, acc=acc, tau=tau,
        lam=lam, mu=mu, max_prompt_len=int(r["p_cap"]), first_token_mode=first_token_mode, seed=seed)


def poisson_arrivals(num_queries: int, rate_qps: float, seed: int) -> np.ndarray:
    """Arrival times (s, fp64) of a Poisson process: exponential gaps with mean 1/rate."""
    rng = np.random.default_rng(np.random.SeedSequence([seed, 0x5eed]))
    return np.cumsum(rng.exponential(1.0 / rate_qps, num_queries))


def mmpp2_rates(mean_qps: float, ratio: float, p_high: float = 0.2):
    """Low- and high-state rates of a two-state MMPP with long-run mean `mean_qps`,
    high/low rate ratio `ratio` and a fraction `p_high` of time in the high state."""
    low = mean_qps / ((1.0 - p_high) + p_high * ratio)
    return low, ratio * low


def mmpp2_arrivals(num_queries: int, mean_qps: float, ratio: float, seed: int, z_lh: float = 0.1,
                   z_hl: float = 0.4) -> np.ndarray:
    """Arrival times (s, fp64) of a two-state Markov-modulated Poisson process.

    The latent state switches low->high at rate z_lh and high->low at z_hl (so it
    spends z_lh / (z_lh + z_hl) of the time high); within a sojourn of length d at
    rate a, the arrivals are a Poisson(a d) count of uniform times.  The state
    starts from its stationary law."""
    p_high = z_lh / (z_lh + z_hl)
    low, high_rate = mmpp2_rates(mean_qps, ratio, p_high)
    rng = np.random.default_rng(np.random.SeedSequence([seed, 0x3A77]))
    high = bool(rng.random() < p_high)
    t, total, parts = 0.0, 0, []
    while total < num_queries:
        d = rng.exponential(1.0 / (z_hl if high else z_lh))
        k = int(rng.poisson((high_rate if high else low) * d))
        if k:
            parts.append(t + np.sort(rng.uniform(0.0, d, k)))
            total += k
        t += d
        high = not high
    return np.concatenate(parts)[:num_queries]


def batch_log(num_batches: int, num_models: int, seed: int, coef: np.ndarray, noise: float = 0.04,
              grouped: bool = True):
    """A synthetic log of executed token batches, as calibration input.

    Each row is one batch of some model: F0 = 1, up to 256 decode tokens at
    contexts 128..4096 (F2, F3), and up to two prefill chunks of 1..2048 tokens at
    contexts 0..8192 (F1, F4 = sum of x c + x(x+1)/2).  The synthetic engine's
    observed time is coef[model] . F (the batch-time form being calibrated) times
    (1 + noise * N(0, 1)).  grouped: rows sorted by model, as per-instance logs are.
    Returns features [N][5] int64, model [N] int32, time [N] fp64."""
    rng = np.random.default_rng(np.random.SeedSequence([seed, 0xCA1B]))
    n = num_batches
    mdl = rng.integers(0, num_models, n)
    if grouped:
        mdl = np.sort(mdl)
    ndec = rng.integers(0, 257, n)
    ctx = rng.integers(128, 4097, n)
    F = np.zeros((n, 5), np.int64)
    F[:, 0] = 1
    F[:, 2] = ndec
    F[:, 3] = ndec * ctx
    for _ in range(2):
        has = rng.random(n) < 0.5
        x = np.where(has, rng.integers(1, 2049, n), 0)
        c = rng.integers(0, 8193, n)
        F[:, 1] += x
        F[:, 4] += x * c + x * (x + 1) // 2
    cf = np.asarray(coef, np.float64)[mdl]
    t = np.einsum("nk,nk->n", cf, F.astype(np.float64)) * (1.0 + noise * rng.standard_normal(n))
    return F, mdl.astype(np.int32), t


def kv_limits(wl: Workload, seed: int, block_sizes=(16,), tightness=(0.3, 1.0), ctx_limited: float = 0.5,
              ctx_slack=(1, 64), unlimited: int = 1 << 40, max_new: int = 1):
    """Seeded per-instance KV-cache limits for a workload's snapshot: block sizes drawn
    from `block_sizes`; a context limit on a `ctx_limited` share of the instances, just
    above the longest context any request or query already needs (so that decoding runs
    into it), else `unlimited`; and a block count that a `tightness` draw places between
    the most any single request (or the longest query with `max_new` output tokens: 1
    for an estimate up to the first token, the longest response for a stream that runs
    queries to their end) can need and the residents' whole demand, never below the
    blocks the running requests hold.
    Returns (block_size [I] int32, num_blocks [I] int64, max_ctx [I] int64).  Token
    counts are turned into blocks by the bound tokens // bs + 1 >= ceil(tokens / bs)."""
    rng = np.random.default_rng(seed)
    I = wl.num_instances
    bs = rng.choice(np.asarray(block_sizes, np.int64), I).astype(np.int32)
    nb = np.zeros(I, np.int64)
    mctx = np.zeros(I, np.int64)
    for j in range(I):
        b = int(bs[j])
        nr, nw = int(wl.n_run[j]), int(wl.n_wait[j])
        ctx = wl.run_ctx[j, :nr].astype(np.int64)
        pre = wl.run_pre[j, :nr].astype(np.int64)
        dec = wl.run_dec[j, :nr].astype(np.int64)
        wpre = wl.wait_pre[j, :nw].astype(np.int64)
        wdec = wl.wait_dec[j, :nw].astype(np.int64)
        lo = max([wl.max_prompt_len] + list(ctx + pre) + list(wpre)) + 1
        if rng.random() < ctx_limited:
            mctx[j] = lo + int(rng.integers(ctx_slack[0], ctx_slack[1] + 1))
        else:
            mctx[j] = unlimited
        whole = np.concatenate([np.minimum(ctx + pre + dec, mctx[j]), np.minimum(wpre + wdec, mctx[j]),
                                [min(wl.max_prompt_len + max_new, int(mctx[j]))]])
        one = int((whole // b + 1).max())
        held = int((ctx // b + 1).sum())
        demand = int((whole // b + 1).sum())
        u = rng.uniform(*tightness)
        nb[j] = max(one, held, int(one + u * (demand - one)))
    return bs, nb, mctx


def sweep_pairs():
    """The trade-off grid: 4 lambda values (log 0.1..10) x 8 mu values (log 0.01..1 /s), lambda-major."""
    lam = np.logspace(-1, 1, 4)
    mu = np.logspace(-2, 0, 8)
    L, Mu = np.meshgrid(lam, mu, indexing="ij")
    return L.ravel().astype(np.float32), Mu.ravel().astype(np.float32)


def random_small_state(rng: np.random.Generator, num_instances: int, cap_running: int, cap_waiting: int,
                       budget_range=(4, 64), with_tail_prefill: bool = True,
                       max_ctx: int = 300, max_pre: int = 200, max_dec: int = 40, min_gap: int = 1,
                       wait_max: Optional[int] = None):
    """Small random pools for property tests.

    Returns per-instance budget B, cap S (1 <= S <= B - min_gap + 1), and a
    state whose running list holds at most one request with remaining
    prefill, placed last, and never more requests than S.
    """
    I = num_instances
    B = rng.integers(max(budget_range[0], min_gap), budget_range[1] + 1, I).astype(np.int32)
    S = np.array([rng.integers(1, b - min_gap + 2) for b in B], np.int32)
    S = np.minimum(S, cap_running).astype(np.int32)
    n_run = np.array([rng.integers(0, s + 1) for s in S], np.int32)
    n_wait = rng.integers(0, (cap_waiting if wait_max is None else wait_max) + 1, I).astype(np.int32)
    run_ctx = np.zeros((I, cap_running), np.int32)
    run_pre = np.zeros((I, cap_running), np.int32)
    run_dec = np.zeros((I, cap_running), np.int32)
    wait_pre = np.zeros((I, cap_waiting), np.int32)
    wait_dec = np.zeros((I, cap_waiting), np.int32)
    for j in range(I):
        n = n_run[j]
        run_ctx[j, :n] = rng.integers(0, max_ctx + 1, n)
        run_dec[j, :n] = rng.integers(1, max_dec + 1, n)
        if with_tail_prefill and n > 0 and rng.random() < 0.4:
            run_pre[j, n - 1] = rng.integers(1, max_pre + 1)
        w = n_wait[j]
        wait_pre[j, :w] = rng.integers(1, max_pre + 1, w)
        wait_dec[j, :w] = rng.integers(1, max_dec + 1, w)
    return B, S, n_run, run_ctx, run_pre, run_dec, n_wait, wait_pre, wait_dec


def small_workload(seed: int, num_instances: int = 6, num_models: int = 3, num_queries: int = 24,
                   cap_running: int = 8, cap_waiting: int = 8, max_prompt_len: int = 160,
                   first_token_mode: int = FIRST_TOKEN_SEPARATE_DECODE, budget_range=(4, 64),
                   with_tail_prefill: bool = True, min_gap: int = 1, wait_max: Optional[int] = None) -> Workload:
    """A random small pool (for property and parity tests on tiny inputs)."""
    rng = np.random.default_rng(seed)
    B, S, n_run, run_ctx, run_pre, run_dec, n_wait, wait_pre, wait_dec = random_small_state(
        rng, num_instances, cap_running, cap_waiting, budget_range=budget_range,
        with_tail_prefill=with_tail_prefill, min_gap=min_gap, wait_max=wait_max)
    alpha = rng.uniform(1.0, 10.0, num_models)
    beta = rng.uniform(0.01, 0.2, num_models)
    gamma = beta + rng.uniform(0.05, 0.5, num_models)
    coef = coefficients(alpha, beta, gamma)
    price = (rng.uniform(0.05, 3.0, num_models) * 1e-6).astype(np.float32)
    p = rng.integers(1, max_prompt_len + 1, num_queries).astype(np.int32)
    dec_hat = rng.integers(1, 50, (num_queries, num_models)).astype(np.int32)
    acc = rng.uniform(0, 1, (num_queries, num_models)).astype(np.float32)
    tau = ttft_targets(rng, p)
    moi = rng.integers(0, num_models, num_instances).astype(np.int32)
    return Workload(
        name=f"small{seed}", model_of_instance=moi, coef=coef, price_in=price.copy(),
        price_out=(price * 2).astype(np.float32), max_batched_tokens=B, max_seqs=S,
        cap_running=cap_running, cap_waiting=cap_waiting, n_run=n_run, run_ctx=run_ctx, run_pre=run_pre,
        run_dec=run_dec, n_wait=n_wait, wait_pre=wait_pre, wait_dec=wait_dec, prompt_len=p, dec_hat=dec_hat,
        acc=acc, tau=tau, lam=np.array([1.0], np.float32), mu=np.array([0.1], np.float32),
        max_prompt_len=max_prompt_len, first_token_mode=first_token_mode, seed=seed)
