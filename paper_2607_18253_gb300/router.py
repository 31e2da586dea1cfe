"""Thin Python binding of the C ABI in include/latency_router.h.

Argument marshalling only: every step of the estimator and the router runs in
the CUDA library (liblr.so).  PyTorch supplies device memory and the current
stream.  There is no CPU fallback: if the library is missing, construction
raises.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional, Sequence

import numpy as np
import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "_lib", "liblr.so")

LR_OK, LR_EINVAL, LR_ENOMEM, LR_ECUDA, LR_ECAPACITY, LR_ETRAJ, LR_ESTATE, LR_ENOSTATE = range(8)
FIRST_TOKEN_SEPARATE_DECODE = 0
FIRST_TOKEN_WITH_LAST_CHUNK = 1
LR_TTFT_SFS, LR_TTFT_THROUGHPUT, LR_TTFT_LPS = 0, 1, 2
LR_POLICY_ROUND_ROBIN, LR_POLICY_SHORTEST_QUEUE, LR_POLICY_LATENCY_AGNOSTIC = 0, 1, 2

EXPORTED_SYMBOLS = ("lr_create", "lr_destroy", "lr_load_state", "lr_estimate_ttft", "lr_estimate_features",
                    "lr_route", "lr_route_frontier_static", "lr_advance", "lr_read_state", "lr_status",
                    "lr_set_queue_params", "lr_set_ttft_source", "lr_calibrate", "lr_route_baseline",
                    "lr_on_time_utility", "lr_set_kv_limits", "lr_strerror", "lr_last_error",
                    "lr_track_first_tokens", "lr_advance_tracked")

_P = ctypes.c_void_p
_I32 = ctypes.c_int32


class _Config(ctypes.Structure):
    _fields_ = [("num_instances", _I32), ("num_models", _I32), ("model_of_instance", _P), ("coef", _P),
                ("price_in", _P), ("price_out", _P), ("max_batched_tokens", _P), ("max_seqs", _P),
                ("cap_running", _I32), ("cap_waiting", _I32), ("max_queries", _I32), ("max_pairs", _I32),
                ("max_prompt_len", _I32), ("first_token_mode", _I32), ("max_iters", _I32)]


class _QueueParams(ctypes.Structure):
    _fields_ = [("prefill_tput", _P), ("decode_batch_time", _P), ("arrival_rate", _P), ("service_rate", _P),
                ("parallelism", _P), ("arrival_scv", _P), ("service_scv", _P)]


class _StateView(ctypes.Structure):
    _fields_ = [("n_run", _P), ("run_ctx", _P), ("run_pre", _P), ("run_dec", _P), ("n_wait", _P),
                ("wait_pre", _P), ("wait_dec", _P)]


_lib = None


def load_library(path: str = LIB_PATH):
    """Load liblr.so (raises if it has not been built)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise RuntimeError(f"CUDA library not built: {path} is missing (run __graft_entry__.build())")
    lib = ctypes.CDLL(path)
    lib.lr_create.argtypes = [ctypes.POINTER(_Config), ctypes.POINTER(_P)]
    lib.lr_destroy.argtypes = [_P]
    lib.lr_load_state.argtypes = [_P, ctypes.POINTER(_StateView), _P]
    lib.lr_estimate_ttft.argtypes = [_P, _I32, _P, _P, _P, _P]
    lib.lr_estimate_features.argtypes = [_P, _I32, _P, _P, _P]
    lib.lr_route.argtypes = [_P, _I32, _P, _P, _P, _P, _I32, _P, _P, _P, _P, _P, _P, _P, _P]
    lib.lr_route_frontier_static.argtypes = [_P, _I32, _P, _P, _P, _P, _I32, _P, _P, _P, _P, _P, _P]
    lib.lr_advance.argtypes = [_P, _I32, _P, _P, _P, _I32, ctypes.c_double, _P]
    lib.lr_advance_tracked.argtypes = [_P, _I32, _P, _P, _P, _I32, ctypes.c_int64, ctypes.c_double, _P]
    lib.lr_track_first_tokens.argtypes = [_P, _P, ctypes.c_int64]
    lib.lr_set_queue_params.argtypes = [_P, ctypes.POINTER(_QueueParams), _P]
    lib.lr_set_ttft_source.argtypes = [_P, _I32]
    lib.lr_calibrate.argtypes = [_P, ctypes.c_int64, _P, _P, _P, _I32, _P, _P]
    lib.lr_route_baseline.argtypes = [_P, _I32, _I32, _P, _P, _P, ctypes.c_float, ctypes.c_int64, _P, _P, _P, _P]
    lib.lr_on_time_utility.argtypes = [_P, _I32, _P, _P, _P, _P, _P, _P]
    lib.lr_set_kv_limits.argtypes = [_P, _P, _P, _P, _I32]
    lib.lr_read_state.argtypes = [_P, _P, _P, _P, _P, _P, _P, _P, _P, _P]
    lib.lr_status.argtypes = [_P, _P]
    lib.lr_strerror.argtypes = [ctypes.c_int]
    lib.lr_strerror.restype = ctypes.c_char_p
    lib.lr_last_error.argtypes = [_P]
    lib.lr_last_error.restype = ctypes.c_char_p
    for name in ("lr_create", "lr_destroy", "lr_load_state", "lr_estimate_ttft", "lr_estimate_features",
                 "lr_route", "lr_route_frontier_static", "lr_advance", "lr_read_state", "lr_status",
                 "lr_set_queue_params", "lr_set_ttft_source", "lr_calibrate", "lr_route_baseline",
                 "lr_on_time_utility", "lr_set_kv_limits", "lr_advance_tracked", "lr_track_first_tokens"):
        getattr(lib, name).restype = ctypes.c_int
    _lib = lib
    return lib


class LRError(RuntimeError):
    def __init__(self, code: int, detail: str = ""):
        lib = load_library()
        msg = lib.lr_strerror(code).decode()
        super().__init__(f"{msg} (code {code})" + (f": {detail}" if detail else ""))
        self.code = code


def _dev(t: Optional[torch.Tensor], dtype: torch.dtype, name: str, numel: Optional[int] = None):
    if t is None:
        return None
    if not isinstance(t, torch.Tensor) or not t.is_cuda:
        raise TypeError(f"{name} must be a CUDA tensor")
    if t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if numel is not None and t.numel() != numel:
        raise ValueError(f"{name} must have {numel} elements, got {t.numel()}")
    return ctypes.c_void_p(t.data_ptr())


def _stream(stream) -> ctypes.c_void_p:
    s = torch.cuda.current_stream() if stream is None else stream
    return ctypes.c_void_p(s.cuda_stream)


class LatencyRouter:
    """A router context: pool description, a live snapshot and the kernels."""

    def __init__(self, *, model_of_instance, coef, price_in, price_out, max_batched_tokens, max_seqs,
                 cap_running: int, cap_waiting: int, max_queries: int, max_prompt_len: int, max_pairs: int = 1,
                 first_token_mode: int = FIRST_TOKEN_SEPARATE_DECODE, max_iters: int = 1 << 22):
        self._lib = load_library()
        self._keep = [np.ascontiguousarray(model_of_instance, np.int32), np.ascontiguousarray(coef, np.float32),
                      np.ascontiguousarray(price_in, np.float32), np.ascontiguousarray(price_out, np.float32),
                      np.ascontiguousarray(max_batched_tokens, np.int32), np.ascontiguousarray(max_seqs, np.int32)]
        moi, cf, pin, pout, B, S = self._keep
        self.num_instances = int(moi.shape[0])
        self.num_models = int(cf.shape[0])
        self.cap_running, self.cap_waiting = int(cap_running), int(cap_waiting)
        self.max_queries, self.max_pairs = int(max_queries), int(max_pairs)
        cfg = _Config(self.num_instances, self.num_models, *(a.ctypes.data_as(_P) for a in (moi, cf, pin, pout, B, S)),
                      self.cap_running, self.cap_waiting, self.max_queries, self.max_pairs, int(max_prompt_len),
                      int(first_token_mode), int(max_iters))
        torch.cuda.init()
        h = _P()
        rc = self._lib.lr_create(ctypes.byref(cfg), ctypes.byref(h))
        if rc != LR_OK:
            raise LRError(rc, "lr_create")
        self._h = h

    @classmethod
    def from_workload(cls, wl, max_queries: Optional[int] = None, max_pairs: Optional[int] = None,
                      max_iters: int = 1 << 22) -> "LatencyRouter":
        return cls(model_of_instance=wl.model_of_instance, coef=wl.coef, price_in=wl.price_in,
                   price_out=wl.price_out, max_batched_tokens=wl.max_batched_tokens, max_seqs=wl.max_seqs,
                   cap_running=wl.cap_running, cap_waiting=wl.cap_waiting,
                   max_queries=max(1, wl.num_queries if max_queries is None else max_queries),
                   max_prompt_len=wl.max_prompt_len, max_pairs=max(1, wl.num_pairs if max_pairs is None else max_pairs),
                   first_token_mode=wl.first_token_mode, max_iters=max_iters)

    def close(self):
        if getattr(self, "_h", None):
            self._lib.lr_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def _check(self, rc: int, what: str):
        if rc != LR_OK:
            raise LRError(rc, f"{what}: {self._lib.lr_last_error(self._h).decode()}")

    def load_state(self, n_run, run_ctx, run_pre, run_dec, n_wait, wait_pre, wait_dec, stream=None):
        I, R, W = self.num_instances, self.cap_running, self.cap_waiting
        v = _StateView(_dev(n_run, torch.int32, "n_run", I), _dev(run_ctx, torch.int32, "run_ctx", I * R),
                       _dev(run_pre, torch.int32, "run_pre", I * R), _dev(run_dec, torch.int32, "run_dec", I * R),
                       _dev(n_wait, torch.int32, "n_wait", I), _dev(wait_pre, torch.int32, "wait_pre", I * W),
                       _dev(wait_dec, torch.int32, "wait_dec", I * W))
        self._check(self._lib.lr_load_state(self._h, ctypes.byref(v), _stream(stream)), "lr_load_state")

    def estimate_ttft(self, prompt_len: torch.Tensor, out: Optional[torch.Tensor] = None,
                      first_batch: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
        Q, I = int(prompt_len.numel()), self.num_instances
        if out is None:
            out = torch.empty((Q, I), dtype=torch.float32, device=prompt_len.device)
        self._check(self._lib.lr_estimate_ttft(self._h, Q, _dev(prompt_len, torch.int32, "prompt_len"),
                                               _dev(out, torch.float32, "ttft_out", Q * I),
                                               _dev(first_batch, torch.int32, "first_batch_out", Q * I),
                                               _stream(stream)), "lr_estimate_ttft")
        return out

    def estimate_features(self, prompt_len: torch.Tensor, out: Optional[torch.Tensor] = None,
                          stream=None) -> torch.Tensor:
        Q, I = int(prompt_len.numel()), self.num_instances
        if out is None:
            out = torch.empty((Q, I, 5), dtype=torch.int64, device=prompt_len.device)
        self._check(self._lib.lr_estimate_features(self._h, Q, _dev(prompt_len, torch.int32, "prompt_len"),
                                                   _dev(out, torch.int64, "features_out", Q * I * 5),
                                                   _stream(stream)), "lr_estimate_features")
        return out

    def route(self, prompt_len: torch.Tensor, dec_hat: torch.Tensor, acc: torch.Tensor, lam: Sequence[float],
              mu: Optional[Sequence[float]] = None, tau: Optional[torch.Tensor] = None,
              ttft_chosen: bool = True, frontier: bool = False, ttft_matrix: Optional[torch.Tensor] = None,
              out: Optional[dict] = None, stream=None) -> dict:
        """Route every query for each (lambda, mu) pair; returns a dict of device tensors."""
        Q, M = int(prompt_len.numel()), self.num_models
        lam_h = np.ascontiguousarray(np.atleast_1d(np.asarray(lam, np.float32)))
        P = int(lam_h.shape[0])
        mu_h = None if mu is None else np.ascontiguousarray(np.atleast_1d(np.asarray(mu, np.float32)))
        if mu_h is not None and mu_h.shape[0] != P:
            raise ValueError("lam and mu must have the same length")
        dev = prompt_len.device
        o = {} if out is None else out
        if "assign" not in o:
            o["assign"] = torch.empty((P, Q), dtype=torch.int32, device=dev)
            o["util"] = torch.empty((P, Q), dtype=torch.float32, device=dev)
        if ttft_chosen and "ttft_chosen" not in o:
            o["ttft_chosen"] = torch.empty((P, Q), dtype=torch.float32, device=dev)
        if frontier and "frontier" not in o:
            o["frontier"] = torch.empty((P, 3), dtype=torch.float64, device=dev)
        if ttft_matrix is not None:
            o["ttft_matrix"] = ttft_matrix
        rc = self._lib.lr_route(
            self._h, Q, _dev(prompt_len, torch.int32, "prompt_len"), _dev(dec_hat, torch.int32, "dec_hat", Q * M),
            _dev(acc, torch.float32, "acc", Q * M), _dev(tau, torch.float32, "tau", Q), P,
            lam_h.ctypes.data_as(_P), None if mu_h is None else mu_h.ctypes.data_as(_P),
            _dev(o["assign"], torch.int32, "assign_out", P * Q), _dev(o["util"], torch.float32, "util_out", P * Q),
            _dev(o.get("ttft_chosen") if ttft_chosen else None, torch.float32, "ttft_chosen_out", P * Q),
            _dev(o.get("frontier") if frontier else None, torch.float64, "frontier_out", P * 3),
            _dev(ttft_matrix, torch.float32, "ttft_matrix_out", Q * self.num_instances), _stream(stream))
        self._check(rc, "lr_route")
        return o

    def route_frontier_static(self, prompt_len: torch.Tensor, dec_hat: torch.Tensor, acc: torch.Tensor,
                              lam: Sequence[float], mu: Optional[Sequence[float]] = None,
                              tau: Optional[torch.Tensor] = None, out: Optional[dict] = None, stream=None) -> dict:
        """route(..., frontier=True, ttft_chosen=False) whose intermediate lives in static device memory.

        The C call allocates nothing; pass preallocated tensors in `out` ("assign",
        "util", "frontier") to keep this wrapper from allocating them."""
        Q, M = int(prompt_len.numel()), self.num_models
        lam_h = np.ascontiguousarray(np.atleast_1d(np.asarray(lam, np.float32)))
        P = int(lam_h.shape[0])
        mu_h = None if mu is None else np.ascontiguousarray(np.atleast_1d(np.asarray(mu, np.float32)))
        if mu_h is not None and mu_h.shape[0] != P:
            raise ValueError("lam and mu must have the same length")
        dev = prompt_len.device
        o = {} if out is None else out
        if "assign" not in o:
            o["assign"] = torch.empty((P, Q), dtype=torch.int32, device=dev)
            o["util"] = torch.empty((P, Q), dtype=torch.float32, device=dev)
        if "frontier" not in o:
            o["frontier"] = torch.empty((P, 3), dtype=torch.float64, device=dev)
        rc = self._lib.lr_route_frontier_static(
            self._h, Q, _dev(prompt_len, torch.int32, "prompt_len"), _dev(dec_hat, torch.int32, "dec_hat", Q * M),
            _dev(acc, torch.float32, "acc", Q * M), _dev(tau, torch.float32, "tau", Q), P,
            lam_h.ctypes.data_as(_P), None if mu_h is None else mu_h.ctypes.data_as(_P),
            _dev(o["assign"], torch.int32, "assign_out", P * Q), _dev(o["util"], torch.float32, "util_out", P * Q),
            _dev(o["frontier"], torch.float64, "frontier_out", P * 3), _stream(stream))
        self._check(rc, "lr_route_frontier_static")
        return o

    def route_baseline(self, policy: int, prompt_len: torch.Tensor, dec_hat: torch.Tensor, acc: torch.Tensor,
                       lam: float, rr_start: int = 0, out: Optional[dict] = None, stream=None) -> dict:
        """A baseline router (LR_POLICY_*): {"assign", "util", "ttft_chosen"} [Q] on the device."""
        Q, M = int(prompt_len.numel()), self.num_models
        dev = prompt_len.device
        o = {} if out is None else out
        if "assign" not in o:
            o["assign"] = torch.empty(Q, dtype=torch.int32, device=dev)
            o["util"] = torch.empty(Q, dtype=torch.float32, device=dev)
            o["ttft_chosen"] = torch.empty(Q, dtype=torch.float32, device=dev)
        rc = self._lib.lr_route_baseline(
            self._h, int(policy), Q, _dev(prompt_len, torch.int32, "prompt_len"),
            _dev(dec_hat, torch.int32, "dec_hat", Q * M), _dev(acc, torch.float32, "acc", Q * M), float(lam),
            int(rr_start), _dev(o["assign"], torch.int32, "assign_out", Q), _dev(o["util"], torch.float32, "util_out", Q),
            _dev(o.get("ttft_chosen"), torch.float32, "ttft_chosen_out", Q), _stream(stream))
        self._check(rc, "lr_route_baseline")
        return o

    def on_time_utility(self, util: torch.Tensor, ttft: torch.Tensor, tau: torch.Tensor,
                        delay: Optional[torch.Tensor] = None, out: Optional[torch.Tensor] = None,
                        stream=None) -> torch.Tensor:
        """[OnTimeUtility (Eq. 4), SLO attainment] as a float64 device tensor of 2."""
        Q = int(util.numel())
        o = torch.empty(2, dtype=torch.float64, device=util.device) if out is None else out
        rc = self._lib.lr_on_time_utility(
            self._h, Q, _dev(util, torch.float32, "util", Q), _dev(ttft, torch.float32, "ttft", Q),
            _dev(tau, torch.float32, "tau", Q), _dev(delay, torch.float32, "delay", Q),
            _dev(o, torch.float64, "out", 2), _stream(stream))
        self._check(rc, "lr_on_time_utility")
        return o

    def set_queue_params(self, prefill_tput, decode_batch_time, arrival_rate=None, service_rate=None,
                         parallelism=None, arrival_scv=None, service_scv=None, stream=None):
        """Per-instance parameters of the average-case TTFT sources (host arrays of length I)."""
        I = self.num_instances

        def arr(x, dt):
            return None if x is None else np.ascontiguousarray(np.broadcast_to(np.asarray(x, dt), (I,)))

        keep = [arr(prefill_tput, np.float64), arr(decode_batch_time, np.float64), arr(arrival_rate, np.float64),
                arr(service_rate, np.float64), arr(parallelism, np.int32), arr(arrival_scv, np.float64),
                arr(service_scv, np.float64)]
        qp = _QueueParams(*(None if k is None else k.ctypes.data_as(_P) for k in keep))
        self._check(self._lib.lr_set_queue_params(self._h, ctypes.byref(qp), _stream(stream)), "lr_set_queue_params")

    def set_ttft_source(self, source: int):
        """LR_TTFT_SFS (default), LR_TTFT_THROUGHPUT or LR_TTFT_LPS."""
        self._check(self._lib.lr_set_ttft_source(self._h, int(source)), "lr_set_ttft_source")

    def set_kv_limits(self, block_size=None, num_blocks=None, max_ctx=None, horizon: int = 4096):
        """KV-cache block limits, context limits and preemption in the simulated step rule
        (host arrays of length I, or scalars for every instance); all None turns them off.
        Drops the live snapshot: load one again before estimating."""
        I = self.num_instances
        if block_size is None and num_blocks is None and max_ctx is None:
            self._check(self._lib.lr_set_kv_limits(self._h, None, None, None, 0), "lr_set_kv_limits")
            return
        keep = [np.ascontiguousarray(np.broadcast_to(np.asarray(x, dt), (I,)))
                for x, dt in ((block_size, np.int32), (num_blocks, np.int64), (max_ctx, np.int64))]
        self._check(self._lib.lr_set_kv_limits(self._h, *(k.ctypes.data_as(_P) for k in keep), int(horizon)),
                    "lr_set_kv_limits")

    def calibrate(self, features: torch.Tensor, model: torch.Tensor, time: torch.Tensor, shared_beta1: bool = True,
                  out: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
        """Least-squares batch-time coefficients per model, [M, 5] fp64, from a batch log."""
        N = int(model.numel())
        if out is None:
            out = torch.empty((self.num_models, 5), dtype=torch.float64, device=model.device)
        self._check(self._lib.lr_calibrate(self._h, N, _dev(features, torch.int64, "features", N * 5),
                                           _dev(model, torch.int32, "model", N), _dev(time, torch.float64, "time", N),
                                           1 if shared_beta1 else 0, _dev(out, torch.float64, "coef_out", self.num_models * 5),
                                           _stream(stream)), "lr_calibrate")
        return out

    def advance(self, assign: torch.Tensor, prompt_len: torch.Tensor, dec: torch.Tensor, t_now: float,
                stream=None, id_base: Optional[int] = None):
        """Append routed queries (assign[i] >= 0) and advance every instance to t_now.

        dec is [Q] (one output length per query) or [Q, M] (the chosen model's column is used).
        id_base: track query i of this call as id id_base + i (lr_advance_tracked)."""
        Q = int(assign.numel())
        cols = 1 if dec.dim() == 1 else int(dec.shape[1])
        args = (_dev(assign, torch.int32, "assign"), _dev(prompt_len, torch.int32, "prompt_len", Q),
                _dev(dec, torch.int32, "dec", Q * cols), cols)
        if id_base is None:
            rc = self._lib.lr_advance(self._h, Q, *args, float(t_now), _stream(stream))
        else:
            rc = self._lib.lr_advance_tracked(self._h, Q, *args, int(id_base), float(t_now), _stream(stream))
        self._check(rc, "lr_advance")

    def track_first_tokens(self, first_token_time: Optional[torch.Tensor]):
        """Record tracked queries' first-token times into first_token_time [N] fp64 (None: off)."""
        if first_token_time is None:
            self._check(self._lib.lr_track_first_tokens(self._h, None, 0), "lr_track_first_tokens")
            return
        self._check(self._lib.lr_track_first_tokens(self._h, _dev(first_token_time, torch.float64,
                                                                  "first_token_time"),
                                                    int(first_token_time.numel())),
                    "lr_track_first_tokens")

    def read_state(self, device="cuda", stream=None) -> dict:
        """The live snapshot as device tensors (n_run, run_ctx, ..., wait_dec, clock)."""
        I, R, W = self.num_instances, self.cap_running, self.cap_waiting
        out = {"n_run": torch.empty(I, dtype=torch.int32, device=device),
               "run_ctx": torch.empty((I, R), dtype=torch.int32, device=device),
               "run_pre": torch.empty((I, R), dtype=torch.int32, device=device),
               "run_dec": torch.empty((I, R), dtype=torch.int32, device=device),
               "n_wait": torch.empty(I, dtype=torch.int32, device=device),
               "wait_pre": torch.empty((I, W), dtype=torch.int32, device=device),
               "wait_dec": torch.empty((I, W), dtype=torch.int32, device=device),
               "clock": torch.empty(I, dtype=torch.float64, device=device)}
        rc = self._lib.lr_read_state(self._h, *(ctypes.c_void_p(out[k].data_ptr()) for k in
                                                ("n_run", "run_ctx", "run_pre", "run_dec", "n_wait", "wait_pre",
                                                 "wait_dec", "clock")), _stream(stream))
        self._check(rc, "lr_read_state")
        return out

    def status(self, stream=None) -> int:
        """Synchronize the stream; return and clear the device status word."""
        rc = self._lib.lr_status(self._h, _stream(stream))
        return int(rc)


def state_tensors(wl, device="cuda"):
    """The snapshot arrays of a workload as device tensors (in lr_state_view order)."""
    return [torch.from_numpy(np.ascontiguousarray(a, np.int32)).to(device)
            for a in (wl.n_run, wl.run_ctx, wl.run_pre, wl.run_dec, wl.n_wait, wl.wait_pre, wl.wait_dec)]


def query_tensors(wl, device="cuda"):
    """prompt_len, dec_hat, acc, tau of a workload as device tensors."""
    return (torch.from_numpy(np.ascontiguousarray(wl.prompt_len, np.int32)).to(device),
            torch.from_numpy(np.ascontiguousarray(wl.dec_hat, np.int32)).to(device),
            torch.from_numpy(np.ascontiguousarray(wl.acc, np.float32)).to(device),
            torch.from_numpy(np.ascontiguousarray(wl.tau, np.float32)).to(device))
