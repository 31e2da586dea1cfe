"""Benchmark of the router hot path on one GB300 (or N independent replicas).

A step is one pass of the whole hot path over one batch: ingest the instance
snapshot (copy + per-instance trajectory summary) and route every query of the
batch -- SFS TTFT for every (query, instance) candidate written as the full
estimate matrix, utility, Lagrangian argmax.  Workload: "pool256", 256
instances (8 models x 32 replicas) and 65,536 queries, seeded synthetic.  As in
a serving loop (App. F), the snapshot ingest of a step runs on one stream while
its batch is routed on another against the most recent complete snapshot; the
same steps run back to back on one stream give the per-kernel times.

value      = candidates (query x instance) per second, device time, inputs resident
e2e        = same metric through the public API from pinned host buffers, with the
             host->device copy of the snapshot and queries and the device->host copy
             of the routing result inside each timed step
roofline   = the SFS estimate call (lr_estimate_ttft, the full Q x I matrix) on the same
             workload against measured HBM bandwidth; per-kernel figures of the step
             (route, K1) under "kernels"
configs    = the other single-GPU configurations (tiny, pool64, the 32-pair sweep)
cpu_baseline / --impl reference = the CPU oracle (literal per-candidate simulation) on
             every host core (and one core), with the host's core count and CPU model
"""
import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "TTFT estimates/sec (query×instance) on 1 GB300; p50 per-batch route latency"
UNIT = "estimates/s"
WORKLOAD = "pool256"
# DRAM bytes (read + write) per launch of the step's kernels on this workload, from one
# ncu capture of the kernels as they are built now (summaries under profiles/); they
# are retaken whenever one of the kernels changes.
NCU_TRAFFIC = {"k_route": 4_577_792 + 8_019_712, "k_trajectory": 1_401_344, "k_estimate": 357_888 + 7_386_624,
               "k_calibrate": 208_430_848 + 3_465_728}


def _peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


def _dist():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def _max_over_ranks(x: float, world: int) -> float:
    """The largest of the ranks' values (the slowest rank's time); x itself on one rank."""
    if world <= 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def _job_rate(units_per_rank: float, world: int, ms: float) -> float:
    """Whole-job throughput: the units every rank processed over the slowest rank's time."""
    return units_per_rank * world / (ms * 1e-3)


def _config_desc(wl, extra=None):
    d = {"workload": f"{WORKLOAD}: {wl.num_instances} instances ({wl.num_models} models x "
                     f"{wl.num_instances // wl.num_models} replicas) x {wl.num_queries} queries, "
                     f"B={int(wl.max_batched_tokens[0])}, S={int(wl.max_seqs[0])}, prompts <= {wl.max_prompt_len}",
         "instances": wl.num_instances, "queries_per_batch": wl.num_queries,
         "step": "lr_load_state (K1, new snapshot) on one stream overlapped with lr_route (K2: full TTFT "
                 "matrix, Lagrangian argmax) on a second, routing against the most recent complete snapshot "
                 "(App. F); one CUDA graph per step",
         "l2": "flushed (256 MiB write) between timed steps",
         "parallelism": "replicas"}
    if extra:
        d.update(extra)
    return d


class Clocks:
    """nvidia-smi sampling of SM clocks and throttle reasons during the timed region."""

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        # the raw samples (one CSV per rank) go to LR_CLOCK_DIR, else the system temp dir
        self.path = os.path.join(os.environ.get("LR_CLOCK_DIR", tempfile.gettempdir()), f"lr_clocks_rank{index}.csv")

    def __enter__(self):
        try:
            os.makedirs(os.path.dirname(self.path), exist_ok=True)
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.index}",
                 "--query-gpu=index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
                 "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
                 "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap",
                 "--format=csv,noheader,nounits", "-lms", "100"], stdout=self.f, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()
            self.f.close()

    def summary(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        sm, smax, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        try:
            for line in open(self.path):
                parts = [x.strip() for x in line.split(",")]
                if len(parts) < 9:
                    continue
                try:
                    sm.append(float(parts[1]))
                    smax = float(parts[2])
                except ValueError:
                    continue
                for n, v in zip(names, parts[5:9]):
                    if v.lower() == "active":
                        reasons.add(n)
        except OSError:
            pass
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": smax, "samples": len(sm),
                "reasons": sorted(reasons)}


def run_gpu(args):
    import torch
    import torch.distributed as dist

    import __graft_entry__
    from paper_2607_18253_gb300 import router as R
    from paper_2607_18253_gb300 import workloads as W

    rank, world, local = _dist()
    if world > 1:
        dist.init_process_group("gloo")
    torch.cuda.set_device(local)
    if rank == 0:
        __graft_entry__.build()
    if world > 1:
        dist.barrier()
    dev = torch.device("cuda", local)

    wl = W.make_workload(WORKLOAD)
    Q, I, M = wl.num_queries, wl.num_instances, wl.num_models
    rt = R.LatencyRouter.from_workload(wl)
    state = R.state_tensors(wl, dev)
    p, dh, acc, _ = R.query_tensors(wl, dev)
    mat = torch.empty((Q, I), dtype=torch.float32, device=dev)
    out = {"assign": torch.empty((1, Q), dtype=torch.int32, device=dev),
           "util": torch.empty((1, Q), dtype=torch.float32, device=dev),
           "ttft_chosen": torch.empty((1, Q), dtype=torch.float32, device=dev)}
    flush = torch.empty(64 << 20, dtype=torch.float32, device=dev)  # 256 MiB > L2
    stream = torch.cuda.current_stream()

    # The step is captured once into CUDA graphs (snapshot ingest, routing) and
    # replayed, so the timed region holds no host-side launch work.
    side = torch.cuda.Stream(device=dev)
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        for _ in range(args.warmup):
            rt.load_state(*state)
            rt.route(p, dh, acc, wl.lam, wl.mu, ttft_matrix=mat, out=out)
    torch.cuda.current_stream().wait_stream(side)
    torch.cuda.synchronize()
    st = rt.status()
    if st != R.LR_OK:
        raise RuntimeError(f"device status {st} after warm-up")
    g_load, g_route = torch.cuda.CUDAGraph(), torch.cuda.CUDAGraph()
    with torch.cuda.graph(g_load):
        rt.load_state(*state)
    with torch.cuda.graph(g_route):
        rt.route(p, dh, acc, wl.lam, wl.mu, ttft_matrix=mat, out=out)
    for _ in range(args.warmup):
        flush.fill_(1.0)
        g_load.replay()
        g_route.replay()
    torch.cuda.synchronize()

    # The step as a serving loop runs it (App. F): the snapshot is summarized (K1) on
    # this stream while the batch is routed (K2) on a second one against the most
    # recent complete snapshot; one graph per step (fork, K1 || K2, join), so the next
    # step's load starts only after this step's routing has finished.
    g_pipe = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g_pipe):
        main = torch.cuda.current_stream()
        side.wait_stream(main)
        rt.load_state(*state, stream=main)
        with torch.cuda.stream(side):
            rt.route(p, dh, acc, wl.lam, wl.mu, ttft_matrix=mat, out=out, stream=side)
        main.wait_stream(side)
    for _ in range(args.warmup):
        flush.fill_(1.0)
        g_pipe.replay()
    torch.cuda.synchronize()

    K = args.steps
    evp = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(K)]
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    with Clocks(local) as clk:
        # the same step replayed back to back for args.sustain_seconds first, so that the
        # clock sampler (one sample per 100 ms) sees the GPU under this load; then the K
        # timed steps
        t_s0 = time.perf_counter()
        ev_s = (torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
        ev_s[0].record(stream)
        sustained = 0
        while time.perf_counter() - t_s0 < args.sustain_seconds:
            for _ in range(256):
                flush.fill_(1.0)
                g_pipe.replay()
            sustained += 256
            torch.cuda.synchronize()
        ev_s[1].record(stream)
        t_wall0 = time.perf_counter()
        for k in range(K):
            flush.fill_(float(k))
            evp[k][0].record(stream)
            g_pipe.replay()
            evp[k][1].record(stream)
        torch.cuda.synchronize()
        t_wall = time.perf_counter() - t_wall0
    sustained_ms = ev_s[0].elapsed_time(ev_s[1])
    if world > 1:
        dist.barrier()
    assert rt.status() == R.LR_OK
    step_ms = [e0.elapsed_time(e1) for e0, e1 in evp]
    total_ms = _max_over_ranks(sum(step_ms), world)
    ms_per_step = total_ms / K

    # The same steps with K1 and K2 in sequence: each kernel's own duration (roofline,
    # shares) and the non-overlapped step time.
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(K)]
    for k in range(K):
        flush.fill_(float(k))
        ev[k][0].record(stream)
        g_load.replay()
        ev[k][1].record(stream)
        g_route.replay()
        ev[k][2].record(stream)
    torch.cuda.synchronize()
    assert rt.status() == R.LR_OK
    load_ms = [ev[k][0].elapsed_time(ev[k][1]) for k in range(K)]
    route_ms = [ev[k][1].elapsed_time(ev[k][2]) for k in range(K)]
    seq_ms = sum(a + b for a, b in zip(load_ms, route_ms)) / K
    cands = Q * I
    value = _job_rate(cands, world, ms_per_step)

    # End to end, as a serving loop runs it: every step copies its snapshot and queries
    # from pinned host memory, ingests and routes them (K1 || K2 as above) and copies
    # the routing result back to pinned host memory, which the host reads.  NB buffer
    # sets rotate, so step k+1's upload (copy stream) overlaps step k's compute, and the
    # host waits for each step's result HOST_LAG steps later (NB > HOST_LAG keeps that
    # result's host buffer from being overwritten before it is read).
    # The step's inputs (snapshot arrays, then prompts, predicted lengths and accuracies)
    # sit in one pinned host buffer and arrive with one copy; the routing results go back
    # with one copy too (one large copy moves ~200 GB/s here, ten separate ones far less).
    ins = list(state) + [p, dh, acc]
    sizes = [t.numel() for t in ins]
    offs = np.concatenate([[0], np.cumsum(sizes)]).astype(np.int64)
    host_in = torch.empty(int(offs[-1]), dtype=torch.int32).pin_memory()
    for t, o, n in zip(ins, offs[:-1], sizes):
        host_in[o:o + n].copy_(t.reshape(-1).view(torch.int32).cpu())

    def views(flat):
        # int32 views in the order of `ins`; the last one (accuracies) as fp32
        v = [flat[o:o + n].view(t.shape) for t, o, n in zip(ins, offs[:-1], sizes)]
        v[-1] = v[-1].view(torch.float32)
        return v[:len(state)], v[len(state):]

    res_keys = ("assign", "util", "ttft_chosen")
    NB, HOST_LAG = 3, 2
    dev_in = [torch.empty(int(offs[-1]), dtype=torch.int32, device=dev) for _ in range(NB)]
    bufs = [views(f) for f in dev_in]
    dev_out = [torch.empty(3 * Q, dtype=torch.int32, device=dev) for _ in range(NB)]
    outs = [{"assign": f[:Q].view(1, Q), "util": f[Q:2 * Q].view(torch.float32).view(1, Q),
             "ttft_chosen": f[2 * Q:].view(torch.float32).view(1, Q)} for f in dev_out]
    host_out_flat = [torch.empty(3 * Q, dtype=torch.int32).pin_memory() for _ in range(NB)]
    host_outs = [{"assign": f[:Q].view(1, Q)} for f in host_out_flat]
    h2d = int(offs[-1]) * 4
    d2h = 3 * Q * 4
    copy_stream = torch.cuda.Stream(device=dev)
    g_up, g_step = [], []
    for b in range(NB):
        dst, dqq = bufs[b]

        def upload(b=b):
            dev_in[b].copy_(host_in, non_blocking=True)

        def step(b=b, dst=dst, dqq=dqq):
            main = torch.cuda.current_stream()
            side.wait_stream(main)
            rt.load_state(*dst, stream=main)
            with torch.cuda.stream(side):
                rt.route(dqq[0], dqq[1], dqq[2], wl.lam, wl.mu, ttft_matrix=mat, out=outs[b], stream=side)
            main.wait_stream(side)

        upload()
        step()
        host_out_flat[b].copy_(dev_out[b], non_blocking=True)
        torch.cuda.synchronize()
        gu, gs = torch.cuda.CUDAGraph(), torch.cuda.CUDAGraph()
        with torch.cuda.graph(gu):
            upload()
        with torch.cuda.graph(gs):
            step()
        g_up.append(gu)
        g_step.append(gs)

    d2h_stream = torch.cuda.Stream(device=dev)

    def run_e2e(steps):
        # `steps` pipelined steps with no L2 flush inside the loop (each step's inputs
        # arrive by their own host->device copy).  Three streams: uploads, compute and
        # read-backs, so that step k's read-back and step k+1's upload overlap step
        # k+1's compute; the host waits for step k - HOST_LAG's result after issuing
        # step k.  Returns the span from the first upload's issue to the last result's
        # arrival in host memory, and each step's latency from its upload's issue to
        # its result's arrival.
        ev_up0 = [torch.cuda.Event(enable_timing=True) for _ in range(steps)]
        ev1 = [torch.cuda.Event() for _ in range(steps)]          # compute done
        ev2 = [torch.cuda.Event(enable_timing=True) for _ in range(steps)]  # result in host memory
        up = [torch.cuda.Event() for _ in range(steps)]
        for k in range(steps):
            b = k % NB
            if k >= NB:
                copy_stream.wait_event(ev1[k - NB])  # step k-NB has read buffer set b's inputs
            ev_up0[k].record(copy_stream)
            with torch.cuda.stream(copy_stream):
                g_up[b].replay()
            up[k].record(copy_stream)
            stream.wait_event(up[k])
            if k >= NB:
                stream.wait_event(ev2[k - NB])  # step k-NB's results have left buffer set b
            g_step[b].replay()
            ev1[k].record(stream)
            d2h_stream.wait_event(ev1[k])
            with torch.cuda.stream(d2h_stream):
                host_out_flat[b].copy_(dev_out[b], non_blocking=True)
            ev2[k].record(d2h_stream)
            if k >= HOST_LAG:
                ev2[k - HOST_LAG].synchronize()  # the host has step k-HOST_LAG's result
        torch.cuda.synchronize()
        return ev_up0[0].elapsed_time(ev2[-1]), [ev_up0[k].elapsed_time(ev2[k]) for k in range(steps)]

    run_e2e(max(3, args.warmup))
    KE = max(3, min(K, 2000))
    e2e_span, e2e_lat = run_e2e(KE)
    e2e_mean = _max_over_ranks(e2e_span / KE, world)
    host_out = host_outs[(KE - 1) % NB]
    out = outs[(KE - 1) % NB]
    assert rt.status() == R.LR_OK
    ok = torch.equal(host_out["assign"].to(dev), out["assign"])
    if not ok:
        raise RuntimeError("end-to-end result differs from the device result")

    # roofline of the dominant kernel (algorithmic bytes / event-timed duration)
    hbm, peak_src = _peaks()
    load_avg = sum(load_ms) / K
    route_avg = sum(route_ms) / K
    route_bytes = cands * 4 + Q * (4 + 8 * M) + Q * 12
    load_bytes = 2 * 4 * (I * (3 * wl.cap_running + 2 * wl.cap_waiting) + 2 * I)
    kernels = {
        "k_route (TTFT matrix + utility + argmax)": {
            "ms": route_avg, "share": route_avg / seq_ms, "algorithmic_bytes": route_bytes,
            "hbm_frac": route_bytes / (route_avg * 1e-3) / 1e9 / hbm, "dram_bytes_ncu": NCU_TRAFFIC["k_route"]},
        "k_trajectory (snapshot copy + summary)": {
            "ms": load_avg, "share": load_avg / seq_ms, "algorithmic_bytes": load_bytes,
            "hbm_frac": load_bytes / (load_avg * 1e-3) / 1e9 / hbm, "dram_bytes_ncu": NCU_TRAFFIC["k_trajectory"],
            "bound": "dependency-latency chain of the slowest instance"},
    }
    # the line's roofline: the SFS estimate call (lr_estimate_ttft) on this workload,
    # HBM-bound (the full Q x I fp32 matrix written, the prompts and the summary read)
    estimate = run_estimate(args, dev, wl, flush)
    roof = dict(estimate["roofline"])
    roof["call"] = estimate["call"]
    roof["target"] = "frac >= 0.5 (the 256-instance x 65,536-query configuration)"
    roof["target_met"] = bool(roof["frac"] >= 0.5)
    configs = run_configs(args, dev, flush)
    kv = run_kv(args, dev, wl, flush)
    avgcase = run_avgcase(args, dev, wl, flush)
    calibration = run_calibration(args, dev, flush)
    stream = None if args.no_stream else run_stream(args, dev)
    policy_eval = None if args.no_stream else run_policy_eval(args, dev)

    if rank == 0:
        cpu = cpu_baseline(wl, args.cpu_seconds) if (world == 1 and not args.no_cpu) else None
        srt = sorted(step_ms)
        elat = sorted(e2e_lat)
        clocks = clk.summary()
        if clocks.get("sm_mhz"):
            clocks["ms_x_mhz_per_step"] = ms_per_step * clocks["sm_mhz"]
        clocks["sampled_region"] = (f"{sustained} back-to-back steps ({sustained_ms / 1e3:.2f} s) then the "
                                    f"{K} timed steps")
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": K, "warmup": args.warmup,
            "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "f32+i64", "data": "synthetic (seeded lognormal/uniform stand-ins for the paper's workloads)",
            "config": _config_desc(wl),
            "p50_step_ms": srt[len(srt) // 2], "p99_step_ms": srt[min(len(srt) - 1, int(0.99 * len(srt)))],
            "roofline": roof, "kernels": kernels, "cpu_baseline": cpu,
            "e2e": {"value": _job_rate(cands, world, e2e_mean), "unit": UNIT, "ms_per_step": e2e_mean,
                    "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "steps": KE,
                    "p50_latency_ms": elat[len(elat) // 2],
                    "p99_latency_ms": elat[min(len(elat) - 1, int(0.99 * len(elat)))],
                    "note": "through the public API (lr_load_state + lr_route): per step the snapshot and "
                            "queries are copied from pinned host memory on an upload stream (one packed copy), "
                            "ingested and routed (K1 || K2), and the result copied back to pinned host memory "
                            f"on a read-back stream (one copy), which the host waits for {HOST_LAG} steps later; "
                            f"{NB} device and host buffer sets rotate, so a step's upload and the previous step's "
                            "read-back overlap its compute.  ms_per_step = span from the first upload's issue to the last result's "
                            "arrival / steps (no L2 flush inside the loop: every step's inputs arrive by copy); "
                            "latency = a step's upload issue to its result's arrival"},
            "gpu_launches": 2 * K, "clocks": clocks, "wall_s_timed_region": t_wall,
            "sequential": {"ms_per_step": seq_ms, "value": _job_rate(cands, world, seq_ms), "unit": UNIT,
                           "note": "K1 then K2 on one stream, same steps (kernel shares are of this time)"},
            "estimate": estimate,
            "configs": configs,
            "kv": kv,
            "avgcase": avgcase,
            "calibration": calibration,
            "stream": stream,
            "policy_eval": policy_eval,
        }
        print(json.dumps(line), flush=True)
    rt.close()
    if world > 1:
        dist.destroy_process_group()


def run_calibration(args, dev, flush):
    """Least-squares calibration of the batch-time coefficients (Sec. 4.1) over a
    synthetic log of 4M executed batches of 8 models, grouped by model."""
    import torch
    from paper_2607_18253_gb300 import router as R
    from paper_2607_18253_gb300 import workloads as W

    M, N = 8, 4_000_000
    alpha, beta, gamma, _ = W.model_pool(M)
    coef = W.coefficients(alpha, beta, gamma).astype(np.float64)
    F, mdl, t = W.batch_log(N, M, seed=5, coef=coef, noise=0.04)
    wl = W.small_workload(0, num_instances=M, num_models=M, budget_range=(8, 96), min_gap=8)
    rt = R.LatencyRouter.from_workload(wl)
    Fd, md, td = (torch.from_numpy(np.ascontiguousarray(x)).to(dev) for x in (F, mdl, t))
    out = torch.empty((M, 5), dtype=torch.float64, device=dev)
    for _ in range(3):
        rt.calibrate(Fd, md, td, out=out)
    torch.cuda.synchronize()
    K = max(3, min(args.steps, 100))
    ms = []
    for k in range(K):
        flush.fill_(float(k))
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        rt.calibrate(Fd, md, td, out=out)
        e1.record()
        e1.synchronize()
        ms.append(e0.elapsed_time(e1))
    if rt.status() != R.LR_OK:
        raise RuntimeError("calibration failed")
    rel = float(np.max(np.abs(out.cpu().numpy() - coef) / coef))
    rt.close()
    ms_avg = sum(ms) / K
    hbm, src = _peaks()
    nbytes = N * (5 * 8 + 4 + 8)
    ach = nbytes / (ms_avg * 1e-3) / 1e9
    return {"log": f"{N} batches of {M} models, grouped by model, 4% noise", "ms": ms_avg,
            "value": N / (ms_avg * 1e-3), "unit": "batches/s", "max_rel_error_vs_generating_coef": rel,
            "gpu_launches": K,
            "roofline": {"kernel": "k_calibrate (one pass over the log, then the last CTA's solve)", "bound": "hbm", "achieved": ach, "peak": hbm, "unit": "GB/s",
                         "frac": ach / hbm, "peak_source": f"{src} (MEASURED_PEAKS.json hbm_gbs, copy)",
                         "algorithmic_bytes": nbytes, "traffic": NCU_TRAFFIC["k_calibrate"]}}


def run_estimate(args, dev, wl, flush):
    """The SFS estimate alone (Eq. 8-9, lr_estimate_ttft) on the same workload: the full
    TTFT matrix from the live snapshot, timed against HBM (4 B per candidate, 4 B per
    query and the ~64 KiB summary).  The snapshot is loaded on the capture stream, so
    the call runs alone with a static row split."""
    import torch
    from paper_2607_18253_gb300 import router as R

    Q, I = wl.num_queries, wl.num_instances
    rt = R.LatencyRouter.from_workload(wl)
    state = R.state_tensors(wl, dev)
    p = torch.from_numpy(np.ascontiguousarray(wl.prompt_len)).to(dev)
    mat = torch.empty((Q, I), dtype=torch.float32, device=dev)
    cap = torch.cuda.Stream(device=dev)
    cap.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(cap):
        rt.load_state(*state)
        for _ in range(3):
            rt.estimate_ttft(p, out=mat)
    cap.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=cap):
        rt.estimate_ttft(p, out=mat)
    for _ in range(args.warmup):
        flush.fill_(1.0)
        g.replay()
    torch.cuda.synchronize()
    K = max(3, min(args.steps, 500))
    ms = []
    for k in range(K):
        flush.fill_(float(k))
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        g.replay()
        e1.record()
        e1.synchronize()
        ms.append(e0.elapsed_time(e1))
    if rt.status() != R.LR_OK:
        raise RuntimeError("SFS estimate failed")
    rt.close()
    ms_avg = sum(ms) / K
    hbm, src = _peaks()
    nbytes = Q * I * 4 + Q * 4 + 64 * 1024
    ach = nbytes / (ms_avg * 1e-3) / 1e9
    return {"call": "lr_estimate_ttft (SFS), full Q x I matrix", "ms": ms_avg, "value": Q * I / (ms_avg * 1e-3),
            "unit": UNIT, "steps": K, "gpu_launches": K,
            "roofline": {"kernel": "k_cand<0, 1>", "bound": "hbm", "achieved": ach, "peak": hbm, "unit": "GB/s",
                         "frac": ach / hbm, "peak_source": f"{src} (MEASURED_PEAKS.json hbm_gbs, copy)",
                         "algorithmic_bytes": nbytes, "traffic": NCU_TRAFFIC["k_estimate"]}}


def run_configs(args, dev, flush):
    """The other single-GPU configurations, one router each, every call captured in a
    CUDA graph and timed with CUDA events after an L2 flush:
      tiny   -- 8 instances (2 models x 4 replicas) x 16 queries, B = 2048, S = 64;
      pool64 -- 64 instances (4 models x 16) x 4,096 queries, B = 4096, S = 64;
      sweep  -- the pool64 state and queries routed for 32 (lambda, mu) pairs (4 x 8 on a log
                grid) with the per-pair frontier.
    For each: the route call alone (lr_route: the full TTFT matrix, utility, argmax) and the
    step (lr_load_state + lr_route on one stream); estimates/s counts query x instance TTFT
    estimates (the sweep's 32 pairs reuse one matrix; pair evaluations are given beside)."""
    import torch
    from paper_2607_18253_gb300 import router as R
    from paper_2607_18253_gb300 import workloads as W

    lam5, mu5 = W.sweep_pairs()
    cases = (("tiny", W.make_workload("tiny"), False),
             ("pool64", W.make_workload("pool64"), False),
             ("sweep_pool64_32pairs", W.make_workload("pool64", lam=lam5, mu=mu5), True))
    K = max(3, min(args.steps, 200))
    out = {}
    for label, wl, frontier in cases:
        Q, I, P = wl.num_queries, wl.num_instances, wl.num_pairs
        rt = R.LatencyRouter.from_workload(wl)
        state = R.state_tensors(wl, dev)
        p, dh, acc, _ = R.query_tensors(wl, dev)
        mat = torch.empty((Q, I), dtype=torch.float32, device=dev)
        res = {"assign": torch.empty((P, Q), dtype=torch.int32, device=dev),
               "util": torch.empty((P, Q), dtype=torch.float32, device=dev),
               "ttft_chosen": torch.empty((P, Q), dtype=torch.float32, device=dev)}
        if frontier:
            res["frontier"] = torch.empty((P, 3), dtype=torch.float64, device=dev)
        cap = torch.cuda.Stream(device=dev)
        cap.wait_stream(torch.cuda.current_stream())

        def route():
            rt.route(p, dh, acc, wl.lam, wl.mu, ttft_matrix=mat, frontier=frontier, out=res)

        with torch.cuda.stream(cap):
            for _ in range(3):
                rt.load_state(*state)
                route()
        cap.synchronize()
        graphs = {}
        for name in ("route", "step"):
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=cap):
                if name == "step":
                    rt.load_state(*state)
                route()
            graphs[name] = g
        ms = {}
        for name, g in graphs.items():
            for _ in range(args.warmup):
                flush.fill_(1.0)
                g.replay()
            torch.cuda.synchronize()
            t = []
            for k in range(K):
                flush.fill_(float(k))
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                e0.record()
                g.replay()
                e1.record()
                e1.synchronize()
                t.append(e0.elapsed_time(e1))
            ms[name] = sorted(t)
        if rt.status() != R.LR_OK:
            raise RuntimeError(f"{label}: device status after the timed calls")
        rt.close()
        mean = {k: sum(v) / len(v) for k, v in ms.items()}
        out[label] = {"queries": Q, "instances": I, "pairs": P, "steps": K,
                      "route_us": mean["route"] * 1e3, "route_p50_us": ms["route"][K // 2] * 1e3,
                      "step_us": mean["step"] * 1e3, "step_p50_us": ms["step"][K // 2] * 1e3,
                      "value": Q * I / (mean["route"] * 1e-3), "step_value": Q * I / (mean["step"] * 1e-3),
                      "unit": UNIT, "pair_evaluations_per_s": Q * I * P / (mean["route"] * 1e-3),
                      # route: the candidate kernel (+ the frontier kernel); step: K1 and the route
                      "gpu_launches": K * (2 * (1 + int(frontier)) + 1)}
    return out


KV_SEED = 11
KV_BLOCK = 16
KV_HORIZON = 4096


def run_kv(args, dev, wl, flush):
    """The SFS estimate under KV-cache block limits, context limits and preemption
    (App. F) on the same workload: seeded limits (16-token blocks, each instance's
    block count between its largest request and its residents' whole demand, half the
    instances with a context limit).  A step is the snapshot load (residents alone
    with per-batch records, k_kv_load) then the full Q x I TTFT matrix (per-candidate
    walk over the records, k_kv_estimate), on one stream; each kernel is also timed
    alone.  The estimate is timed against HBM: 4 B per candidate, 4 B per query, the
    instance headers and the records up to each instance's last first-token batch."""
    import torch
    from paper_2607_18253_gb300 import router as R
    from paper_2607_18253_gb300 import workloads as W

    Q, I = wl.num_queries, wl.num_instances
    limits = W.kv_limits(wl, KV_SEED, block_sizes=(KV_BLOCK,))
    rt = R.LatencyRouter.from_workload(wl)
    rt.set_kv_limits(*limits, horizon=KV_HORIZON)
    state = R.state_tensors(wl, dev)
    p = torch.from_numpy(np.ascontiguousarray(wl.prompt_len)).to(dev)
    mat = torch.empty((Q, I), dtype=torch.float32, device=dev)
    fb = torch.empty((Q, I), dtype=torch.int32, device=dev)
    cap = torch.cuda.Stream(device=dev)
    cap.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(cap):
        for _ in range(3):
            rt.load_state(*state)
            rt.estimate_ttft(p, out=mat, first_batch=fb)
    cap.synchronize()
    if rt.status() != R.LR_OK:
        raise RuntimeError("KV estimate failed")
    last = fb.amax(dim=0).to(torch.int64).sum().item()  # records up to each instance's last first token
    graphs = {}
    for name in ("load", "estimate", "step"):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=cap):
            if name != "estimate":
                rt.load_state(*state)
            if name != "load":
                rt.estimate_ttft(p, out=mat)
        graphs[name] = g
    K = max(3, min(args.steps, 300))
    out = {}
    for name, g in graphs.items():
        for _ in range(args.warmup):
            flush.fill_(1.0)
            g.replay()
        torch.cuda.synchronize()
        ms = []
        for k in range(K):
            flush.fill_(float(k))
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            g.replay()
            e1.record()
            e1.synchronize()
            ms.append(e0.elapsed_time(e1))
        out[name] = sum(ms) / K
    if rt.status() != R.LR_OK:
        raise RuntimeError("KV estimate failed")
    rt.close()
    hbm, src = _peaks()
    nbytes = Q * I * 4 + Q * 4 + I * 64 + last * 64
    ach = nbytes / (out["estimate"] * 1e-3) / 1e9
    return {"call": "lr_set_kv_limits, then per step lr_load_state + lr_estimate_ttft (SFS with KV limits)",
            "limits": {"block_size": KV_BLOCK, "seed": KV_SEED, "horizon": KV_HORIZON,
                       "ctx_limited_instances": int((limits[2] < (1 << 40)).sum()),
                       "blocks_median": int(np.median(limits[1]))},
            "ms_per_step": out["step"], "value": Q * I / (out["step"] * 1e-3), "unit": UNIT, "steps": K,
            "gpu_launches": 14 * K, "load_ms": out["load"], "estimate_ms": out["estimate"],
            "estimate_value": Q * I / (out["estimate"] * 1e-3),
            "roofline": {"kernel": "lr_estimate_ttft with KV limits (count, tile sums, scan, scatter, "
                                   "k_kv_estimate, k_kv_expand)", "bound": "hbm", "achieved": ach, "peak": hbm, "unit": "GB/s",
                         "frac": ach / hbm, "peak_source": f"{src} (MEASURED_PEAKS.json hbm_gbs, copy)",
                         "algorithmic_bytes": nbytes, "traffic": None,
                         "note": "the call's six kernels together; k_kv_estimate alone read 2.35 MB and wrote "
                                 "0.85 MB per launch (ncu); the load is one dependency chain per instance"}}


def run_avgcase(args, dev, wl, flush):
    """The average-case LPS source (App. E) on the same workload: the full TTFT matrix.

    No snapshot is involved; the estimate is affine in the prompt length per
    instance, so the kernel is a pure matrix write and is timed against HBM."""
    import torch
    from paper_2607_18253_gb300 import router as R

    Q, I = wl.num_queries, wl.num_instances
    rng = np.random.default_rng(17)
    mu = rng.uniform(5.0, 30.0, I)
    qp = dict(prefill_tput=rng.uniform(3e3, 4e4, I), decode_batch_time=rng.uniform(0.004, 0.06, I),
              arrival_rate=mu * rng.uniform(0.3, 0.9, I), service_rate=mu, parallelism=np.full(I, 25, np.int32))
    rt = R.LatencyRouter.from_workload(wl)
    rt.set_queue_params(**qp)
    rt.set_ttft_source(R.LR_TTFT_LPS)
    p = torch.from_numpy(np.ascontiguousarray(wl.prompt_len)).to(dev)
    mat = torch.empty((Q, I), dtype=torch.float32, device=dev)
    side = torch.cuda.Stream(device=dev)
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        for _ in range(3):
            rt.estimate_ttft(p, out=mat)
    torch.cuda.current_stream().wait_stream(side)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        rt.estimate_ttft(p, out=mat)
    for _ in range(args.warmup):
        flush.fill_(1.0)
        g.replay()
    torch.cuda.synchronize()
    K = max(3, min(args.steps, 500))
    ms = []
    for k in range(K):
        flush.fill_(float(k))
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        g.replay()
        e1.record()
        e1.synchronize()
        ms.append(e0.elapsed_time(e1))
    if rt.status() != R.LR_OK:
        raise RuntimeError("average-case estimate failed")
    rt.close()
    ms_avg = sum(ms) / K
    hbm, src = _peaks()
    nbytes = Q * I * 4 + Q * 4 + I * 32
    ach = nbytes / (ms_avg * 1e-3) / 1e9
    return {"source": "LPS (App. E), k = 25, rho in [0.3, 0.9], no snapshot", "ms": ms_avg,
            "value": Q * I / (ms_avg * 1e-3), "unit": UNIT, "steps": K, "gpu_launches": K,
            "roofline": {"kernel": "k_cand<2, 1>", "bound": "hbm", "achieved": ach, "peak": hbm, "unit": "GB/s",
                         "frac": ach / hbm, "peak_source": f"{src} (MEASURED_PEAKS.json hbm_gbs, copy)",
                         "algorithmic_bytes": nbytes}}


STREAM_WORKLOAD = "pool64"
STREAM_SEED = 3
STREAM_QUERIES = 1_000_000
STREAM_SIZES = (1, 16, 256)


def pool_capacity(R, W, wl, dev, horizon=300.0, warm=30.0, dt=2.0, depth=256):
    """Completions/s of every instance fed a saturating FCFS stream of the workload's queries.

    Each instance starts empty.  Before every advance of dt seconds its waiting queue
    is topped up to `depth` with the workload's next queries (each with the predicted
    output length of the instance's model), so the scheduler never runs dry;
    completions are counted between t = warm and t = horizon.  The simulation is the
    library's own stream step (lr_advance)."""
    import dataclasses

    import torch
    I, M = wl.num_instances, wl.num_models
    z = np.zeros(I, np.int32)
    empty = dataclasses.replace(wl, n_run=z, n_wait=z.copy(), cap_waiting=depth,
                                run_ctx=np.zeros((I, wl.cap_running), np.int32),
                                run_pre=np.zeros((I, wl.cap_running), np.int32),
                                run_dec=np.zeros((I, wl.cap_running), np.int32),
                                wait_pre=np.zeros((I, depth), np.int32), wait_dec=np.zeros((I, depth), np.int32))
    rt = R.LatencyRouter.from_workload(empty, max_queries=I * depth)
    rt.load_state(*R.state_tensors(empty, dev))
    appended = np.zeros(I, np.int64)
    nq = wl.num_queries
    nxt, t, c_warm = 0, 0.0, None
    while True:
        st = rt.read_state(device=dev)
        n_run, n_wait = st["n_run"].cpu().numpy(), st["n_wait"].cpu().numpy()
        completed = appended - n_run - n_wait
        if c_warm is None and t >= warm:
            c_warm = completed.copy()
        if t >= horizon:
            break
        need = depth - n_wait
        a = np.repeat(np.arange(I, dtype=np.int32), need)
        idx = (nxt + np.arange(a.shape[0])) % nq
        nxt += a.shape[0]
        appended += need
        t += dt
        rt.advance(torch.from_numpy(a).to(dev), torch.from_numpy(wl.prompt_len[idx]).to(dev),
                   torch.from_numpy(np.ascontiguousarray(wl.dec_hat[idx, wl.model_of_instance[a]])).to(dev), t)
    torch.cuda.synchronize()
    if rt.status() != R.LR_OK:
        raise RuntimeError("capacity run failed")
    rt.close()
    return (completed - c_warm) / (horizon - warm)


def run_stream(args, dev):
    """Online stream: arrivals at 0.8 x pool capacity (Poisson, and bursty MMPP-2), routed in micro-batches.

    At each decision time (the arrival of the batch's last query) the pool is advanced
    to that time with the previous batch appended to its chosen instances (K3 + K1),
    then the batch is routed on the new snapshot (K2, Lagrangian argmax).  The latency
    of a batch is the device time of those three launches, from CUDA events around them;
    the arguments are marshalled once, so the loop issues the C calls directly."""
    import ctypes

    import torch
    from paper_2607_18253_gb300 import router as R
    from paper_2607_18253_gb300 import workloads as W

    wl = W.make_workload(STREAM_WORKLOAD, num_queries=STREAM_QUERIES, seed=STREAM_SEED, cap_waiting=512)
    I, M = wl.num_instances, wl.num_models
    cap = pool_capacity(R, W, wl, dev)
    rate = 0.8 * float(cap.sum())
    traces = [("poisson", W.poisson_arrivals(STREAM_QUERIES, rate, STREAM_SEED), STREAM_SIZES),
              ("mmpp2_r6", W.mmpp2_arrivals(STREAM_QUERIES, rate, 6.0, STREAM_SEED), (16, 256))]
    mmax = max(STREAM_SIZES)
    rt = R.LatencyRouter.from_workload(wl, max_queries=mmax)
    state = R.state_tensors(wl, dev)
    p, dh, acc, _ = R.query_tensors(wl, dev)
    assign = torch.full((2, mmax), -1, dtype=torch.int32, device=dev)  # ping-pong: batch b, batch b-1
    util = torch.empty((1, mmax), dtype=torch.float32, device=dev)
    lam = np.ascontiguousarray(wl.lam[:1], np.float32)
    mu = np.ascontiguousarray(wl.mu[:1], np.float32)
    lib, h = rt._lib, rt._h
    sp = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    pp, dhp, accp = p.data_ptr(), dh.data_ptr(), acc.data_ptr()
    ap = [assign[0].data_ptr(), assign[1].data_ptr()]
    lamp, mup = lam.ctypes.data_as(ctypes.c_void_p), mu.ctypes.data_as(ctypes.c_void_p)
    V = ctypes.c_void_p
    out = {"workload": f"{STREAM_WORKLOAD} state and pool (seed {STREAM_SEED}), {STREAM_QUERIES} arrivals: Poisson, "
                       f"and MMPP-2 (rate ratio 6, 20% of time in the high state, switching 0.1/s and 0.4/s)",
           "capacity_qps": float(cap.sum()), "arrival_qps": rate,
           "capacity_reading": "completions/s of each instance under a saturating FCFS stream, t = 30..300 s",
           "latency": "device time of advance (K3 + K1) + route (K2) per micro-batch, CUDA events",
           "sizes": {}, "mmpp2_r6": {}}
    launches = 0
    for label, arr, sizes in traces:
        for m in sizes:
            nq = STREAM_QUERIES if m > 1 else min(STREAM_QUERIES, args.stream_queries_b1)
            nb = nq // m
            rt.load_state(*state)
            chunk = 4096
            ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(chunk)]
            lat = []
            torch.cuda.synchronize()
            w0 = time.perf_counter()
            for b in range(nb):
                lo = b * m
                cur, prev = ap[b & 1], ap[(b - 1) & 1]
                e0, e1 = ev[b % chunk]
                e0.record()
                # previous batch joins its instances' queues; every instance advances to now
                pm = m if b > 0 else 0
                plo = (b - 1) * m
                rc = lib.lr_advance(h, pm, V(prev), V(pp + 4 * max(plo, 0)), V(dhp + 4 * M * max(plo, 0)), M,
                                    ctypes.c_double(float(arr[lo + m - 1])), sp)
                rc |= lib.lr_route(h, m, V(pp + 4 * lo), V(dhp + 4 * M * lo), V(accp + 4 * M * lo), None, 1, lamp,
                                   mup, V(cur), V(util.data_ptr()), None, None, None, sp)
                e1.record()
                if rc:
                    raise RuntimeError(f"stream call failed: {lib.lr_last_error(h).decode()}")
                if b % chunk == chunk - 1 or b == nb - 1:
                    torch.cuda.synchronize()
                    lat += [ev[k][0].elapsed_time(ev[k][1]) for k in range(b % chunk + 1)]
            wall = time.perf_counter() - w0
            st = rt.status()
            if st != R.LR_OK:
                raise RuntimeError(f"stream run ({label}, micro-batch {m}) ended with device status {st}")
            launches += 3 * nb
            q = np.percentile(np.asarray(lat) * 1e3, [50, 99])
            fin = rt.read_state(device=dev)
            res = {"batches": nb, "queries": nb * m, "p50_us": float(q[0]), "p99_us": float(q[1]),
                   "mean_us": float(np.mean(lat) * 1e3), "wall_s": wall, "simulated_s": float(arr[nb * m - 1]),
                   "final_mean_waiting": float(fin["n_wait"].float().mean().item())}
            out["sizes" if label == "poisson" else label][str(m)] = res
    # A Poisson stream under KV-cache limits (App. F; the stream step executes the KV
    # rule and the KV load summarizes each snapshot): STREAM_KV_QUERIES arrivals at 0.5 x
    # the plain pool's capacity (the limits lower it), micro-batches of 16.  Limits:
    # 16-token blocks, each instance's block count between its largest request (a
    # query's whole response included) and its residents' demand, a context limit on
    # half the instances.
    limits = W.kv_limits(wl, KV_SEED, block_sizes=(KV_BLOCK,), max_new=int(wl.dec_hat.max()))
    rt.set_kv_limits(*limits, horizon=KV_HORIZON)
    rt.load_state(*state)
    arr = W.poisson_arrivals(STREAM_KV_QUERIES, 0.5 * float(cap.sum()), STREAM_SEED)
    m = 16
    nb = STREAM_KV_QUERIES // m
    lat = []
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(nb)]
    torch.cuda.synchronize()
    w0 = time.perf_counter()
    for b in range(nb):
        lo = b * m
        cur, prev = ap[b & 1], ap[(b - 1) & 1]
        ev[b][0].record()
        pm = m if b > 0 else 0
        plo = (b - 1) * m
        rc = lib.lr_advance(h, pm, V(prev), V(pp + 4 * max(plo, 0)), V(dhp + 4 * M * max(plo, 0)), M,
                            ctypes.c_double(float(arr[lo + m - 1])), sp)
        rc |= lib.lr_route(h, m, V(pp + 4 * lo), V(dhp + 4 * M * lo), V(accp + 4 * M * lo), None, 1, lamp,
                           mup, V(cur), V(util.data_ptr()), None, None, None, sp)
        ev[b][1].record()
        if rc:
            raise RuntimeError(f"KV stream call failed: {lib.lr_last_error(h).decode()}")
    torch.cuda.synchronize()
    wall = time.perf_counter() - w0
    st = rt.status()
    if st != R.LR_OK:
        raise RuntimeError(f"KV stream run ended with device status {st}")
    lat = [e0.elapsed_time(e1) for e0, e1 in ev]
    q = np.percentile(np.asarray(lat) * 1e3, [50, 99])
    fin = rt.read_state(device=dev)
    # launches per decision: advance (K3 KV, KV load) + route (count, tile sums, scan,
    # scatter, walk, expand, route)
    launches += 9 * nb
    out["kv_poisson_16"] = {"arrival_qps": 0.5 * float(cap.sum()), "batches": nb, "queries": nb * m, "p50_us": float(q[0]), "p99_us": float(q[1]),
                            "mean_us": float(np.mean(lat) * 1e3), "wall_s": wall,
                            "simulated_s": float(arr[nb * m - 1]),
                            "final_mean_waiting": float(fin["n_wait"].float().mean().item()),
                            "limits": {"block_size": KV_BLOCK, "seed": KV_SEED, "horizon": KV_HORIZON,
                                       "ctx_limited_instances": int((limits[2] < (1 << 40)).sum())}}
    out["gpu_launches"] = launches
    rt.close()
    return out


STREAM_KV_QUERIES = 32_768
POLICY_WORKLOAD = "paper3"
POLICY_LOADS = (0.2, 0.4, 0.6, 0.8)
POLICY_QUERIES = 4096
POLICY_BATCH = 1  # every query is routed on arrival, as in the paper
POLICIES = (("sfs_constrained", None), ("round_robin", 0), ("shortest_queue", 1), ("latency_agnostic", 2))


def run_policy_eval(args, dev):
    """Routing quality of the SFS router and the baselines on synthetic streams (Sec. 6, Eq. 4).

    A pool of one instance per model, as in the paper (the Latency-Agnostic baseline sends
    every query of a model to one instance, so replicas would only stand idle), starting
    empty, fed Poisson arrivals at 0.2 .. 0.8 x its capacity (the paper's OnTimeUtility
    against arrival rate) and MMPP-2 arrivals at 0.6 x.  "auc" is the mean OnTimeUtility
    over the Poisson rates (trapezoids on the evenly spaced grid)."""
    import dataclasses

    from paper_2607_18253_gb300 import router as R
    from paper_2607_18253_gb300 import workloads as W

    wl = W.make_workload(POLICY_WORKLOAD, num_queries=POLICY_QUERIES, cap_waiting=1024)
    cap = pool_capacity(R, W, wl, dev)
    I = wl.num_instances
    wl = dataclasses.replace(wl, n_run=np.zeros(I, np.int32), n_wait=np.zeros(I, np.int32))
    rt = R.LatencyRouter.from_workload(wl, max_queries=POLICY_BATCH)
    p, dh, acc, _ = R.query_tensors(wl, dev)
    out = {"workload": f"{POLICY_WORKLOAD}: 3 models, one instance each, starting empty; {POLICY_QUERIES} arrivals "
                       f"per trace, TTFT targets of App. B.2", "capacity_qps": float(cap.sum()), "poisson": {}}
    launches = 0
    for f in POLICY_LOADS:
        rate = f * float(cap.sum())
        r = _policy_eval(rt, wl, W.poisson_arrivals(POLICY_QUERIES, rate, wl.seed), dev, p, dh, acc)
        out["poisson"][f"{f:.1f}"] = r
        launches += r["gpu_launches"]
    rate = 0.6 * float(cap.sum())
    out["mmpp2_r6_0.6"] = _policy_eval(rt, wl, W.mmpp2_arrivals(POLICY_QUERIES, rate, 6.0, wl.seed), dev, p, dh, acc)
    launches += out["mmpp2_r6_0.6"]["gpu_launches"]
    auc = {}
    for name, _ in POLICIES:
        y = [out["poisson"][f"{f:.1f}"]["policies"][name]["on_time_utility"] for f in POLICY_LOADS]
        auc[name] = float(np.mean([(a + b) / 2 for a, b in zip(y[:-1], y[1:])]))
    out["auc"] = auc
    best = max(v for k, v in auc.items() if k != "sfs_constrained")
    out["sfs_auc_over_best_baseline"] = auc["sfs_constrained"] / best if best > 0 else None
    out["gpu_launches"] = launches
    rt.close()
    return out


def _policy_eval(rt, wl, arr, dev, p, dh, acc):
    """One trace: every policy routes the same arrivals from the same initial state.

    The first POLICY_QUERIES arrivals are routed in micro-batches of POLICY_BATCH at the
    arrival of each batch's last query, by the constrained objective (Eq. 3) on SFS
    estimates or by a baseline policy; every batch joins its chosen instances before the
    next is routed, tracked to its first output token (lr_advance_tracked), and the
    pool is finally run until every query has one.  A query's realized TTFT is its
    first-token time in that executed stream minus its arrival: it includes the wait for
    the decision and the batches that later queries lengthened, which no estimate made
    at the decision can see.  On time if within its target; OnTimeUtility and SLO
    attainment come from lr_on_time_utility.  Also reported: the same two metrics with
    the decision-time view (decision delay + the chosen instance's SFS estimate), mean
    utility, mean realized TTFT, and the device time per micro-batch (advance + route)."""
    import ctypes

    import torch
    from paper_2607_18253_gb300 import router as R

    m, n = POLICY_BATCH, POLICY_QUERIES
    nb = n // m
    M = wl.num_models
    lib, h = rt._lib, rt._h
    sp = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    V = ctypes.c_void_p
    td = np.repeat(arr[m - 1:nb * m:m], m)  # decision time of each query's batch
    delay = torch.from_numpy((td - arr[:nb * m]).astype(np.float32)).to(dev)
    tau = torch.from_numpy(np.ascontiguousarray(wl.tau[:nb * m], np.float32)).to(dev)
    util = torch.empty(nb * m, dtype=torch.float32, device=dev)
    ttft = torch.empty(nb * m, dtype=torch.float32, device=dev)
    assign = torch.full((2, m), -1, dtype=torch.int32, device=dev)
    lam = np.ascontiguousarray(wl.lam[:1], np.float32)
    lamp = lam.ctypes.data_as(V)
    pp, dhp, accp, taup = p.data_ptr(), dh.data_ptr(), acc.data_ptr(), tau.data_ptr()
    up, tp = util.data_ptr(), ttft.data_ptr()
    ap = [assign[0].data_ptr(), assign[1].data_ptr()]
    state = R.state_tensors(wl, dev)
    ftt = torch.empty(nb * m, dtype=torch.float64, device=dev)
    arr_d = torch.from_numpy(np.ascontiguousarray(arr[:nb * m], np.float64)).to(dev)
    res = {}
    for name, pol in POLICIES:
        ftt.fill_(float("nan"))
        rt.track_first_tokens(ftt)
        rt.load_state(*state)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        e0.record()
        for b in range(nb):
            lo = b * m
            cur, prev = ap[b & 1], ap[(b - 1) & 1]
            pm = m if b > 0 else 0
            plo = max((b - 1) * m, 0)
            rc = lib.lr_advance_tracked(h, pm, V(prev), V(pp + 4 * plo), V(dhp + 4 * M * plo), M,
                                        ctypes.c_int64(plo), ctypes.c_double(float(td[lo])), sp)
            if pol is None:
                rc |= lib.lr_route(h, m, V(pp + 4 * lo), V(dhp + 4 * M * lo), V(accp + 4 * M * lo), V(taup + 4 * lo),
                                   1, lamp, None, V(cur), V(up + 4 * lo), V(tp + 4 * lo), None, None, sp)
            else:
                rc |= lib.lr_route_baseline(h, pol, m, V(pp + 4 * lo), V(dhp + 4 * M * lo), V(accp + 4 * M * lo),
                                            ctypes.c_float(float(lam[0])), ctypes.c_int64(lo), V(cur),
                                            V(up + 4 * lo), V(tp + 4 * lo), sp)
            if rc:
                raise RuntimeError(f"policy run {name} failed: {lib.lr_last_error(h).decode()}")
        e1.record()
        fin = rt.read_state(device=dev)
        # the last batch joins, then the pool runs until every routed query has its first token
        plo = (nb - 1) * m
        rc = lib.lr_advance_tracked(h, m, V(ap[(nb - 1) & 1]), V(pp + 4 * plo), V(dhp + 4 * M * plo), M,
                                    ctypes.c_int64(plo), ctypes.c_double(1e9), sp)
        if rc:
            raise RuntimeError(f"policy run {name} failed: {lib.lr_last_error(h).decode()}")
        torch.cuda.synchronize()
        st = rt.status()
        if st != R.LR_OK:
            raise RuntimeError(f"policy run {name} ended with device status {st}")
        if torch.isnan(ftt).any():
            raise RuntimeError(f"policy run {name}: a query never produced its first token")
        realized = (ftt - arr_d).to(torch.float32)
        otu, slo = (float(x) for x in rt.on_time_utility(util, realized, tau).cpu().numpy())
        otu_e, slo_e = (float(x) for x in rt.on_time_utility(util, ttft, tau, delay).cpu().numpy())
        gap = (realized - (delay + ttft)).double()
        res[name] = {"on_time_utility": otu, "slo_attainment": slo, "mean_utility": float(util.mean().item()),
                     "mean_realized_ttft_s": float(realized.double().mean().item()),
                     "decision_view": {"on_time_utility": otu_e, "slo_attainment": slo_e,
                                       "mean_ttft_s": float((delay + ttft).double().mean().item())},
                     "realized_minus_decision_view_s": {"mean": float(gap.mean().item()),
                                                        "max": float(gap.max().item()),
                                                        "min": float(gap.min().item())},
                     "us_per_batch": e0.elapsed_time(e1) * 1e3 / nb,
                     "final_max_waiting": int(fin["n_wait"].max().item())}
    rt.track_first_tokens(None)
    return {"queries": nb * m, "micro_batch": m, "lambda": float(lam[0]),
            "objective": "SFS router: Eq. 3 (max utility within the TTFT target, else least TTFT)",
            "realized_ttft": "first-token time in the executed stream (lr_advance_tracked) - arrival; "
                             "decision_view: decision delay + SFS estimate of the chosen instance",
            "policies": res, "gpu_launches": len(POLICIES) * (3 * nb + 3 + 2)}


def _host_cpu():
    """Core count and CPU model of this host (lscpu, else /proc/cpuinfo)."""
    import platform
    model = None
    try:
        txt = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        names = [ln.split(":", 1)[1].strip() for ln in txt.splitlines() if ln.startswith("Model name:")]
        model = " / ".join(dict.fromkeys(names)) or None
    except Exception:
        pass
    if not model:
        try:
            for ln in open("/proc/cpuinfo"):
                if ln.lower().startswith("model name"):
                    model = ln.split(":", 1)[1].strip()
                    break
        except OSError:
            pass
    try:
        usable = len(os.sched_getaffinity(0))
    except (AttributeError, OSError):
        usable = os.cpu_count()
    return {"nproc": os.cpu_count(), "usable_cores": usable, "cpu_model": model or platform.machine(),
            "arch": platform.machine()}


def _oracle_rows(wl, nq, seed, threads):
    """Full TTFT rows for nq sampled queries, then the oracle's argmax over them."""
    import oracle
    rng = np.random.default_rng(seed)
    qs = np.sort(rng.choice(wl.num_queries, nq, replace=False))
    sub = wl.with_queries(qs)
    t0 = time.perf_counter()
    _, _, t32, _ = oracle.estimate_matrix(sub, threads=threads)
    oracle.route(sub, t32)
    return nq * wl.num_instances, time.perf_counter() - t0


def _sized_rows(wl, seconds, seed, threads):
    """About `seconds` of oracle work on whole rows: (candidates, seconds, queries)."""
    probe = 8 if threads == 1 else 64
    cands, dt = _oracle_rows(wl, probe, seed, threads)
    per_row = dt / probe
    nq = max(probe, min(wl.num_queries, int(seconds / per_row)))
    cands, dt = _oracle_rows(wl, nq, seed + 1, threads)
    return cands, dt, nq


def _repeat_for(fn, seconds):
    """Run fn() (which returns units of work) until `seconds` have passed: (units, seconds)."""
    units, t0 = 0, time.perf_counter()
    while True:
        units += fn()
        dt = time.perf_counter() - t0
        if dt >= seconds:
            return units, dt


def _oracle_configs(threads, seconds):
    """The oracle on the other configurations, on `threads` host threads."""
    import dataclasses

    import oracle
    from paper_2607_18253_gb300 import workloads as W
    out = {}
    lam5, mu5 = W.sweep_pairs()
    for label, wl in (("tiny", W.make_workload("tiny")), ("pool64", W.make_workload("pool64")),
                      ("sweep_pool64_32pairs", W.make_workload("pool64", lam=lam5, mu=mu5))):
        def one(wl=wl, label=label):
            _, _, t32, _ = oracle.estimate_matrix(wl, threads=threads)
            a, _, tc = oracle.route(wl, t32)
            if label.startswith("sweep"):
                oracle.frontier(wl, a, tc)
            return wl.num_queries * wl.num_instances
        units, dt = _repeat_for(one, min(seconds, 2.0))
        out[label] = {"value": units / dt, "unit": UNIT, "seconds": dt,
                      "sample": f"the whole configuration ({wl.num_queries} x {wl.num_instances}"
                                f"{', 32 pairs + frontier' if label.startswith('sweep') else ''}), repeated"}
    # the online stream: decisions of the Poisson trace at micro-batch 256, each the
    # oracle's advance to the decision time, then the batch's rows and argmax
    wl = W.make_workload(STREAM_WORKLOAD, num_queries=STREAM_QUERIES, seed=STREAM_SEED, cap_waiting=512)
    rate = 0.8 * float(oracle.pool_capacity(wl).sum())
    arr = W.poisson_arrivals(STREAM_QUERIES, rate, STREAM_SEED)
    m, st, clk, prev = 256, wl, np.zeros(wl.num_instances), None
    none = np.zeros(0, np.int32)
    t0, b = time.perf_counter(), 0
    while time.perf_counter() - t0 < seconds and (b + 1) * m <= STREAM_QUERIES:
        lo = b * m
        t_now = float(arr[lo + m - 1])
        if prev is None:
            st, clk = oracle.advance(st, clk, none, none, none, t_now)
        else:
            pa, pq = prev
            d = np.ascontiguousarray(pq.dec_hat[np.arange(m), wl.model_of_instance[pa]])
            st, clk = oracle.advance(st, clk, pa, pq.prompt_len, d, t_now)
        q = dataclasses.replace(st, prompt_len=wl.prompt_len[lo:lo + m], dec_hat=wl.dec_hat[lo:lo + m],
                                acc=wl.acc[lo:lo + m], tau=wl.tau[lo:lo + m])
        _, _, t32, _ = oracle.estimate_matrix(q, threads=threads)
        a, _, _ = oracle.route(q, t32, lam=wl.lam[:1], mu=wl.mu[:1])
        prev = (a[0], q)
        b += 1
    dt = time.perf_counter() - t0
    out["stream_pool64_b256"] = {"value": b * m * wl.num_instances / dt, "unit": UNIT, "seconds": dt,
                                 "decisions_per_s": b / dt,
                                 "sample": f"the first {b} decisions of the Poisson trace at micro-batch {m} "
                                           f"(advance + rows + argmax)"}
    return out


def cpu_baseline(wl, seconds: float):
    """The oracle as it stands on this host's cores, on bounded samples of each workload.

    value: the headline workload on every core (one thread per core, candidates split
    into contiguous slices); one_core: the same on one thread; configs: the other
    configurations on every core."""
    import oracle
    n = oracle.host_threads()
    c1, d1, q1 = _sized_rows(wl, seconds, 2, 1)
    cn, dn, qn = _sized_rows(wl, seconds, 4, n)
    sample = (f"{qn} random queries of {WORKLOAD} x all {wl.num_instances} instances ({cn} candidates, "
              f"{dn:.1f} s): literal per-candidate simulation + brute-force argmax, {n} threads; estimates/s "
              f"extrapolate to the whole {wl.num_queries}-query batch")
    return {"value": cn / dn, "unit": UNIT, "cores": n, "kind": "oracle", "sample": sample,
            "host": _host_cpu(),
            "one_core": {"value": c1 / d1, "unit": UNIT, "cores": 1,
                         "sample": f"{q1} random queries x all instances ({c1} candidates, {d1:.1f} s)"},
            "configs": _oracle_configs(n, min(seconds, 5.0))}


def run_reference(args):
    rank, world, _ = _dist()
    if rank != 0:
        return
    import oracle
    from paper_2607_18253_gb300 import workloads as W
    oracle.build()
    n = oracle.host_threads()
    wl = W.make_workload(WORKLOAD)
    probe = 64
    _, dt = _oracle_rows(wl, probe, 0, n)
    per_row = dt / probe
    # about two minutes in total, whatever K and W are
    step_s = min(args.ref_step_seconds, 120.0 / max(1, args.steps + args.warmup))
    nq = max(2, min(wl.num_queries, int(step_s / per_row)))
    for w in range(args.warmup):
        _oracle_rows(wl, nq, 100 + w, n)
    times = []
    for k in range(args.steps):
        c, t = _oracle_rows(wl, nq, 1000 + k, n)
        times.append(t)
    ms = 1e3 * sum(times) / len(times)
    v = nq * wl.num_instances / (ms * 1e-3)
    sample = (f"each step: {nq} random queries of {WORKLOAD} x all {wl.num_instances} instances, literal "
              f"per-candidate simulation + brute-force argmax, {n} host threads (one per core)")
    line = {"impl": "reference", "metric": METRIC, "value": v, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f32+i64", "data": "synthetic", "config": _config_desc(wl),
            "cpu_baseline": {"value": v, "unit": UNIT, "cores": n, "kind": "oracle", "sample": sample,
                             "host": _host_cpu()},
            "e2e": {"value": v, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="gb300", choices=["gb300", "reference"])
    ap.add_argument("--cpu-seconds", type=float, default=15.0)
    ap.add_argument("--ref-step-seconds", type=float, default=2.0)
    ap.add_argument("--sustain-seconds", type=float, default=1.5,
                    help="back-to-back steps before the timed ones, while the clocks are sampled")
    ap.add_argument("--no-cpu", action="store_true")
    ap.add_argument("--no-stream", action="store_true", help="skip the online-stream latency run")
    ap.add_argument("--stream-queries-b1", type=int, default=STREAM_QUERIES,
                    help="queries of the trace routed one at a time (default: the whole trace)")
    ap.add_argument("--traffic", type=float, default=None,
                    help="dram bytes per launch of the dominant kernel from an ncu capture of this build")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    if args.impl == "reference":
        run_reference(args)
    else:
        run_gpu(args)


if __name__ == "__main__":
    main()
