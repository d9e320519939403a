#!/usr/bin/env python3
"""Throughput of the CompressKV prefill-end compression path on GB300.

One step = every layer of the workload compressed once (scoring with the SRH
heads, pooling, budgeted top-k, K/V gather), inputs resident in HBM.  The
default workload is 32 layers of a Llama-3.1-8B GQA shape at L = 32768
(bf16, W = 32, P = 7, budgets with mean 256).  Prints one JSON line.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME]
  python bench.py --impl reference ...     # the float64 oracle on host cores

Multi-GPU (torchrun, one process per GPU): every rank compresses its own
replica of the workload (the path has no exchange step); value = tokens of
all ranks / slowest rank's time.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import re
import statistics
import subprocess
import sys
import time
import types

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402
import torch  # noqa: E402

import workloads as wl  # noqa: E402

METRIC = ("prompt tokens compressed/sec per GB300 and achieved HBM GB/s vs peak at "
          "L=32K–128K")
UNIT = "tokens/s"
PROFILE_TRAFFIC = os.path.join(ROOT, "profiles", "fused_llama8b_L32k.md")
# the timed kernel's own source: a committed traffic figure is shown only
# while it matches
KERNEL_SOURCES = ["paper_2606_24467_gb300/csrc/fused_kernel.cu"]


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--workload", default="c2")
    ap.add_argument("--layers", type=int, default=0,
                    help="compress only the first N layers (small profiling runs)")
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--e2e-steps", type=int, default=5)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-secondary", action="store_true",
                    help="skip the L=128K workload measured after the L=32K headline")
    ap.add_argument("--no-lse", action="store_true",
                    help="skip the given-LSE (log-sum-exp supplied) measurement")
    ap.add_argument("--streams", type=int, default=1,
                    help="calls in flight: call c runs on stream c %% S with its own workspace")
    ap.add_argument("--layers-per-call", type=int, default=0,
                    help="layers compressed by one compress_layers call; 0 = every layer of the "
                         "workload in one call (one launch of the persistent kernel per step)")
    return ap.parse_args()


# --------------------------------------------------------------------- distributed
def dist_env():
    return (int(os.environ.get("RANK", 0)), int(os.environ.get("WORLD_SIZE", 1)),
            int(os.environ.get("LOCAL_RANK", 0)))


def init_dist(world: int, backend: str):
    if world <= 1:
        return None
    import torch.distributed as dist

    os.environ.setdefault("MASTER_ADDR", "127.0.0.1")
    dist.init_process_group(backend=backend)
    return dist


def reduce_max(dist, value: float, device) -> float:
    """Max of a float over ranks (identity without a process group)."""
    if dist is None:
        return value
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def barrier(dist):
    if dist is not None:
        dist.barrier()


# --------------------------------------------------------------------- clocks
_CLOCK_FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
                 "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
                 "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
_REASON_NAMES = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")


class ClockSampler:
    """nvidia-smi sampling (read-only) while the timed region runs."""

    def __init__(self, device):
        self.proc = None
        self.lines = []
        ident = []
        try:
            uuid = str(torch.cuda.get_device_properties(device).uuid)
            ident = [f"--id=GPU-{uuid}" if not uuid.startswith("GPU-") else f"--id={uuid}"]
        except Exception:
            ident = []
        self.cmd = ["nvidia-smi", *ident, f"--query-gpu={_CLOCK_FIELDS}",
                    "--format=csv,noheader,nounits", "-lms", "100"]

    def start(self):
        try:
            self.proc = subprocess.Popen(self.cmd, stdout=subprocess.PIPE,
                                         stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
        time.sleep(0.25)

    def stop(self) -> dict | None:
        if self.proc is None:
            return None
        time.sleep(0.15)
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
            out, _ = self.proc.communicate()
        sm, mx, reasons = [], [], set()
        for line in out.strip().splitlines():
            parts = [x.strip() for x in line.split(",")]
            if len(parts) < 8:
                continue
            try:
                sm.append(float(parts[0]))
                mx.append(float(parts[1]))
            except ValueError:
                continue
            for name, val in zip(_REASON_NAMES, parts[4:8]):
                if val.lower().startswith("active"):
                    reasons.add(name)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx),
                "reasons": sorted(reasons), "samples": len(sm)}


# --------------------------------------------------------------------- helpers
def measured_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


def kernel_source_hash() -> str:
    h = hashlib.sha256()
    for rel in KERNEL_SOURCES:
        with open(os.path.join(ROOT, rel), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def profiled_traffic(workload: str, layers_per_call: int):
    """DRAM bytes per launch of the scoring kernel from the committed
    ncu summary, if it was taken on the current kernel sources with the same
    workload and layers per call."""
    try:
        text = open(PROFILE_TRAFFIC).read()
    except OSError:
        return None
    m = re.search(r"traffic_bytes_per_launch:\s*(\d+)", text)
    h = re.search(r"kernel_source_sha256_16:\s*([0-9a-f]+)", text)
    w = re.search(r"workload:\s*(\S+)", text)
    c = re.search(r"layers_per_call:\s*(\d+)", text)
    if not (m and h and w and c) or h.group(1) != kernel_source_hash() or \
            w.group(1) != workload or int(c.group(1)) != layers_per_call:
        return None
    return int(m.group(1))


def cpu_cores() -> int:
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


def build_layers(cfg, device):
    lengths = wl.sequence_lengths(cfg)
    masks = wl.srh_masks(cfg)
    budgets = wl.layer_budgets(cfg, lengths)
    layers = [wl.make_layer(cfg, l, device=device, lengths=lengths, masks=masks, budgets=budgets)
              for l in range(cfg.n_layers)]
    return lengths, masks, budgets, layers


# Most layers one per-group compress_layers call takes (one SRH mask each).
MAX_LAYERS_PER_CALL = 256


def layers_per_call(cfg, layers, lengths) -> int:
    """Every layer of the step in one call: the persistent kernel then
    streams K from the first layer to the last without a break."""
    return max(1, min(MAX_LAYERS_PER_CALL, cfg.n_layers))


def algorithmic_bytes(cfg, layers, lengths):
    """K read once for scoring + retained K and V read and written, per step,
    plus the window-query rows of the SRH heads."""
    d = cfg.head_dim
    esz = 2
    k_bytes = sum(lengths) * cfg.num_kv_heads * d * esz
    total = 0
    score_bytes = 0
    for lay in layers:
        kept = sum(min(int(b), L) for b, L in zip(lay["budgets"], lengths))
        q_rows = int(lay["srh_mask"].sum()) * cfg.window * cfg.batch
        score_bytes += k_bytes + q_rows * d * esz
        total += k_bytes + q_rows * d * esz + 4 * kept * cfg.num_kv_heads * d * esz
    return total, score_bytes


def workload_config(cfg, budgets, lengths) -> dict:
    """The workload's keys, identical in both arms (run-specific settings go
    to the line's `run` object)."""
    kv_bytes = sum(lengths) * cfg.num_kv_heads * cfg.head_dim * 2 * 2 * cfg.n_layers
    return {"workload": cfg.name, "layers": cfg.n_layers, "batch": cfg.batch,
            "seq_len": cfg.seq_len if cfg.length_range is None else "ragged",
            "q_heads": cfg.num_q_heads, "kv_heads": cfg.num_kv_heads,
            "head_dim": cfg.head_dim, "window": cfg.window, "pool_width": cfg.pool_width,
            "mean_budget": float(np.mean(budgets)),
            "l2": f"inputs larger than L2: {kv_bytes / 1e9:.2f} GB of K/V per step, each "
                  "layer's K read cold; no flush"}


# --------------------------------------------------------------------- our arm
# The headline workload is L = 32K; the metric spans 32K-128K, so the same
# run also measures this one (same method, reported under `workloads`).
SECONDARY = {"c2": "c3"}


def run_ours(args):
    import paper_2606_24467_gb300 as ckv

    rank, world, local_rank = dist_env()
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    dist = init_dist(world, "nccl")
    ckv.load(build_if_missing=(rank == 0 and world == 1))
    cfg = wl.get(args.workload)
    if args.layers:
        cfg = cfg.scaled(n_layers=args.layers)
    result = bench_workload(args, cfg, dev, dist, world, rank, headline=True)
    second = SECONDARY.get(args.workload)
    if second and not args.layers and not args.no_secondary:
        torch.cuda.empty_cache()
        sub = bench_workload(args, wl.get(second), dev, dist, world, rank, headline=False)
        result["workloads"] = {sub["config"]["workload"]: {
            k: sub[k] for k in ("value", "unit", "ms_per_step", "config", "roofline", "path",
                                "kernels", "gpu_launches", "clocks", "timed_blocks",
                                "parity_layer0") if k in sub}}
    if rank == 0:
        print(json.dumps(result), flush=True)
    if dist is not None:
        dist.destroy_process_group()


def bench_workload(args, cfg, dev, dist, world, rank, headline: bool) -> dict:
    """Times the step of one workload; with `headline`, also the CPU
    baseline, the end-to-end and the given-LSE measurements."""
    import paper_2606_24467_gb300 as ckv

    lengths, masks, budgets, layers = build_layers(cfg, dev)
    tokens = sum(lengths)

    # The step's K, V and window queries live in one allocation each, like a
    # model's cache [n_layers][T][H_kv][d]; each layer is a view into it.
    B, T = cfg.batch, layers[0]["k"].shape[0]
    k_all = torch.cat([lay["k"] for lay in layers])
    v_all = torch.cat([lay["v"] for lay in layers])
    q_all = torch.cat([lay["q_win"] for lay in layers])
    for l, lay in enumerate(layers):
        lay["k"], lay["v"] = k_all[l * T:(l + 1) * T], v_all[l * T:(l + 1) * T]
        lay["q_win"] = q_all[l * B:(l + 1) * B]
    torch.cuda.empty_cache()

    # library objects: one compress_layers call per `layers_per_call` layers
    # (the layers packed as one batch, one SRH mask per layer), a workspace
    # per stream, per-call outputs.  Two graphs of the same step: `graph`
    # (timed; consecutive kernels overlap through programmatic dependent
    # launch) and `traced` (every launch bracketed by CUDA events, which
    # serialises the kernels) for the per-kernel durations.
    trace = ckv.Trace(capacity=16 * cfg.n_layers)
    counter = ckv.Trace(capacity=0)
    lpc = args.layers_per_call if args.layers_per_call > 0 else layers_per_call(cfg, layers,
                                                                                  lengths)
    calls = [(l0, min(l0 + lpc, cfg.n_layers)) for l0 in range(0, cfg.n_layers, lpc)]

    def call_problem(l0, l1, tr):
        m = l1 - l0
        cu = np.concatenate([np.asarray(layers[0]["cu_seqlens"][:-1], np.int64) + j * T
                             for j in range(m)] + [[m * T]]).astype(np.int32)
        return ckv.Problem(q_all[l0 * B:l1 * B], k_all[l0 * T:l1 * T], cu, cfg.window,
                           cfg.pool_width, trace=tr)

    probs = [call_problem(l0, l1, counter) for l0, l1 in calls]
    tprobs = [call_problem(l0, l1, trace) for l0, l1 in calls]
    c_budgets = [np.concatenate([np.asarray(layers[l]["budgets"]).reshape(-1)
                                 for l in range(l0, l1)]) for l0, l1 in calls]
    c_masks = [np.stack([np.asarray(layers[l]["srh_mask"]) for l in range(l0, l1)])
               for l0, l1 in calls]
    # Calls are independent: with S streams, call c runs on stream c % S with
    # that stream's workspace, so one call's latency-bound select overlaps
    # the next call's K stream.  Each stream's kernels still chain through
    # programmatic dependent launch.
    n_streams = max(1, args.streams)
    wss = [ckv.workspace(probs[0], dev) for _ in range(n_streams)]
    ws = wss[0]
    lanes = [torch.cuda.Stream() for _ in range(n_streams)]
    outs = [ckv.LayerOutputs(probs[c], c_budgets[c], cfg.head_dim, k_all.dtype, dev,
                             scores=False) for c in range(len(calls))]
    # per-layer problems for the single-layer calls of the e2e measurement
    lprobs = [ckv.Problem(lay["q_win"], lay["k"], lay["cu_seqlens"], cfg.window, cfg.pool_width)
              for lay in layers]

    def run_call(pr, c, wsp, stream=None):
        l0, l1 = calls[c]
        o = outs[c]
        ckv.compress_layers(pr[c], l1 - l0, q_all[l0 * B:l1 * B], k_all[l0 * T:l1 * T],
                            v_all[l0 * T:l1 * T], c_masks[c], c_budgets[c], o.indices, o.k_out,
                            o.v_out, wsp, stream=stream)

    def step(pr, streams=n_streams):
        if streams == 1:
            for c in range(len(calls)):
                run_call(pr, c, ws)
            return
        cur = torch.cuda.current_stream()
        fork = torch.cuda.Event()
        fork.record(cur)
        for st in lanes[:streams]:
            st.wait_event(fork)
        for c in range(len(calls)):
            run_call(pr, c, wss[c % streams], stream=lanes[c % streams])
        for st in lanes[:streams]:
            done = torch.cuda.Event()
            done.record(st)
            cur.wait_event(done)

    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        for _ in range(2):
            step(probs)
    torch.cuda.current_stream().wait_stream(side)
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    counter.reset()
    with torch.cuda.graph(graph, capture_error_mode="thread_local"):
        step(probs)
    launches_per_step = counter.launches
    traced = torch.cuda.CUDAGraph()
    trace.reset()
    with torch.cuda.graph(traced, capture_error_mode="thread_local"):
        step(tprobs, streams=1)
    torch.cuda.synchronize()

    w0 = torch.cuda.Event(enable_timing=True)
    w1 = torch.cuda.Event(enable_timing=True)
    w0.record()
    for _ in range(max(args.warmup, 3)):
        graph.replay()
    w1.record()
    torch.cuda.synchronize()
    warm_ms = w0.elapsed_time(w1) / max(args.warmup, 3)
    # Exactly `steps` steps per timed block, bracketed by a barrier and a
    # synchronize; the block is repeated until about two seconds of timed
    # work have run (so the clock sampler sees the GPU under load) and the
    # median block is reported.
    blocks = int(min(50, max(1, math.ceil(2000.0 / max(warm_ms * args.steps, 1e-3)))))
    barrier(dist)
    sampler = ClockSampler(dev)
    sampler.start()
    block_ms = []
    for _ in range(blocks):
        t0 = torch.cuda.Event(enable_timing=True)
        t1 = torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        barrier(dist)
        t0.record()
        for _ in range(args.steps):
            graph.replay()
        t1.record()
        torch.cuda.synchronize()
        barrier(dist)
        block_ms.append(reduce_max(dist, t0.elapsed_time(t1), dev))
    clocks = sampler.stop()
    elapsed_ms = statistics.median(block_ms)
    ms_per_step = elapsed_ms / args.steps
    value = world * tokens * args.steps / (elapsed_ms / 1e3)
    for w in wss:
        assert ckv.read_device_status(w) == 0, "device status set during the bench"

    # per-kernel durations: a second timed region replaying the traced graph
    for _ in range(3):
        traced.replay()
    torch.cuda.synchronize()
    t2 = torch.cuda.Event(enable_timing=True)
    t3 = torch.cuda.Event(enable_timing=True)
    n_traced = max(3, min(args.steps, 20))
    t2.record()
    for _ in range(n_traced):
        traced.replay()
    t3.record()
    torch.cuda.synchronize()
    traced_ms_per_step = t2.elapsed_time(t3) / n_traced

    per_kind: dict[str, list[float]] = {}
    for kind, ms in trace.records():
        per_kind.setdefault(kind, []).append(ms)
    step_bytes, score_bytes = algorithmic_bytes(cfg, layers, lengths)
    peak, peak_src = measured_peaks()
    if "fused" in per_kind:
        # the persistent kernel does the whole path: its algorithmic bytes are
        # the path's (K once, the SRH query rows, retained K/V read + written)
        kname, stats_ms, path_bytes = ("fused (scoring, pooling, top-k and gather of every "
                                       "unit of the call; persistent)"), per_kind["fused"], step_bytes
    else:
        kname, stats_ms, path_bytes = ("score (one pass over K)", per_kind.get("score", [float("nan")]),
                                       score_bytes)
    n_stats = len(stats_ms)
    avg_stats_ms = sum(stats_ms) / max(n_stats, 1)
    bytes_per_launch = path_bytes / max(n_stats, 1)
    achieved = bytes_per_launch / (avg_stats_ms / 1e3) / 1e9
    roofline = {"bound": "hbm", "kernel": kname, "achieved": round(achieved, 1),
                "peak": peak, "unit": "GB/s", "frac": round(achieved / peak, 4),
                "peak_source": f"{peak_src} (MEASURED_PEAKS.json hbm_gbs)" if peak_src == "measured"
                else "fallback 6.8 TB/s",
                "bytes_per_launch": int(bytes_per_launch), "launches_per_step": n_stats,
                "avg_launch_us": round(avg_stats_ms * 1e3, 2),
                "timing": f"CUDA events around each launch in a traced replay of the step "
                          f"({n_traced} steps, {traced_ms_per_step:.3f} ms/step serialised); the "
                          "timed step overlaps consecutive kernels",
                "traffic": profiled_traffic(cfg.name, lpc)}
    path_gbs = step_bytes / (ms_per_step / 1e3) / 1e9
    kernels = {k: {"launches_per_step": len(v), "avg_us": round(1e3 * sum(v) / len(v), 2),
                   "total_us_per_step": round(1e3 * sum(v), 1)} for k, v in per_kind.items()}

    result = {
        "metric": METRIC, "value": round(value, 1), "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": max(args.warmup, 3), "ms_per_step": round(ms_per_step, 4),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (seeded generator: Gaussian Q/K/V, sinks, planted needles)",
        "config": workload_config(cfg, budgets, lengths),
        "run": {"cuda_graph": True, "parallelism": f"replicas x{world}",
                "layers_per_call": lpc, "call_streams": n_streams,
                "l2_bytes": torch.cuda.get_device_properties(dev).L2_cache_size,
                "sms": torch.cuda.get_device_properties(dev).multi_processor_count},
        "roofline": roofline,
        "path": {"algorithmic_bytes_per_step": step_bytes, "achieved_gbs": round(path_gbs, 1),
                 "frac_of_peak": round(path_gbs / peak, 4),
                 "frac_of_8tbs_nominal": round(path_gbs / 8000.0, 4),
                 "layer_tokens_per_s": round(value * cfg.n_layers, 1)},
        "kernels": kernels,
        "gpu_launches": int(launches_per_step * args.steps),
        "clocks": clocks,
        "timed_blocks": {"blocks": blocks, "steps_per_block": args.steps,
                         "ms_per_block": [round(x, 3) for x in block_ms],
                         "reported": "median block"},
    }

    # layer 0's block of the first call's outputs
    first = types.SimpleNamespace(indices=outs[0].indices[:, :int(outs[0].cu_out[B])])
    if not headline:
        if rank == 0 and not args.no_cpu_baseline:
            result["parity_layer0"] = sampled_parity(cfg, layers[0], first, max_units=2)
        return result
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        result["cpu_baseline"], result["parity_layer0"] = cpu_baseline(cfg, layers[0], first)
    if not args.no_e2e:
        result["e2e"] = run_e2e(args, cfg, layers, lprobs, ws, dev, dist, world)
    if not args.no_lse:
        result["lse_fed"] = run_lse_fed(args, cfg, layers, (q_all, k_all, v_all, T, B), dev, dist,
                                        world, tokens)
    return result


def cpu_baseline(cfg, layer, out):
    """The float64 oracle, as it stands, on one layer (every unit) of the same
    workload; extrapolated to all layers.  Also checks that layer's device
    result against the oracle."""
    import oracle
    from oracle import compare

    q = layer["q_win"].float().cpu().numpy()
    k = layer["k"].float().cpu().numpy()
    v = layer["v"].float().cpu().numpy()
    t = time.perf_counter()
    res = oracle.compress_layer(q, k, v, layer["cu_seqlens"], layer["srh_mask"],
                                layer["budgets"], cfg.window, cfg.pool_width)
    dt = time.perf_counter() - t
    tokens = int(layer["cu_seqlens"][-1])
    value = tokens / (dt * cfg.n_layers)
    parity = "ok"
    try:
        idx = out.indices.cpu().numpy()
        ties = 0
        for (s, g), unit in res.units.items():
            L = int(layer["cu_seqlens"][s + 1] - layer["cu_seqlens"][s])
            o0, o1 = int(res.cu_out[s]), int(res.cu_out[s + 1])
            ties += compare.check_unit_indices(idx[g, o0:o1], unit, L, cfg.window)
        parity = f"ok ({ties} near-tie differences)"
    except AssertionError as e:
        parity = f"FAILED: {e}"
    base = {"value": round(value, 2), "unit": UNIT, "cores": cpu_cores(), "kind": "oracle",
            "sample": f"layer 0 of {cfg.n_layers} ({len(res.units)} units, {tokens} tokens) in "
                      f"{dt:.2f} s, extrapolated x{cfg.n_layers} layers; numpy float64 "
                      "(BLAS threads for q.k^T, one core for the rest)"}
    return base, parity


def sampled_parity(cfg, layer, out, max_units: int) -> str:
    """Layer 0's first `max_units` units (sequence 0, groups 0, 1, ...)
    against the float64 oracle, unit by unit."""
    import oracle
    from oracle import compare

    q = layer["q_win"].float().cpu().numpy()
    k = layer["k"].float().cpu().numpy()
    cu = layer["cu_seqlens"]
    idx = out.indices.cpu().numpy()
    L = int(cu[1] - cu[0])
    budget = int(np.asarray(layer["budgets"]).reshape(-1)[0])
    ties = 0
    try:
        for g in range(min(max_units, cfg.num_kv_heads)):
            heads = oracle.srh_heads(layer["srh_mask"], g, cfg.group_size)
            unit = oracle.compress_unit(q[0, heads], k[cu[0]:cu[1], g], cfg.window,
                                        cfg.pool_width, budget, oracle.default_scale(cfg.head_dim))
            ties += compare.check_unit_indices(idx[g, :unit.indices.size], unit, L, cfg.window)
    except AssertionError as e:
        return f"FAILED: {e}"
    return f"ok ({min(max_units, cfg.num_kv_heads)} units of sequence 0, {ties} near-tie differences)"


def window_lse_torch(lay, cfg, dev):
    """Natural-log softmax denominators of every window query (what a
    prefill attention kernel returns as its log-sum-exp), computed with plain
    PyTorch fp32 matmuls as input preparation, outside any timed region."""
    q = lay["q_win"].to(dev).float()  # [B, Hq, W, d]
    k = lay["k"].to(dev).float()      # [T, Hkv, d]
    cu = [int(x) for x in lay["cu_seqlens"]]
    B, Hq, W, d = q.shape
    Hkv = k.shape[1]
    G = Hq // Hkv
    scale = 1.0 / math.sqrt(d)
    lse = torch.zeros((B, Hq, W), dtype=torch.float32, device=dev)
    for s in range(B):
        L = cu[s + 1] - cu[s]
        if L == 0:
            continue
        ks = k[cu[s]:cu[s + 1]].permute(1, 0, 2)                 # [Hkv, L, d]
        qs = q[s].reshape(Hkv, G * W, d)                         # [Hkv, G*W, d]
        z = torch.bmm(qs, ks.transpose(1, 2)) * scale            # [Hkv, G*W, L]
        pos = torch.arange(L, device=dev)
        wpos = (L - W + torch.arange(W, device=dev)).repeat(G)   # row -> its position
        z = z.masked_fill(pos[None, None, :] > wpos[None, :, None], float("-inf"))
        lse[s] = torch.logsumexp(z, dim=-1).reshape(Hq, W)
        if L < W:
            lse[s, :, :W - L] = 0.0
    return lse


def run_lse_fed(args, cfg, layers, packed, dev, dist, world, tokens):
    """The same step through compresskv_compress_layers_lse: the window
    queries' log-sum-exp is an input (a prefill attention kernel produces it),
    so the persistent kernel skips its first pass over K.  Every layer in one
    call, as the headline.  Reported beside the headline, which computes
    everything itself."""
    import paper_2606_24467_gb300 as ckv

    q_all, k_all, v_all, T, B = packed
    lse_all = torch.cat([window_lse_torch(lay, cfg, dev) for lay in layers])
    lpc = layers_per_call(cfg, layers, None)
    calls = [(l0, min(l0 + lpc, cfg.n_layers)) for l0 in range(0, cfg.n_layers, lpc)]
    n_streams = 1
    trace = ckv.Trace(capacity=8 * cfg.n_layers)

    def call_problem(l0, l1, tr=None):
        m = l1 - l0
        cu = np.concatenate([np.asarray(layers[0]["cu_seqlens"][:-1], np.int64) + j * T
                             for j in range(m)] + [[m * T]]).astype(np.int32)
        return ckv.Problem(q_all[l0 * B:l1 * B], k_all[l0 * T:l1 * T], cu, cfg.window,
                           cfg.pool_width, trace=tr)

    probs = [call_problem(l0, l1) for l0, l1 in calls]
    tprobs = [call_problem(l0, l1, trace) for l0, l1 in calls]
    budgets = [np.concatenate([np.asarray(layers[l]["budgets"]).reshape(-1) for l in range(l0, l1)])
               for l0, l1 in calls]
    masks = [np.stack([np.asarray(layers[l]["srh_mask"]) for l in range(l0, l1)])
             for l0, l1 in calls]
    outs = [ckv.LayerOutputs(probs[c], budgets[c], cfg.head_dim, k_all.dtype, dev, scores=False)
            for c in range(len(calls))]
    wss = [ckv.workspace(probs[0], dev) for _ in range(n_streams)]
    lanes = [torch.cuda.Stream() for _ in range(n_streams)]

    def step(pr, streams):
        cur = torch.cuda.current_stream()
        fork = torch.cuda.Event()
        fork.record(cur)
        for st in lanes[:streams]:
            st.wait_event(fork)
        for c, (l0, l1) in enumerate(calls):
            o = outs[c]
            ckv.compress_layers_lse(pr[c], l1 - l0, q_all[l0 * B:l1 * B], k_all[l0 * T:l1 * T],
                                    v_all[l0 * T:l1 * T], lse_all[l0 * B:l1 * B], masks[c],
                                    budgets[c], o.indices, o.k_out, o.v_out, wss[c % streams],
                                    stream=lanes[c % streams])
        for st in lanes[:streams]:
            done = torch.cuda.Event()
            done.record(st)
            cur.wait_event(done)

    step(probs, n_streams)
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, capture_error_mode="thread_local"):
        step(probs, n_streams)
    traced = torch.cuda.CUDAGraph()
    trace.reset()
    with torch.cuda.graph(traced, capture_error_mode="thread_local"):
        step(tprobs, 1)
    for _ in range(max(args.warmup, 3)):
        graph.replay()
    torch.cuda.synchronize()
    barrier(dist)
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    t0.record()
    for _ in range(args.steps):
        graph.replay()
    t1.record()
    torch.cuda.synchronize()
    el = reduce_max(dist, t0.elapsed_time(t1), dev)
    for _ in range(3):
        traced.replay()
    torch.cuda.synchronize()
    per_kind: dict[str, list[float]] = {}
    for kind, ms in trace.records():
        per_kind.setdefault(kind, []).append(ms)
    for w in wss:
        assert ckv.read_device_status(w) == 0, "device status set during the LSE-fed bench"
    # the persistent kernel (given-LSE mode) does the whole path: its bytes
    # are the headline's path bytes
    kern_ms = per_kind.get("fused", per_kind.get("score", [float("nan")]))
    step_bytes, _ = algorithmic_bytes(cfg, layers, [int(x) for x in np.diff(layers[0]["cu_seqlens"])])
    path_bytes = step_bytes / max(len(kern_ms), 1)
    peak, _ = measured_peaks()
    achieved = path_bytes / (sum(kern_ms) / len(kern_ms) / 1e3) / 1e9
    return {"value": round(world * tokens * args.steps / (el / 1e3), 1), "unit": UNIT,
            "ms_per_step": round(el / args.steps, 4), "layers_per_call": lpc,
            "call_streams": n_streams,
            "kernels": {k: {"launches_per_step": len(v), "avg_us": round(1e3 * sum(v) / len(v), 2)}
                        for k, v in per_kind.items()},
            "roofline": {"bound": "hbm", "kernel": "fused (given LSE: one pass over K)",
                         "achieved": round(achieved, 1), "peak": peak, "unit": "GB/s",
                         "frac": round(achieved / peak, 4),
                         "bytes_per_launch": int(path_bytes)},
            "note": "window-query log-sum-exp supplied (prepared with PyTorch outside the timed "
                    "region, as a prefill attention kernel would return it); not the headline"}


def run_e2e(args, cfg, layers, probs, ws, dev, dist, world):
    """The same metric through the public API with host buffers: every step
    copies each layer's Q window and K from pinned host memory, compresses it
    with V left in pinned host memory (the gather reads only the kept rows
    over the host link) and reads the compressed cache and indices back.
    Copies of layer l+1 overlap the compression of layer l (two device slots;
    K split over two copy streams, one per copy engine)."""
    import paper_2606_24467_gb300 as ckv

    host = []
    for lay in layers:
        host.append({k: lay[k].cpu().pin_memory() for k in ("q_win", "k", "v")})
    slots = [{k: torch.empty_like(layers[0][k]) for k in ("q_win", "k")} for _ in range(2)]
    outs_h, outs_d = [], []
    for l, lay in enumerate(layers):
        o = ckv.LayerOutputs(probs[l], lay["budgets"], cfg.head_dim, lay["k"].dtype, dev,
                             scores=False)
        outs_d.append(o)
        outs_h.append({"indices": torch.empty(o.indices.shape, dtype=o.indices.dtype, pin_memory=True),
                       "k_out": torch.empty(o.k_out.shape, dtype=o.k_out.dtype, pin_memory=True),
                       "v_out": torch.empty(o.v_out.shape, dtype=o.v_out.dtype, pin_memory=True)})
    # host->device bytes: Q and K copied, plus the V rows the gather reads in
    # place (as many as it writes)
    h2d = sum(h[key].numel() * h[key].element_size() for h in host for key in ("q_win", "k"))
    h2d += sum(o.v_out.numel() * o.v_out.element_size() for o in outs_d)
    d2h = sum(t.numel() * t.element_size() for h in outs_h for t in h.values())
    comp = torch.cuda.current_stream()
    copies = [torch.cuda.Stream(), torch.cuda.Stream()]
    T = layers[0]["k"].shape[0]
    halves = [(0, T // 2), (T // 2, T)]
    # Problems built on the slot tensors (same shapes/strides as the resident ones)
    sprobs = [[ckv.Problem(slots[i]["q_win"], slots[i]["k"], lay["cu_seqlens"], cfg.window,
                           cfg.pool_width) for i in range(2)] for lay in layers]

    def step():
        done = [torch.cuda.Event() for _ in range(2)]
        ready = [[torch.cuda.Event() for _ in range(2)] for _ in range(len(layers))]
        for l in range(len(layers) + 1):
            if l < len(layers):
                i = l % 2
                for c, (a, b) in enumerate(halves):
                    with torch.cuda.stream(copies[c]):
                        if l >= 2:
                            copies[c].wait_event(done[i])
                        if c == 0:
                            slots[i]["q_win"].copy_(host[l]["q_win"], non_blocking=True)
                        slots[i]["k"][a:b].copy_(host[l]["k"][a:b], non_blocking=True)
                        ready[l][c].record(copies[c])
            if l >= 1:
                j = l - 1
                i = j % 2
                for c in range(2):
                    comp.wait_event(ready[j][c])
                o = outs_d[j]
                ckv.compress_layer(sprobs[j][i], slots[i]["q_win"], slots[i]["k"], host[j]["v"],
                                   layers[j]["srh_mask"], layers[j]["budgets"], o.indices,
                                   o.k_out, o.v_out, ws, stream=comp)
                done[i].record(comp)
                for key in ("indices", "k_out", "v_out"):
                    outs_h[j][key].copy_(getattr(o, key), non_blocking=True)
        comp.synchronize()

    step()
    torch.cuda.synchronize()
    barrier(dist)
    t = time.perf_counter()
    for _ in range(args.e2e_steps):
        step()
    torch.cuda.synchronize()
    el = reduce_max(dist, time.perf_counter() - t, dev)
    tokens = sum(int(lay["cu_seqlens"][-1]) for lay in layers[:1])
    return {"value": round(world * tokens * args.e2e_steps / el, 1), "unit": UNIT,
            "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h),
            "steps": args.e2e_steps, "ms_per_step": round(1e3 * el / args.e2e_steps, 3),
            "note": "pinned host buffers; Q and K copied (K in two halves on two copy "
                    "streams), overlapped with compression of the previous layer; V stays "
                    "in pinned host memory and the gather reads only the kept rows "
                    "(counted in h2d_bytes_per_step)"}


# --------------------------------------------------------------------- reference arm
def run_reference(args):
    """The float64 oracle on the host cores, as it stands: each step is one
    unit (sequence x KV group) of layer 0 of the workload, extrapolated to the
    whole workload (all units of all layers)."""
    rank, world, _ = dist_env()
    if rank != 0:
        return
    import oracle

    cfg = wl.get(args.workload)
    lengths = wl.sequence_lengths(cfg)
    masks = wl.srh_masks(cfg)
    budgets = wl.layer_budgets(cfg, lengths)
    lay = wl.make_layer(cfg, 0, lengths=lengths, masks=masks, budgets=budgets)
    q = lay["q_win"].float().numpy()
    k = lay["k"].float().numpy()
    G = cfg.group_size
    cu = lay["cu_seqlens"]
    units = [(s, g) for s in range(cfg.batch) for g in range(cfg.num_kv_heads)]

    def one(i):
        s, g = units[i % len(units)]
        heads = oracle.srh_heads(lay["srh_mask"], g, G)
        return oracle.compress_unit(q[s, heads], k[cu[s]:cu[s + 1], g], cfg.window,
                                    cfg.pool_width, int(lay["budgets"][s]),
                                    oracle.default_scale(cfg.head_dim))

    for i in range(max(args.warmup, 1)):
        one(i)
    times = []
    for i in range(args.steps):
        t = time.perf_counter()
        one(i)
        times.append(time.perf_counter() - t)
    per_unit = statistics.mean(times)
    tokens = sum(lengths)
    n_units_total = len(units) * cfg.n_layers
    # a unit is 1/n_units_total of the workload's tokens x layers: the rate in
    # workload tokens per second is the same whether measured per unit or per
    # whole step
    value = tokens / (per_unit * n_units_total)
    line = {
        "impl": "reference", "metric": METRIC, "value": round(value, 3), "unit": UNIT,
        "n_gpus": world, "steps": args.steps, "warmup": max(args.warmup, 1),
        "ms_per_step": round(per_unit * 1e3, 3), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic (same seeded generator)",
        "config": workload_config(cfg, budgets, lengths),
        "step": "one unit (1 sequence x 1 KV group of layer 0) per step, as timed",
        "extrapolated_ms_per_workload_step": round(per_unit * n_units_total * 1e3, 1),
        "cpu_baseline": {"value": round(value, 3), "unit": UNIT, "cores": cpu_cores(),
                         "kind": "oracle",
                         "sample": f"each step = 1 unit (1 sequence x 1 KV group, L={lengths[0]}) "
                                   f"of layer 0, mean {per_unit:.3f} s, extrapolated to "
                                   f"{n_units_total} units"},
        "e2e": {"value": round(value, 3), "unit": UNIT, "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def main():
    args = parse_args()
    if args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
