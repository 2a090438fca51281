#!/usr/bin/env python
"""Throughput of the interaction-network edge classifier on GB300.

One step = one gnn_infer call on one synthetic full event (300,000 nodes,
1,000,000 candidate edges, 12 node features, H=128, T=8, 3-layer MLPs):
device-side CSR build, encoders, eight message-passing iterations and the
classifier, inputs resident in HBM.  Prints one JSON line (rank 0).  The
headline steps are timed with nothing but their own CUDA events; the
per-kernel split (`kernels`, and the dominant kernel's `roofline`) comes from a
second pass with the library's profiling events between kernel groups.  After
the timed steps, and outside `value`: `pipeline` times every stage of the
tracking pipeline once on the same event (embedding, graph building,
filtering, the network, track labels), `bf16` times the bf16 model on the same
event and `batch16` one call on 16 events (4.8M nodes, 16M edges), each with
its own step roofline.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl gb300|reference]

N > 1 runs under torchrun: every rank scores its own event (independent
events, no data-path collective), so scaling is weak and `value` is the sum
over ranks.  `--impl reference` times the fp64 CPU oracle on a bounded sample
of the same workload (rank 0 only)."""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2402_09633_gb300 import synthetic as S  # noqa: E402

METRIC = "GNN inference edges/sec and events/sec (300k-node/1M-edge) on 1 GB300; % of roofline"
UNIT = "edges/s"
L2_FLUSH_BYTES = 256 << 20          # > 2x the 129 MB L2, written between timed steps
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
NOMINAL_HBM_GBS = 7900.0       # GB300 HBM3e datasheet bandwidth; fractions against it are a second line


def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            d = json.load(f)
        return d, "measured"
    return dict(FALLBACK_PEAKS), "fallback"


# ------------------------------------------------------------------ traffic model
def step_roofline(model, peaks, mean_ms: float, **extra):
    """Step-level roofline: the algorithmic bytes and flops of one step against the measured
    peaks (the headline fraction), and the bytes against the nominal HBM bandwidth."""
    t_roof_ms = 1e3 * max(model["bytes"] / (peaks["hbm_gbs"] * 1e9), model["flops"] / (peaks["bf16_tflops"] * 1e12))
    t_nom_ms = 1e3 * max(model["bytes"] / (NOMINAL_HBM_GBS * 1e9), model["flops"] / (peaks["bf16_tflops"] * 1e12))
    return {"t_roof_ms": t_roof_ms, "frac": t_roof_ms / mean_ms, "bytes_alg": model["bytes"],
            "flops_alg": model["flops"], "t_roof_nominal_hbm_ms": t_nom_ms, "frac_of_nominal_hbm": t_nom_ms / mean_ms,
            **extra}


def step_model(w: S.Workload):
    """Algorithmic bytes and flops of one step (whole path) and of the two iteration kernels."""
    m, ev = w.model, w.event
    N, E = ev.n_nodes * w.n_events, ev.n_edges * w.n_events
    bf16 = m.precision == S.PRECISION_BF16
    # s: bytes of a stored activation (the step model); the projections P_s, P_d are fp32 in both models
    H, T, L, Fn, s, sp = m.hidden, m.n_iters, m.mlp_layers, m.n_node_feat, (2 if bf16 else 4), 4
    bytes_step = (32 * E + 4 * N + 4 * Fn * N + (E + N) * H * s
                  + T * ((3 * E + 2 * N) * H * s + 4 * E + 4 * N) + (2 * E + N) * H * s + 8 * E)
    mac_edge_iter = E * H * H * L                           # e * W_e, then L-1 H x H layers
    mac_node_iter = N * (2 * H * H + 2 * H * H + H * H * (L - 1))   # P_s, P_d, [h,a] layer, rest
    flops_step = 2 * (T * (mac_edge_iter + mac_node_iter)
                      + N * (Fn * H + H * H * (L - 1) + 2 * H * H)      # node encoder + projections
                      + E * (2 * H + H * H * (L - 1))                   # edge encoder
                      + E * (H * H * L + H))                            # classifier (+ head)
    edge_update = {"bytes": E * (2 * H * s + H * sp + 8) + N * H * sp, "flops": 2 * mac_edge_iter,
                   "bytes_note": "per edge: e read + e write + gathered W_s h_src row (fp32) + 2 indices; "
                                 "per node: W_d h_dst + b1 row (fp32)"}
    node_update = {"bytes": N * (3 * H * s + 2 * H * sp), "flops": 2 * mac_node_iter,
                   "bytes_note": "per node: h and a read, h write, P_s and P_d (fp32) write"}
    return {"bytes": bytes_step, "flops": flops_step, "N": N, "E": E,
            "edge_update": edge_update, "node_update": node_update}


# ------------------------------------------------------------------ ncu traffic
PROFILE_FOR_KERNEL = {("edge_update", False): "edge_update_full_event.md",
                      ("edge_update", True): "edge_update_bf16_full_event.md"}
KERNEL_SOURCES = ("ptx.cuh", "csr.cuh", "mlp_tiles.cuh")


def source_hash() -> str:
    """First 16 hex digits of a sha256 over the code of the sources that define the profiled
    kernels and their launch geometry (the host API around them is left out): `//` comments,
    trailing blanks and empty lines are skipped, so editing a comment does not void a profile."""
    import hashlib
    h = hashlib.sha256()
    for f in KERNEL_SOURCES:
        with open(os.path.join(ROOT, "paper_2402_09633_gb300", "csrc", f)) as fh:
            for line in fh:
                code = line.split("//", 1)[0].rstrip()
                if code:
                    h.update(code.encode() + b"\n")
    return h.hexdigest()[:16]


def profiled_traffic(kernel: str, bf16: bool = False):
    """DRAM bytes per launch from the committed ncu summary of `kernel` (fp32 or bf16 model), or
    None when there is none or the kernel sources changed since the counters were taken."""
    name = PROFILE_FOR_KERNEL.get((kernel, bf16))
    path = os.path.join(ROOT, "profiles", name) if name else None
    if not path or not os.path.exists(path):
        return None
    fields = {}
    with open(path) as f:
        for line in f:
            if ":" in line and line.split(":", 1)[0].strip() in ("source_sha256", "dram_bytes_per_launch"):
                k, v = line.split(":", 1)
                fields[k.strip()] = v.split()[0]
    if fields.get("source_sha256") != source_hash() or "dram_bytes_per_launch" not in fields:
        return None
    return int(fields["dram_bytes_per_launch"])


# ------------------------------------------------------------------ clocks
def gpu_index_for(local_rank: int) -> str:
    vis = os.environ.get("CUDA_VISIBLE_DEVICES")
    if vis:
        items = [v.strip() for v in vis.split(",") if v.strip()]
        if local_rank < len(items):
            return items[local_rank]
    return str(local_rank)


class ClockSampler:
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu: str):
        self.proc = None
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", gpu, f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "100"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"], "samples": 0}
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
            out, _ = self.proc.communicate()
        sm, smax, power, reasons = [], [], [], set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for line in out.strip().splitlines():
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 8:
                continue
            try:
                sm.append(float(parts[0])); smax.append(float(parts[1])); power.append(float(parts[2]))
            except ValueError:
                continue
            for n, v in zip(names, parts[4:8]):
                if v.lower() == "active":
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(smax) if smax else None,
                "power_w_max": max(power) if power else None,
                "reasons": sorted(reasons), "samples": len(sm)}


# ------------------------------------------------------------------ CPU oracle sample
def oracle_sample(w: S.Workload, scale: float, seed: int = 0):
    """A bounded sample of the workload: the same generator and model at `scale` of the event."""
    ev = w.event
    spec = S.EventSpec(max(int(ev.n_nodes * scale), 20), ev.n_extra_feat, ev.mode, ev.dphi_window,
                       ev.fanout, max(int(ev.n_edges * scale), 1) if ev.mode == "powerlaw" else 0)
    x, ei = S.generate_event(spec, seed)
    W = S.init_weights(w.model, w.weight_seed)
    return W, x, ei


def time_oracle(w: S.Workload, scale: float, repeats: int = 1):
    from oracle import gnn_oracle as O       # CPU baseline leg only
    W, x, ei = oracle_sample(w, scale)
    bf16 = w.model.precision == S.PRECISION_BF16
    O.forward(W, x[:50], ei[:, :0], w.model.n_iters, bf16=bf16)          # import / allocator warm-up
    times = []
    for _ in range(repeats):
        t0 = time.perf_counter()
        O.forward(W, x, ei, w.model.n_iters, w.model.ln_eps, bf16=bf16)
        times.append(time.perf_counter() - t0)
    return ei.shape[1], x.shape[0], times


def cpu_cores() -> int:
    for var in ("OPENBLAS_NUM_THREADS", "OMP_NUM_THREADS"):
        if os.environ.get(var, "").isdigit():
            return int(os.environ[var])
    return os.cpu_count() or 1


# ------------------------------------------------------------------ reference arm
def run_reference(args, rank: int):
    if rank != 0:
        return
    w = S.WORKLOADS[args.workload]
    total = args.steps + args.warmup
    scale = 0.01 if total <= 60 else 0.003
    edges_per_step = []
    times = []
    for k in range(total):
        e, n, t = time_oracle(w, scale, 1)
        if k >= args.warmup:
            times.append(t[0]); edges_per_step.append(e)
    sec = sum(times)
    value = sum(edges_per_step) / sec
    sample = (f"{n} nodes / {e} edges from the '{w.name}' generator ({scale:g} of the event), "
              f"same model (H={w.model.hidden}, T={w.model.n_iters}, L={w.model.mlp_layers}), fp64 numpy")
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * sec / len(times),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": workload_config(w),
            "events_per_s": value / w.event.n_edges,
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cpu_cores(), "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line))


def workload_config(w: S.Workload):
    m, ev = w.model, w.event
    return {"workload": w.name, "description": w.description, "n_nodes": ev.n_nodes * w.n_events,
            "n_edges": ev.n_edges * w.n_events, "events_per_step": w.n_events,
            "node_features": m.n_node_feat, "hidden": m.hidden, "n_iters": m.n_iters,
            "mlp_layers": m.mlp_layers, "l2": "256 MB buffer written between timed steps",
            "parallelism": "replicas (one event per GPU per step)"}


# ------------------------------------------------------------------ ranks
def whole_job(local_s: float, local_units: float, world: int, device=None):
    """Whole-job figures of a step that every rank runs on its own events (replicas, no data-path
    collective): the slowest rank's time and the units summed over ranks, so throughput is
    units / time.  All ranks must call it (two all-reduces)."""
    if world == 1:
        return local_s, local_units
    import torch
    import torch.distributed as dist
    t = torch.tensor([local_s], dtype=torch.float64, device=device)
    u = torch.tensor([local_units], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    dist.all_reduce(u, op=dist.ReduceOp.SUM)
    return float(t.item()), float(u.item())


# ------------------------------------------------------------------ GB300 arm
def run_pipeline(net, w: S.Workload, x, dev, reps: int = 5):
    """Every stage of the tracking pipeline on the bench event, each timed with CUDA events on the
    current stream (mean of `reps` after one untimed call): embedding, fixed-radius graph building,
    filtering, the interaction network on the kept edges, track labels.  Random-init embedding and
    filter weights; the radius is the median distance to the 4th nearest neighbour of 2,000 sampled
    hits, the filter threshold the median filter score (setup, outside the timed calls)."""
    import torch
    net.load_embedding(S.pack_embed_blob(w.model, S.init_embed_weights(w.model, 8, 2)))
    net.load_filter(S.pack_filter_blob(w.model, S.init_filter_weights(w.model, 1)))
    N = x.shape[0]
    out = {}

    def timed(name, fn):
        res = fn()
        torch.cuda.synchronize(dev)
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        for _ in range(reps):
            res = fn()
        b.record()
        torch.cuda.synchronize(dev)
        out[name + "_ms"] = a.elapsed_time(b) / reps
        return res

    emb = timed("embed", lambda: net.embed(x))
    sample = emb[torch.randperm(N, generator=torch.Generator().manual_seed(0))[:2000].to(dev)]
    radius = float(torch.cdist(sample, emb).kthvalue(5, dim=1).values.median())
    cand, n_cand = timed("build_graph", lambda: net.build_graph(emb, x, radius, 40 * N))
    cand = cand.contiguous()
    fsc, _, _ = net.filter_edges(x, cand, 0.5)
    thr = float(fsc.median())
    _, kept, _ = timed("filter", lambda: net.filter_edges(x, cand, thr))
    kept = kept.contiguous()
    scores = timed("infer", lambda: net.infer(x, kept))
    timed("track_labels", lambda: net.track_labels(scores, kept, N, 0.5))
    out.update({"total_ms": sum(v for k, v in out.items() if k.endswith("_ms")), "n_hits": N,
                "embedding_dim": 8, "radius": radius, "candidate_edges": n_cand,
                "filter_threshold": thr, "kept_edges": int(kept.shape[1]), "device_status": net.status()})
    return out


def time_steps(net, x, ei, scores, flush, stream, steps: int):
    """Device time (ms) of `steps` gnn_infer calls, one CUDA event pair per call on the launching
    stream, with the L2 flushed (a buffer of twice its size written) before each call."""
    import torch
    starts = [torch.cuda.Event(enable_timing=True) for _ in range(steps)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(steps)]
    for k in range(steps):
        flush.fill_(float(k))
        starts[k].record(stream)
        net.infer(x, ei, scores)
        ends[k].record(stream)
    torch.cuda.synchronize()
    return [a.elapsed_time(b) for a, b in zip(starts, ends)]


def kernel_split(net, x, ei, scores, flush, stream, steps: int):
    """Per-kernel-group device time from a separate pass of `steps` calls with the library's
    profiling events on (they sit between kernel groups, so the headline is timed without them)."""
    net.profile(True)
    net.profile_read()                                   # clear
    ms = time_steps(net, x, ei, scores, flush, stream, steps)
    prof = net.profile_read()
    net.profile(False)
    groups = {g: {"ms_total": t, "launches": n, "ms_per_launch": t / n} for g, (t, n) in prof.items() if n}
    return groups, sum(ms) / len(ms)


def cpu_model() -> str:
    """Host CPU model name, from lscpu or /proc/cpuinfo."""
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.lower().startswith("model name"):
                return line.split(":", 1)[1].strip()
    except (OSError, subprocess.SubprocessError):
        pass
    try:
        with open("/proc/cpuinfo") as f:
            for line in f:
                if line.lower().startswith(("model name", "cpu model")):
                    return line.split(":", 1)[1].strip()
    except OSError:
        pass
    import platform
    return platform.machine()


def side_workload(name: str, steps: int, dev, peaks, x_dev=None, ei_dev=None):
    """One more workload timed after the headline (outside its timed region): the bf16 model on the
    same event, or the 16-event batch in one call.  Returns its sub-object of the JSON line."""
    import torch
    from paper_2402_09633_gb300 import InteractionNetwork
    w = S.WORKLOADS[name]
    if x_dev is None:
        x_np, ei_np = (S.generate_batch(w.event, list(w.seeds)) if w.n_events > 1
                       else S.generate_event(w.event, w.seeds[0]))
        x_dev, ei_dev = torch.from_numpy(x_np).to(dev), torch.from_numpy(ei_np).to(dev)
    N, E = x_dev.shape[0], ei_dev.shape[1]
    net = InteractionNetwork(w.model, S.pack_blob(w.model, S.init_weights(w.model, w.weight_seed)))
    net.reserve(N, E)
    scores = torch.empty(E, dtype=torch.float32, device=dev)
    flush = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream(dev)
    time_steps(net, x_dev, ei_dev, scores, flush, stream, 3)
    ms = time_steps(net, x_dev, ei_dev, scores, flush, stream, steps)
    status = net.status()
    groups, _ = kernel_split(net, x_dev, ei_dev, scores, flush, stream, min(steps, 5))
    net.close()
    mean_ms = sum(ms) / len(ms)
    model = step_model(w)
    out = {"workload": name, "description": w.description, "n_nodes": N, "n_edges": E,
           "steps": steps, "ms_per_step": mean_ms, "edges_per_s": E / (mean_ms * 1e-3),
           "events_per_s": w.n_events / (mean_ms * 1e-3),
           "dtype": "bf16->f32" if w.model.precision == S.PRECISION_BF16 else "bf16x3->f32",
           "step_roofline": step_roofline(model, peaks, mean_ms, bytes_per_activation=2 if w.model.precision else 4),
           "kernels": {g: v["ms_per_launch"] for g, v in groups.items()}, "device_status": status}
    if w.model.precision == S.PRECISION_BF16:
        out["tolerance"] = ("stated 1e-2 max on logits is not met: the GPU's max logit error against the "
                            "fp64 oracle exceeds it on the full event, as does the oracle's own fp64-vs-fp32 "
                            "evaluation of the same bf16 model; tests/test_gpu_bf16.py checks the error's "
                            "distribution against that envelope")
    return out


def run_gb300(args, rank: int, world: int, local: int):
    import torch
    import torch.distributed as dist
    from paper_2402_09633_gb300 import InteractionNetwork
    from paper_2402_09633_gb300 import build as B

    if rank == 0 or world == 1:
        B.build()
    if world > 1:
        dist.init_process_group("nccl")
        dist.barrier()
        B.build()                       # no-op once rank 0 finished
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    w = S.WORKLOADS[args.workload]
    x_np, ei_np = (S.generate_batch(w.event, [s + rank * w.n_events for s in w.seeds])
                   if w.n_events > 1 else S.generate_event(w.event, w.seeds[0] + rank))
    N, E = x_np.shape[0], ei_np.shape[1]
    W = S.init_weights(w.model, w.weight_seed)
    net = InteractionNetwork(w.model, S.pack_blob(w.model, W))
    net.reserve(N, E)
    x = torch.from_numpy(x_np).to(dev)
    ei = torch.from_numpy(ei_np).to(dev)
    scores = torch.empty(E, dtype=torch.float32, device=dev)
    flush = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream(dev)

    time_steps(net, x, ei, scores, flush, stream, args.warmup)
    if net.status() != 0:
        raise RuntimeError("device error during warm-up")

    # headline: exactly `steps` timed calls, no profiling events inside
    sampler = ClockSampler(gpu_index_for(local))
    time.sleep(0.3)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize(dev)
    t_wall = time.perf_counter()
    step_ms = time_steps(net, x, ei, scores, flush, stream, args.steps)
    if world > 1:
        dist.barrier()
    wall = time.perf_counter() - t_wall
    clocks = sampler.stop()
    status = net.status()
    step_s, job_edges = whole_job(sum(step_ms) / len(step_ms) * 1e-3, E, world, dev)
    mean_ms = step_s * 1e3
    value = job_edges / step_s

    # per-kernel split: a second pass with the library's profiling events
    split_steps = max(3, min(args.steps, 20))
    groups, profiled_ms = kernel_split(net, x, ei, scores, flush, stream, split_steps)

    # end to end through the host-buffer entry point (copies inside the timed region)
    x_h = torch.from_numpy(x_np).pin_memory()
    ei_h = torch.from_numpy(ei_np).pin_memory()
    s_h = torch.empty(E, dtype=torch.float32).pin_memory()
    n_e2e = max(3, min(args.steps, 50))
    net.infer_host(x_h, ei_h, s_h)
    if world > 1:
        dist.barrier()
    t0 = time.perf_counter()
    for _ in range(n_e2e):
        net.infer_host(x_h, ei_h, s_h)
    e2e_s, _ = whole_job((time.perf_counter() - t0) / n_e2e, E, world, dev)
    e2e_ok = bool(np.array_equal(s_h.numpy(), scores.cpu().numpy()))

    if rank != 0:
        if world > 1:
            dist.destroy_process_group()
        return

    peaks, peak_src = load_peaks()
    side = {}
    if world == 1 and not args.no_side_workloads and args.workload == "full":
        pipeline = run_pipeline(net, w, x, dev)
        net.close()
        side["bf16"] = side_workload("full_bf16", max(3, min(args.steps, 50)), dev, peaks, x, ei)
        side["batch16"] = side_workload("batch16", max(3, min(args.steps, 10)), dev, peaks)
    else:
        pipeline = run_pipeline(net, w, x, dev) if w.n_events == 1 and not args.no_side_workloads else None
        net.close()

    model = step_model(w)
    kernels_only = {g: v for g, v in groups.items() if g != "host_copies"}
    dom = max(kernels_only, key=lambda g: kernels_only[g]["ms_total"])
    dom_avg_s = kernels_only[dom]["ms_per_launch"] * 1e-3
    dom_model = model.get(dom, None)
    roofline = None
    if dom_model is not None:
        achieved = dom_model["bytes"] / dom_avg_s / 1e9
        roofline = {"kernel": dom, "bound": "hbm", "achieved": achieved, "peak": peaks["hbm_gbs"],
                    "unit": "GB/s", "frac": achieved / peaks["hbm_gbs"],
                    "frac_of_nominal_hbm": achieved / NOMINAL_HBM_GBS,
                    "traffic": profiled_traffic(dom, w.model.precision == S.PRECISION_BF16),
                    "peak_source": f"{peak_src} (hbm_gbs, copy burst) -- of {peak_src}",
                    "bytes_per_launch": dom_model["bytes"], "avg_launch_ms": dom_avg_s * 1e3,
                    "launch_timing": f"CUDA events around each launch on the launching stream, "
                                     f"{split_steps} profiled steps after the headline",
                    "tensor_tflops_executed": (1 if w.model.precision == S.PRECISION_BF16 else 3)
                                              * dom_model["flops"] / dom_avg_s / 1e12}
    launches_per_step = sum(v["launches"] for v in kernels_only.values()) / split_steps

    cpu = None
    if world == 1 and not args.no_cpu_baseline:
        scale = 0.1
        e_s, n_s, t = time_oracle(w, scale, 1)
        cpu = {"value": e_s / t[0], "unit": UNIT, "cores": cpu_cores(), "kind": "oracle",
               "cpu_model": cpu_model(), "threads": cpu_cores(),
               "sample": f"{n_s} nodes / {e_s} edges from the '{w.name}' generator ({scale:g} of the "
                         f"event), same model, fp64 numpy, one pass of {t[0]:.1f} s"}

    line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": mean_ms, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16->f32" if w.model.precision == S.PRECISION_BF16 else "bf16x3->f32",
            "data": "synthetic",
            "config": workload_config(w),
            "events_per_s": value / E * w.n_events,                 # every rank scores events of E edges
            "roofline": roofline,
            "step_roofline": step_roofline(model, peaks, mean_ms),
            "kernels": groups,
            "kernels_pass": {"steps": split_steps, "ms_per_step_with_events": profiled_ms},
            **side,
            "pipeline": pipeline,
            "cpu_baseline": cpu,
            "e2e": {"value": job_edges / e2e_s, "unit": UNIT,
                    "h2d_bytes_per_step": int(x_np.nbytes + ei_np.nbytes),
                    "d2h_bytes_per_step": int(E * 4), "ms_per_step": e2e_s * 1e3,
                    "matches_device_path": e2e_ok},
            "gpu_launches": int(round(launches_per_step * args.steps)),
            "clocks": clocks,
            "device_status": status,
            "wall_s_timed_region": wall}
    print(json.dumps(line))
    if world > 1:
        dist.destroy_process_group()


def main():
    ap = argparse.ArgumentParser(description=__doc__)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=("gb300", "reference"), default="gb300")
    ap.add_argument("--workload", choices=tuple(S.WORKLOADS), default="full")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-side-workloads", action="store_true",
                    help="skip what is timed after the headline: the pipeline stages and the bf16-model and "
                         "16-event-batch sub-objects")
    args = ap.parse_args()
    rank = int(os.environ.get("RANK", 0))
    world = int(os.environ.get("WORLD_SIZE", 1))
    local = int(os.environ.get("LOCAL_RANK", 0))
    if args.warmup < 3:
        args.warmup = 3
    if args.impl == "reference":
        run_reference(args, rank)
    else:
        run_gb300(args, rank, world, local)


if __name__ == "__main__":
    main()
