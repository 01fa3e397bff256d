"""Benchmark: ResNet-50 inference with the DPRS-selected routine path on GB300.

One step = one inference of a 32 x 3 x 224 x 224 bf16 batch through the whole
routine path (every layer routine and adapt), replayed as a CUDA graph.
Tuning (profiling + DPRS) runs once before the timed region and is reported
separately.  Inputs are seeded synthetic tensors shaped like the paper's
workloads (no trained weights or datasets are available).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

--impl reference times the CPU oracle (plain fp64) on the same workload and
metric, one image per step as a bounded sample.  Multi-GPU: independent
replicas (one batch per rank, no collective on the data path).
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

METRIC = "ResNet-50 b1 latency (ms), b32 images/s; conv TFLOP/s & GB/s vs peak"
WORKLOAD = ("ResNet-50 v1.5 inference, batch 32, 3x224x224 bf16, residual adds fused into the conv that feeds "
            "them, DPRS path over {bf16 NCHW, bf16 NHWC}")
FALLBACK = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0, "sm_max_mhz": 2070.0}


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return d, "measured"
    return FALLBACK, "fallback"


def job_throughput(ms_local, ws, batch, dist=None, device="cpu"):
    """Replicas: every rank runs its own batch with no exchange on the data
    path; the job's step time is the slowest rank's (max over ranks, the one
    collective) and its throughput the images of all ranks over that time.
    Returns (ms_per_step, images_per_s)."""
    ms = ms_local
    if dist is not None:
        import torch
        t = torch.tensor([ms_local], dtype=torch.float64, device=device)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        ms = float(t.item())
    return ms, ws * batch / (ms / 1e3)


def dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled during the timed region."""
    Q = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
         "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
         "clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.proc = None
        self.lines = []  # (arrival time, csv line)
        self.t0 = self.t1 = None

    def start(self):
        """Start sampling and wait (up to 15 s) for the first sample, so that
        the timed region that follows is covered."""
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.Q}",
                                          "--format=csv,noheader,nounits", "-lms", "10"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
            deadline = time.monotonic() + 15.0
            while not self.lines and time.monotonic() < deadline:
                time.sleep(0.01)
        except Exception:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append((time.monotonic(), line.strip()))

    def begin(self):
        self.t0 = time.monotonic()

    def end(self):
        self.t1 = time.monotonic()

    def stop(self):
        if not self.proc:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        # samples that arrived while the timed region ran (plus the first one
        # after it, which nvidia-smi took during its last interval)
        inside = [l for (t, l) in self.lines if self.t0 is not None and self.t0 <= t <= (self.t1 or t)]
        after = [l for (t, l) in self.lines if self.t1 is not None and t > self.t1][:1]
        for l in inside + after:
            f = [x.strip() for x in l.split(",")]
            if len(f) < 7:
                continue
            try:
                sm.append(float(f[0]))
                mx.append(float(f[1]))
            except ValueError:
                continue
            for n, v in zip(names, f[3:7]):
                if v.lower() == "active":
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": sorted(reasons), "samples": len(sm)}


TRAFFIC_FILE = os.path.join(ROOT, "profiles", "conv_tc_r50_b32_bf16_traffic.md")


def tc_sources_digest():
    """sha256 over the tensor-core conv kernel sources: a DRAM-traffic figure
    measured with ncu is reported only while these are unchanged."""
    h = hashlib.sha256()
    for f in ("tc_conv.cuh", "kernels_tc.cu", "kernels_tc_sk.cu", "kernels_tc_halo.cu", "tc_common.cuh"):
        with open(os.path.join(ROOT, "paper_2110_06037_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()


def tc_traffic_per_step():
    """DRAM bytes (read + write) of the step's conv2/igemm_tc launches from the
    committed ncu summary, or None when it is missing or the kernel changed."""
    try:
        kv = {}
        with open(TRAFFIC_FILE) as fh:
            for line in fh:
                if ":" in line:
                    k, v = line.split(":", 1)
                    kv[k.strip().strip("`- ")] = v.strip().strip("`")
        if kv.get("kernel_sources_sha256") != tc_sources_digest():
            return None
        return float(kv["igemm_tc_dram_bytes_per_step"])
    except (OSError, KeyError, ValueError):
        return None


def conv_work(layers, in_shape, elem=2):
    """Algorithmic FLOPs and bytes of every layer (inputs, weights, output once)."""
    shapes = []
    work = []
    for l in layers:
        ins = [in_shape if j < 0 else shapes[j] for j in l["inputs"]]
        n, c, h, w = ins[0]
        p = l["params"]
        if l["type"] in ("conv2", "dwconv2"):
            g = p["groups"]
            P = (h + 2 * p["ph"] - p.get("dh", 1) * (p["kh"] - 1) - 1) // p["sh"] + 1
            Q = (w + 2 * p["pw"] - p.get("dw", 1) * (p["kw"] - 1) - 1) // p["sw"] + 1
            K = p["c_out"]
            out = (n, K, P, Q)
            fl = 2 * n * K * P * Q * (c // g) * p["kh"] * p["kw"]
            by = elem * (n * c * h * w + n * K * P * Q + K * (c // g) * p["kh"] * p["kw"]) + 4 * K
            if len(ins) == 2:  # residual input (fused add): one more read and one add per output
                fl += n * K * P * Q
                by += elem * n * K * P * Q
        elif l["type"] == "maxpool":
            P = (h + 2 * p["ph"] - p["kh"]) // p["sh"] + 1
            Q = (w + 2 * p["pw"] - p["kw"]) // p["sw"] + 1
            out = (n, c, P, Q)
            fl, by = 0, elem * (n * c * h * w + n * c * P * Q)
        elif l["type"] == "gap":
            out = (n, c, 1, 1)
            fl, by = n * c * h * w, elem * (n * c * h * w + n * c)
        elif l["type"] == "add":
            out = ins[0]
            fl, by = n * c * h * w, 3 * elem * n * c * h * w
        elif l["type"] == "mul":  # per-channel scale: the blob in and out, one scale per (n, c)
            out = ins[0]
            fl, by = n * c * h * w, elem * (2 * n * c * h * w + n * c)
        else:  # dense
            out = (n, p["out_features"], 1, 1)
            fl = 2 * n * p["in_features"] * p["out_features"]
            by = elem * (n * p["in_features"] + n * p["out_features"] + p["in_features"] * p["out_features"])
        shapes.append(out)
        work.append((fl, by))
    return work, shapes


def run_reference(args, ws, rank):
    """The CPU oracle on the same workload: one image per step (bounded sample)."""
    if rank != 0:
        return
    import synth
    from oracle.net import run_net
    x, layers = synth.resnet50(32)
    xs = x[:1]
    for _ in range(max(0, args.warmup and 1)):
        run_net(layers, xs, "bf16")
    times = []
    for _ in range(args.steps):
        t0 = time.perf_counter()
        run_net(layers, xs, "bf16")
        times.append(time.perf_counter() - t0)
    sec = sum(times) / len(times)
    v = 1.0 / sec
    cores = os.cpu_count()
    line = {"impl": "reference", "metric": METRIC, "value": v, "unit": "images/s", "n_gpus": ws,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": sec * 1e3, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": WORKLOAD + " (oracle: 1 image per step)", "batch": 32},
            "cpu_baseline": {"value": v, "unit": "images/s", "cores": cores, "kind": "oracle",
                             "sample": "1 of the 32 images per step, fp64 oracle, OpenMP over all host cores"},
            "e2e": {"value": v, "unit": "images/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line))


def cpu_baseline_sample():
    import synth
    from oracle.net import run_net
    x, layers = synth.resnet50(32)
    xs = x[:1]
    t0 = time.perf_counter()
    n = 0
    while True:
        run_net(layers, xs, "bf16")
        n += 1
        if time.perf_counter() - t0 > 10.0 or n >= 3:
            break
    sec = (time.perf_counter() - t0) / n
    return {"value": 1.0 / sec, "unit": "images/s", "cores": os.cpu_count(), "kind": "oracle",
            "sample": f"{n} single-image passes of the 32-image batch, fp64 oracle, OpenMP over all host cores"}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--batch", type=int, default=32)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-b1", action="store_true")
    ap.add_argument("--no-extras", action="store_true",
                    help="skip the extra rows of the benchmark line (bandwidth, MobileNetV2 / tiny CNN latency, "
                         "sweep summary, oracle timings)")
    ap.add_argument("--config", default="r50_b32",
                    choices=["r50_b32", "bandwidth", "sweep", "mbv2_b1", "r50_b1", "tiny", "layer", "vgg16_b32",
                             "vgg16_b1", "mbv3_b1", "hybrid", "q8_dense", "dw_band_14", "transpose_14", "wino_14"],
                    help="r50_b32 is the benchmark line; the others print one extra JSON line each")
    ap.add_argument("--layer", default="32,512,56,512,3,1",
                    help="--config layer: N,C,H,K,k,s of one bf16 NHWC conv (C -> K channels, HxH input)")
    ap.add_argument("--plan", default="",
                    help="tuned-state file (cost table + path): loaded if it exists, else written after tuning, "
                         "so that a profiler run times the same path as a plain run")
    ap.add_argument("--variant", type=int, default=-1,
                    help="--config layer: conv2/igemm_tc routine parameter index (-1: every one)")
    args = ap.parse_args()
    args.warmup = max(args.warmup, 3)
    ws, rank, local = dist_env()
    if args.impl == "reference":
        return run_reference(args, ws, rank)
    if args.config == "hybrid":
        return run_hybrid(args)
    if args.config != "r50_b32":
        return run_extra_config(args)

    import torch
    import synth
    import paper_2110_06037_gb300 as sn
    from paper_2110_06037_gb300 import routine_name

    torch.cuda.set_device(local)
    dist = None
    if ws > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")
    pk, pk_kind = peaks()

    # ---------------- tune: profile + DPRS ----------------
    x, layers0 = synth.resnet50(args.batch)
    sch = [("bf16", "nchw"), ("bf16", "nhwc")]
    stream = torch.cuda.Stream()
    t_tune0 = time.perf_counter()
    with torch.cuda.stream(stream):
        # the library's residual-add fusion pass runs before tuning
        g = sn.build_graph(layers0, x.shape, ("bf16", "nchw"), ("bf16", "nchw"), sch, fuse=True)
        layers = sn.fused_description(layers0, g.fused_ids)
        plan_loaded = bool(args.plan) and os.path.exists(args.plan)
        if plan_loaded:  # the saved cost table; DPRS on it gives the saved path again
            g.load_plan(args.plan)
        else:
            # 20 back-to-back launches per unit timing, the best 3 candidates per
            # (layer, schema) re-timed in 5 whole-net passes: three runs each of
            # (10, 2, 3), (20, 3, 5) and (40, 3, 8) tuned to 0.770-0.787,
            # 0.766-0.770 and 0.765-0.779 ms per step on GB300
            g.profile(warmup=3, iters=20, topk=3, passes=5)
        total, schemas, cands = g.select_path(sn.SN_SELECT_DPRS)
        if args.plan and not plan_loaded:
            g.save_plan(args.plan)
    stream.synchronize()
    tune_s = time.perf_counter() - t_tune0

    xd = torch.from_numpy(x).to(torch.bfloat16).cuda()
    out = g.new_output()
    flush = torch.empty(256 * 1024 * 1024, dtype=torch.uint8, device="cuda")  # > L2 (129 MB)
    g.set_option(sn.SN_OPT_CUDA_GRAPH, 1)
    with torch.cuda.stream(stream):
        for _ in range(args.warmup):
            g.run(xd, out)
    stream.synchronize()
    n_ops, n_kern = g.plan_stats(stream)
    arena_b, unshared_b = g.plan_memory(stream)

    # ---------------- timed region (device, per-step events, L2 flushed between steps) -------
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
    clocks = ClockSampler(local)
    if dist:
        dist.barrier()
    torch.cuda.synchronize()
    clocks.start()
    clocks.begin()
    torch.cuda.nvtx.range_push("sn_timed")
    with torch.cuda.stream(stream):
        for i in range(args.steps):
            flush.zero_()
            ev[i][0].record(stream)
            g.run(xd, out)
            ev[i][1].record(stream)
    torch.cuda.synchronize()
    torch.cuda.nvtx.range_pop()
    clocks.end()
    if dist:
        dist.barrier()
    clk = clocks.stop()
    step_ms = [a.elapsed_time(b) for a, b in ev]
    ms, value = job_throughput(sum(step_ms) / len(step_ms), ws, args.batch, dist, "cuda")

    # ---------------- e2e through the C ABI with host buffers ----------------
    # Every step is one sn_run_host call: the library uploads the batch from
    # pinned host memory (on its own copy stream, into one of two landing
    # buffers, so that the upload overlaps the previous step's net), runs the
    # net and copies the logits back to pinned host memory, in order on the
    # stream, so the timed region holds each step's host->device and
    # device->host copies.
    xh = torch.from_numpy(x).to(torch.bfloat16).pin_memory()
    oh = torch.empty(out.shape, dtype=out.dtype).pin_memory()
    with torch.cuda.stream(stream):
        for _ in range(3):
            g.run_host(xh, oh)
    stream.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        e0.record(stream)
        for _ in range(args.steps):
            g.run_host(xh, oh)
        e1.record(stream)
    stream.synchronize()
    e2e_ms = e0.elapsed_time(e1) / args.steps
    e2e = {"value": args.batch / (e2e_ms / 1e3), "unit": "images/s",
           "h2d_bytes_per_step": xh.numel() * xh.element_size(),
           "d2h_bytes_per_step": oh.numel() * oh.element_size(),
           "path": "sn_run_host (C ABI): copies from and to pinned host memory inside each call; the upload of "
                   "one call overlaps the net of the previous one (library copy stream, two landing buffers)"}

    # ---------------- per-op shares of the step ----------------
    # One replay of the step with a timing node around every op gives each
    # op's device time run on its own; the ops overlap in the timed replay
    # (programmatic dependent launch), so these times sum to more than the
    # step.  Each routine's time in the step is its share of that sum times
    # the measured ms_per_step, which by construction cannot exceed the step.
    g.set_option(sn.SN_OPT_CUDA_GRAPH, 0)
    t = g.cost_table()
    layer_ms = np.zeros(t["n_layers"])
    edge_ms = np.zeros(len(t["edges"]))
    reps = max(3, min(args.steps, 10))
    with torch.cuda.stream(stream):
        for _ in range(reps):
            flush.zero_()
            _, lm, em = g.run_timed(xd, out)
            layer_ms += lm
            edge_ms += em[: len(edge_ms)]
    layer_ms /= reps
    edge_ms /= reps
    op_sum = float(layer_ms[1:-1].sum() + edge_ms.sum())
    scale = ms / op_sum
    work, shapes = conv_work(layers, x.shape)
    per_routine = {}
    for i in range(1, t["n_layers"] - 1):
        c = int(cands[i])
        r = routine_name(int(t["routine"][c]))
        d = per_routine.setdefault(r, {"ms": 0.0, "flop": 0, "bytes": 0, "launches": 0})
        d["ms"] += float(layer_ms[i]) * scale
        d["flop"] += work[i - 1][0]
        d["bytes"] += work[i - 1][1]
        d["launches"] += 1
    if edge_ms.sum() > 0:
        per_routine["adapt/convert"] = {"ms": float(edge_ms.sum()) * scale, "flop": 0, "bytes": 0,
                                        "launches": int((edge_ms > 0).sum())}
    dom = max(per_routine, key=lambda r: per_routine[r]["ms"])
    d = per_routine[dom]
    sustained = pk.get("bf16_tflops_sustained", pk["bf16_tflops"])
    share = {"share_of_step": d["ms"] / ms, "time_ms": d["ms"],
             "method": "the routine's share of the per-op device times of one replay with a timing node around "
                       "every op (CUDA events on the launching stream), times ms_per_step"}
    if dom == "conv2/igemm_tc":
        achieved = d["flop"] / (d["ms"] / 1e3) / 1e12
        roof = {"bound": "tensor", "achieved": achieved, "peak": sustained, "unit": "TFLOP/s",
                "frac": achieved / sustained, "traffic": tc_traffic_per_step(),
                "traffic_unit": "DRAM bytes per step over the igemm_tc launches (ncu, cold L2 per kernel)",
                "algorithmic_flop": d["flop"], "algorithmic_bytes": d["bytes"], **share}
    elif dom in ("conv2/igemm_simt", "conv2/direct", "conv2/wino_f2x2_3x3"):
        ffma_peak = 2 * 128 * 152 * pk.get("sm_max_mhz", 2070.0) / 1e6  # TFLOP/s fp32 FFMA
        achieved = d["flop"] / (d["ms"] / 1e3) / 1e12
        roof = {"bound": "alu", "achieved": achieved, "peak": ffma_peak, "unit": "TFLOP/s",
                "frac": achieved / ffma_peak, "traffic": None, **share}
    else:
        achieved = d["bytes"] / (d["ms"] / 1e3) / 1e9
        roof = {"bound": "hbm", "achieved": achieved, "peak": pk["hbm_gbs"], "unit": "GB/s",
                "frac": achieved / pk["hbm_gbs"], "traffic": None, **share}
    roof["kernel"] = dom
    roof["peak_source"] = f"{pk_kind} (MEASURED_PEAKS.json)" if pk_kind == "measured" else "fallback"
    # every conv layer of the path: its share-derived time, TFLOP/s and the
    # fraction of the roofline its arithmetic intensity puts it under
    ridge = sustained * 1e12 / (pk["hbm_gbs"] * 1e9)  # FLOP per byte where the two roofs meet
    per_layer = []
    for i in range(1, t["n_layers"] - 1):
        lay = layers[i - 1]
        if lay["type"] != "conv2":
            continue
        fl, by = work[i - 1]
        us = float(layer_ms[i]) * scale * 1e3
        if us <= 0:
            continue
        p_ = lay["params"]
        ins = [x.shape if j < 0 else shapes[j] for j in lay["inputs"]]
        ai = fl / by
        row = {"layer": lay.get("name", str(i)),
               "shape": f"{ins[0][1]}->{p_['c_out']} {ins[0][2]}x{ins[0][3]} k{p_['kh']} s{p_['sh']}" +
                        (" +res" if len(lay["inputs"]) == 2 else ""),
               "routine": g.candidate_desc(int(cands[i])), "us": round(us, 2),
               "tflops": round(fl / us / 1e6, 1), "gbs": round(by / us / 1e3, 1), "ai": round(ai, 1),
               "bound": "tensor" if ai > ridge else "hbm"}
        row["frac"] = round(row["tflops"] / sustained if ai > ridge else row["gbs"] / pk["hbm_gbs"], 3)
        per_layer.append(row)

    # ---------------- ResNet-50 b1 latency (fp16, CUDA graph) ----------------
    b1 = None
    if not args.no_b1:
        x1, layers1 = synth.resnet50(1)
        s16 = [("f16", "nchw"), ("f16", "nhwc")]
        with torch.cuda.stream(stream):
            g1 = sn.build_graph(layers1, x1.shape, ("f16", "nchw"), ("f16", "nchw"), s16, fuse=True)
            g1.profile(warmup=3, iters=10, topk=2, passes=3)
            g1.select_path(sn.SN_SELECT_DPRS)
            g1.set_option(sn.SN_OPT_CUDA_GRAPH, 1)
            x1d = torch.from_numpy(x1).to(torch.float16).cuda()
            o1 = g1.new_output()
            for _ in range(5):
                g1.run(x1d, o1)
        stream.synchronize()
        lat = []
        for _ in range(20):
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            with torch.cuda.stream(stream):
                flush.zero_()
                a.record(stream)
                g1.run(x1d, o1)
                b.record(stream)
            stream.synchronize()
            lat.append(a.elapsed_time(b))
        b1 = {"mean_ms": statistics.mean(lat), "std_ms": statistics.pstdev(lat), "median_ms": statistics.median(lat)}

    # ---------------- the other rooflines and configurations (one GPU, rank 0) ----------------
    extras = None
    if rank == 0 and not args.no_extras:
        extras = {}
        t_ex = time.perf_counter()
        extras["bandwidth"] = _bandwidth_rows(sn, torch, synth, pk["hbm_gbs"], compact=True)
        lat_graphs = {}
        for name in ("mbv2_b1", "tiny"):
            extras[name] = _latency_config(sn, torch, synth, name, keep=lat_graphs)
        extras["sweep"] = _sweep_summary(sn, torch, synth, pk)
        if ws == 1:
            extras["oracle"] = _oracle_times(sn, synth, lat_graphs, g1_table=(g1.cost_table() if b1 else None))
        extras["seconds"] = time.perf_counter() - t_ex

    cpu = None
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline_sample()

    if rank == 0:
        line = {"metric": METRIC, "value": value, "unit": "images/s", "n_gpus": ws, "steps": args.steps,
                "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
                "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
                "config": {"workload": WORKLOAD, "batch": args.batch, "parallelism": f"replicas x{ws}",
                           "l2": "flushed between steps (256 MB write outside the step events)",
                           "timing": "CUDA events around each step on the launching stream, CUDA-graph replay"},
                "e2e": e2e, "gpu_launches": n_kern * args.steps, "roofline": roof, "cpu_baseline": cpu,
                "clocks": clk, "tuning_s": tune_s, "path_cost_ns": total,
                "plan": ("loaded from " + os.path.basename(args.plan)) if plan_loaded else "tuned in this run",
                "r50_b1_fp16_latency": b1,
                "activation_memory": {"arena_bytes": arena_b, "unshared_bytes": unshared_b},
                "per_routine_ms": {k: round(v["ms"], 4) for k, v in per_routine.items()},
                "per_layer": per_layer, "extras": extras}
        print(json.dumps(line))
    if dist:
        dist.destroy_process_group()



# ----------------------------------------------------------------------------
# the other configurations (one JSON line each; not the benchmark line)
# ----------------------------------------------------------------------------

def _single_layer_graph(sn, layer, in_shape, schema):
    return sn.build_graph([dict(layer, inputs=[-1])], in_shape, schema, schema, [schema])


def _time_back_to_back(torch, fn, reps=50, warm=5):
    """Mean device time of `reps` back-to-back launches (CUDA events resolve ~2 us on this GPU)."""
    for _ in range(warm):
        fn()
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record()
    for _ in range(reps):
        fn()
    b.record()
    torch.cuda.synchronize()
    return a.elapsed_time(b) / reps


def _time_graph(torch, fn, reps=20):
    """Mean device time of one fn() from `reps` calls captured into a CUDA graph
    and replayed (no host launch cost; events resolve ~2 us, so many launches
    are timed together).  Median of five replays."""
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        for _ in range(3):
            fn()
    s.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=s):
        for _ in range(reps):
            fn()
    graph.replay()
    torch.cuda.synchronize()
    ts = []
    for _ in range(5):
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        graph.replay()
        b.record()
        torch.cuda.synchronize()
        ts.append(a.elapsed_time(b) / reps)
    return statistics.median(ts)


L2_BYTES = 129 << 20


def _sets_for(nbytes):
    """Buffer sets to rotate through so that one pass over them moves at least
    four L2 capacities: every launch then starts with its operands out of L2."""
    return max(2, min(64, -(-4 * L2_BYTES // max(1, nbytes))))


def _time_cold(torch, fns, reps=40):
    """Mean device time of one call from a CUDA-graph replay of `reps` calls that
    cycle through `fns` (each bound to its own buffers, together larger than L2).
    Median of five replays."""
    return _time_graph(torch, _Cycle(fns), reps=max(reps, len(fns)))


class _Cycle:
    def __init__(self, fns):
        self.fns, self.i = fns, 0

    def __call__(self):
        self.fns[self.i % len(self.fns)]()
        self.i += 1


def _forced(sn, g, routine, variant=0):
    import numpy as _np
    t = g.cost_table()
    c = [i for i in range(len(t["cost"])) if t["layer"][i] == 1 and sn.routine_name(int(t["routine"][i])) == routine
         and t["variant"][i] == variant][0]
    g.set_path([int(_np.flatnonzero(t["layer"] == 0)[0]), c, int(_np.flatnonzero(t["layer"] == 2)[0])])


def _latency_ms(torch, g, xd, y, stream, flush, reps=20):
    """Median CUDA-event latency of one CUDA-graph replay of the net, L2 flushed before each."""
    with torch.cuda.stream(stream):
        for _ in range(3):
            g.run(xd, y)
    stream.synchronize()
    lat = []
    for _ in range(reps):
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        with torch.cuda.stream(stream):
            flush.zero_()
            a.record(stream)
            g.run(xd, y)
            b.record(stream)
        stream.synchronize()
        lat.append(a.elapsed_time(b))
    return statistics.median(lat)


def run_hybrid(args):
    """Hybrid float/qint8 tuning (section V-C, Table I) on the paper's four nets
    at batch 1: (1) no tuning: every layer's first routine in fp16 NCHW;
    (2) tuning over the fp16 schemas; (3) over the qint8 schemas; (4) over both
    (hybrid).  Scales come from calibration on the synthetic input."""
    import torch
    import synth
    import paper_2110_06037_gb300 as sn
    torch.cuda.set_device(0)
    F16 = [("f16", "nchw"), ("f16", "nhwc")]
    Q8 = [("qi8", "nchw"), ("qi8", "nhwc")]
    io = ("f16", "nchw")
    stream = torch.cuda.Stream()
    flush = torch.empty(256 << 20, dtype=torch.uint8, device="cuda")
    nets = {"vgg16": lambda: synth.vgg16(1), "resnet50": lambda: synth.resnet50(1),
            "mobilenet_v2": lambda: synth.mobilenet_v2(1), "mobilenet_v3": lambda: synth.mobilenet_v3(1)}
    rows = {}
    for name, make in nets.items():
        x, layers = make()
        if name != "vgg16":
            layers = sn.fuse_residual(layers, x.shape)
        xd = torch.from_numpy(x).to(torch.float16).cuda()
        row = {}
        outs = {}

        def tuned(schemas, scales_from=None):
            with torch.cuda.stream(stream):
                g = sn.build_graph(layers, x.shape, io, io, schemas)
                if scales_from is not None:
                    for i in range(-1, len(layers)):
                        g.set_qscale(i, scales_from.get_qscale(i))
                g.profile(warmup=3, iters=10, topk=2, passes=3)
                if scales_from is None and any(d == "qi8" for d, _ in schemas):
                    g.calibrate(xd)
                total, sch, cands = g.select_path(sn.SN_SELECT_DPRS)
            stream.synchronize()
            g.set_option(sn.SN_OPT_CUDA_GRAPH, 1)
            return g, total, sch, cands

        # (1) no tuning
        g0 = sn.build_graph(layers, x.shape, io, io, [F16[0]])
        t = g0.cost_table()
        g0.set_path([int(np.flatnonzero(t["layer"] == i)[0]) for i in range(t["n_layers"])])
        g0.set_option(sn.SN_OPT_CUDA_GRAPH, 1)
        y = g0.new_output()
        row["untuned_ms"] = _latency_ms(torch, g0, xd, y, stream, flush, reps=5)
        del g0
        # (4) hybrid first: its calibration gives the scales for (3)
        gh, th, sch_h, cand_h = tuned(F16 + Q8)
        gf, tf, _, _ = tuned(F16)
        gq, tq, _, _ = tuned(Q8, scales_from=gh)
        for key, g in (("float_ms", gf), ("qint8_ms", gq), ("hybrid_ms", gh)):
            y = g.new_output()
            row[key] = _latency_ms(torch, g, xd, y, stream, flush)
            outs[key] = y.float().cpu().numpy().ravel()
        uni = gh.schema_universe()
        t = gh.cost_table()
        row["qint8_layers"] = [[i - 1, layers[i - 1]["type"], sn.routine_name(int(t["routine"][int(cand_h[i])]))]
                               for i in range(1, t["n_layers"] - 1) if uni[int(sch_h[i])][0] == "qi8"]
        row["path_cost_ns"] = {"float": int(tf), "qint8": int(tq), "hybrid": int(th)}
        ref = outs["float_ms"]
        den = max(float(np.abs(ref).max()), 1e-30)
        row["out_maxrel_vs_float"] = {k: float(np.abs(outs[k] - ref).max()) / den for k in ("qint8_ms", "hybrid_ms")}
        row["hybrid_vs_float"] = row["float_ms"] / row["hybrid_ms"]
        rows[name] = row
        del gh, gf, gq
        torch.cuda.empty_cache()
    print(json.dumps({"config": "hybrid", "metric": "batch-1 latency (ms) by tuning case, CUDA-graph replay, "
                      "L2 flushed: untuned / fp16-tuned / qint8-tuned / hybrid (section V-C, Table I)",
                      "data": "synthetic inputs and random weights", "nets": rows}))


_COPY_US = {}


def _copy_ref_us(torch, nbytes):
    """Size-matched reference: PyTorch's vectorised element-wise kernel (a
    bitwise NOT of int16) reading half the bytes and writing the other half,
    timed like the kernels (cold operands, CUDA-graph replay).  It pays the
    same launch ramp and tail as a kernel of that size."""
    if nbytes not in _COPY_US:
        n = max(8, nbytes // 4 // 8 * 8)
        bufs = [(torch.zeros(n, dtype=torch.int16, device="cuda"), torch.empty(n, dtype=torch.int16, device="cuda"))
                for _ in range(_sets_for(4 * n))]
        _COPY_US[nbytes] = _time_cold(torch, [(lambda a=a, b=b: torch.bitwise_not(a, out=b)) for a, b in bufs]) * 1e3
        del bufs
    return _COPY_US[nbytes]


def _dw_rows(sn, torch, synth, hbm, shapes, variants=(0, 1, 2), layouts=("nhwc", "nchw")):
    rows = []
    for (N, C, H, s_) in shapes:
        for lay in layouts:
            for var in variants:
                if var == 2 and lay == "nchw":
                    continue
                sch = ("f16", lay)
                layer = synth.dwconv(C, 3, s_, act="relu6")
                layer["weight"] = np.zeros((C, 1, 3, 3), np.float32)
                layer["bias"] = np.zeros(C, np.float32)
                g = _single_layer_graph(sn, layer, (N, C, H, H), sch)
                try:
                    _forced(sn, g, "dwconv2/direct", var)
                except IndexError:  # this routine parameter is not offered for the shape
                    continue
                P = (H + 2 - 3) // s_ + 1
                bufs = [(torch.zeros(sn.storage_shape((N, C, H, H), lay), dtype=torch.float16, device="cuda"),
                         g.new_output()) for _ in range(_sets_for(2 * N * C * (H * H + P * P)))]
                ms = _time_cold(torch, [(lambda xb=xb, yb=yb: g.run(xb, yb)) for xb, yb in bufs])
                del bufs, g
                by = 2 * (N * C * H * H + N * C * P * P) + 2 * 9 * C + 4 * C
                cu = _copy_ref_us(torch, by)
                rows.append({"kernel": "dwconv2/direct", "variant": sn.variant_name(5, var), "layout": lay,
                             "shape": [N, C, H, H], "stride": s_, "us": ms * 1e3, "gbs": by / ms / 1e6,
                             "frac": by / ms / 1e6 / hbm, "copy_us": cu, "frac_of_copy": cu / (ms * 1e3)})
    return rows


def _adapt_rows(sn, torch, hbm, shapes, pairs):
    rows = []
    dt = {"f32": torch.float32, "bf16": torch.bfloat16, "f16": torch.float16}
    for shp in shapes:
        for (a_, b_) in pairs:
            x = torch.zeros(sn.storage_shape(shp, a_[1]), dtype=dt[a_[0]], device="cuda")
            y = torch.empty(sn.storage_shape(shp, b_[1]), dtype=dt[b_[0]], device="cuda")
            bufs = [(x, y)] + [(torch.zeros_like(x), torch.empty_like(y))
                               for _ in range(_sets_for(x.nbytes + y.nbytes) - 1)]
            ms = _time_cold(torch, [(lambda xb=xb, yb=yb: sn.convert(xb, a_, b_, shp, out=yb)) for xb, yb in bufs])
            del bufs
            by = x.numel() * x.element_size() + y.numel() * y.element_size()
            cu = _copy_ref_us(torch, by)
            rows.append({"kernel": "adapt/convert", "from": "%s.%s" % a_, "to": "%s.%s" % b_, "shape": list(shp),
                         "us": ms * 1e3, "gbs": by / ms / 1e6, "frac": by / ms / 1e6 / hbm, "copy_us": cu,
                         "frac_of_copy": cu / (ms * 1e3)})
    return rows


DW_SHAPES = [(128, 144, 56, 1), (128, 96, 112, 2), (128, 192, 28, 1), (128, 576, 14, 1), (128, 960, 7, 1)]
ADAPT_SHAPES = [(32, 64, 112, 112), (32, 256, 56, 56), (32, 1024, 14, 14)]
ADAPT_PAIRS = [(("bf16", "nchw"), ("bf16", "nhwc")), (("bf16", "nhwc"), ("bf16", "nchw")),
               (("f32", "nchw"), ("bf16", "nhwc")), (("bf16", "nhwc"), ("f32", "nchw"))]


def _bandwidth_rows(sn, torch, synth, hbm, compact=False):
    """Depthwise 3x3 at MobileNetV2 shapes (batch 128) and the adapt conversions
    on ResNet-50 b32 activations, each timed from CUDA-graph replays that rotate
    through buffer sets totalling four L2 capacities (cold operands).  compact:
    the best routine parameter and layout per depthwise shape (what DPRS would
    take), and the conversions of the ResNet-50 b32 path."""
    dw = _dw_rows(sn, torch, synth, hbm, DW_SHAPES)
    ad = _adapt_rows(sn, torch, hbm, ADAPT_SHAPES, ADAPT_PAIRS)
    if not compact:
        return dw + ad
    best = {}
    for r in dw:
        k = (tuple(r["shape"]), r["stride"])
        if k not in best or r["gbs"] > best[k]["gbs"]:
            best[k] = r
    rnd = lambda r: {k: (round(v, 3) if isinstance(v, float) else v) for k, v in r.items()}
    return {"metric": "achieved HBM GB/s (algorithmic bytes / event time), cold L2; copy_us: PyTorch's "
                      "element-wise kernel moving the same bytes, timed the same way", "peak_gbs": hbm,
            "depthwise_best": [rnd(r) for r in best.values()], "adapt": [rnd(r) for r in ad]}


def _latency_config(sn, torch, synth, name, keep=None):
    """Profile + DPRS + CUDA-graph latency of one net at batch 1 (or the given config)."""
    if name == "tiny":
        x, layers = synth.tiny_cnn()
        sch, io, dt = [("f32", "nchw"), ("f32", "nhwc")], ("f32", "nchw"), torch.float32
    elif name == "mbv2_b1":
        x, layers = synth.mobilenet_v2(1)
        sch, io, dt = [("f16", "nchw"), ("f16", "nhwc")], ("f16", "nchw"), torch.float16
    elif name == "mbv3_b1":
        x, layers = synth.mobilenet_v3(1)
        sch, io, dt = [("f16", "nchw"), ("f16", "nhwc")], ("f16", "nchw"), torch.float16
    elif name == "vgg16_b32":
        x, layers = synth.vgg16(32)
        sch, io, dt = [("bf16", "nchw"), ("bf16", "nhwc")], ("bf16", "nchw"), torch.bfloat16
    elif name == "vgg16_b1":
        x, layers = synth.vgg16(1)
        sch, io, dt = [("f16", "nchw"), ("f16", "nhwc")], ("f16", "nchw"), torch.float16
    else:
        x, layers = synth.resnet50(1)
        sch, io, dt = [("f16", "nchw"), ("f16", "nhwc")], ("f16", "nchw"), torch.float16
    stream = torch.cuda.Stream()
    t0 = time.perf_counter()
    with torch.cuda.stream(stream):
        # residual adds fused by the library's pass before tuning (no-op where there are none)
        g = sn.build_graph(layers, x.shape, io, io, sch, fuse=True)
        layers = sn.fused_description(layers, g.fused_ids)
        g.profile(warmup=3, iters=10, topk=2, passes=3)
        total, schemas, cands = g.select_path(sn.SN_SELECT_DPRS)
    stream.synchronize()
    tune = time.perf_counter() - t0
    g.set_option(sn.SN_OPT_CUDA_GRAPH, 1)
    xd = torch.from_numpy(x).to(dt).cuda()
    y = g.new_output()
    flush = torch.empty(256 << 20, dtype=torch.uint8, device="cuda")
    with torch.cuda.stream(stream):
        for _ in range(5):
            g.run(xd, y)
    stream.synchronize()
    lat = []
    for _ in range(20):
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        with torch.cuda.stream(stream):
            flush.zero_()
            a.record(stream)
            g.run(xd, y)
            b.record(stream)
        stream.synchronize()
        lat.append(a.elapsed_time(b))
    t = g.cost_table()
    path = {}
    for i in range(1, t["n_layers"] - 1):
        r = sn.routine_name(int(t["routine"][int(cands[i])]))
        path[r] = path.get(r, 0) + 1
    work, _ = conv_work(layers, x.shape)
    fl = sum(w[0] for w in work)
    out = {"batch": int(x.shape[0]), "images_per_s": x.shape[0] / statistics.median(lat) * 1e3,
           "gflop": fl / 1e9, "tflops": fl / statistics.median(lat) / 1e9,
           "metric": "latency (ms), CUDA-graph replay, L2 flushed", "mean_ms": statistics.mean(lat),
           "std_ms": statistics.pstdev(lat), "median_ms": statistics.median(lat), "tuning_s": tune,
           "path_cost_ns": total, "routines_on_path": path,
           "schemas_on_path": {str(s_): int((schemas == i).sum()) for i, s_ in enumerate(g.schema_universe())}}
    if keep is not None:
        keep[name] = (t, layers, x)
    del g
    return out


def _sweep_rows(sn, torch, synth, Ns, Hs, Cs, ks, ss, lays):
    rows = []
    for N in Ns:
        for H in Hs:
            for C in Cs:
                for k in ks:
                    for s_ in ss:
                        for lay in lays:
                            sch = ("f16", lay)
                            x, layers = synth.single_conv(N, H, C, C, k, s_)
                            g = _single_layer_graph(sn, layers[0], x.shape, sch)
                            g.profile(warmup=2, iters=5, topk=0, passes=1)
                            total, schemas, cands = g.select_path(sn.SN_SELECT_DPRS)
                            t = g.cost_table()
                            c = int(cands[1])
                            xd = torch.zeros(sn.storage_shape(x.shape, lay), dtype=torch.float16, device="cuda")
                            y = g.new_output()
                            ms = _time_back_to_back(torch, lambda: g.run(xd, y), reps=10, warm=2)
                            P = (H + 2 * (k // 2) - k) // s_ + 1
                            fl = 2 * N * C * P * P * C * k * k
                            by = 2 * (N * C * H * H + N * C * P * P + C * C * k * k)
                            rows.append({"N": N, "H": H, "C": C, "k": k, "s": s_, "layout": lay,
                                         "routine": g.candidate_desc(c), "us": ms * 1e3,
                                         "tflops": fl / ms / 1e9, "gbs": by / ms / 1e6, "ai": fl / by})
                            del g
    return rows


def _sweep_summary(sn, torch, synth, pk):
    """A cut of the single-layer sweep (batch 32, NHWC, stride 1, every H, C and
    kernel size): per shape the DPRS-chosen routine, and each shape's fraction
    of the roofline its arithmetic intensity puts it under (back-to-back
    launches; --config sweep runs the whole sweep)."""
    sustained = pk.get("bf16_tflops_sustained", pk["bf16_tflops"])
    ridge = sustained * 1e12 / (pk["hbm_gbs"] * 1e9)
    rows = _sweep_rows(sn, torch, synth, (32,), (7, 14, 28, 56), (64, 128, 256, 512), (1, 3), (1,), ("nhwc",))
    out = []
    for r in rows:
        tb = r["ai"] > ridge
        out.append({"H": r["H"], "C": r["C"], "k": r["k"], "us": round(r["us"], 2), "tflops": round(r["tflops"], 1),
                    "bound": "tensor" if tb else "hbm",
                    "frac": round(r["tflops"] / sustained if tb else r["gbs"] / pk["hbm_gbs"], 3),
                    "routine": r["routine"]})
    tens = [r["frac"] for r in out if r["bound"] == "tensor"]
    mem = [r["frac"] for r in out if r["bound"] == "hbm"]
    return {"metric": "single-layer conv, fp16 NHWC, batch 32, stride 1; frac of the sustained tensor peak "
                      "(AI above the ridge) or of the HBM peak", "ridge_flop_per_byte": ridge,
            "tensor_bound_median_frac": statistics.median(tens) if tens else None,
            "hbm_bound_median_frac": statistics.median(mem) if mem else None, "rows": out}


def _oracle_times(sn, synth, graphs, g1_table=None):
    """The oracle on the host cores: one ResNet-50 image with every core and
    with one thread (a child process with OMP_NUM_THREADS=1), the exhaustive
    path search on the tiny CNN's profiled cost table and the block-wise exact
    search on ResNet-50 b1's (section IV problem sizes), with the library's
    DPRS time on the same tables for comparison."""
    import oracle
    from oracle.net import run_net
    from oracle.paths import blockwise_search
    out = {"cores": os.cpu_count()}
    x, layers = synth.resnet50(1)
    t0 = time.perf_counter()
    run_net(layers, x, "bf16")
    out["r50_image_all_cores_s"] = time.perf_counter() - t0
    code = ("import sys, time; sys.path.insert(0, %r); import synth; from oracle.net import run_net; "
            "x, l = synth.resnet50(1); t0 = time.perf_counter(); run_net(l, x, 'bf16'); "
            "print(time.perf_counter() - t0)") % ROOT
    env = dict(os.environ, OMP_NUM_THREADS="1", CUDA_VISIBLE_DEVICES="")
    try:
        r = subprocess.run([sys.executable, "-c", code], env=env, capture_output=True, text=True, timeout=300)
        out["r50_image_1_thread_s"] = float(r.stdout.strip().splitlines()[-1])
    except Exception as e:  # noqa: BLE001
        out["r50_image_1_thread_s"] = None
        out["r50_image_1_thread_error"] = str(e)[:200]

    def layer_cost(t):
        n, ns = t["n_layers"], t["n_schemas"]
        return np.array([oracle.fastest_per_schema(t["schema"][t["layer"] == i], t["cost"][t["layer"] == i], ns)
                         for i in range(n)])
    if "tiny" in graphs:
        t = graphs["tiny"][0]
        lc = layer_cost(t)
        t0 = time.perf_counter()
        tot, _, _ = oracle.brute_force(lc, t["edges"], t["adapt"])
        out["tiny_exhaustive_search_s"] = time.perf_counter() - t0
        out["tiny_assignments"] = int(t["n_schemas"]) ** int(t["n_layers"] - 2)
    if g1_table is not None:
        lc = layer_cost(g1_table)
        t0 = time.perf_counter()
        blockwise_search(lc, g1_table["edges"], g1_table["adapt"])
        out["r50_b1_blockwise_search_s"] = time.perf_counter() - t0
    return out


def run_extra_config(args):
    import torch
    import synth
    import paper_2110_06037_gb300 as sn
    pk, pk_kind = peaks()
    hbm = pk["hbm_gbs"]
    torch.cuda.set_device(0)
    out = {"config": args.config, "peaks": pk_kind}
    if args.config == "bandwidth":
        rows = _bandwidth_rows(sn, torch, synth, hbm)
        # qint8 schema: the quantise / dequantise adapts on ResNet-50 b32 activations
        # and the int8 dense routine at batch 1 (VGG16's fully connected shapes),
        # where the weight codes are the bytes that matter
        for shp in [(32, 256, 56, 56), (32, 1024, 14, 14)]:
            for (a_, b_) in [(("f16", "nchw"), ("qi8", "nhwc")), (("f16", "nhwc"), ("qi8", "nhwc")),
                             (("qi8", "nhwc"), ("f16", "nhwc"))]:
                dt = {"f16": torch.float16, "qi8": torch.int8}
                x = torch.zeros(sn.storage_shape(shp, a_[1]), dtype=dt[a_[0]], device="cuda")
                y = torch.empty(sn.storage_shape(shp, b_[1]), dtype=dt[b_[0]], device="cuda")
                bufs = [(x, y)] + [(torch.zeros_like(x), torch.empty_like(y))
                                   for _ in range(_sets_for(x.nbytes + y.nbytes) - 1)]
                ms = _time_cold(torch, [(lambda xb=xb, yb=yb: sn.convert_q(xb, a_, b_, shp, 0.05, out=yb))
                                        for xb, yb in bufs])
                del bufs
                by = x.numel() * x.element_size() + y.numel() * y.element_size()
                rows.append({"kernel": "adapt/convert (qi8)", "from": "%s.%s" % a_, "to": "%s.%s" % b_,
                             "shape": list(shp), "us": ms * 1e3, "gbs": by / ms / 1e6, "frac": by / ms / 1e6 / hbm})
        for (fi, fo) in [(25088, 4096), (4096, 4096)]:
            layer = {"type": "dense", "params": dict(in_features=fi, out_features=fo, act="relu"),
                     "weight": np.zeros((fo, fi), np.float32), "bias": np.zeros(fo, np.float32)}
            sets = _sets_for(fi * fo)
            gs = []
            for _ in range(sets):
                g = _single_layer_graph(sn, layer, (1, fi, 1, 1), ("qi8", "nhwc"))
                g.set_qscale(-1, 0.05)
                g.set_qscale(0, 0.05)
                _forced(sn, g, "dense/simt")
                gs.append((g, torch.zeros((1, 1, 1, fi), dtype=torch.int8, device="cuda"), g.new_output()))
                gs[-1][0].run(gs[-1][1], gs[-1][2])  # plan and weights built before the capture
            torch.cuda.synchronize()
            ms = _time_cold(torch, [(lambda g=g, xb=xb, yb=yb: g.run(xb, yb)) for g, xb, yb in gs])
            del gs
            by = fi * fo + fi + fo + 8 * fo  # codes, input, output, weight scales + bias
            rows.append({"kernel": "dense/simt (qi8)", "shape": [1, fi, fo], "us": ms * 1e3, "gbs": by / ms / 1e6,
                         "frac": by / ms / 1e6 / hbm})
        out.update({"metric": "achieved HBM GB/s (algorithmic bytes / event time)", "peak_gbs": hbm, "rows": rows})
    elif args.config == "q8_dense":
        # the int8 dense routine on VGG16's first fully connected shape at batch 1
        # (102.8 MB of weight codes, read once per launch): a small case for ncu
        fi, fo = 25088, 4096
        layer = {"type": "dense", "params": dict(in_features=fi, out_features=fo, act="relu"),
                 "weight": np.zeros((fo, fi), np.float32), "bias": np.zeros(fo, np.float32)}
        g = _single_layer_graph(sn, layer, (1, fi, 1, 1), ("qi8", "nhwc"))
        g.set_qscale(-1, 0.05)
        g.set_qscale(0, 0.05)
        _forced(sn, g, "dense/simt")
        xb = torch.zeros((1, 1, 1, fi), dtype=torch.int8, device="cuda")
        yb = g.new_output()
        ms = _time_back_to_back(torch, lambda: g.run(xb, yb), reps=20, warm=3)
        by = fi * fo + fi + fo + 8 * fo
        out.update({"metric": "dense/simt (qi8), batch 1, back-to-back launches of one weight set (102.8 MB, "
                              "within L2; --config bandwidth gives the cold-L2 figure)",
                    "shape": [1, fi, fo], "us": ms * 1e3, "gbs": by / ms / 1e6, "frac": by / ms / 1e6 / hbm})
    elif args.config in ("dw_band_14", "transpose_14", "wino_14"):
        # small single-kernel cases for ncu captures, four back-to-back runs each:
        #   dw_band_14   MobileNetV2's 14x14 depthwise 3x3 at batch 128 (576 channels, fp16 NHWC)
        #                on the band kernel (dwconv2/direct routine parameter 2)
        #   transpose_14 the NHWC -> NCHW adapt of a ResNet-50 b32 stage-3 activation (bf16)
        #   wino_14      conv2/wino_f2x2_3x3 on 32 x 256 -> 256, 14x14, fp16 NHWC
        if args.config == "dw_band_14":
            N, C_, H = 128, 576, 14
            layer = dict(synth.dwconv(C_, 3, 1, act="relu6"), weight=np.zeros((C_, 1, 3, 3), np.float32),
                         bias=np.zeros(C_, np.float32))
            g = _single_layer_graph(sn, layer, (N, C_, H, H), ("f16", "nhwc"))
            _forced(sn, g, "dwconv2/direct", 2)
            xb = torch.zeros(N, H, H, C_, dtype=torch.float16, device="cuda")
            yb = g.new_output()
            fn = lambda: g.run(xb, yb)
        elif args.config == "transpose_14":
            shp = (32, 1024, 14, 14)
            xb = torch.zeros(32, 14, 14, 1024, dtype=torch.bfloat16, device="cuda")
            yb = torch.empty(32, 1024, 14, 14, dtype=torch.bfloat16, device="cuda")
            fn = lambda: sn.convert(xb, ("bf16", "nhwc"), ("bf16", "nchw"), shp, out=yb)
        else:
            x0, layers = synth.single_conv(32, 14, 256, 256, 3, 1)
            g = _single_layer_graph(sn, layers[0], x0.shape, ("f16", "nhwc"))
            _forced(sn, g, "conv2/wino_f2x2_3x3", 0)
            xb = torch.zeros(32, 14, 14, 256, dtype=torch.float16, device="cuda")
            yb = g.new_output()
            fn = lambda: g.run(xb, yb)
        for _ in range(4):
            fn()
        torch.cuda.synchronize()
        out.update({"metric": "single-kernel case for a profiler capture (four back-to-back runs, not timed)"})
    elif args.config == "layer":
        # one bf16 NHWC conv layer on the tensor-core routine: every routine-parameter
        # combination (or the one given), timed back to back
        N, C, H, K, k, s_ = map(int, args.layer.split(","))
        sch = ("bf16", "nhwc")
        x, layers = synth.single_conv(N, H, C, K, k, s_)
        g = _single_layer_graph(sn, layers[0], x.shape, sch)
        t = g.cost_table()
        xd = torch.from_numpy(x).to(torch.bfloat16).cuda().permute(0, 2, 3, 1).contiguous()
        y = g.new_output()
        P = (H + 2 * (k // 2) - k) // s_ + 1
        fl = 2 * N * K * P * P * C * k * k
        by = 2 * (N * C * H * H + N * K * P * P + K * C * k * k)
        sustained = pk.get("bf16_tflops_sustained", pk["bf16_tflops"])
        rows = []
        nvar = sum(1 for c in range(len(t["cost"])) if t["layer"][c] == 1 and
                   sn.routine_name(int(t["routine"][c])) == "conv2/igemm_tc")
        for var in ([args.variant] if args.variant >= 0 else range(nvar)):
            _forced(sn, g, "conv2/igemm_tc", var)
            ms = _time_graph(torch, lambda: g.run(xd, y), reps=max(3, min(args.steps, 20)))
            rows.append({"variant": var, "us": ms * 1e3, "tflops": fl / ms / 1e9, "gbs": by / ms / 1e6,
                         "frac_tensor": fl / ms / 1e9 / sustained, "frac_hbm": by / ms / 1e6 / hbm})
        best = min(rows, key=lambda r: r["us"])
        out.update({"metric": "single-layer conv2/igemm_tc, bf16 NHWC, device time per launch (CUDA-graph replay)",
                    "layer": [N, C, H, K, k, s_], "gflop": fl / 1e9, "bytes": by, "best": best, "rows": rows})
    elif args.config == "sweep":
        rows = _sweep_rows(sn, torch, synth, (1, 8, 32), (7, 14, 28, 56), (64, 128, 256, 512), (1, 3), (1, 2),
                           ("nhwc", "nchw"))
        out.update({"metric": "single-layer conv, fp16, best routine by profiling + DPRS", "rows": rows})
    else:
        out.update(_latency_config(sn, torch, synth, args.config))
    print(json.dumps(out))


if __name__ == "__main__":
    main()
