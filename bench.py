#!/usr/bin/env python3
"""Throughput benchmark of the SGD-KV compression step on GB300.

One step = the whole hot path for one model's prefilled cache: the head-level budget
allocation (host, Eq. 2 + Algorithm 1) and, for every layer, window scoring + max-pool
(sgdkv_score) and top-b_h selection + K/V gather (sgdkv_compact) over all KV heads.
Metric: compressed context tokens per second per layer = n_layers * L / step time.
Inputs are seeded synthetic caches shaped like the paper's models (no datasets/weights).

Prints one JSON line (rank 0).  Also reports the roofline of the dominant kernel stage,
the end-to-end figure through the C-ABI from pinned host buffers, and the CPU oracle
timed on this machine's host cores on a bounded sample.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME] [--frac F]
  python bench.py --impl reference ...   # the CPU oracle as the reference arm
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

DEFAULT_WORKLOAD = "c3_qwen25_7b_L128k"
METRIC = "compressed context tokens/sec per layer"
UNIT = "tokens/s/layer"


def parse_args(argv=None):
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=20)
    p.add_argument("--warmup", type=int, default=3)
    p.add_argument("--impl", choices=["ours", "reference"], default="ours")
    p.add_argument("--workload", default=DEFAULT_WORKLOAD)
    p.add_argument("--frac", type=float, default=0.25)
    p.add_argument("--layers", type=int, default=0, help="layers per step (0 = all)")
    p.add_argument("--e2e-steps", type=int, default=4)
    p.add_argument("--no-e2e", action="store_true")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--no-decode", action="store_true",
                   help="skip the decode-attention measurement over the compressed caches")
    p.add_argument("--cpu-child", action="store_true", help=argparse.SUPPRESS)
    return p.parse_args(argv)


# ------------------------------------------------------------------------------------------
# multi-process plumbing (one process per GPU; replicas, no data-path collective)
# ------------------------------------------------------------------------------------------

def dist_env():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def dist_init(world):
    if world > 1:
        import torch.distributed as dist
        if not dist.is_initialized():
            dist.init_process_group("gloo")


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(x: float, world: int) -> float:
    if world == 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


# ------------------------------------------------------------------------------------------
# clocks during the timed region
# ------------------------------------------------------------------------------------------

class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_id: str | None):
        self.gpu_id = gpu_id
        self.proc = None
        self.path = None

    def start(self):
        try:
            fd, self.path = tempfile.mkstemp(prefix="clocks_", suffix=".csv")
            os.close(fd)
            cmd = ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                   "-lms", "100"]
            if self.gpu_id is not None:
                cmd += ["-i", self.gpu_id]
            self.proc = subprocess.Popen(cmd, stdout=open(self.path, "w"),
                                         stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        rows = []
        with open(self.path) as f:
            for line in f:
                parts = [x.strip() for x in line.split(",")]
                if len(parts) != 9:
                    continue
                try:
                    rows.append(dict(sm=float(parts[1]), max=float(parts[2]),
                                     hw=parts[5], hwt=parts[6], swt=parts[7], swp=parts[8]))
                except ValueError:
                    continue
        os.unlink(self.path)
        if not rows:
            return None
        reasons = set()
        for r in rows:
            for key, name in (("hw", "hw_slowdown"), ("hwt", "hw_thermal_slowdown"),
                              ("swt", "sw_thermal_slowdown"), ("swp", "sw_power_cap")):
                if r[key].lower() == "active":
                    reasons.add(name)
        return {"sm_mhz": statistics.median(r["sm"] for r in rows),
                "sm_max_mhz": max(r["max"] for r in rows), "samples": len(rows),
                "reasons": sorted(reasons)}


def nvsmi_id(dev_index: int) -> str | None:
    try:
        import torch
        props = torch.cuda.get_device_properties(dev_index)
        u = getattr(props, "uuid", None)
        if u is not None:
            s = str(u)
            return s if s.startswith("GPU-") else "GPU-" + s
    except Exception:
        pass
    vis = os.environ.get("CUDA_VISIBLE_DEVICES", "")
    ids = [v for v in vis.split(",") if v.strip()]
    return ids[dev_index] if dev_index < len(ids) else None


def measured_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            m = json.load(f)
        return dict(hbm=float(m["hbm_gbs"]), bf16=float(m["bf16_tflops"]),
                    bf16_sus=float(m["bf16_tflops_sustained"]), source="measured")
    except Exception:
        return dict(hbm=6800.0, bf16=1900.0, bf16_sus=1700.0, source="fallback")


# ------------------------------------------------------------------------------------------
# algorithmic work (per layer)
# ------------------------------------------------------------------------------------------

def score_flops(wl) -> float:
    """Two passes over every (window row, key) pair: 2 * (2 * G * W * d) per key per KV head."""
    return 2.0 * 2.0 * wl.G * wl.W * wl.d * wl.L * wl.Hkv


def pass_flops(wl) -> float:
    """One scoring pass: the window logits q.k of every (window row, key) pair, 2*G*W*d per key
    per KV head (Eq. 1's numerator; pass 1 and pass 2 each form them once)."""
    return 2.0 * wl.G * wl.W * wl.d * wl.L * wl.Hkv


DIAG_STEPS = 3
TIMED_EVERY = 4          # the dominant kernel is event-bracketed in every 4th layer
N_SCORE_WS = 3           # scoring workspaces in rotation (layers in flight on them)
KERNEL_NAMES = ("score_pass1_tc", "score_pass2_tc", "maxpool_sum_kernel", "sel_cluster_kernel",
                "gather_kernel")

# DRAM traffic per launch (dram__bytes_read.sum + dram__bytes_write.sum) from one ncu capture
# of the 128K-context Qwen2.5-7B layer (28 query / 4 KV heads, W=64), keyed by the SHA-256 of
# the kernel source it was taken on; a source that has changed since reads as null.
_SCORE_SHA = "e7936773fbe7ce70c3b7e0ac5c4f49450047f96a7e980040dce6593adc033e28"
_SELECT_SHA = "95ec997644c3fdfdf93a0671515bfdb607f37f72d5ada6e648711d459661f0be"
MEASURED_TRAFFIC = {
    ("score_pass1_tc", "c3_qwen25_7b_L128k"):
        {"bytes": 134755072 + 3629568, "source": "score_tc.cu", "sha256": _SCORE_SHA},
    ("score_pass2_tc", "c3_qwen25_7b_L128k"):
        {"bytes": 135312896 + 4008448, "source": "score_tc.cu", "sha256": _SCORE_SHA},
    ("sel_cluster_kernel", "c3_qwen25_7b_L128k"):
        {"bytes": 8444416 + 0, "source": "select.cu", "sha256": _SELECT_SHA},
    ("gather_kernel", "c3_qwen25_7b_L128k"):
        {"bytes": 40768768 + 1776896, "source": "select.cu", "sha256": _SELECT_SHA},
}


def _source_sha(name):
    import hashlib
    p = os.path.join(os.path.dirname(os.path.abspath(__file__)), "paper_2609_03235_gb300", "csrc", name)
    with open(p, "rb") as f:
        return hashlib.sha256(f.read()).hexdigest()


def measured_traffic(kernel, workload):
    rec = MEASURED_TRAFFIC.get((kernel, workload))
    if rec is None or rec["sha256"] != _source_sha(rec["source"]):
        return None
    return rec["bytes"]


def path_bytes(wl, budgets_layer) -> float:
    """K read once (d*2 B/key), score written and read (8 B/key), and per kept row: K and V
    read and written (4*d*2 B) plus its int32 index."""
    per_key = wl.d * 2 + 8
    return float(wl.Hkv * wl.L * per_key + sum(int(b) for b in budgets_layer) * (4 * wl.d * 2 + 4))


# ------------------------------------------------------------------------------------------
# our arm
# ------------------------------------------------------------------------------------------

def workload_config(wl, args, world, n_layers):
    """The `config` object of both arms' JSON lines (the same workload for both)."""
    from paper_2609_03235_gb300 import configs
    n_sink, n_recent = configs.sink_recent_split(wl.floor)
    return {"workload": wl.name, "model_shape": "Qwen2.5-7B-1M" if wl.Hkv == 4 else "Qwen3-32B",
            "n_layers": n_layers, "Hq": wl.Hq, "Hkv": wl.Hkv, "head_dim": wl.d,
            "context_len": wl.L, "window": wl.W, "pool": wl.pool,
            "budget_frac": args.frac, "floor": wl.floor, "n_sink": n_sink,
            "n_recent": n_recent, "parallelism": f"replicas x{world}",
            "streams": "scoring passes on one stream, max-pool + selection (one kernel) and "
                       "gather on a second; layer l's pooling and compaction overlap layer "
                       "l+1's scoring",
            "l2": "inputs larger than L2 (K+V of one layer = %d MiB)" %
                  (2 * wl.Hkv * wl.L * wl.d * 2 >> 20)}



def run_ours(args, world, rank, local):
    import numpy as np
    import torch

    from paper_2609_03235_gb300 import configs, synth
    from paper_2609_03235_gb300 import sgdkv as sg

    wl = configs.BY_NAME[args.workload]
    dev = torch.device(f"cuda:{local}")
    torch.cuda.set_device(dev)
    sg.lib()
    n_sink, n_recent = configs.sink_recent_split(wl.floor)
    hs = synth.head_scores(wl)
    T = wl.total_budget(args.frac)
    b_all = sg.sgdkv_allocate_budgets(hs, wl.L, T, wl.floor)
    Ls = wl.n_layers if args.layers <= 0 else min(args.layers, wl.n_layers)
    layers = [synth.layer_inputs_device(wl, l, dev) for l in range(Ls)]
    outs = []
    for l in range(Ls):
        b = b_all[l * wl.Hkv:(l + 1) * wl.Hkv]
        tot = int(b.sum())
        outs.append(dict(
            b=b, scores=torch.empty((wl.Hkv, wl.L), dtype=torch.float32, device=dev),
            idx=torch.empty(tot, dtype=torch.int32, device=dev),
            cu=torch.empty(wl.Hkv + 1, dtype=torch.int32, device=dev),
            ko=torch.empty((tot, wl.d), dtype=torch.bfloat16, device=dev),
            vo=torch.empty((tot, wl.d), dtype=torch.bfloat16, device=dev)))
    # One step = the host budget allocation (a1), then the launches of every layer: the two
    # scoring passes on the capturing stream, sgdkv_pool_compact (the max-pool inside the
    # selection kernel, then the gather) on `sel_stream`; layer l's pooling and compaction
    # wait for layer l's passes only, so they overlap layer l+1's scoring, whose CTAs claim
    # key tiles dynamically and absorb the SMs the other stream leaves.  The raw scores of
    # layer l stay in scoring workspace l % 3 until its compaction has read them (layer
    # l + 3's scoring waits for that: with two workspaces, layer l + 2's scoring would wait
    # for layer l's gather as well).  The launches of a step are
    # captured into a CUDA graph (per-kernel launch cost ~1 us instead of ~3 us on a stream)
    # and the graph is replayed; the allocation still runs on the host every step and must
    # reproduce the budgets the graph was captured with.
    ws_score = [sg.make_workspace(wl.Hq, wl.Hkv, wl.L, wl.W, dev) for _ in range(N_SCORE_WS)]
    ws_sel = sg.make_workspace(wl.Hq, wl.Hkv, wl.L, wl.W, dev)
    stream = torch.cuda.current_stream(dev)
    lo_prio, hi_prio = torch.cuda.Stream.priority_range()
    sel_stream = torch.cuda.Stream(dev, priority=hi_prio)
    fork = torch.cuda.Event()
    scored = [torch.cuda.Event() for _ in range(Ls)]
    pooled = [torch.cuda.Event() for _ in range(Ls)]     # workspace l % N_SCORE_WS read
    done = torch.cuda.Event()

    def launches(ball, s, kinds=(), every=1, first=0):
        fork.record(s)
        sel_stream.wait_event(fork)
        for l in range(Ls):
            inp, o = layers[l], outs[l]
            b = ball[l * wl.Hkv:(l + 1) * wl.Hkv]
            sg.sgdkv_debug_enable_kernel_timing(kinds if l % every == first % every else ())
            wsl = ws_score[l % N_SCORE_WS]
            if l >= N_SCORE_WS:
                s.wait_event(pooled[l - N_SCORE_WS])   # its workspace read by that compaction
            sg.sgdkv_score_raw(inp["q"], inp["K"], wl.W, wsl, s)
            scored[l].record(s)
            sel_stream.wait_event(scored[l])
            sg.sgdkv_pool_compact(wsl, wl.pool, inp["K"], inp["V"], b, n_sink, n_recent,
                                  o["scores"], o["idx"], o["cu"], o["ko"], o["vo"], ws_sel,
                                  sel_stream)
            pooled[l].record(sel_stream)
        done.record(sel_stream)
        s.wait_event(done)

    def allocate():
        ball = sg.sgdkv_allocate_budgets(hs, wl.L, T, wl.floor)      # a1 (host)
        if not np.array_equal(ball, b_all):
            raise RuntimeError("budget allocation changed between steps")
        return ball

    def capture(kinds, every=1, first=0):
        """One step's launches as a CUDA graph; the kernels of `kinds` in every `every`-th
        layer from layer `first` on are bracketed by timing events."""
        g = torch.cuda.CUDAGraph()
        n0 = sg.sgdkv_launch_count()
        with torch.cuda.graph(g):
            launches(b_all, torch.cuda.current_stream(dev), kinds, every, first)
        sg.sgdkv_debug_enable_kernel_timing(())
        return g, sg.sgdkv_launch_count() - n0

    def drain_timers():
        return [sg.sgdkv_debug_kernel_timing(kind) for kind in range(len(KERNEL_NAMES))]

    def check(where):
        st = max(max(sg.sgdkv_last_error(w, stream) for w in ws_score),
                 sg.sgdkv_last_error(ws_sel, sel_stream))
        if st != sg.OK:
            raise RuntimeError(f"device-side error {where}: {sg.status_string(st)}")

    launches(allocate(), stream)                 # one eager step (first-use setup), then graphs
    torch.cuda.synchronize(dev)
    check("in the first step")
    g_warm, _ = capture(())
    for _ in range(max(args.warmup, 0)):
        allocate()
        g_warm.replay()
    torch.cuda.synchronize(dev)
    check("during warm-up")

    # Diagnostic window (untimed for the headline): every kernel bracketed by CUDA events,
    # giving each kernel's share of the step and picking the dominant kernel.
    drain_timers()
    diag = [capture(range(len(KERNEL_NAMES)))[0] for _ in range(DIAG_STEPS)]
    for g in diag:
        allocate()
        g.replay()
    torch.cuda.synchronize(dev)
    kern = {}
    for name, (tot_ms, n) in zip(KERNEL_NAMES, drain_timers()):
        kern[name] = {"launches": n, "us_per_launch": 1e3 * tot_ms / max(n, 1), "ms_total": tot_ms,
                      "dram_bytes_ncu": measured_traffic(name, wl.name)}
    del diag
    kern = {k: v for k, v in kern.items() if v["launches"] > 0}   # no pool kernel at this size
    all_ms = sum(v["ms_total"] for v in kern.values())
    for v in kern.values():
        v["share"] = v["ms_total"] / all_ms if all_ms > 0 else None
    top_kind = max(range(2), key=lambda k: kern[KERNEL_NAMES[k]]["ms_total"])
    top = KERNEL_NAMES[top_kind]

    # Timed region: K graphs of one step each.  The dominant kernel is bracketed by two event
    # nodes in every TIMED_EVERY-th layer (each pair costs about 1 us of step time), starting
    # one layer later in each successive step so that every layer position is sampled alike;
    # the events are distinct per graph, so every bracketed launch of the timed region is read.
    K = args.steps
    timed = [capture([top_kind], TIMED_EVERY, k) for k in range(K)]
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    clocks = ClockSampler(nvsmi_id(local))
    barrier(world)
    torch.cuda.synchronize(dev)
    clocks.start()
    time.sleep(0.3)                      # let the sampler attach before the timed region
    start.record(stream)
    for g, _ in timed:
        allocate()
        g.replay()
    end.record(stream)
    torch.cuda.synchronize(dev)
    launches_timed = sum(n for _, n in timed)
    top_ms, top_n = sg.sgdkv_debug_kernel_timing(top_kind)
    clk = clocks.stop()
    barrier(world)
    check("in the timed region")
    del timed, g_warm
    ms = start.elapsed_time(end) / K
    ms_max = max_over_ranks(ms, world)

    peaks = measured_peaks()
    top_us = 1e3 * top_ms / max(top_n, 1)
    achieved_tf = pass_flops(wl) / (top_us * 1e-6) / 1e12
    stage_us = sum(kern[n]["us_per_launch"] for n in KERNEL_NAMES[:3] if n in kern)
    stage_tf = score_flops(wl) / (stage_us * 1e-6) / 1e12
    bytes_step = sum(path_bytes(wl, o["b"]) for o in outs)
    value = world * wl.L * Ls / (ms_max * 1e-3)

    dec = None if args.no_decode else run_decode(args, wl, outs, dev, stream, peaks)

    e2e = None
    if not args.no_e2e and args.e2e_steps > 0:
        e2e = run_e2e(args, wl, layers, outs, n_sink, n_recent, dev, world)

    rec = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": K,
        "warmup": args.warmup, "ms_per_step": ms_max, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (seeded N(0,1) K/V/Q with planted sink and salient keys)",
        "config": workload_config(wl, args, world, Ls),
        "roofline": {"kernel": top, "bound": "tensor", "achieved": achieved_tf,
                     "peak": peaks["bf16_sus"], "unit": "TFLOP/s",
                     "frac": achieved_tf / peaks["bf16_sus"],
                     "traffic": measured_traffic(top, wl.name),
                     "peak_source": peaks["source"] + " bf16 sustained",
                     "us_per_launch": top_us, "launches_timed": top_n,
                     "timed_launches": f"every {TIMED_EVERY}th layer of every timed step, "
                                       "rotating by one layer per step",
                     "flops_per_launch": pass_flops(wl)},
        "score_stage": {"us_per_layer": stage_us, "tflops": stage_tf,
                        "frac": stage_tf / peaks["bf16_sus"]},
        "kernels": {"window": f"{DIAG_STEPS} steps after warm-up, every launch bracketed",
                    **kern},
        "hbm_path": {"achieved_gbs": bytes_step / (ms_max * 1e-3) / 1e9,
                     "peak_gbs": peaks["hbm"], "frac": bytes_step / (ms_max * 1e-3) / 1e9 / peaks["hbm"],
                     "bytes_per_step": bytes_step},
        "decode_attention": dec,
        "gpu_launches": int(launches_timed),
        "schedule": "each step: budget allocation on the host, then one CUDA-graph launch of "
                    "the step's kernels (the scoring passes on one stream, max-pool + "
                    "selection in one kernel and the gather on a second inside the graph); "
                    "one graph per timed step",
        "clocks": clk,
        "e2e": e2e,
    }
    return rec


def run_decode(args, wl, outs, dev, stream, peaks):
    """Decode attention over the compressed caches the step wrote (one new token per query
    head, every layer): the layers' calls captured into one CUDA graph, W untimed and K
    timed replays between CUDA events on the stream.  The caches of all layers (1.9 GB at
    25 %) are larger than L2, so each layer's cache comes from HBM.  Bytes per layer: the
    kept K and V rows read once, plus the queries and the fp32 outputs."""
    import numpy as np
    import torch
    from paper_2609_03235_gb300 import sgdkv as sg
    Ls = len(outs)
    g = torch.Generator(device=dev).manual_seed(20260902)
    qd = (torch.randn((wl.Hq, 1, wl.d), device=dev, generator=g) * 2.0).to(torch.bfloat16)
    od = torch.empty((wl.Hq, 1, wl.d), dtype=torch.float32, device=dev)
    rows = [int(np.sum(o["b"])) for o in outs]
    ws = sg.make_decode_workspace(wl.Hq, wl.Hkv, 1, max(rows), dev)

    def step(s):
        for o in outs:
            sg.sgdkv_decode_attention(qd, o["ko"], o["vo"], o["b"], od, ws, s)

    step(stream)                                 # first-use setup outside the capture
    torch.cuda.synchronize(dev)
    graph = torch.cuda.CUDAGraph()
    n0 = sg.sgdkv_launch_count()
    with torch.cuda.graph(graph):
        step(torch.cuda.current_stream(dev))
    launches = sg.sgdkv_launch_count() - n0
    for _ in range(max(args.warmup, 3)):
        graph.replay()
    torch.cuda.synchronize(dev)
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    reps = max(args.steps, 5)
    t0.record(stream)
    for _ in range(reps):
        graph.replay()
    t1.record(stream)
    torch.cuda.synchronize(dev)
    us_layer = 1e3 * t0.elapsed_time(t1) / reps / Ls
    byts = sum(r * wl.d * 2 * 2 for r in rows) / Ls + wl.Hq * wl.d * (2 + 4)
    gbs = byts / (us_layer * 1e-6) / 1e9
    return {"what": "one decode token per query head attending over each layer's compressed "
                    "cache (sgdkv_decode_attention: partials + merge kernels)",
            "us_per_layer": us_layer, "bytes_per_layer": byts, "achieved_gbs": gbs,
            "peak_gbs": peaks["hbm"], "frac": gbs / peaks["hbm"], "bound": "hbm",
            "layers": Ls, "replays": reps, "launches_per_replay": int(launches)}


def run_e2e(args, wl, layers, outs, n_sink, n_recent, dev, world):
    """Same metric through the public API with host buffers: every step copies each layer's
    q and K from pinned host memory, compresses the layer (the gather reads the kept V rows
    straight from pinned host memory, so only those cross the host link), and copies the
    compressed cache back."""
    import torch

    from paper_2609_03235_gb300 import sgdkv as sg

    Ls = len(layers)
    hq = [l["q"].cpu().pin_memory() for l in layers]
    hk = [l["K"].cpu().pin_memory() for l in layers]
    hv = [l["V"].cpu().pin_memory() for l in layers]
    ho = [dict(idx=torch.empty(o["idx"].shape, dtype=torch.int32).pin_memory(),
               cu=torch.empty(o["cu"].shape, dtype=torch.int32).pin_memory(),
               ko=torch.empty(o["ko"].shape, dtype=torch.bfloat16).pin_memory(),
               vo=torch.empty(o["vo"].shape, dtype=torch.bfloat16).pin_memory()) for o in outs]
    slots = []
    maxtot = max(o["idx"].numel() for o in outs)
    for _ in range(2):
        slots.append(dict(
            q=torch.empty_like(layers[0]["q"]), K=torch.empty_like(layers[0]["K"]),
            idx=torch.empty(maxtot, dtype=torch.int32, device=dev),
            cu=torch.empty(wl.Hkv + 1, dtype=torch.int32, device=dev),
            ko=torch.empty((maxtot, wl.d), dtype=torch.bfloat16, device=dev),
            vo=torch.empty((maxtot, wl.d), dtype=torch.bfloat16, device=dev),
            ws=sg.make_workspace(wl.Hq, wl.Hkv, wl.L, wl.W, dev)))
    s_h2d, s_cmp, s_d2h = torch.cuda.Stream(dev), torch.cuda.Stream(dev), torch.cuda.Stream(dev)
    ev = lambda: torch.cuda.Event()
    h2d_done = [ev(), ev()]
    cmp_done = [ev(), ev()]
    d2h_done = [ev(), ev()]
    hs = None
    from paper_2609_03235_gb300 import synth
    hs = synth.head_scores(wl)
    T = wl.total_budget(args.frac)
    h2d_bytes = sum(hq[l].numel() * 2 + hk[l].numel() * 2 for l in range(Ls))
    # kept V rows read by the gather from pinned host memory (not a copy)
    host_read_bytes = sum(int(o["b"].sum()) * wl.d * 2 for o in outs)
    d2h_bytes = sum(ho[l]["idx"].numel() * 4 + ho[l]["cu"].numel() * 4 +
                    ho[l]["ko"].numel() * 2 + ho[l]["vo"].numel() * 2 for l in range(Ls))

    def step():
        ball = sg.sgdkv_allocate_budgets(hs, wl.L, T, wl.floor)
        for l in range(Ls):
            s = l % 2
            sl = slots[s]
            b = ball[l * wl.Hkv:(l + 1) * wl.Hkv]
            tot = int(b.sum())
            s_h2d.wait_event(cmp_done[s])
            with torch.cuda.stream(s_h2d):
                sl["q"].copy_(hq[l], non_blocking=True)
                sl["K"].copy_(hk[l], non_blocking=True)
                h2d_done[s].record(s_h2d)
            s_cmp.wait_event(h2d_done[s])
            s_cmp.wait_event(d2h_done[s])
            sg.sgdkv_compress_layer(sl["q"], sl["K"], hv[l], b, wl.W, wl.pool, n_sink,
                                    n_recent, None, sl["idx"], sl["cu"], sl["ko"], sl["vo"],
                                    sl["ws"], s_cmp)
            cmp_done[s].record(s_cmp)
            s_d2h.wait_event(cmp_done[s])
            with torch.cuda.stream(s_d2h):
                ho[l]["idx"].copy_(sl["idx"][:tot], non_blocking=True)
                ho[l]["cu"].copy_(sl["cu"], non_blocking=True)
                ho[l]["ko"].copy_(sl["ko"][:tot], non_blocking=True)
                ho[l]["vo"].copy_(sl["vo"][:tot], non_blocking=True)
                d2h_done[s].record(s_d2h)

    for _ in range(2):                       # warm-up: first use of the pinned pages
        step()
    torch.cuda.synchronize(dev)
    K = args.e2e_steps
    barrier(world)
    torch.cuda.synchronize(dev)
    t0 = time.perf_counter()
    for _ in range(K):
        step()
    torch.cuda.synchronize(dev)
    dt = (time.perf_counter() - t0) / K
    barrier(world)
    dt = max_over_ranks(dt, world)
    for sl in slots:
        st = sg.sgdkv_last_error(sl["ws"])
        if st != sg.OK:
            raise RuntimeError(f"device-side error in the e2e run: {sg.status_string(st)}")
    return {"value": world * wl.L * Ls / dt, "unit": UNIT, "h2d_bytes_per_step": int(h2d_bytes),
            "d2h_bytes_per_step": int(d2h_bytes),
            "host_read_bytes_per_step": int(host_read_bytes),
            "ms_per_step": dt * 1e3, "steps": K,
            "overlap": "H2D (q, K) / compute / D2H on three streams, two device slots; V stays "
                       "in pinned host memory and the gather reads only the kept rows"}


# ------------------------------------------------------------------------------------------
# the CPU oracle (reported baseline; also the reference arm)
# ------------------------------------------------------------------------------------------

def cpu_child(args):
    """Runs in a fresh process: times the oracle on one layer (all KV heads) of the workload."""
    import numpy as np

    from oracle import sgdkv_oracle as O
    from paper_2609_03235_gb300 import configs, synth
    wl = configs.BY_NAME[args.workload]
    heads = int(os.environ.get("SGDKV_ORACLE_HEADS", str(wl.Hkv)))
    inp = synth.layer_inputs_host(wl, 0)
    n_sink, n_recent = configs.sink_recent_split(wl.floor)
    b_all = O.allocate_budgets(synth.head_scores(wl), wl.L, wl.total_budget(args.frac), wl.floor)
    b = b_all[:wl.Hkv][:heads]
    G = wl.G
    reps = int(os.environ.get("SGDKV_ORACLE_REPS", "1"))
    times = []
    for _ in range(reps):
        t0 = time.perf_counter()
        O.allocate_budgets(synth.head_scores(wl), wl.L, wl.total_budget(args.frac), wl.floor)
        O.compress_layer(inp["q"][:heads * G], inp["K"][:heads], inp["V"][:heads], b, n_sink,
                         n_recent, pool=wl.pool)
        times.append(time.perf_counter() - t0)
    print(json.dumps({"seconds": times, "heads": heads, "Hkv": wl.Hkv,
                      "threads": int(os.environ.get("OMP_NUM_THREADS", "0"))}))


def run_cpu_oracle(args, heads=None, reps=1):
    cores = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else os.cpu_count()
    env = dict(os.environ)
    for v in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS"):
        env[v] = str(cores)
    env["CUDA_VISIBLE_DEVICES"] = ""
    if heads is not None:
        env["SGDKV_ORACLE_HEADS"] = str(heads)
    env["SGDKV_ORACLE_REPS"] = str(reps)
    cmd = [sys.executable, os.path.join(ROOT, "bench.py"), "--cpu-child", "--workload",
           args.workload, "--frac", str(args.frac)]
    r = subprocess.run(cmd, env=env, capture_output=True, text=True, timeout=1800)
    if r.returncode != 0:
        raise RuntimeError("oracle child failed:\n" + r.stderr[-2000:])
    out = json.loads(r.stdout.strip().splitlines()[-1])
    return out, cores


def cpu_baseline(args):
    from paper_2609_03235_gb300 import configs
    wl = configs.BY_NAME[args.workload]
    out, cores = run_cpu_oracle(args, reps=3)
    sec = statistics.mean(out["seconds"])
    per_layer = sec * wl.Hkv / out["heads"]
    return {"value": wl.L / per_layer, "unit": UNIT, "cores": cores, "kind": "oracle",
            "sample": f"1 of {wl.n_layers} layers ({out['heads']} of {wl.Hkv} KV heads), "
                      f"mean of 3 runs, {sec:.1f} s each, NumPy float64 oracle, BLAS threads = {cores}"}


def run_reference(args, world, rank):
    from paper_2609_03235_gb300 import configs
    wl = configs.BY_NAME[args.workload]
    if rank != 0:
        return None
    # each step: one KV head of one layer (a bounded sample of the workload)
    out, cores = run_cpu_oracle(args, heads=1, reps=args.warmup + args.steps)
    secs = out["seconds"][args.warmup:] or out["seconds"]
    step_s = statistics.mean(secs)
    value = wl.L / (step_s * wl.Hkv)
    return {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": step_s * 1e3,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic (seeded, host-generated)", "impl": "reference",
            "config": workload_config(wl, args, world,
                                      wl.n_layers if args.layers <= 0 else min(args.layers, wl.n_layers)),
            "cpu_baseline": {"value": value, "unit": UNIT, "kind": "oracle", "cores": cores,
                             "sample": f"each step: 1 KV head of 1 layer of {wl.name}"},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}


def main(argv=None):
    args = parse_args(argv)
    if args.cpu_child:
        cpu_child(args)
        return 0
    world, rank, local = dist_env()
    if args.gpus != world and world > 1:
        print(f"warning: --gpus {args.gpus} but WORLD_SIZE {world}", file=sys.stderr)
    if args.impl == "reference":
        rec = run_reference(args, world, rank)
        if rec is not None:
            print(json.dumps(rec))
        return 0
    dist_init(world)
    rec = run_ours(args, world, rank, local)
    if rank == 0:
        if world == 1 and not args.no_cpu_baseline:
            rec["cpu_baseline"] = cpu_baseline(args)
        print(json.dumps(rec))
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
