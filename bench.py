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
    p.add_argument("--no-sweep", action="store_true",
                   help="skip the per-workload measurements beside the headline")
    p.add_argument("--deterministic", action="store_true",
                   help="score with SGDKV_SCORE_DETERMINISTIC (bit-reproducible scores)")
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
_SCORE_SHA = "fa49b3044063c5da7cdd915f5f3c6a294dadf9df04c9006fa9bb616fb448e6c1"
_SELECT_SHA = "5ae20f0374e7f88753406f17f0b0eee0c6453579642823a0f79678d0246f1390"
MEASURED_TRAFFIC = {
    ("score_pass1_tc", "c3_qwen25_7b_L128k"):
        {"bytes": 134765312 + 2956544, "source": "score_tc.cu", "sha256": _SCORE_SHA},
    ("score_pass2_tc", "c3_qwen25_7b_L128k"):
        {"bytes": 135362304 + 1843712, "source": "score_tc.cu", "sha256": _SCORE_SHA},
    ("sel_cluster_kernel", "c3_qwen25_7b_L128k"):
        {"bytes": 8444672 + 0, "source": "select.cu", "sha256": _SELECT_SHA},
    ("gather_kernel", "c3_qwen25_7b_L128k"):
        {"bytes": 40771328 + 528128, "source": "select.cu", "sha256": _SELECT_SHA},
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
                  (2 * wl.Hkv * wl.L * wl.d * 2 >> 20),
            "scores": "bit-reproducible (SGDKV_SCORE_DETERMINISTIC)"
                      if getattr(args, "deterministic", False) else
                      "dynamic key-tile claims (reproducible to fp32 rounding)"}



class StepRunner:
    """One workload's compression step on this GPU: inputs of every layer resident in HBM,
    the step's launches captured into CUDA graphs and replayed.

    One step = the host budget allocation (a1), then the launches of every layer: the two
    scoring passes on the capturing stream, sgdkv_pool_compact (the max-pool inside the
    selection kernel, then the gather) on `sel_stream`; layer l's pooling and compaction
    wait for layer l's passes only, so they overlap layer l+1's scoring, whose CTAs claim
    key tiles dynamically and absorb the SMs the other stream leaves.  The raw scores of
    layer l stay in scoring workspace l % 3 until its compaction has read them (layer
    l + 3's scoring waits for that: with two workspaces, layer l + 2's scoring would wait
    for layer l's gather as well).  The launches of a step are captured into a CUDA graph
    (per-kernel launch cost ~1 us instead of ~3 us on a stream) and the graph is replayed;
    the allocation still runs on the host every step and must reproduce the budgets the
    graph was captured with."""

    def __init__(self, wl, frac, n_layers, dev, score_flags=0):
        import numpy as np
        import torch

        from paper_2609_03235_gb300 import configs, synth
        from paper_2609_03235_gb300 import sgdkv as sg
        self.np, self.torch, self.sg = np, torch, sg
        self.wl, self.frac, self.dev = wl, frac, dev
        self.score_flags = score_flags
        self.n_sink, self.n_recent = configs.sink_recent_split(wl.floor)
        self.hs = synth.head_scores(wl)
        self.T = wl.total_budget(frac)
        self.b_all = sg.sgdkv_allocate_budgets(self.hs, wl.L, self.T, wl.floor)
        self.Ls = n_layers
        self.layers = [synth.layer_inputs_device(wl, l, dev) for l in range(n_layers)]
        self.outs = []
        for l in range(n_layers):
            b = self.b_all[l * wl.Hkv:(l + 1) * wl.Hkv]
            tot = int(b.sum())
            self.outs.append(dict(
                b=b, scores=torch.empty((wl.Hkv, wl.L), dtype=torch.float32, device=dev),
                idx=torch.empty(tot, dtype=torch.int32, device=dev),
                cu=torch.empty(wl.Hkv + 1, dtype=torch.int32, device=dev),
                ko=torch.empty((tot, wl.d), dtype=torch.bfloat16, device=dev),
                vo=torch.empty((tot, wl.d), dtype=torch.bfloat16, device=dev)))
        self.ws_score = [sg.make_workspace(wl.Hq, wl.Hkv, wl.L, wl.W, dev)
                         for _ in range(N_SCORE_WS)]
        self.ws_sel = sg.make_workspace(wl.Hq, wl.Hkv, wl.L, wl.W, dev)
        self.stream = torch.cuda.current_stream(dev)
        lo_prio, hi_prio = torch.cuda.Stream.priority_range()
        self.sel_stream = torch.cuda.Stream(dev, priority=hi_prio)
        self.fork = torch.cuda.Event()
        self.scored = [torch.cuda.Event() for _ in range(n_layers)]
        self.pooled = [torch.cuda.Event() for _ in range(n_layers)]  # workspace l % N read
        self.done = torch.cuda.Event()

    def launches(self, s, kinds=(), every=1, first=0):
        sg, wl = self.sg, self.wl
        self.fork.record(s)
        self.sel_stream.wait_event(self.fork)
        for l in range(self.Ls):
            inp, o = self.layers[l], self.outs[l]
            sg.sgdkv_debug_enable_kernel_timing(kinds if l % every == first % every else ())
            wsl = self.ws_score[l % N_SCORE_WS]
            if l >= N_SCORE_WS:
                s.wait_event(self.pooled[l - N_SCORE_WS])   # its workspace read by then
            sg.sgdkv_score_raw(inp["q"], inp["K"], wl.W, wsl, s, flags=self.score_flags)
            self.scored[l].record(s)
            self.sel_stream.wait_event(self.scored[l])
            sg.sgdkv_pool_compact(wsl, wl.pool, inp["K"], inp["V"], o["b"], self.n_sink,
                                  self.n_recent, o["scores"], o["idx"], o["cu"], o["ko"],
                                  o["vo"], self.ws_sel, self.sel_stream)
            self.pooled[l].record(self.sel_stream)
        sg.sgdkv_debug_enable_kernel_timing(())
        self.done.record(self.sel_stream)
        s.wait_event(self.done)

    def allocate(self):
        ball = self.sg.sgdkv_allocate_budgets(self.hs, self.wl.L, self.T, self.wl.floor)   # a1
        if not self.np.array_equal(ball, self.b_all):
            raise RuntimeError("budget allocation changed between steps")
        return ball

    def capture(self, kinds, every=1, first=0):
        """One step's launches as a CUDA graph; the kernels of `kinds` in every `every`-th
        layer from layer `first` on are bracketed by timing events."""
        torch, sg = self.torch, self.sg
        g = torch.cuda.CUDAGraph()
        n0 = sg.sgdkv_launch_count()
        with torch.cuda.graph(g):
            self.launches(torch.cuda.current_stream(self.dev), kinds, every, first)
        return g, sg.sgdkv_launch_count() - n0

    def drain_timers(self):
        return [self.sg.sgdkv_debug_kernel_timing(kind) for kind in range(len(KERNEL_NAMES))]

    def check(self, where):
        sg = self.sg
        st = max(max(sg.sgdkv_last_error(w, self.stream) for w in self.ws_score),
                 sg.sgdkv_last_error(self.ws_sel, self.sel_stream))
        if st != sg.OK:
            raise RuntimeError(f"device-side error {where}: {sg.status_string(st)}")

    def measure(self, steps, warmup, diag_steps, world, local):
        """Warm-up, a diagnostic window (every launch bracketed: per-kernel shares and the
        dominant scoring pass), then `steps` timed graph replays between barrier +
        synchronize and CUDA events on the launching stream, with the dominant pass
        bracketed in every TIMED_EVERY-th layer (rotating by one layer per step) and
        nvidia-smi clocks sampled meanwhile."""
        torch = self.torch
        dev = self.dev
        self.launches(self.stream)         # one eager step (first-use setup), then graphs
        torch.cuda.synchronize(dev)
        self.check("in the first step")
        g_warm, _ = self.capture(())
        for _ in range(max(warmup, 0)):
            self.allocate()
            g_warm.replay()
        torch.cuda.synchronize(dev)
        self.check("during warm-up")
        self.drain_timers()
        diag = [self.capture(range(len(KERNEL_NAMES)))[0] for _ in range(diag_steps)]
        for g in diag:
            self.allocate()
            g.replay()
        torch.cuda.synchronize(dev)
        kern = {}
        for name, (tot_ms, n) in zip(KERNEL_NAMES, self.drain_timers()):
            kern[name] = {"launches": n, "us_per_launch": 1e3 * tot_ms / max(n, 1),
                          "ms_total": tot_ms, "dram_bytes_ncu": measured_traffic(name, self.wl.name)}
        del diag
        kern = {k: v for k, v in kern.items() if v["launches"] > 0}
        all_ms = sum(v["ms_total"] for v in kern.values())
        for v in kern.values():
            v["share"] = v["ms_total"] / all_ms if all_ms > 0 else None
        # the compaction kernels against their roofs: the selection's algorithmic bytes are
        # the raw planes it pools (16 B per key) and the pooled scores and indices it writes;
        # the gather's, the kept rows read and written plus their indices
        wl, hbm = self.wl, measured_peaks()["hbm"]
        kept = sum(int(o["b"].sum()) for o in self.outs) / max(self.Ls, 1)
        copied = "gather_kernel" not in kern     # the selection copied the rows itself
        roof_bytes = {"sel_cluster_kernel": wl.Hkv * wl.L * (16 + 4) + kept * 4 +
                      (kept * 4 * wl.d * 2 if copied else 0),
                      "gather_kernel": kept * (4 * wl.d * 2 + 4)}
        bound = {"sel_cluster_kernel": "latency (cluster barriers and histogram exchange; "
                                       "inputs L2-resident)" +
                                       ("; plus the HBM copy of the kept rows" if copied else ""),
                 "gather_kernel": "hbm"}
        for name, byts in roof_bytes.items():
            if name in kern:
                gbs = byts / (kern[name]["us_per_launch"] * 1e-6) / 1e9
                kern[name]["roofline"] = {"bound": bound[name], "bytes_per_launch": byts,
                                          "achieved_gbs": gbs, "peak_gbs": hbm,
                                          "frac_of_hbm": gbs / hbm,
                                          "note": "live duration, sharing SMs with the "
                                                  "scoring stream"}
        top_kind = max(range(2), key=lambda k: kern[KERNEL_NAMES[k]]["ms_total"])
        timed = [self.capture([top_kind], TIMED_EVERY, k) for k in range(steps)]
        start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        clocks = ClockSampler(nvsmi_id(local))
        barrier(world)
        torch.cuda.synchronize(dev)
        clocks.start()
        time.sleep(0.3)                  # let the sampler attach before the timed region
        start.record(self.stream)
        for g, _ in timed:
            self.allocate()
            g.replay()
        end.record(self.stream)
        torch.cuda.synchronize(dev)
        launches_timed = sum(n for _, n in timed)
        top_ms, top_n = self.sg.sgdkv_debug_kernel_timing(top_kind)
        clk = clocks.stop()
        barrier(world)
        self.check("in the timed region")
        del timed, g_warm
        ms = start.elapsed_time(end) / steps
        return dict(ms=ms, ms_max=max_over_ranks(ms, world), kern=kern,
                    top=KERNEL_NAMES[top_kind], top_us=1e3 * top_ms / max(top_n, 1),
                    top_n=top_n, launches=int(launches_timed), clocks=clk)

    def free(self):
        self.layers = self.outs = self.ws_score = self.ws_sel = None


def roofs(wl, outs, ms_step, n_layers, peaks):
    """The step against its two roofs (per layer): HBM for the algorithmic bytes and the
    tensor pipe for the two scoring passes' flops.  The binding roof is the larger of the two
    floor times; its fraction is floor time / measured time."""
    bytes_step = sum(path_bytes(wl, o["b"]) for o in outs)
    us_layer = 1e3 * ms_step / n_layers
    hbm_us = bytes_step / n_layers / (peaks["hbm"] * 1e9) * 1e6
    tensor_us = score_flops(wl) / (peaks["bf16"] * 1e12) * 1e6
    bound = "tensor" if tensor_us > hbm_us else "hbm"
    roof_us = max(hbm_us, tensor_us)
    hbm_gbs = bytes_step / (ms_step * 1e-3) / 1e9
    return bytes_step, {
        "hbm_path": {"achieved_gbs": hbm_gbs, "peak_gbs": peaks["hbm"],
                     "frac": hbm_gbs / peaks["hbm"], "bytes_per_step": bytes_step},
        "binding_roof": {"bound": bound, "floor_us_per_layer": roof_us,
                         "hbm_floor_us_per_layer": hbm_us, "tensor_floor_us_per_layer": tensor_us,
                         "us_per_layer": us_layer, "frac": roof_us / us_layer,
                         "peaks": f"{peaks['source']}: HBM {peaks['hbm']} GB/s, bf16 burst "
                                  f"{peaks['bf16']} TFLOP/s (two scoring passes of "
                                  "2*G*W*d flops per key per KV head)"}}


# Workloads measured beside the headline by the default run: every configuration the
# compression step is specified on, the 128K Qwen2.5-7B shape at each of its total budgets.
E2E_ROUNDS = 3                # timed rounds of the end-to-end run (median reported)
SWEEP_STEPS, SWEEP_WARMUP = 5, 3
SWEEP_MIN_LAYER_STEPS = 112   # timed steps x layers at least this: a one-layer step is ~50 us,
                              # and five of them would be mostly the timed region's start-up


def sweep_cases():
    from paper_2609_03235_gb300 import configs
    return [(w.name, f) for w in configs.WORKLOADS for f in w.budget_fracs]


def run_sweep(args, world, local, dev, peaks, skip):
    """One entry per (workload, total budget): tokens/s/layer, us/layer, the HBM and binding
    roof fractions, the dominant pass's CUDA-event time and the clocks of its timed region."""
    import torch

    from paper_2609_03235_gb300 import configs
    out = {}
    for name, frac in sweep_cases():
        key = f"{name}@{frac:g}"
        if (name, frac) == skip:
            out[key] = "headline (top-level fields of this line)"
            continue
        wl = configs.BY_NAME[name]
        r = StepRunner(wl, frac, wl.n_layers, dev)
        steps = max(SWEEP_STEPS, -(-SWEEP_MIN_LAYER_STEPS // wl.n_layers))
        m = r.measure(steps, SWEEP_WARMUP, 1, world, local)
        _, rf = roofs(wl, r.outs, m["ms_max"], r.Ls, peaks)
        tf = pass_flops(wl) / (m["top_us"] * 1e-6) / 1e12
        out[key] = {
            "value": world * wl.L * r.Ls / (m["ms_max"] * 1e-3), "unit": UNIT,
            "us_per_layer": 1e3 * m["ms_max"] / r.Ls, "ms_per_step": m["ms_max"],
            "n_layers": r.Ls, "steps": steps, "warmup": SWEEP_WARMUP,
            "model_shape": "Qwen2.5-7B-1M" if wl.Hkv == 4 else "Qwen3-32B",
            "context_len": wl.L, "window": wl.W, "budget_frac": frac,
            **rf,
            "dominant_pass": {"kernel": m["top"], "us_per_launch": m["top_us"],
                              "launches_timed": m["top_n"], "tflops": tf,
                              "frac_of_bf16_burst": tf / peaks["bf16"]},
            "gpu_launches": m["launches"], "clocks": m["clocks"]}
        r.free()
        del r
        torch.cuda.synchronize(dev)
        torch.cuda.empty_cache()
    return out


def run_ours(args, world, rank, local):
    import torch

    from paper_2609_03235_gb300 import configs
    from paper_2609_03235_gb300 import sgdkv as sg

    wl = configs.BY_NAME[args.workload]
    dev = torch.device(f"cuda:{local}")
    torch.cuda.set_device(dev)
    sg.lib()
    Ls = wl.n_layers if args.layers <= 0 else min(args.layers, wl.n_layers)
    r = StepRunner(wl, args.frac, Ls, dev,
                   sg.SCORE_DETERMINISTIC if args.deterministic else 0)
    m = r.measure(args.steps, args.warmup, DIAG_STEPS, world, local)
    ms_max = m["ms_max"]
    kern = m["kern"]

    peaks = measured_peaks()
    # The timed region lasts well under a second at full clocks, so the dominant pass is
    # set against the burst bf16 peak (the sustained figure is for seconds-long loops).
    achieved_tf = pass_flops(wl) / (m["top_us"] * 1e-6) / 1e12
    stage_us = sum(kern[n]["us_per_launch"] for n in KERNEL_NAMES[:3] if n in kern)
    stage_tf = score_flops(wl) / (stage_us * 1e-6) / 1e12
    bytes_step, rf = roofs(wl, r.outs, ms_max, Ls, peaks)
    value = world * wl.L * Ls / (ms_max * 1e-3)

    dec = None if args.no_decode else run_decode(args, wl, r.outs, dev, r.stream, peaks)

    e2e = None
    if not args.no_e2e and args.e2e_steps > 0:
        e2e = run_e2e(args, wl, r.layers, r.outs, r.n_sink, r.n_recent, dev, world)
    r.free()
    del r
    torch.cuda.synchronize(dev)
    torch.cuda.empty_cache()

    sweep = None
    if not args.no_sweep and world == 1:      # replicas (N > 1) time the headline only
        sweep = run_sweep(args, world, local, dev, peaks, skip=(wl.name, args.frac)
                          if Ls == wl.n_layers else None)

    rec = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_max, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (seeded N(0,1) K/V/Q with planted sink and salient keys)",
        "config": workload_config(wl, args, world, Ls),
        "roofline": {"kernel": m["top"], "bound": "tensor", "achieved": achieved_tf,
                     "peak": peaks["bf16"], "unit": "TFLOP/s",
                     "frac": achieved_tf / peaks["bf16"],
                     "traffic": measured_traffic(m["top"], wl.name),
                     "peak_source": peaks["source"] + " bf16 burst (timed region < 1 s)",
                     "frac_of_sustained": achieved_tf / peaks["bf16_sus"],
                     "us_per_launch": m["top_us"], "launches_timed": m["top_n"],
                     "timed_launches": f"every {TIMED_EVERY}th layer of every timed step, "
                                       "rotating by one layer per step",
                     "flops_per_launch": pass_flops(wl)},
        "score_stage": {"us_per_layer": stage_us, "tflops": stage_tf,
                        "frac": stage_tf / peaks["bf16"]},
        "kernels": {"window": f"{DIAG_STEPS} steps after warm-up, every launch bracketed",
                    **kern},
        **rf,
        "decode_attention": dec,
        "gpu_launches": m["launches"],
        "schedule": "each step: budget allocation on the host, then one CUDA-graph launch of "
                    "the step's kernels (the scoring passes on one stream, max-pool + "
                    "selection in one kernel and the gather on a second inside the graph); "
                    "one graph per timed step",
        "clocks": m["clocks"],
        "e2e": e2e,
        "workloads": sweep,
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
    rounds = []          # the host link is shared with other jobs: three rounds, the median
    for _ in range(E2E_ROUNDS):
        barrier(world)
        torch.cuda.synchronize(dev)
        t0 = time.perf_counter()
        for _ in range(K):
            step()
        torch.cuda.synchronize(dev)
        dt = (time.perf_counter() - t0) / K
        barrier(world)
        rounds.append(max_over_ranks(dt, world))
    dt = sorted(rounds)[len(rounds) // 2]
    for sl in slots:
        st = sg.sgdkv_last_error(sl["ws"])
        if st != sg.OK:
            raise RuntimeError(f"device-side error in the e2e run: {sg.status_string(st)}")
    return {"value": world * wl.L * Ls / dt, "unit": UNIT, "h2d_bytes_per_step": int(h2d_bytes),
            "d2h_bytes_per_step": int(d2h_bytes),
            "host_read_bytes_per_step": int(host_read_bytes),
            "ms_per_step": dt * 1e3, "steps": K,
            "rounds_ms_per_step": [x * 1e3 for x in rounds], "of_rounds": "median",
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
