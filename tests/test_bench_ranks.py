"""The benchmark's multi-process path on CPU (gloo, world size 2): ranks run replicas,
meet at barriers and report the maximum of their timings; only rank 0 runs the reference
arm.  Uses 127.0.0.1 for the rendezvous."""
import os
import socket

import pytest
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    import bench
    w, r, local = bench.dist_env()
    assert (w, r, local) == (world, rank, rank)
    bench.dist_init(w)
    bench.barrier(w)
    out[rank] = bench.max_over_ranks(1.5 + rank, w)
    ref = bench.run_reference(bench.parse_args(["--impl", "reference"]), w, r) if r != 0 else None
    assert ref is None
    bench.barrier(w)
    import torch.distributed as dist
    dist.destroy_process_group()


def test_max_over_two_gloo_ranks():
    world = 2
    port = _free_port()
    manager = mp.Manager()
    out = manager.dict()
    mp.spawn(_worker, args=(world, port, out), nprocs=world, join=True)
    assert out[0] == out[1] == 2.5


def test_single_process_needs_no_group():
    import bench
    assert bench.max_over_ranks(3.25, 1) == 3.25
    bench.barrier(1)


def test_roofs_pick_the_binding_roof():
    """The step's floor per layer is the larger of the HBM and tensor floors; W = 32 shapes
    are bound by HBM, W = 64 shapes by the tensor pipe at these budgets."""
    import numpy as np

    import bench
    from paper_2609_03235_gb300 import configs
    peaks = dict(hbm=6678.5, bf16=1897.4, bf16_sus=1723.5, source="measured")
    for name, frac, bound in [("c2_qwen25_7b_L32k", 0.25, "hbm"),
                              ("c3_qwen25_7b_L128k", 0.25, "tensor"),
                              ("c4_qwen3_32b_L128k", 0.25, "tensor")]:
        wl = configs.BY_NAME[name]
        b = np.full(wl.Hkv, int(frac * wl.L), np.int64)
        outs = [dict(b=b)]
        _, rf = bench.roofs(wl, outs, 1.0, 1, peaks)
        br = rf["binding_roof"]
        assert br["bound"] == bound
        assert br["floor_us_per_layer"] == max(br["hbm_floor_us_per_layer"],
                                               br["tensor_floor_us_per_layer"])
        assert abs(br["frac"] - br["floor_us_per_layer"] / 1000.0) < 1e-12
        hbm = rf["hbm_path"]
        assert abs(hbm["achieved_gbs"] - hbm["bytes_per_step"] / 1e-3 / 1e9) < 1e-6


def test_sweep_covers_every_workload_and_budget():
    import bench
    cases = bench.sweep_cases()
    assert ("c3_qwen25_7b_L128k", 0.125) in cases and ("c3_qwen25_7b_L128k", 0.5) in cases
    assert {n for n, _ in cases} == {"c1_single_layer_L4k", "c2_qwen25_7b_L32k",
                                     "c3_qwen25_7b_L128k", "c4_qwen3_32b_L128k",
                                     "c5_qwen25_7b_L1m"}
    assert len(cases) == 7
