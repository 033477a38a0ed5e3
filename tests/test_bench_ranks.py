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
