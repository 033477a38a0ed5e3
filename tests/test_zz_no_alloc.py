"""sgdkv_score_static: scoring for callers that cannot allocate device memory.

It uses a static scratch array inside the library instead of a caller workspace.  Two
calls in a row must each give the scores of the oracle and of sgdkv_score with a workspace
(within the score tolerance), report a clean device status, and take no device memory;
shapes beyond the scratch must be refused before any device work, leaving the output as
it was.  Named to be collected last; it also passes on its own.
"""
import ctypes

import numpy as np
import pytest
import torch

from oracle import sgdkv_oracle as O
from paper_2609_03235_gb300 import synth
from paper_2609_03235_gb300 import sgdkv as sg

pytestmark = pytest.mark.gpu
RTOL, ATOL = 2e-3, 1e-5


def _within(got, exp):
    return np.abs(got - exp) <= ATOL + RTOL * np.abs(exp)


def test_static_scratch_matches_oracle_and_workspace_path_twice():
    dev = torch.device("cuda:0")
    wl = synth.tiny_workload(Hq=28, Hkv=4, d=128, L=5000, W=64, n_salient=16)
    inp = synth.tiny_inputs(wl, tag=900)
    q = synth.to_torch_bf16(inp["q"], dev)
    K = synth.to_torch_bf16(inp["K"], dev)
    ws = sg.make_workspace(wl.Hq, wl.Hkv, wl.L, wl.W, dev)
    ref = torch.empty((wl.Hkv, wl.L), dtype=torch.float32, device=dev)
    sg.sgdkv_score(q, K, wl.W, 7, ref, ws)
    torch.cuda.synchronize()
    assert sg.sgdkv_last_error(ws) == sg.OK
    from_ws = ref.cpu().numpy().astype(np.float64)
    oracle = O.max_pool(O.window_scores(inp["q"], inp["K"]), 7)
    assert _within(from_ws, oracle).all()
    outs = [torch.full((wl.Hkv, wl.L), -1.0, dtype=torch.float32, device=dev) for _ in range(2)]
    stats = [torch.full((1,), 12345, dtype=torch.int32, device=dev) for _ in range(2)]
    torch.cuda.synchronize()
    mem = None
    for i in range(2):
        if i == 1:
            # after the first call (which looks the scratch up and loads what it launches),
            # a call takes no device memory at all
            mem = (torch.cuda.memory_allocated(dev), torch.cuda.mem_get_info(dev)[0])
        sg.sgdkv_score_static(q, K, wl.W, 7, outs[i], stats[i])
        torch.cuda.synchronize()
        assert int(stats[i].item()) == sg.OK
        got = outs[i].cpu().numpy().astype(np.float64)
        assert _within(got, oracle).all(), f"call {i}: off the oracle"
        assert _within(got, from_ws).all(), f"call {i}: off the workspace path"
    assert (torch.cuda.memory_allocated(dev), torch.cuda.mem_get_info(dev)[0]) == mem


def test_static_scratch_rejects_oversized_shape():
    dev = torch.device("cuda:0")
    Hq, Hkv, L, W = 28, 4, 1 << 20, 64          # needs about 69 MiB of scratch
    q = torch.zeros((Hq, W, 128), dtype=torch.bfloat16, device=dev)
    K = torch.zeros((1, 128), dtype=torch.bfloat16, device=dev)   # never read: refused first
    out = torch.full((64,), 7.0, dtype=torch.float32, device=dev)
    status = torch.full((1,), 12345, dtype=torch.int32, device=dev)
    torch.cuda.synchronize()
    st = sg.lib().sgdkv_score_static(ctypes.c_void_p(q.data_ptr()), ctypes.c_void_p(K.data_ptr()),
                                     Hq, Hkv, L, 128, W, 7, ctypes.c_void_p(out.data_ptr()),
                                     ctypes.c_void_p(status.data_ptr()), sg._stream(None))
    assert st == sg.ERR_WORKSPACE
    torch.cuda.synchronize()
    assert bool((out == 7.0).all()), "the refused call wrote its output"
    assert int(status.item()) == 12345, "the refused call wrote its status"
