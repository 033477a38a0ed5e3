"""Failure detection on the GPU without a fault: every mbarrier wait in the scoring
kernels is bounded.  The test hook makes the MMA issuer wait on a barrier nothing
signals; the wait must run out after the configured bound, the kernels must record
SGDKV_ERR_TIMEOUT, drain their in-flight copies, free TMEM and exit, and the context must
stay usable: the next call with the hook off gives correct scores."""
import numpy as np
import pytest
import torch

from oracle import sgdkv_oracle as O
from paper_2609_03235_gb300 import synth
from paper_2609_03235_gb300 import sgdkv as sg

pytestmark = pytest.mark.gpu


def test_bounded_wait_times_out_and_recovers():
    dev = torch.device("cuda:0")
    wl = synth.tiny_workload(Hq=14, Hkv=2, d=128, L=3000, W=32, n_salient=8)
    inp = synth.tiny_inputs(wl, tag=77)
    q = synth.to_torch_bf16(inp["q"], dev)
    K = synth.to_torch_bf16(inp["K"], dev)
    ws = sg.make_workspace(wl.Hq, wl.Hkv, wl.L, wl.W, dev)
    out = torch.zeros((wl.Hkv, wl.L), dtype=torch.float32, device=dev)
    try:
        sg.sgdkv_debug_set_score_hooks(1, 2_000_000)        # stall the MMA issuer, 2 ms bound
        sg.sgdkv_score(q, K, wl.W, 7, out, ws)
        assert sg.sgdkv_last_error(ws) == sg.ERR_TIMEOUT
    finally:
        sg.sgdkv_debug_set_score_hooks(0, 0)
    assert sg.sgdkv_last_error(ws) == sg.OK                # cleared by the previous read
    sg.sgdkv_score(q, K, wl.W, 7, out, ws)
    torch.cuda.synchronize()
    assert sg.sgdkv_last_error(ws) == sg.OK
    exp = O.max_pool(O.window_scores(inp["q"], inp["K"]), 7)
    got = out.cpu().numpy()
    assert np.all(np.abs(got - exp) <= 1e-5 + 2e-3 * np.abs(exp))
