"""GPU parity of the decode attention over the compressed cache, through the C-ABI.

Bar (from the arithmetic): logits from bf16 products summed in fp32, the softmax in fp32,
the weights rounded to bf16 (relative error <= 2^-9 each) and normalised by the sum of the
rounded weights, so the output is a convex combination of the head's value rows whose
weights are off by at most 2 * 2^-9 relative: |gpu - oracle| <= 2^-8 * max|v| over the
head's rows, plus 1e-5 for the fp32 sums.  The output must also lie within the rows'
per-column range.
"""
import numpy as np
import pytest
import torch

from oracle import sgdkv_oracle as O
from paper_2609_03235_gb300 import configs, synth
from paper_2609_03235_gb300 import sgdkv as sg

from _guard import guarded

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dev():
    sg.lib()
    return torch.device("cuda:0")


def _case(Hq, Hkv, n_tok, budgets, seed, q_scale=1.0):
    rng = np.random.default_rng(seed)
    R = int(np.sum(budgets))
    q = synth.bf16_round(rng.standard_normal((Hq, n_tok, 128)).astype(np.float32) * q_scale)
    K = synth.bf16_round(rng.standard_normal((max(R, 1), 128)).astype(np.float32))
    V = synth.bf16_round(rng.standard_normal((max(R, 1), 128)).astype(np.float32))
    return q, K[:R], V[:R]


def _run(dev, q, K, V, budgets):
    Hq, n_tok, _ = q.shape
    Hkv = len(budgets)
    R = int(np.sum(budgets))
    qt = synth.to_torch_bf16(q, dev)
    Kt = synth.to_torch_bf16(K, dev) if R else None
    Vt = synth.to_torch_bf16(V, dev) if R else None
    g_out = guarded((Hq, n_tok, 128), torch.float32, dev, fill=float("nan"))
    ws = sg.make_decode_workspace(Hq, Hkv, n_tok, R, dev)
    sg.sgdkv_decode_attention(qt, Kt, Vt, budgets, g_out.t, ws)
    torch.cuda.synchronize()
    g_out.check("decode output")
    return g_out.t.cpu().numpy()


def _check(got, q, K, V, budgets):
    cu = np.concatenate([[0], np.cumsum(budgets)]).astype(np.int64)
    exp = O.decode_attention(q, K, V, cu)
    Hq = q.shape[0]
    G = Hq // len(budgets)
    vf = O.bf16_bits_to_f64(V) if len(V) else np.zeros((0, 128))
    for qh in range(Hq):
        h = qh // G
        seg = vf[cu[h]:cu[h + 1]]
        if seg.shape[0] == 0:
            assert np.array_equal(got[qh], np.zeros_like(got[qh])), f"head {qh}: not zero"
            continue
        tol = 2.0 ** -8 * np.abs(seg).max() + 1e-5
        err = np.abs(got[qh] - exp[qh]).max()
        assert err <= tol, f"query head {qh}: error {err} > {tol}"
        assert np.all(got[qh] >= seg.min(axis=0) - 1e-5) and np.all(got[qh] <= seg.max(axis=0) + 1e-5)


CASES = [
    # Hq, Hkv, n_tok, budgets                  (what it covers)
    (28, 4, 1, [1250, 700, 2400, 256]),        # GQA group of 7, ragged chunks
    (64, 8, 1, [0, 517, 3, 1024, 32, 33, 31, 4000]),   # group of 8, an empty head, tile +-1
    (4, 4, 1, [1, 64, 0, 1000]),               # one query row per head, single-row head
    (8, 1, 2, [5000]),                         # 16 query rows (the most)
    (14, 2, 1, [96, 7000]),                    # uneven heads
    (2, 2, 3, [0, 0]),                         # no rows at all
    (8, 2, 1, [3, 150000]),                    # one head holds 147 of the 149 chunks
]


@pytest.mark.parametrize("Hq,Hkv,n_tok,budgets", CASES)
@pytest.mark.parametrize("q_scale", [1.0, 8.0])
def test_decode_parity(dev, Hq, Hkv, n_tok, budgets, q_scale):
    b = np.asarray(budgets, np.int64)
    q, K, V = _case(Hq, Hkv, n_tok, b, seed=int(b.sum()) + Hq, q_scale=q_scale)
    _check(_run(dev, q, K, V, b), q, K, V, b)


def test_decode_over_a_compressed_layer(dev):
    """End to end: compress a layer, then decode over the cache the GPU wrote (its rows are
    bit-exact with the oracle's gather of the GPU's indices)."""
    wl = synth.tiny_workload(Hq=28, Hkv=4, d=128, L=5000, W=64, n_salient=32, floor=256)
    inp = synth.tiny_inputs(wl, tag=301)
    q = synth.to_torch_bf16(inp["q"], dev)
    K = synth.to_torch_bf16(inp["K"], dev)
    V = synth.to_torch_bf16(inp["V"], dev)
    b = np.array([1250, 700, 2400, 256], np.int64)
    ws = sg.make_workspace(wl.Hq, wl.Hkv, wl.L, wl.W, dev)
    out = sg.compress_layer_alloc(q, K, V, b, wl.W, 7, 128, 128, ws)
    rng = np.random.default_rng(5)
    qd = synth.bf16_round(rng.standard_normal((28, 1, 128)).astype(np.float32) * 2.0)
    got = _run(dev, qd, synth.from_torch_bf16(out["K_out"]), synth.from_torch_bf16(out["V_out"]), b)
    assert sg.sgdkv_last_error(ws) == sg.OK
    ko, vo = O.gather(inp["K"], inp["V"], out["indices"].cpu().numpy(), out["cu_seqlens"].cpu().numpy())
    _check(got, qd, ko, vo, b)


def test_decode_full_size_layer(dev):
    """The 128K-context Qwen2.5-7B layer at 25 %: the budgets the benchmark allocates for
    its last layer, every query head against the oracle."""
    wl = configs.BY_NAME["c3_qwen25_7b_L128k"]
    all_b = sg.sgdkv_allocate_budgets(synth.head_scores(wl), wl.L, wl.total_budget(0.25), wl.floor)
    b = np.asarray(all_b[(wl.n_layers - 1) * wl.Hkv: wl.n_layers * wl.Hkv], np.int64)
    q, K, V = _case(wl.Hq, wl.Hkv, 1, b, seed=77, q_scale=2.0)
    _check(_run(dev, q, K, V, b), q, K, V, b)


def test_decode_reuses_its_workspace(dev):
    """One workspace through several calls of different budgets, eager and captured into a
    CUDA graph (replayed twice): every call gives the oracle's output."""
    ws = sg.make_decode_workspace(28, 4, 1, 20000, dev)
    cases = [(28, 4, [1250, 700, 2400, 256], 1), (28, 4, [0, 5000, 3, 9000], 2),
             (28, 4, [20000, 0, 0, 0], 3)]
    for Hq, Hkv, budgets, seed in cases:
        b = np.asarray(budgets, np.int64)
        q, K, V = _case(Hq, Hkv, 1, b, seed=seed)
        qt = synth.to_torch_bf16(q, dev)
        Kt, Vt = synth.to_torch_bf16(K, dev), synth.to_torch_bf16(V, dev)
        for graph in (False, True):
            g_out = guarded((Hq, 1, 128), torch.float32, dev, fill=float("nan"))
            if graph:
                g = torch.cuda.CUDAGraph()
                with torch.cuda.graph(g):
                    sg.sgdkv_decode_attention(qt, Kt, Vt, b, g_out.t, ws)
                for _ in range(2):
                    g.replay()
            else:
                sg.sgdkv_decode_attention(qt, Kt, Vt, b, g_out.t, ws)
            torch.cuda.synchronize()
            g_out.check("decode output")
            _check(g_out.t.cpu().numpy(), q, K, V, b)
