"""GPU parity of the CUDA path against the CPU oracle, through the C-ABI.

Bars: scores |gpu - oracle| <= 1e-5 + 2e-3 |oracle| element by element; given identical
scores, indices and cu_seqlens bit-exact; gathered K/V rows bit-exact.  End to end (each
side with its own scores), the GPU's selection must equal the oracle's selection applied
to the GPU's scores, and every position where it differs from the oracle's own selection
must have an oracle score within tolerance of that head's threshold.
"""
import numpy as np
import pytest
import torch

from oracle import sgdkv_oracle as O
from paper_2609_03235_gb300 import configs, synth
from paper_2609_03235_gb300 import sgdkv as sg

from _guard import guarded, check_all

pytestmark = pytest.mark.gpu
RTOL, ATOL = 2e-3, 1e-5


@pytest.fixture(scope="module")
def dev():
    sg.lib()
    return torch.device("cuda:0")


def _within(got, exp):
    return np.abs(got.astype(np.float64) - exp) <= ATOL + RTOL * np.abs(exp.astype(np.float64))


def _upload(inp, dev):
    return (synth.to_torch_bf16(inp["q"], dev), synth.to_torch_bf16(inp["K"], dev),
            synth.to_torch_bf16(inp["V"], dev))


SCORE_SHAPES = [
    # Hq, Hkv, L, W    (G*W = 224, 448, 512, 32, 224 ...)
    (14, 2, 1000, 32),
    (28, 4, 3000, 64),
    (16, 2, 2049, 64),
    (1, 1, 300, 32),
    (7, 1, 32, 32),        # L == W: every key is a window key
    (8, 8, 640, 32),
    (28, 4, 129, 64),
    (9, 1, 1000, 32),      # G*W = 288: three row tiles, N chunks of 144 split 80 / 64
    (28, 4, 20000, 64),    # several key tiles per CTA
]


@pytest.mark.parametrize("Hq,Hkv,L,W", SCORE_SHAPES)
@pytest.mark.parametrize("pool", [1, 7, 63])
def test_score_parity(dev, Hq, Hkv, L, W, pool):
    wl = synth.tiny_workload(Hq=Hq, Hkv=Hkv, d=128, L=L, W=W, n_salient=min(8, max(0, L - W - 4)))
    inp = synth.tiny_inputs(wl, tag=200 + L)
    q, K, _ = _upload(inp, dev)
    ws = sg.make_workspace(Hq, Hkv, L, W, dev)
    out = torch.empty((Hkv, L), dtype=torch.float32, device=dev)
    sg.sgdkv_score(q, K, W, pool, out, ws)
    torch.cuda.synchronize()
    assert sg.sgdkv_last_error(ws) == sg.OK
    raw = O.window_scores(inp["q"], inp["K"])
    exp = O.max_pool(raw, pool)
    got = out.cpu().numpy()
    ok = _within(got, exp)
    assert ok.all(), f"{(~ok).sum()} of {ok.size} off; worst {np.max(np.abs(got - exp))}"


def test_score_output_not_16_byte_aligned_is_refused(dev):
    """scores_out 4 bytes past a 16-byte boundary: INVALID_ARG, nothing launched, the buffer
    untouched (the pooled scores are written with 16-byte stores)."""
    Hq, Hkv, L, W = 28, 4, 4096, 64
    wl = synth.tiny_workload(Hq=Hq, Hkv=Hkv, d=128, L=L, W=W, n_salient=8)
    inp = synth.tiny_inputs(wl, tag=77)
    q, K, _ = _upload(inp, dev)
    ws = sg.make_workspace(Hq, Hkv, L, W, dev)
    buf = torch.full((Hkv * L + 1,), float("nan"), dtype=torch.float32, device=dev)
    out = buf[1:].view(Hkv, L)
    assert out.data_ptr() % 16 == 4
    with pytest.raises(sg.SgdkvError) as e:
        sg.sgdkv_score(q, K, W, 7, out, ws)
    assert e.value.status == sg.ERR_INVALID_ARG
    torch.cuda.synchronize()
    assert torch.isnan(buf).all()


PROXY_SHAPES = [
    # Hq, Hkv, L, W    (W external query rows per query head; every row sees all L keys)
    (14, 2, 1000, 32),
    (28, 4, 3000, 64),
    (16, 2, 2049, 64),
    (1, 1, 300, 32),
    (9, 1, 1000, 32),
    (28, 4, 20000, 64),
]


@pytest.mark.parametrize("Hq,Hkv,L,W", PROXY_SHAPES)
@pytest.mark.parametrize("pool", [1, 7])
def test_proxy_query_score_parity(dev, Hq, Hkv, L, W, pool):
    """Proxy-query scoring (no causal mask) against the oracle's non-causal scores."""
    wl = synth.tiny_workload(Hq=Hq, Hkv=Hkv, d=128, L=L, W=W, n_salient=min(8, max(0, L - W - 4)))
    inp = synth.tiny_inputs(wl, tag=600 + L)
    q, K, _ = _upload(inp, dev)
    ws = sg.make_workspace(Hq, Hkv, L, W, dev)
    out = torch.empty((Hkv, L), dtype=torch.float32, device=dev)
    sg.sgdkv_score(q, K, W, pool, out, ws, flags=sg.SCORE_PROXY_QUERY)
    torch.cuda.synchronize()
    assert sg.sgdkv_last_error(ws) == sg.OK
    exp = O.max_pool(O.window_scores(inp["q"], inp["K"], causal=False), pool)
    got = out.cpu().numpy()
    ok = _within(got, exp)
    assert ok.all(), f"{(~ok).sum()} of {ok.size} off; worst {np.max(np.abs(got - exp))}"
    # every row sees every key: the raw scores of a head sum to G*W
    if pool == 1:
        assert np.allclose(got.astype(np.float64).sum(axis=1), Hq // Hkv * W, rtol=1e-4)


IPT_SHAPES = [
    # Hq, Hkv, L, W
    (14, 2, 1000, 32),     # G*W = 224: one row chunk
    (28, 4, 3000, 64),     # G*W = 448: two chunks, head 3 split across them
    (16, 2, 2049, 64),     # G = 8, G*W = 512
    (4, 4, 700, 32),       # G = 1
]
IPT_MODES = [("max", 2, "AGG_IPT_MAX"), ("mean", 4, "AGG_IPT_MEAN"), ("only", 6, "AGG_IPT_ONLY")]


def _ipt_weights(Hq, seed):
    w = np.random.default_rng(seed).random(Hq).astype(np.float32)
    w[0] = 0.0                              # a head that contributes nothing
    if Hq > 3:
        w[3] = w[2]                         # a tie (Ipt only: lower head wins)
    return w


@pytest.mark.parametrize("Hq,Hkv,L,W", IPT_SHAPES)
@pytest.mark.parametrize("mode", IPT_MODES, ids=[m[0] for m in IPT_MODES])
@pytest.mark.parametrize("proxy", [False, True])
def test_ipt_aggregation_parity(dev, Hq, Hkv, L, W, mode, proxy):
    """Summarization-weighted GQA aggregation against the oracle (appendix variants)."""
    name, flag, omode = mode
    wl = synth.tiny_workload(Hq=Hq, Hkv=Hkv, d=128, L=L, W=W, n_salient=min(8, max(0, L - W - 4)))
    inp = synth.tiny_inputs(wl, tag=700 + L)
    q, K, _ = _upload(inp, dev)
    w = _ipt_weights(Hq, L)
    ws = sg.make_workspace(Hq, Hkv, L, W, dev)
    out = torch.empty((Hkv, L), dtype=torch.float32, device=dev)
    flags = flag | (sg.SCORE_PROXY_QUERY if proxy else 0)
    sg.sgdkv_score(q, K, W, 7, out, ws, flags=flags, head_weights=torch.from_numpy(w).to(dev))
    torch.cuda.synchronize()
    assert sg.sgdkv_last_error(ws) == sg.OK
    raw = O.window_scores_ipt(inp["q"], inp["K"], w, getattr(O, omode), causal=not proxy)
    exp = O.max_pool(raw, 7)
    got = out.cpu().numpy()
    ok = _within(got, exp)
    assert ok.all(), f"{(~ok).sum()} of {ok.size} off; worst {np.max(np.abs(got - exp))}"


@pytest.mark.parametrize("flags_name", ["sum", "proxy", "ipt_max", "ipt_mean"])
def test_score_raw_then_pool_equals_score(dev, flags_name):
    """sgdkv_score_raw + sgdkv_pool_raw (pooling on a second stream) give what
    sgdkv_score_ex gives (to within the run-to-run rounding of the dynamically claimed
    row sums), and match the oracle."""
    Hq, Hkv, L, W = 28, 4, 3000, 64
    flags = {"sum": 0, "proxy": sg.SCORE_PROXY_QUERY, "ipt_max": sg.SCORE_AGG_IPT_MAX,
             "ipt_mean": sg.SCORE_AGG_IPT_MEAN}[flags_name]
    wl = synth.tiny_workload(Hq=Hq, Hkv=Hkv, d=128, L=L, W=W, n_salient=8)
    inp = synth.tiny_inputs(wl, tag=1234)
    q, K, _ = _upload(inp, dev)
    w = _ipt_weights(Hq, 5)
    hw = torch.from_numpy(w).to(dev) if flags_name.startswith("ipt") else None
    ws_one = sg.make_workspace(Hq, Hkv, L, W, dev)
    ws_two = sg.make_workspace(Hq, Hkv, L, W, dev)
    one = torch.empty((Hkv, L), dtype=torch.float32, device=dev)
    two = torch.full((Hkv, L), float("nan"), dtype=torch.float32, device=dev)
    sg.sgdkv_score(q, K, W, 7, one, ws_one, flags=flags, head_weights=hw)
    s_a = torch.cuda.current_stream(dev)
    s_b = torch.cuda.Stream(dev)
    sg.sgdkv_score_raw(q, K, W, ws_two, s_a, flags=flags, head_weights=hw)
    ev = torch.cuda.Event()
    ev.record(s_a)
    s_b.wait_event(ev)
    sg.sgdkv_pool_raw(ws_two, Hkv, L, 7, two, s_b, flags=flags)
    torch.cuda.synchronize()
    assert sg.sgdkv_last_error(ws_one) == sg.OK and sg.sgdkv_last_error(ws_two) == sg.OK
    torch.testing.assert_close(two, one, rtol=1e-5, atol=1e-9)
    if flags_name.startswith("ipt"):
        omode = O.AGG_IPT_MAX if flags_name == "ipt_max" else O.AGG_IPT_MEAN
        raw = O.window_scores_ipt(inp["q"], inp["K"], w, omode, causal=True)
    else:
        raw = O.window_scores(inp["q"], inp["K"], causal=flags_name == "sum")
    exp = O.max_pool(raw, 7)
    got = two.cpu().numpy()
    ok = _within(got, exp)
    assert ok.all(), f"{(~ok).sum()} of {ok.size} off; worst {np.max(np.abs(got - exp))}"


@pytest.mark.parametrize("flags_name", ["sum", "proxy", "ipt_max"])
def test_window_stats_then_sums_two_layers_in_flight(dev, flags_name):
    """sgdkv_window_stats / sgdkv_window_sums / sgdkv_pool_raw as separate calls, two
    layers in flight on two streams (layer 1's statistics beside layer 0's sums, one
    workspace each), against the oracle."""
    Hq, Hkv, L, W = 28, 4, 3000, 64
    flags = {"sum": 0, "proxy": sg.SCORE_PROXY_QUERY, "ipt_max": sg.SCORE_AGG_IPT_MAX}[flags_name]
    wl = synth.tiny_workload(Hq=Hq, Hkv=Hkv, d=128, L=L, W=W, n_salient=8)
    w = _ipt_weights(Hq, 11)
    hw = torch.from_numpy(w).to(dev) if flags_name == "ipt_max" else None
    s_a, s_b = torch.cuda.current_stream(dev), torch.cuda.Stream(dev)
    layers = []
    for tag in (501, 502):
        inp = synth.tiny_inputs(wl, tag=tag)
        q, K, _ = _upload(inp, dev)
        layers.append((inp, q, K, sg.make_workspace(Hq, Hkv, L, W, dev),
                       torch.full((Hkv, L), float("nan"), dtype=torch.float32, device=dev)))
    torch.cuda.synchronize()
    for inp, q, K, ws, out in layers:
        sg.sgdkv_window_stats(q, K, W, ws, s_a, flags=flags, head_weights=hw)
        ev = torch.cuda.Event()
        ev.record(s_a)
        s_b.wait_event(ev)
        sg.sgdkv_window_sums(q, K, W, ws, s_b, flags=flags, head_weights=hw)
        sg.sgdkv_pool_raw(ws, Hkv, L, 7, out, s_b, flags=flags)
    torch.cuda.synchronize()
    for inp, q, K, ws, out in layers:
        assert sg.sgdkv_last_error(ws) == sg.OK
        if flags_name == "ipt_max":
            raw = O.window_scores_ipt(inp["q"], inp["K"], w, O.AGG_IPT_MAX, causal=True)
        else:
            raw = O.window_scores(inp["q"], inp["K"], causal=flags_name == "sum")
        exp = O.max_pool(raw, 7)
        got = out.cpu().numpy()
        ok = _within(got, exp)
        assert ok.all(), f"{(~ok).sum()} of {ok.size} off; worst {np.max(np.abs(got - exp))}"


def test_ipt_negative_weight_is_reported(dev):
    wl = synth.tiny_workload(Hq=14, Hkv=2, d=128, L=500, W=32, n_salient=4)
    inp = synth.tiny_inputs(wl, tag=799)
    q, K, _ = _upload(inp, dev)
    w = np.ones(14, np.float32)
    w[5] = -1.0
    ws = sg.make_workspace(14, 2, 500, 32, dev)
    out = torch.empty((2, 500), dtype=torch.float32, device=dev)
    sg.sgdkv_score(q, K, 32, 7, out, ws, flags=sg.SCORE_AGG_IPT_MEAN,
                   head_weights=torch.from_numpy(w).to(dev))
    torch.cuda.synchronize()
    assert sg.sgdkv_last_error(ws) == sg.ERR_INVALID_ARG
    assert sg.sgdkv_last_error(ws) == sg.OK                   # reading clears it


def _tie_heavy_scores(rng, Hkv, L):
    return (rng.integers(0, 6, size=(Hkv, L)) * 0.125).astype(np.float32)


COMPACT_CASES = [
    # Hkv, L, n_sink, n_recent, budget rule
    (4, 4096, 64, 64, "quarter"),
    (2, 1000, 16, 16, "random"),
    (3, 777, 0, 0, "random"),
    (2, 300, 150, 150, "all"),        # no middle at all
    (2, 5000, 10, 20, "floor"),       # nothing selected from the middle
    (2, 5000, 10, 20, "full"),        # the whole middle selected
    (5, 9000, 100, 28, "random"),     # several selection chunks, ragged tail
    (1, 1, 0, 0, "full"),
    (2, 200000, 64, 64, "random"),    # 16 positions per thread
    (1, 600000, 64, 64, "random"),    # streaming selection: several ordered-write rounds
    (8, 5000, 16, 16, "random"),      # 8 x 16 CTAs: the selection copies the rows itself
    (12, 3001, 0, 32, "quarter"),     # the same, ragged slices
    (3, 80000, 64, 64, "random"),     # 10-CTA clusters (the smallest that holds 8 a thread)
    (2, 100001, 32, 32, "quarter"),   # 13-CTA clusters, ragged last slice
    (13, 80000, 16, 16, "random"),    # 13 x 10 CTAs: rows copied inside the selection kernel
]


def _budgets_for(rule, rng, Hkv, L, n_sink, n_recent):
    lo, hi = n_sink + n_recent, L
    if rule == "quarter":
        return np.full(Hkv, max(lo, L // 4), np.int64)
    if rule == "all" or rule == "full":
        return np.full(Hkv, hi, np.int64)
    if rule == "floor":
        return np.full(Hkv, lo, np.int64)
    return rng.integers(lo, hi + 1, size=Hkv).astype(np.int64)


@pytest.mark.parametrize("Hkv,L,n_sink,n_recent,rule", COMPACT_CASES)
@pytest.mark.parametrize("ties", [False, True])
def test_compact_parity_identical_scores(dev, Hkv, L, n_sink, n_recent, rule, ties):
    rng = np.random.default_rng(L * 7 + Hkv + int(ties))
    scores = _tie_heavy_scores(rng, Hkv, L) if ties else rng.random((Hkv, L)).astype(np.float32)
    K = synth.bf16_round(rng.standard_normal((Hkv, L, 128), dtype=np.float32))
    V = synth.bf16_round(rng.standard_normal((Hkv, L, 128), dtype=np.float32))
    b = _budgets_for(rule, rng, Hkv, L, n_sink, n_recent)
    total = int(b.sum())
    ws = sg.make_workspace(Hkv, Hkv, L, 32, dev) if L >= 32 else sg.make_workspace(1, 1, 32, 32, dev)
    Kt, Vt = synth.to_torch_bf16(K, dev), synth.to_torch_bf16(V, dev)
    st = torch.from_numpy(scores).to(dev)
    g_idx = guarded((total,), torch.int32, dev, fill=-1)
    g_cu = guarded((Hkv + 1,), torch.int32, dev, fill=-1)
    g_ko = guarded((total, 128), torch.bfloat16, dev, fill=0)
    g_vo = guarded((total, 128), torch.bfloat16, dev, fill=0)
    idx, cu, ko, vo = g_idx.t, g_cu.t, g_ko.t, g_vo.t
    for _ in range(2):       # the same workspace twice in a row
        sg.sgdkv_compact(Kt, Vt, st, b, n_sink, n_recent, idx, cu, ko, vo, ws)
        torch.cuda.synchronize()
        assert sg.sgdkv_last_error(ws) == sg.OK
        check_all(g_idx, g_cu, g_ko, g_vo)
        e_idx, e_cu = O.select_indices(scores, b, n_sink, n_recent)
        assert np.array_equal(cu.cpu().numpy(), e_cu)
        assert np.array_equal(idx.cpu().numpy(), e_idx)
        e_ko, e_vo = O.gather(K, V, e_idx, e_cu)
        assert np.array_equal(synth.from_torch_bf16(ko), e_ko)
        assert np.array_equal(synth.from_torch_bf16(vo), e_vo)


def test_compact_negative_zero_scores_count_as_zero(dev):
    """-0.0 compares equal to +0.0: a row of zeros with some -0.0 keeps the lowest middle
    positions, as the oracle's (score desc, position asc) order does."""
    Hkv, L = 2, 5000
    rng = np.random.default_rng(3)
    scores = np.zeros((Hkv, L), np.float32)
    scores[:, rng.choice(L, 400, replace=False)] = np.float32(-0.0)
    scores[1, rng.choice(L, 50, replace=False)] = 0.5
    K = synth.bf16_round(rng.standard_normal((Hkv, L, 128), dtype=np.float32))
    V = synth.bf16_round(rng.standard_normal((Hkv, L, 128), dtype=np.float32))
    b = np.array([300, 200], np.int64)
    total = int(b.sum())
    ws = sg.make_workspace(Hkv, Hkv, L, 32, dev)
    g_idx = guarded((total,), torch.int32, dev, fill=-1)
    g_cu = guarded((Hkv + 1,), torch.int32, dev, fill=-1)
    g_ko = guarded((total, 128), torch.bfloat16, dev, fill=0)
    g_vo = guarded((total, 128), torch.bfloat16, dev, fill=0)
    sg.sgdkv_compact(synth.to_torch_bf16(K, dev), synth.to_torch_bf16(V, dev),
                     torch.from_numpy(scores).to(dev), b, 16, 16, g_idx.t, g_cu.t, g_ko.t,
                     g_vo.t, ws)
    torch.cuda.synchronize()
    assert sg.sgdkv_last_error(ws) == sg.OK
    check_all(g_idx, g_cu, g_ko, g_vo)
    e_idx, e_cu = O.select_indices(scores, b, 16, 16)
    assert np.array_equal(g_cu.t.cpu().numpy(), e_cu)
    assert np.array_equal(g_idx.t.cpu().numpy(), e_idx)
    assert np.array_equal(e_idx[:b[0]], np.concatenate([np.arange(300 - 16), np.arange(L - 16, L)]))


def _check_end_to_end(inp, out, budgets, n_sink, n_recent, pool, raw=None):
    if raw is None:
        raw = O.window_scores(inp["q"], inp["K"])
    exp = O.max_pool(raw, pool) if pool > 1 else raw
    got = out["scores"].cpu().numpy()
    ok = _within(got, exp)
    assert ok.all(), f"{(~ok).sum()} scores off; worst {np.max(np.abs(got - exp))}"
    g_idx = out["indices"].cpu().numpy()
    g_cu = out["cu_seqlens"].cpu().numpy()
    s_idx, s_cu = O.select_indices(got, budgets, n_sink, n_recent)
    assert np.array_equal(g_cu, s_cu)
    assert np.array_equal(g_idx, s_idx)
    o_idx, o_cu = O.select_indices(exp, budgets, n_sink, n_recent)
    for h in range(len(budgets)):
        a = set(g_idx[g_cu[h]:g_cu[h + 1]].tolist())
        b = set(o_idx[o_cu[h]:o_cu[h + 1]].tolist())
        diff = np.array(sorted(a ^ b), dtype=np.int64)
        if diff.size:
            kept = np.array(sorted(b - set(range(n_sink)) - set(range(len(exp[h]) - n_recent,
                                                                      len(exp[h])))))
            tau = exp[h, kept].min() if kept.size else 0.0
            assert np.all(np.abs(exp[h, diff] - tau) <= ATOL + RTOL * abs(tau))
    ko, vo = O.gather(inp["K"], inp["V"], g_idx, g_cu)
    assert np.array_equal(synth.from_torch_bf16(out["K_out"]), ko)
    assert np.array_equal(synth.from_torch_bf16(out["V_out"]), vo)


POOL_COMPACT_CASES = [
    # Hq, Hkv, L, W, pool, flags      (path inside the selection kernel)
    (28, 4, 3000, 64, 7, "sum"),      # 16-byte plane loads, register window
    (14, 2, 3001, 32, 7, "sum"),      # L % 4 != 0: scalar plane loads, ragged last slice
    (16, 2, 2049, 64, 9, "proxy"),    # radius 4: window maxima from shared memory
    (9, 1, 1000, 32, 63, "sum"),      # radius 31 (largest), halo wider than some slices
    (7, 1, 40, 32, 7, "sum"),         # slices of 3 positions, most threads hold none
    (28, 4, 3000, 64, 7, "ipt_max"),  # planes combined by max
    (28, 4, 20000, 64, 1, "sum"),     # no pooling (radius 0)
    (2, 1, 300000, 16, 7, "sum"),     # 32 positions per thread
    (2, 1, 600000, 16, 7, "sum"),     # rows too long for register slices: two kernels
    (64, 8, 3000, 32, 7, "sum"),      # 8 KV heads: rows copied inside the selection kernel
    (28, 4, 72000, 64, 7, "sum"),     # 9-CTA clusters
]


@pytest.mark.parametrize("Hq,Hkv,L,W,pool,flags_name", POOL_COMPACT_CASES)
def test_pool_compact_equals_pool_then_compact(dev, Hq, Hkv, L, W, pool, flags_name):
    """sgdkv_pool_compact (the max-pool inside the selection kernel) writes the pooled
    scores bit for bit as sgdkv_pool_raw does and keeps what sgdkv_compact keeps on them;
    both match the oracle."""
    flags = {"sum": 0, "proxy": sg.SCORE_PROXY_QUERY, "ipt_max": sg.SCORE_AGG_IPT_MAX}[flags_name]
    wl = synth.tiny_workload(Hq=Hq, Hkv=Hkv, d=128, L=L, W=W, n_salient=8)
    inp = synth.tiny_inputs(wl, tag=4321 + L)
    q, K, V = _upload(inp, dev)
    w = _ipt_weights(Hq, 11)
    hw = torch.from_numpy(w).to(dev) if flags_name == "ipt_max" else None
    n_sink, n_recent = min(16, L // 4), min(16, L // 4)
    rng = np.random.default_rng(L + Hkv)
    b = rng.integers(n_sink + n_recent, L + 1, size=Hkv).astype(np.int64)
    total = int(b.sum())
    ws = sg.make_workspace(Hq, Hkv, L, W, dev)
    ws_sel = sg.make_workspace(Hq, Hkv, L, W, dev)
    sg.sgdkv_score_raw(q, K, W, ws, flags=flags, head_weights=hw)

    guards = []

    def outs():
        gs = dict(scores=guarded((Hkv, L), torch.float32, dev, fill=float("nan")),
                  idx=guarded((total,), torch.int32, dev, fill=-1),
                  cu=guarded((Hkv + 1,), torch.int32, dev, fill=-1),
                  ko=guarded((total, 128), torch.bfloat16, dev, fill=0),
                  vo=guarded((total, 128), torch.bfloat16, dev, fill=0))
        guards.extend(gs.values())
        return {k: g.t for k, g in gs.items()}
    a, f = outs(), outs()
    sg.sgdkv_pool_raw(ws, Hkv, L, pool, a["scores"], flags=flags)
    sg.sgdkv_compact(K, V, a["scores"], b, n_sink, n_recent, a["idx"], a["cu"], a["ko"],
                     a["vo"], ws_sel)
    sg.sgdkv_pool_compact(ws, pool, K, V, b, n_sink, n_recent, f["scores"], f["idx"], f["cu"],
                          f["ko"], f["vo"], ws_sel, flags=flags)
    torch.cuda.synchronize()
    assert sg.sgdkv_last_error(ws) == sg.OK and sg.sgdkv_last_error(ws_sel) == sg.OK
    check_all(*guards)
    for k in a:
        if a[k].dtype == torch.bfloat16:
            assert torch.equal(a[k].view(torch.int16), f[k].view(torch.int16)), k
        else:
            assert torch.equal(a[k].view(torch.int32), f[k].view(torch.int32)), k
    if flags_name == "ipt_max":
        raw = O.window_scores_ipt(inp["q"], inp["K"], w, O.AGG_IPT_MAX, causal=True)
    else:
        raw = O.window_scores(inp["q"], inp["K"], causal=flags_name == "sum")
    exp = O.max_pool(raw, pool) if pool > 1 else raw
    got = f["scores"].cpu().numpy()
    ok = _within(got, exp)
    assert ok.all(), f"{(~ok).sum()} of {ok.size} off; worst {np.max(np.abs(got - exp))}"
    e_idx, e_cu = O.select_indices(got, b, n_sink, n_recent)
    assert np.array_equal(f["cu"].cpu().numpy(), e_cu)
    assert np.array_equal(f["idx"].cpu().numpy(), e_idx)
    e_ko, e_vo = O.gather(inp["K"], inp["V"], e_idx, e_cu)
    assert np.array_equal(synth.from_torch_bf16(f["ko"]), e_ko)
    assert np.array_equal(synth.from_torch_bf16(f["vo"]), e_vo)


def test_compress_layer_small(dev):
    wl = synth.tiny_workload(Hq=28, Hkv=4, d=128, L=5000, W=64, n_salient=32, floor=256)
    inp = synth.tiny_inputs(wl, tag=300)
    q, K, V = _upload(inp, dev)
    b = np.array([1250, 700, 2400, 256], np.int64)
    ws = sg.make_workspace(wl.Hq, wl.Hkv, wl.L, wl.W, dev)
    out = sg.compress_layer_alloc(q, K, V, b, wl.W, 7, 128, 128, ws)
    torch.cuda.synchronize()
    assert sg.sgdkv_last_error(ws) == sg.OK
    _check_end_to_end(inp, out, b, 128, 128, 7)


def _compress_guarded(q, K, V, b, W, pool, n_sink, n_recent, ws, stream=None):
    """sgdkv_compress_layer into outputs with guard bands; returns (outputs, guards)."""
    Hkv, L, d = K.shape
    total = int(np.sum(b))
    dev = K.device
    gs = dict(scores=guarded((Hkv, L), torch.float32, dev, fill=float("nan")),
              indices=guarded((total,), torch.int32, dev, fill=-1),
              cu_seqlens=guarded((Hkv + 1,), torch.int32, dev, fill=-1),
              K_out=guarded((total, d), torch.bfloat16, dev, fill=0),
              V_out=guarded((total, d), torch.bfloat16, dev, fill=0))
    out = {k: g.t for k, g in gs.items()}
    sg.sgdkv_compress_layer(q, K, V, b, W, pool, n_sink, n_recent, out["scores"],
                            out["indices"], out["cu_seqlens"], out["K_out"], out["V_out"], ws,
                            stream)
    return out, list(gs.values())


FULL_SIZE_CASES = [(w.name, f) for w in configs.WORKLOADS for f in w.budget_fracs]
_ORACLE_RAW = {}          # the oracle's raw window scores of one full-size layer, by workload


@pytest.mark.parametrize("name,frac", FULL_SIZE_CASES,
                         ids=[f"{n}-{f}" for n, f in FULL_SIZE_CASES])
def test_full_size_layer(dev, name, frac):
    """One layer of each workload at full size, at every total budget the workload is
    measured with (the 128K Qwen2.5-7B shape at 12.5, 25 and 50 %), in the launch
    configuration the benchmark times (sgdkv_compress_layer with the model-wide greedy
    allocation); every output inside guard bands."""
    wl = configs.BY_NAME[name]
    layer = wl.n_layers - 1
    inp = synth.layer_inputs_host(wl, layer)
    all_b = sg.sgdkv_allocate_budgets(synth.head_scores(wl), wl.L, wl.total_budget(frac), wl.floor)
    assert int(all_b.sum()) == wl.total_budget(frac)
    b = all_b[layer * wl.Hkv:(layer + 1) * wl.Hkv]
    n_sink, n_recent = configs.sink_recent_split(wl.floor)
    q, K, V = _upload(inp, dev)
    ws = sg.make_workspace(wl.Hq, wl.Hkv, wl.L, wl.W, dev)
    out, guards = _compress_guarded(q, K, V, b, wl.W, wl.pool, n_sink, n_recent, ws)
    torch.cuda.synchronize()
    assert sg.sgdkv_last_error(ws) == sg.OK
    check_all(*guards)
    if name not in _ORACLE_RAW:
        _ORACLE_RAW.clear()
        _ORACLE_RAW[name] = O.window_scores(inp["q"], inp["K"])
    _check_end_to_end(inp, out, b, n_sink, n_recent, wl.pool, raw=_ORACLE_RAW[name])
    # planted keys (4 sinks + salient) survive whenever the middle budget has room
    g_idx, g_cu = out["indices"].cpu().numpy(), out["cu_seqlens"].cpu().numpy()
    for h in range(wl.Hkv):
        if b[h] - wl.floor >= 7 * len(inp["planted"][h]):
            kept = set(g_idx[g_cu[h]:g_cu[h + 1]].tolist())
            assert set(inp["planted"][h].tolist()) <= kept


def test_rejects_misaligned_pointer(dev):
    wl = synth.tiny_workload(Hq=14, Hkv=2, L=512, W=32)
    inp = synth.tiny_inputs(wl)
    q, K, _ = _upload(inp, dev)
    ws = sg.make_workspace(wl.Hq, wl.Hkv, wl.L, wl.W, dev)
    big = torch.empty(2 * 512 + 1, dtype=torch.float32, device=dev)
    with pytest.raises(sg.SgdkvError) as e:
        sg.sgdkv_score(q, K, wl.W, 7, big[1:], ws)
    assert e.value.status == sg.ERR_INVALID_ARG


SCHED_BYTES = (1024, 2048)     # the scorer's key-tile counters inside the workspace


def test_tile_counters_return_to_zero(dev):
    """Every scoring pass claims key tiles from per-head counters in the workspace; the
    last CTA of each head resets them, so the next call (any shape) starts from zero."""
    for Hq, Hkv, L, W in [(28, 4, 20000, 64), (14, 2, 1000, 32), (8, 8, 640, 32)]:
        wl = synth.tiny_workload(Hq=Hq, Hkv=Hkv, d=128, L=L, W=W, n_salient=4)
        inp = synth.tiny_inputs(wl, tag=400 + L)
        q, K, _ = _upload(inp, dev)
        ws = sg.make_workspace(Hq, Hkv, L, W, dev)
        out = torch.empty((Hkv, L), dtype=torch.float32, device=dev)
        for _ in range(3):
            sg.sgdkv_score(q, K, W, 7, out, ws)
        torch.cuda.synchronize()
        assert sg.sgdkv_last_error(ws) == sg.OK
        assert int(ws[SCHED_BYTES[0]:SCHED_BYTES[1]].count_nonzero()) == 0
        exp = O.max_pool(O.window_scores(inp["q"], inp["K"]), 7)
        assert _within(out.cpu().numpy(), exp).all()


def test_layers_on_two_streams(dev):
    """Two layers scored and compacted at the same time on two streams (one workspace
    each), as the benchmark overlaps consecutive layers: each matches the oracle."""
    wl = synth.tiny_workload(Hq=28, Hkv=4, d=128, L=6000, W=64, n_salient=16, floor=256)
    b = np.array([1500, 700, 2400, 256], np.int64)
    streams = [torch.cuda.Stream(dev), torch.cuda.Stream(dev)]
    runs = []
    for i, s in enumerate(streams):
        inp = synth.tiny_inputs(wl, tag=500 + i)
        q, K, V = _upload(inp, dev)
        ws = sg.make_workspace(wl.Hq, wl.Hkv, wl.L, wl.W, dev)
        runs.append((inp, q, K, V, ws, s))
    torch.cuda.synchronize()
    outs = []
    for inp, q, K, V, ws, s in runs:
        with torch.cuda.stream(s):
            outs.append(sg.compress_layer_alloc(q, K, V, b, wl.W, 7, 128, 128, ws, stream=s))
    torch.cuda.synchronize()
    for (inp, q, K, V, ws, s), out in zip(runs, outs):
        assert sg.sgdkv_last_error(ws) == sg.OK
        _check_end_to_end(inp, out, b, 128, 128, 7)


@pytest.mark.parametrize("Hkv", [3, 8])
def test_compact_reads_kv_from_pinned_host_memory(dev, Hkv):
    """K and V of sgdkv_compact (and V of sgdkv_compress_layer) may be pinned host memory:
    the kept rows are read across the host link (by the gather kernel with 3 KV heads, by
    the selection kernel itself with 8); outputs bit-exact."""
    rng = np.random.default_rng(11 + Hkv)
    L = 3000
    scores = rng.random((Hkv, L)).astype(np.float32)
    K = synth.bf16_round(rng.standard_normal((Hkv, L, 128), dtype=np.float32))
    V = synth.bf16_round(rng.standard_normal((Hkv, L, 128), dtype=np.float32))
    b = np.array(([700, 64, 3000] * 3)[:Hkv], np.int64)
    total = int(b.sum())
    Kh = synth.to_torch_bf16(K, "cpu").pin_memory()
    Vh = synth.to_torch_bf16(V, "cpu").pin_memory()
    ws = sg.make_workspace(Hkv, Hkv, L, 32, dev)
    st = torch.from_numpy(scores).to(dev)
    idx = torch.empty(total, dtype=torch.int32, device=dev)
    cu = torch.empty(Hkv + 1, dtype=torch.int32, device=dev)
    ko = torch.empty((total, 128), dtype=torch.bfloat16, device=dev)
    vo = torch.empty((total, 128), dtype=torch.bfloat16, device=dev)
    sg.sgdkv_compact(Kh, Vh, st, b, 16, 16, idx, cu, ko, vo, ws)
    torch.cuda.synchronize()
    assert sg.sgdkv_last_error(ws) == sg.OK
    e_idx, e_cu = O.select_indices(scores, b, 16, 16)
    assert np.array_equal(idx.cpu().numpy(), e_idx)
    e_ko, e_vo = O.gather(K, V, e_idx, e_cu)
    assert np.array_equal(synth.from_torch_bf16(ko), e_ko)
    assert np.array_equal(synth.from_torch_bf16(vo), e_vo)

    # compress_layer: K on the device, V in pinned host memory
    wl = synth.tiny_workload(Hq=28, Hkv=4, d=128, L=5000, W=64, n_salient=32, floor=256)
    inp = synth.tiny_inputs(wl, tag=301)
    q, Kd, _ = _upload(inp, dev)
    Vh = synth.to_torch_bf16(inp["V"], "cpu").pin_memory()
    b = np.array([1250, 700, 2400, 256], np.int64)
    ws = sg.make_workspace(wl.Hq, wl.Hkv, wl.L, wl.W, dev)
    out = sg.compress_layer_alloc(q, Kd, Vh, b, wl.W, 7, 128, 128, ws)
    torch.cuda.synchronize()
    assert sg.sgdkv_last_error(ws) == sg.OK
    _check_end_to_end(inp, out, b, 128, 128, 7)


@pytest.mark.parametrize("graph", [False, True])
def test_bench_launch_configuration_full_size(dev, graph):
    """The schedule bench.py times, at full size: consecutive layers of the 128K-context
    Qwen2.5-7B workload, the scoring passes on one stream (two alternating workspaces) and
    sgdkv_pool_compact (max-pool inside the selection kernel, then the gather) on a second
    (layer l's pooling and compaction overlapping layer l+1's scoring, layer l+2's scoring
    waiting for layer l's compaction), launched directly or captured into a CUDA graph and
    replayed (bench.py's timed steps); every layer end to end against the oracle."""
    wl = configs.BY_NAME["c3_qwen25_7b_L128k"]
    n_sink, n_recent = configs.sink_recent_split(wl.floor)
    all_b = sg.sgdkv_allocate_budgets(synth.head_scores(wl), wl.L, wl.total_budget(0.25), wl.floor)
    layers = [0, 1, wl.n_layers - 1]
    ws_a = [sg.make_workspace(wl.Hq, wl.Hkv, wl.L, wl.W, dev) for _ in range(2)]
    ws_b = sg.make_workspace(wl.Hq, wl.Hkv, wl.L, wl.W, dev)
    stream_a = torch.cuda.current_stream(dev)
    stream_b = torch.cuda.Stream(dev)
    runs = []
    for layer in layers:
        inp = synth.layer_inputs_host(wl, layer)
        q, K, V = _upload(inp, dev)
        b = all_b[layer * wl.Hkv:(layer + 1) * wl.Hkv]
        tot = int(b.sum())
        out = dict(scores=torch.empty((wl.Hkv, wl.L), dtype=torch.float32, device=dev),
                   indices=torch.empty(tot, dtype=torch.int32, device=dev),
                   cu_seqlens=torch.empty(wl.Hkv + 1, dtype=torch.int32, device=dev),
                   K_out=torch.empty((tot, wl.d), dtype=torch.bfloat16, device=dev),
                   V_out=torch.empty((tot, wl.d), dtype=torch.bfloat16, device=dev))
        runs.append((inp, q, K, V, b, out))
    torch.cuda.synchronize()

    def launches(sa):
        fork = torch.cuda.Event()
        fork.record(sa)
        stream_b.wait_event(fork)
        pooled = []
        for i, (inp, q, K, V, b, out) in enumerate(runs):
            if i >= 2:
                sa.wait_event(pooled[i - 2])
            sg.sgdkv_score_raw(q, K, wl.W, ws_a[i % 2], sa)
            ev = torch.cuda.Event()
            ev.record(sa)
            stream_b.wait_event(ev)
            sg.sgdkv_pool_compact(ws_a[i % 2], wl.pool, K, V, b, n_sink, n_recent,
                                  out["scores"], out["indices"], out["cu_seqlens"],
                                  out["K_out"], out["V_out"], ws_b, stream_b)
            pooled.append(torch.cuda.Event())
            pooled[-1].record(stream_b)
        done = torch.cuda.Event()
        done.record(stream_b)
        sa.wait_event(done)

    if graph:
        launches(stream_a)                       # first-use setup outside the capture
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            launches(torch.cuda.current_stream(dev))
        for inp, q, K, V, b, out in runs:        # the replay must write every output again
            out["scores"].fill_(float("nan"))
            out["indices"].fill_(-1)
            out["cu_seqlens"].fill_(-1)
            out["K_out"].zero_()
            out["V_out"].zero_()
        g.replay()
    else:
        launches(stream_a)
    torch.cuda.synchronize()
    assert all(sg.sgdkv_last_error(w) == sg.OK for w in ws_a)
    assert sg.sgdkv_last_error(ws_b) == sg.OK
    for inp, q, K, V, b, out in runs:
        _check_end_to_end(inp, out, b, n_sink, n_recent, wl.pool)
