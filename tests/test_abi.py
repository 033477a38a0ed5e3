"""Host-side checks of libsgdkv (no GPU needed): the library loads, exports every entry
point declared in include/sgdkv.h, its host allocator equals the oracle bit for bit, and
argument checks reject bad calls before any device work."""
import os
import re

import numpy as np
import pytest

from oracle import sgdkv_oracle as O
from paper_2609_03235_gb300 import sgdkv as sg

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module", autouse=True)
def built_library():
    if not os.path.exists(sg.LIB_PATH):
        from paper_2609_03235_gb300 import build_lib
        build_lib.build()
    return sg.lib()


def _declared_symbols():
    text = open(os.path.join(ROOT, "include", "sgdkv.h")).read()
    return sorted(set(re.findall(r"SGDKV_API[^;]*?\b(sgdkv_\w+)\s*\(", text, re.S)))


def test_exports_every_declared_symbol():
    import ctypes
    declared = _declared_symbols()
    assert set(declared) == set(sg.EXPORTED)
    handle = ctypes.CDLL(sg.LIB_PATH)
    for name in declared:
        assert hasattr(handle, name), name


def test_status_strings_and_version():
    assert sg.status_string(sg.OK) == "ok"
    assert "timed out" in sg.status_string(sg.ERR_TIMEOUT)
    assert sg.status_string(999) == "unknown status"
    assert sg.sgdkv_version() >= 100


def _random_alloc_case(rng):
    n = int(rng.integers(1, 700))
    dist = rng.integers(0, 3)
    if dist == 0:
        s = rng.beta(0.5, 2.0, n)
    elif dist == 1:
        s = rng.random(n)
    else:
        s = rng.integers(0, 3, n) * 0.5        # many exact ties, some zeros
    s = s.astype(np.float32)
    C = int(rng.integers(16, 1 << 21))
    f = int(rng.integers(0, C // 2 + 1))
    T = int(rng.integers(n * f, n * C + 1))
    return s, C, T, f


@pytest.mark.parametrize("mode", [sg.ALLOC_GREEDY, sg.ALLOC_PROPORTIONAL, sg.ALLOC_THRESHOLD,
                                  sg.ALLOC_REVERSE])
def test_allocator_bit_exact_vs_oracle(mode):
    rng = np.random.default_rng(2024 + mode)
    for _ in range(150):
        s, C, T, f = _random_alloc_case(rng)
        got = sg.sgdkv_allocate_budgets(s, C, T, f, mode)
        exp = O.allocate_budgets(s, C, T, f, mode)
        assert np.array_equal(got, exp), (s[:8], C, T, f, mode)


def test_allocator_on_workload_head_scores():
    from paper_2609_03235_gb300 import configs, synth
    for wl in configs.WORKLOADS:
        s = synth.head_scores(wl)
        for frac in wl.budget_fracs:
            T = wl.total_budget(frac)
            got = sg.sgdkv_allocate_budgets(s, wl.L, T, wl.floor)
            assert np.array_equal(got, O.allocate_budgets(s, wl.L, T, wl.floor))
            assert got.sum() == T


@pytest.mark.parametrize("args,status", [
    ((np.array([1.0, -1.0], np.float32), 100, 120, 10), sg.ERR_INVALID_ARG),
    ((np.array([1.0, np.nan], np.float32), 100, 120, 10), sg.ERR_INVALID_ARG),
    ((np.array([1.0, 1.0], np.float32), 100, 19, 10), sg.ERR_INFEASIBLE_BUDGET),
    ((np.array([1.0, 1.0], np.float32), 100, 201, 10), sg.ERR_INFEASIBLE_BUDGET),
    ((np.array([1.0, 1.0], np.float32), 100, 150, 101), sg.ERR_INVALID_ARG),
])
def test_allocator_errors(args, status):
    with pytest.raises(sg.SgdkvError) as e:
        sg.sgdkv_allocate_budgets(*args)
    assert e.value.status == status


def test_mix_head_scores_bit_exact_vs_oracle():
    rng = np.random.default_rng(77)
    for _ in range(100):
        n = int(rng.integers(1, 300))
        a = (rng.gamma(0.6, size=n) * rng.choice([1e-3, 1.0, 1e3])).astype(np.float32)
        b = (rng.gamma(0.6, size=n) * rng.choice([1e-3, 1.0, 1e3])).astype(np.float32)
        if rng.random() < 0.1:
            b[:] = 0.0
        np.testing.assert_array_equal(sg.sgdkv_mix_head_scores(a, b), O.mix_head_scores(a, b))
    # the mixed scores drive the allocator like any other head scores
    a = rng.gamma(0.6, size=112).astype(np.float32)
    b = rng.gamma(0.6, size=112).astype(np.float32)
    mix = sg.sgdkv_mix_head_scores(a, b)
    np.testing.assert_array_equal(sg.sgdkv_allocate_budgets(mix, 4096, 112 * 1024, 256),
                                  O.allocate_budgets(O.mix_head_scores(a, b), 4096, 112 * 1024, 256))


@pytest.mark.parametrize("a,b", [([1.0, -1.0], [1.0, 1.0]), ([1.0, 1.0], [np.inf, 1.0]),
                                 ([np.nan, 1.0], [1.0, 1.0])])
def test_mix_head_scores_errors(a, b):
    with pytest.raises(sg.SgdkvError) as e:
        sg.sgdkv_mix_head_scores(np.float32(a), np.float32(b))
    assert e.value.status == sg.ERR_INVALID_ARG


def test_allocator_bad_mode():
    with pytest.raises(sg.SgdkvError):
        sg.sgdkv_allocate_budgets(np.ones(3, np.float32), 100, 150, 10, mode=7)


def test_workspace_bytes_limits():
    assert sg.sgdkv_workspace_bytes(28, 4, 131072, 128, 64) > 4 * 131072 * 4
    assert sg.sgdkv_workspace_bytes(28, 4, 131072, 64, 64) == 0        # d != 128
    assert sg.sgdkv_workspace_bytes(28, 5, 1000, 128, 32) == 0         # Hq % Hkv != 0
    assert sg.sgdkv_workspace_bytes(28, 4, 1000, 128, 80) == 0         # G*W > 512
    assert sg.sgdkv_workspace_bytes(28, 4, 1000, 128, 12) == 0         # G*W % 32 != 0
    assert sg.sgdkv_workspace_bytes(28, 4, 10, 128, 32) == 0           # W > L


def test_score_rejects_bad_args_before_device_work():
    import ctypes
    L = sg.lib()
    buf = (ctypes.c_uint8 * 4096)()
    p = ctypes.cast(buf, ctypes.c_void_p)
    # null pointers
    assert L.sgdkv_score(None, p, 28, 4, 1024, 128, 32, 7, p, p, 4096, None) == sg.ERR_INVALID_ARG
    # unsupported head dim
    assert L.sgdkv_score(p, p, 28, 4, 1024, 64, 32, 7, p, p, 1 << 30, None) == sg.ERR_UNSUPPORTED
    # even pool kernel
    assert L.sgdkv_score(p, p, 28, 4, 1024, 128, 32, 6, p, p, 1 << 30, None) == sg.ERR_INVALID_ARG
    # workspace too small
    assert L.sgdkv_score(p, p, 28, 4, 1024, 128, 32, 7, p, p, 16, None) == sg.ERR_WORKSPACE
    # sgdkv_score_ex: unknown flag bits, an IPT mode without weights, unsupported IPT max
    # shapes, then the same checks as sgdkv_score
    ex = L.sgdkv_score_ex
    assert ex(p, p, 28, 4, 1024, 128, 32, 7, 16, None, p, p, 1 << 30, None) == sg.ERR_INVALID_ARG
    assert ex(p, p, 28, 4, 1024, 128, 32, 7, 1 << 31, None, p, p, 1 << 30, None) == sg.ERR_INVALID_ARG
    assert ex(p, p, 28, 4, 1024, 128, 32, 7, sg.SCORE_AGG_IPT_MAX, None, p, p, 1 << 30,
              None) == sg.ERR_INVALID_ARG
    assert ex(p, p, 36, 4, 1024, 128, 32, 7, sg.SCORE_AGG_IPT_MAX, p, p, p, 1 << 30,
              None) == sg.ERR_UNSUPPORTED                              # G = 9 > 8
    assert ex(p, p, 4, 4, 1024, 128, 96, 7, sg.SCORE_AGG_IPT_MAX, p, p, p, 1 << 30,
              None) == sg.ERR_UNSUPPORTED                              # W = 96 > 64
    assert ex(p, p, 28, 4, 1024, 128, 32, 6, sg.SCORE_PROXY_QUERY, None, p, p, 1 << 30,
              None) == sg.ERR_INVALID_ARG
    assert ex(p, p, 28, 4, 1024, 128, 32, 7, sg.SCORE_PROXY_QUERY | sg.SCORE_AGG_IPT_MEAN, p, p,
              p, 16, None) == sg.ERR_WORKSPACE
    # the two halves: sgdkv_score_raw checks as sgdkv_score_ex (no pool, no output)...
    raw = L.sgdkv_score_raw
    assert raw(None, p, 28, 4, 1024, 128, 32, 0, None, p, 1 << 30, None) == sg.ERR_INVALID_ARG
    assert raw(p, p, 28, 4, 1024, 64, 32, 0, None, p, 1 << 30, None) == sg.ERR_UNSUPPORTED
    assert raw(p, p, 28, 4, 1024, 128, 32, 16, None, p, 1 << 30, None) == sg.ERR_INVALID_ARG
    assert raw(p, p, 28, 4, 1024, 128, 32, sg.SCORE_AGG_IPT_MAX, None, p, 1 << 30,
               None) == sg.ERR_INVALID_ARG
    assert raw(p, p, 28, 4, 1024, 128, 32, 0, None, p, 16, None) == sg.ERR_WORKSPACE
    # the two passes one at a time check the same
    for fn in (L.sgdkv_window_stats, L.sgdkv_window_sums):
        assert fn(None, p, 28, 4, 1024, 128, 32, 0, None, p, 1 << 30, None) == sg.ERR_INVALID_ARG
        assert fn(p, p, 28, 4, 1024, 64, 32, 0, None, p, 1 << 30, None) == sg.ERR_UNSUPPORTED
        assert fn(p, p, 28, 4, 1024, 128, 32, 16, None, p, 1 << 30, None) == sg.ERR_INVALID_ARG
        assert fn(p, p, 28, 4, 1024, 128, 32, 0, None, p, 16, None) == sg.ERR_WORKSPACE
    # ...and sgdkv_pool_raw its pool kernel, shape, flags, output and workspace
    pr = L.sgdkv_pool_raw
    assert pr(p, 1 << 30, 4, 1024, 6, 0, p, None) == sg.ERR_INVALID_ARG      # even pool
    assert pr(p, 1 << 30, 0, 1024, 7, 0, p, None) == sg.ERR_INVALID_ARG      # Hkv
    assert pr(p, 1 << 30, 4, 0, 7, 0, p, None) == sg.ERR_INVALID_ARG         # L
    assert pr(p, 1 << 30, 4, 1024, 7, 16, p, None) == sg.ERR_INVALID_ARG     # unknown flag
    assert pr(p, 1 << 30, 4, 1024, 7, 0, None, None) == sg.ERR_INVALID_ARG   # no output
    assert pr(p, 1 << 30, 99, 1024, 7, 0, p, None) == sg.ERR_UNSUPPORTED     # Hkv > max
    assert pr(p, 16, 4, 1024, 7, 0, p, None) == sg.ERR_WORKSPACE
    # ...and sgdkv_pool_compact both, before anything reaches the device
    pc = L.sgdkv_pool_compact
    b = np.array([300, 300, 300, 300], np.int64).ctypes.data_as(ctypes.c_void_p)
    bad = np.array([300, 300, 300, 2000], np.int64).ctypes.data_as(ctypes.c_void_p)

    def call(pool=7, flags=0, budgets=b, d=128, scores=p, sws=1 << 30, ws=1 << 30):
        return pc(p, sws, pool, flags, p, p, budgets, 4, 1024, d, 64, 64, scores, p, p, p, p, p,
                  ws, None)
    assert call(pool=6) == sg.ERR_INVALID_ARG                 # even pool
    assert call(pool=65) == sg.ERR_INVALID_ARG                # window wider than 63
    assert call(flags=16) == sg.ERR_INVALID_ARG               # unknown flag
    assert call(scores=None) == sg.ERR_INVALID_ARG            # pooled scores required
    assert call(d=64) == sg.ERR_UNSUPPORTED                   # head dim
    assert call(budgets=bad) == sg.ERR_INVALID_ARG            # budget above L
    assert call(sws=16) == sg.ERR_WORKSPACE                   # scoring workspace too small
    assert call(ws=16) == sg.ERR_WORKSPACE                    # compaction workspace too small


def test_decode_rejects_bad_args_before_device_work():
    import ctypes
    L = sg.lib()
    wb = L.sgdkv_decode_workspace_bytes
    assert wb(28, 4, 1, 128, 131072) > 0
    assert wb(28, 4, 1, 128, 0) > 0
    assert wb(28, 4, 1, 64, 1000) == 0             # head dim
    assert wb(28, 4, 3, 128, 1000) == 0            # G * n_tok = 21 > 16
    assert wb(28, 5, 1, 128, 1000) == 0            # Hq % Hkv
    assert wb(28, 4, 1, 128, -1) == 0
    buf = (ctypes.c_uint8 * 4096)()
    p = ctypes.cast(buf, ctypes.c_void_p)
    good = np.array([100, 200, 0, 50], np.int64)
    neg = np.array([100, -1, 0, 50], np.int64)
    da = L.sgdkv_decode_attention

    def call(q=p, Hq=28, n_tok=1, d=128, b=good, out=p, ws_bytes=1 << 30):
        return da(q, Hq, 4, n_tok, d, p, p, b.ctypes.data_as(ctypes.c_void_p), out, p,
                  ws_bytes, None)
    assert call(q=None) == sg.ERR_INVALID_ARG
    assert call(out=None) == sg.ERR_INVALID_ARG
    assert call(d=64) == sg.ERR_UNSUPPORTED
    assert call(n_tok=3) == sg.ERR_UNSUPPORTED
    assert call(Hq=30) == sg.ERR_INVALID_ARG
    assert call(b=neg) == sg.ERR_INVALID_ARG
    assert call(ws_bytes=16) == sg.ERR_WORKSPACE
    assert da(p, 28, 4, 1, 128, p, p, None, p, p, 1 << 30, None) == sg.ERR_INVALID_ARG


def test_decode_workspace_bound_grows_with_the_cache():
    """A decode workspace sized for the largest cache serves every smaller one: the size is
    non-decreasing in the total kept rows and stops growing at its bound."""
    prev = 0
    for rows in list(range(0, 40000, 61)) + [131072, 524288, 2 ** 31 - 1]:
        n = sg.sgdkv_decode_workspace_bytes(28, 4, 1, 128, rows)
        assert n >= prev > 0 or (prev == 0 and n > 0)
        prev = n
    assert sg.sgdkv_decode_workspace_bytes(28, 4, 1, 128, 2 ** 31 - 1) == \
        sg.sgdkv_decode_workspace_bytes(28, 4, 1, 128, 10 ** 9)
    assert sg.sgdkv_decode_workspace_bytes(28, 4, 1, 128, 2 ** 31) == 0


def test_compact_rejects_bad_budgets():
    import ctypes
    L = sg.lib()
    buf = (ctypes.c_uint8 * 4096)()
    p = ctypes.cast(buf, ctypes.c_void_p)
    b = np.array([10, 3], np.int64)   # second head below n_sink + n_recent
    st = L.sgdkv_compact(p, p, p, b.ctypes.data_as(ctypes.c_void_p), 2, 100, 128, 2, 2, p, p,
                         p, p, p, 1 << 30, None)
    assert st == sg.ERR_INVALID_ARG
    b = np.array([10, 101], np.int64)  # above L
    st = L.sgdkv_compact(p, p, p, b.ctypes.data_as(ctypes.c_void_p), 2, 100, 128, 2, 2, p, p,
                         p, p, p, 1 << 30, None)
    assert st == sg.ERR_INVALID_ARG
