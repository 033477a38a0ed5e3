"""Pins for the oracle's top-b_h selection and gather (Section 3.3).

Selection is checked against a brute-force rule on tiny inputs with many ties: a middle
position is kept iff fewer than k middle positions beat it (higher score, or equal score
at a lower position).  The gather is checked on rows that encode their own (head,
position).  End to end, the planted salient keys of the synthetic recipe must all survive
when the middle budget has room for their 7-wide pooled plateaus.
"""
import numpy as np
import pytest

from oracle import sgdkv_oracle as O
from paper_2609_03235_gb300 import synth


def _brute_keep(x, k, n_sink, n_recent):
    L = x.size
    mid = list(range(n_sink, L - n_recent))
    keep = set(range(n_sink)) | set(range(L - n_recent, L))
    for j in mid:
        beaten = sum(1 for t in mid if x[t] > x[j] or (x[t] == x[j] and t < j))
        if beaten < k:
            keep.add(j)
    return sorted(keep)


@pytest.mark.parametrize("seed", range(30))
def test_select_matches_brute_force(seed):
    rng = np.random.default_rng(seed)
    Hkv = int(rng.integers(1, 4))
    L = int(rng.integers(1, 40))
    n_sink = int(rng.integers(0, L + 1))
    n_recent = int(rng.integers(0, L - n_sink + 1))
    x = rng.integers(0, 4, size=(Hkv, L)).astype(np.float32) * 0.25   # heavy ties
    b = rng.integers(n_sink + n_recent, L + 1, size=Hkv)
    idx, cu = O.select_indices(x, b, n_sink, n_recent)
    assert cu.tolist() == [0] + np.cumsum(b).tolist()
    for h in range(Hkv):
        got = idx[cu[h]:cu[h + 1]].tolist()
        assert got == _brute_keep(x[h], int(b[h]) - n_sink - n_recent, n_sink, n_recent)


def test_select_plateau_ties_take_lowest_positions():
    x = np.zeros((1, 30), np.float32)
    x[0, 10:17] = 1.0      # a 7-wide plateau
    idx, cu = O.select_indices(x, [2 + 3], 1, 1)
    assert idx.tolist() == [0, 10, 11, 12, 29]


def test_select_rejects_bad_budget():
    x = np.zeros((1, 10), np.float32)
    with pytest.raises(ValueError):
        O.select_indices(x, [3], 2, 2)
    with pytest.raises(ValueError):
        O.select_indices(x, [11], 0, 0)


def test_gather_encoded_rows():
    Hkv, L, d = 3, 12, 4
    K = np.zeros((Hkv, L, d), np.uint16)
    V = np.zeros((Hkv, L, d), np.uint16)
    for h in range(Hkv):
        for j in range(L):
            K[h, j] = [h, j, 7, 1]
            V[h, j] = [h, j, 9, 2]
    idx = np.array([0, 5, 11, 2, 3, 1, 4, 6, 10], np.int32)
    cu = np.array([0, 3, 5, 9], np.int32)
    ko, vo = O.gather(K, V, idx, cu)
    heads = [0, 0, 0, 1, 1, 2, 2, 2, 2]
    assert ko[:, 0].tolist() == heads and ko[:, 1].tolist() == idx.tolist()
    assert vo[:, 0].tolist() == heads and vo[:, 1].tolist() == idx.tolist()
    assert np.all(ko[:, 2] == 7) and np.all(vo[:, 2] == 9)


def test_planted_salient_keys_survive():
    wl = synth.tiny_workload(Hq=14, Hkv=2, d=128, L=2048, W=32, n_salient=16, floor=128)
    inp = synth.tiny_inputs(wl)
    n_sink, n_recent = 64, 64
    k_mid = 7 * (wl.n_salient + 4) + 8
    b = np.full(wl.Hkv, n_sink + n_recent + k_mid)
    out = O.compress_layer(inp["q"], inp["K"], inp["V"], b, n_sink, n_recent, pool=7)
    for h in range(wl.Hkv):
        kept = set(out["indices"][out["cu_seqlens"][h]:out["cu_seqlens"][h + 1]].tolist())
        assert set(inp["planted"][h].tolist()) <= kept
