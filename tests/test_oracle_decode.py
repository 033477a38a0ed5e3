"""Pins for the oracle's decode attention over the compressed cache.

Each query head attends, with softmax(q . k / sqrt(d)), over the kept rows of its own KV
head (query head qh reads KV head qh // G: the cache is kept before the values are repeated
for the GQA group, Appendix, Configuration).  The pins below do not retype that formula:
they use special cases with closed forms (one row, equal keys, a zero query, two rows with
a known logit gap), the structure of the answer (a convex combination of the head's value
rows, invariant to row order and to a common shift of the keys along any direction), the
head mapping with per-head constant values, and a pure-Python brute force on tiny inputs.
"""
import math

import numpy as np
import pytest

from oracle import sgdkv_oracle as O


def _cache(rng, rows, d):
    cu = np.concatenate([[0], np.cumsum(rows)]).astype(np.int64)
    K = rng.standard_normal((int(cu[-1]), d))
    V = rng.standard_normal((int(cu[-1]), d))
    return K, V, cu


def test_single_row_returns_its_value():
    rng = np.random.default_rng(1)
    K, V, cu = _cache(rng, [1, 1], 8)
    q = rng.standard_normal((4, 3, 8)) * 10.0
    out = O.decode_attention(q, K, V, cu)
    for qh in range(4):
        for t in range(3):
            assert np.array_equal(out[qh, t], V[qh // 2])


def test_equal_keys_and_zero_query_average_the_values():
    rng = np.random.default_rng(2)
    rows, d = [5, 9], 16
    _, V, cu = _cache(rng, rows, d)
    K = np.tile(rng.standard_normal((1, d)), (int(cu[-1]), 1))     # one key repeated
    q = rng.standard_normal((2, 2, d))
    out = O.decode_attention(q, K, V, cu)
    for h in range(2):
        mean = V[cu[h]:cu[h + 1]].mean(axis=0)
        np.testing.assert_allclose(out[h, 0], mean, rtol=0, atol=1e-12)
        np.testing.assert_allclose(out[h, 1], mean, rtol=0, atol=1e-12)
    K2 = rng.standard_normal(K.shape)
    out0 = O.decode_attention(np.zeros_like(q), K2, V, cu)
    for h in range(2):
        np.testing.assert_allclose(out0[h, 0], V[cu[h]:cu[h + 1]].mean(axis=0), atol=1e-12)


@pytest.mark.parametrize("gap", [0.0, 1.0, -3.5, 12.0])
def test_two_rows_follow_the_logistic_weight(gap):
    d = 4
    q = np.array([[[2.0 * gap, 0.0, 0.0, 0.0]]])       # q . k1 / sqrt(4) = gap, q . k2 = 0
    K = np.array([[1.0, 0.0, 0.0, 0.0], [0.0, 5.0, 0.0, 0.0]])
    V = np.array([[1.0, 2.0, 3.0, 4.0], [-1.0, 0.5, 7.0, 0.0]])
    out = O.decode_attention(q, K, V, np.array([0, 2]))
    w = 1.0 / (1.0 + math.exp(-gap))
    np.testing.assert_allclose(out[0, 0], w * V[0] + (1.0 - w) * V[1], rtol=1e-14, atol=1e-14)


def _brute(q, K, V, cu):
    Hq, T, d = q.shape
    G = Hq // (len(cu) - 1)
    out = [[[0.0] * d for _ in range(T)] for _ in range(Hq)]
    for qh in range(Hq):
        h = qh // G
        for t in range(T):
            s = []
            for i in range(int(cu[h]), int(cu[h + 1])):
                s.append(sum(q[qh][t][e] * K[i][e] for e in range(d)) / math.sqrt(d))
            if not s:
                continue
            top = max(s)
            w = [math.exp(x - top) for x in s]
            z = sum(w)
            for e in range(d):
                out[qh][t][e] = sum(w[k] * V[int(cu[h]) + k][e] for k in range(len(w))) / z
    return np.array(out)


@pytest.mark.parametrize("seed", range(6))
def test_matches_brute_force(seed):
    rng = np.random.default_rng(100 + seed)
    Hkv = int(rng.integers(1, 4))
    G = int(rng.integers(1, 4))
    rows = rng.integers(0, 7, size=Hkv)
    d, T = 6, int(rng.integers(1, 3))
    K, V, cu = _cache(rng, rows, d)
    q = rng.standard_normal((Hkv * G, T, d)) * 3.0
    np.testing.assert_allclose(O.decode_attention(q, K, V, cu), _brute(q, K, V, cu),
                               rtol=1e-12, atol=1e-12)


def test_head_mapping_convexity_order_and_shift():
    rng = np.random.default_rng(7)
    Hkv, G, d = 3, 4, 32
    rows = [11, 1, 30]
    K, V, cu = _cache(rng, rows, d)
    q = rng.standard_normal((Hkv * G, 2, d)) * 2.0
    # per-head constant values: every query head of group h returns exactly h
    Vh = np.concatenate([np.full((r, d), float(h)) for h, r in enumerate(rows)])
    outh = O.decode_attention(q, K, Vh, cu)
    for qh in range(Hkv * G):
        np.testing.assert_allclose(outh[qh], qh // G, atol=1e-12)
    out = O.decode_attention(q, K, V, cu)
    for qh in range(Hkv * G):                  # a convex combination of the head's rows
        seg = V[cu[qh // G]:cu[qh // G + 1]]
        assert np.all(out[qh] >= seg.min(axis=0) - 1e-12)
        assert np.all(out[qh] <= seg.max(axis=0) + 1e-12)
    perm = np.concatenate([cu[h] + rng.permutation(r) for h, r in enumerate(rows)])
    np.testing.assert_allclose(O.decode_attention(q, K[perm], V[perm], cu), out, atol=1e-12)
    shift = rng.standard_normal(d)              # a common key shift moves every logit of a
    np.testing.assert_allclose(O.decode_attention(q, K + shift, V, cu), out, atol=1e-10)


def test_empty_head_gives_zeros_and_bf16_bits_are_read_exactly():
    rng = np.random.default_rng(9)
    K, V, cu = _cache(rng, [0, 4], 8)
    q = rng.standard_normal((2, 1, 8))
    out = O.decode_attention(q, K, V, cu)
    assert np.array_equal(out[0], np.zeros((1, 8)))
    # bf16 bit patterns: 1.0 = 0x3F80, 2.0 = 0x4000; one row per head
    kb = np.array([[0x3F80] * 8], dtype=np.uint16)
    vb = np.array([[0x4000] * 8], dtype=np.uint16)
    qb = np.array([[[0x3F80] * 8]], dtype=np.uint16)
    np.testing.assert_array_equal(O.decode_attention(qb, kb, vb, np.array([0, 1]))[0, 0],
                                  np.full(8, 2.0))
