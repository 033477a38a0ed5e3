"""Pins for the oracle's window scoring and max-pool (Section 3.3, Section 5).

Checked against: the softmax invariant (every visible row sums to one, so the scores of
a head sum to G*W), closed forms for uniform logits (causal and non-causal), a two-key
closed form that fixes the 1/sqrt(d) scale, the limit of one overwhelming key, the GQA
group mapping (query head q -> KV head q // G), torch's float64 softmax with a causal
mask on random tiny shapes (library routine), and torch's max_pool1d (library routine).
"""
import math

import numpy as np
import pytest
import torch

from oracle import sgdkv_oracle as O
from paper_2609_03235_gb300 import synth


def _f(x):
    return np.asarray(x, np.float64)


@pytest.mark.parametrize("Hq,Hkv,L,W,d", [(4, 2, 50, 8, 16), (7, 1, 33, 32, 8), (8, 8, 9, 1, 4)])
@pytest.mark.parametrize("causal", [True, False])
def test_rows_sum_to_one(Hq, Hkv, L, W, d, causal):
    rng = np.random.default_rng(L)
    q = rng.standard_normal((Hq, W, d))
    k = rng.standard_normal((Hkv, L, d)) * 3
    raw = O.window_scores(q, k, causal=causal).astype(np.float64)
    G = Hq // Hkv
    assert np.allclose(raw.sum(axis=1), G * W, rtol=1e-6)


def test_non_causal_sees_the_last_keys_from_every_row():
    """Without the causal mask the first window row's softmax covers keys beyond L - W:
    a key planted at the last position draws mass from every row (it would draw none from
    rows w < W - 1 under the causal mask)."""
    L, W, d = 40, 8, 16
    q = np.zeros((1, W, d)); q[:, :, 0] = 1.0
    k = np.zeros((1, L, d)); k[0, L - 1, 0] = 20.0 * np.sqrt(d)
    nc = O.window_scores(q, k, causal=False).astype(np.float64)
    c = O.window_scores(q, k, causal=True).astype(np.float64)
    assert nc[0, L - 1] > W - 1e-3                   # every row puts ~all its mass on it
    assert c[0, L - 1] < 1 + 1e-3                    # only the last row sees it


@pytest.mark.parametrize("causal", [True, False])
def test_uniform_logits_closed_form(causal):
    Hq, Hkv, L, W, d = 6, 2, 40, 10, 8
    q = np.zeros((Hq, W, d))
    k = np.random.default_rng(0).standard_normal((Hkv, L, d))
    raw = O.window_scores(q, k, causal=causal).astype(np.float64)
    G = Hq // Hkv
    j = np.arange(L)
    if causal:
        # window row w sits at p = L - W + w and spreads 1/(p+1) over keys 0..p
        expect = np.zeros(L)
        for w in range(W):
            p = L - W + w
            expect[: p + 1] += 1.0 / (p + 1)
        expect *= G
        # spot values written out: key 0 is seen by every row, key L-1 only by the last
        assert expect[L - 1] == pytest.approx(G / L)
        assert expect[0] == pytest.approx(G * sum(1.0 / (L - W + w + 1) for w in range(W)))
    else:
        expect = np.full(L, G * W / L)
    for h in range(Hkv):
        assert np.allclose(raw[h], expect, rtol=1e-6, atol=0)
    assert j.size == L


def test_scale_two_keys_closed_form():
    # one query at position 1 (W=1) over keys 0 and 1: p0 = 1 / (1 + exp((b1 - b0) a / sqrt d))
    d, a, b0, b1 = 16, 3.0, 1.5, -0.5
    q = np.zeros((1, 1, d))
    q[0, 0, 0] = a
    k = np.zeros((1, 2, d))
    k[0, 0, 0], k[0, 1, 0] = b0, b1
    raw = O.window_scores(q, k).astype(np.float64)
    p0 = 1.0 / (1.0 + math.exp((b1 - b0) * a / math.sqrt(d)))
    assert raw[0, 0] == pytest.approx(p0, rel=1e-6)
    assert raw[0, 1] == pytest.approx(1 - p0, rel=1e-6)


def test_overwhelming_key_takes_all_mass():
    Hq, Hkv, L, W, d = 4, 1, 64, 8, 32
    rng = np.random.default_rng(5)
    u = rng.standard_normal(d)
    u /= np.linalg.norm(u)
    q = np.tile(u * 8.0, (Hq, W, 1))
    k = rng.standard_normal((Hkv, L, d)) * 0.1
    j_star = 17                                   # visible to every window row
    k[0, j_star] = u * 60.0
    raw = O.window_scores(q, k).astype(np.float64)
    assert raw[0, j_star] > Hq * W * (1 - 1e-6)


def test_gqa_group_mapping_is_contiguous():
    # G = 2: query heads 2, 3 belong to KV head 1.  Only they look along e0, and only KV
    # head 1 holds an e0-aligned key (position 5); head 0 holds one at position 7.
    Hq, Hkv, L, W, d = 4, 2, 32, 4, 8
    q = np.zeros((Hq, W, d))
    q[2:, :, 0] = 10.0
    q[:2, :, 1] = 10.0
    k = np.zeros((Hkv, L, d))
    k[1, 5, 0] = 10.0
    k[0, 7, 0] = 10.0
    raw = O.window_scores(q, k).astype(np.float64)
    assert int(np.argmax(raw[1])) == 5 and raw[1, 5] > 0.99 * 2 * W
    assert raw[0, 7] == pytest.approx(raw[0, 6], rel=1e-9)   # head 0's queries ignore e0


@pytest.mark.parametrize("seed", range(4))
def test_matches_torch_float64_softmax(seed):
    rng = np.random.default_rng(100 + seed)
    Hkv, G, W, d = 2, 3, 6, 16
    L = int(rng.integers(W, 70))
    q = rng.standard_normal((Hkv * G, W, d)) * 2
    k = rng.standard_normal((Hkv, L, d)) * 2
    raw = O.window_scores(q, k).astype(np.float64)
    qt, kt = torch.from_numpy(q), torch.from_numpy(k)
    logits = torch.einsum("hwd,hld->hwl", qt, kt.repeat_interleave(G, dim=0)) / math.sqrt(d)
    pos = torch.arange(L)
    mask = pos[None, :] > (L - W + torch.arange(W))[:, None]
    p = torch.softmax(logits.masked_fill(mask, float("-inf")), dim=-1)
    ref = p.view(Hkv, G, W, L).sum(dim=(1, 2)).numpy()
    assert np.allclose(raw, ref.astype(np.float32), rtol=1e-6, atol=1e-7)


def test_bf16_bits_are_read_exactly():
    x = np.array([1.0, -2.5, 3.140625, 1e-3], np.float32)
    bits = synth.bf16_round(x)
    back = O.bf16_bits_to_f64(bits)
    assert back[0] == 1.0 and back[1] == -2.5 and back[2] == 3.140625
    assert abs(back[3] - 1e-3) < 1e-3 * 2 ** -8


@pytest.mark.parametrize("kernel", [1, 3, 7, 9])
def test_max_pool_matches_torch(kernel):
    rng = np.random.default_rng(kernel)
    x = rng.random((3, 101)).astype(np.float32)
    out = O.max_pool(x, kernel)
    ref = torch.nn.functional.max_pool1d(torch.from_numpy(x)[None], kernel, stride=1,
                                         padding=kernel // 2)[0].numpy()
    assert np.array_equal(out, ref)


def test_max_pool_spike_plateau():
    x = np.zeros((1, 20), np.float32)
    x[0, 1] = 5.0
    x[0, 15] = 2.0
    out = O.max_pool(x, 7)
    assert out[0].tolist() == [5.0] * 5 + [0.0] * 7 + [2.0] * 7 + [0.0]


def test_max_pool_rejects_even_kernel():
    with pytest.raises(ValueError):
        O.max_pool(np.zeros((1, 4), np.float32), 4)


# -- summarization-weighted GQA aggregation ("Ipt." variants of the appendix) --------------

def _ipt_case(seed, Hq=6, Hkv=2, L=40, W=8, d=16):
    rng = np.random.default_rng(seed)
    return rng.standard_normal((Hq, W, d)), rng.standard_normal((Hkv, L, d)) * 2


def test_ipt_head_attention_sums_to_window_scores():
    """Summing the per-head attention over a group gives window_scores (no weights)."""
    q, k = _ipt_case(1)
    A = O.head_window_attention(q, k)
    raw = O.window_scores(q, k).astype(np.float64)
    assert np.allclose(A.reshape(2, 3, -1).sum(axis=1), raw, rtol=1e-6)
    assert np.allclose(A.sum(axis=1), q.shape[1], rtol=1e-9)       # each head: W rows of 1


def test_ipt_modes_on_identical_heads():
    """Every query head of a group equal: max of w_g A = max(w) A, mean = mean(w) A, only = A."""
    q, k = _ipt_case(2, Hq=3, Hkv=1)
    q[1] = q[0]
    q[2] = q[0]
    w = np.array([0.2, 0.9, 0.5])
    A = O.head_window_attention(q, k)[0]
    assert np.allclose(O.window_scores_ipt(q, k, w, O.AGG_IPT_MAX), 0.9 * A, rtol=1e-6)
    assert np.allclose(O.window_scores_ipt(q, k, w, O.AGG_IPT_MEAN), w.mean() * A, rtol=1e-6)
    assert np.allclose(O.window_scores_ipt(q, k, w, O.AGG_IPT_ONLY), A, rtol=1e-6)


def test_ipt_only_picks_the_top_head_lower_index_on_ties():
    q, k = _ipt_case(3, Hq=4, Hkv=1)
    A = O.head_window_attention(q, k)
    assert np.allclose(O.window_scores_ipt(q, k, [0.1, 0.7, 0.7, 0.2], O.AGG_IPT_ONLY)[0],
                       A[1], rtol=1e-6)


def test_ipt_max_takes_the_larger_weighted_head_per_key():
    """Brute force on a tiny case: the weighted maximum per key, and zero weights drop heads."""
    q, k = _ipt_case(4, Hq=4, Hkv=2, L=25)
    w = np.array([0.5, 0.0, 2.0, 1.0])
    A = O.head_window_attention(q, k)
    got = O.window_scores_ipt(q, k, w, O.AGG_IPT_MAX).astype(np.float64)
    for h in range(2):
        for j in range(25):
            assert np.isclose(got[h, j], max(w[2 * h] * A[2 * h, j], w[2 * h + 1] * A[2 * h + 1, j]),
                              rtol=1e-6)
    assert np.allclose(got[0], 0.5 * A[0], rtol=1e-6)              # head 1 has weight 0


def test_ipt_rejects_bad_weights():
    q, k = _ipt_case(5)
    with pytest.raises(ValueError):
        O.window_scores_ipt(q, k, [1, 1, 1, 1, 1, -1], O.AGG_IPT_MAX)
    with pytest.raises(ValueError):
        O.window_scores_ipt(q, k, [1, 1, 1], O.AGG_IPT_MAX)
