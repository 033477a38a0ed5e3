"""Plain, slow CPU oracle of the SGD-KV compression step.

TEST INFRASTRUCTURE ONLY.  Nothing in the library imports this module; only ``tests/``,
``__graft_entry__.smoke()`` and the ``cpu_baseline`` / ``--impl reference`` legs of
``bench.py`` may import or run it.  It shares no code with the CUDA library: its inputs
are plain NumPy arrays (bf16 values given as uint16 bit patterns) and every step is
written from the paper's text in float64.

Steps and the passages they follow (SGD-KV, "Summarization Guided KV Cache Compression"):

* ``allocate_budgets``: Section 3.3 (score normalisation over all layers x KV heads,
  sink + window floor, proportional share of the middle, Eq. 2) and Appendix A.1,
  Algorithm 1 (cap at the middle length, collect the excess, hand it to the remaining
  heads in descending score order).  Integer rounding is not stated by the paper; the
  reading used is largest remainder (ties: higher score, then lower head index).  Modes
  after the appendix's ablation (Table 3): "thr" (scores below the mean zeroed first) and
  "Reverse" (every head's middle share inverted).
* ``mix_head_scores``: the "SGD-KV + HeadKV" row of the same ablation: the normalised
  summarization scores and the normalised HeadKV retrieval-reasoning scores, averaged.
* ``window_scores``: Section 3.3 and Section 5 (token selection from the cumulative
  attention of a final observation window, SnapKV-style): softmax over the causal keys of
  each window query, summed over the window and over the query heads of the KV head's
  GQA group; scale 1/sqrt(d).
* ``window_scores_ipt``: Appendix, "Head Configurations Variants" (last part of the
  ablation table): per query head g, its cumulative window attention A_g[j] weighted by
  the head's summarization score w_g, combined within the GQA group by max ("Ipt., Max")
  or mean ("Ipt., Mean"), or the attention of the group's highest-scoring head alone
  ("Ipt., Only"; ties: lower head).
* ``max_pool``: 1-D max smoothing of the window scores, odd kernel, stride 1, same length,
  the window clipped at the sequence ends.  The paper is silent on pooling; the
  smoothing step is part of the stated problem of this library.
* ``select_indices``: Section 3.3: sink and recent tokens always kept, then the top
  (b_h - n_sink - n_recent) tokens of the middle by pooled score; equal scores are
  broken by the lower position.  Output positions ascending per head, with cu_seqlens.
* ``gather``: keep the selected K/V rows per KV head (Appendix, "allocations occur
  before repeating the KV values": one cache per KV head), concatenated head by head.
* ``decode_attention``: what generation computes over the compressed cache (Section 3.3:
  the retained tokens are the heads' history; Appendix, Configuration: the cache is kept
  per KV head, before the values are repeated for the query heads of a GQA group): for
  each query head and new token, softmax(q . k / sqrt(d)) over its KV head's kept rows,
  times those rows' values.  A head with no kept row gives zeros (the paper is silent).

Parity pins for every function live in ``tests/test_oracle_*.py``.
"""
from __future__ import annotations

import math

import numpy as np

GREEDY, PROPORTIONAL, THRESHOLD, REVERSE = 0, 1, 2, 3
AGG_SUM, AGG_IPT_MAX, AGG_IPT_MEAN, AGG_IPT_ONLY = 0, 1, 2, 3


# ----------------------------------------------------------------------------------------
# Budget allocation (Section 3.3, Eq. 2; Appendix A.1, Algorithm 1)
# ----------------------------------------------------------------------------------------

def normalise(head_scores) -> list:
    """S_h = s_h / sum_h s_h over every (layer, KV head); all-zero scores give uniform S."""
    s = [float(x) for x in np.asarray(head_scores, dtype=np.float32).tolist()]
    if any((not math.isfinite(x)) or x < 0.0 for x in s):
        raise ValueError("head scores must be finite and non-negative")
    total = 0.0
    for x in s:                       # ascending head index
        total += x
    if total == 0.0:
        return [1.0 / len(s)] * len(s)
    return [x / total for x in s]


def _greedy_redistribute(S, x, cap):
    """Algorithm 1: cap every share at the middle length, then give the collected excess
    to the uncapped heads in descending S order (lower head index first on ties), each
    filled up to the cap before the next one is touched."""
    excess = 0.0
    for h in range(len(x)):           # E = sum over heads above the cap of (x_h - cap)
        if x[h] > cap:
            excess += x[h] - cap
    capped = [x[h] > cap for h in range(len(x))]
    xt = [min(v, cap) for v in x]
    order = sorted((h for h in range(len(x)) if not capped[h]), key=lambda h: (-S[h], h))
    for h in order:
        if excess <= 0.0:
            break
        give = min(excess, cap - xt[h])
        xt[h] += give
        excess -= give
    return xt


def _proportional_waterfill(S, pool, cap):
    """Alternative reading of step 5 of Algorithm 1: x_h = min(cap, lam * S_h) with lam
    chosen so that the shares sum to the pool (classic water filling)."""
    n = len(S)
    capped = [False] * n
    while True:
        free = pool - cap * sum(capped)
        ssum = 0.0
        for h in range(n):
            if not capped[h]:
                ssum += S[h]
        if ssum <= 0.0:
            # every remaining head has score zero: spread the rest evenly
            rest = [h for h in range(n) if not capped[h]]
            return [cap if capped[h] else (free / len(rest) if rest else 0.0) for h in range(n)]
        lam = free / ssum
        newly = [h for h in range(n) if not capped[h] and lam * S[h] > cap]
        if not newly:
            return [cap if capped[h] else lam * S[h] for h in range(n)]
        for h in newly:
            capped[h] = True


def _largest_remainder(S, xt, pool, cap):
    """Integer shares summing exactly to ``pool``: floors first, then one more token per
    head in order of (fractional part desc, S desc, head index asc), never above cap."""
    n = len(xt)
    m = [int(math.floor(v)) for v in xt]
    m = [min(max(v, 0), cap) for v in m]
    rest = pool - sum(m)
    frac = [xt[h] - math.floor(xt[h]) for h in range(n)]
    order = sorted(range(n), key=lambda h: (-frac[h], -S[h], h))
    while rest > 0:
        progressed = False
        for h in order:
            if rest == 0:
                break
            if m[h] < cap:
                m[h] += 1
                rest -= 1
                progressed = True
        if not progressed:
            raise ValueError("budget exceeds total capacity")
    return m


def allocate_budgets(head_scores, context_len: int, total_budget: int, floor: int,
                     mode: int = GREEDY) -> np.ndarray:
    """Per-head budgets b_h (int64) for every (layer, KV head), summing exactly to T.

    Section 3.3: b_h = (S_h * L * H * R) * M + b_sink + b_window (Eq. 2).  Here the floor
    f = b_sink + b_window, the middle length M = C - f and the total T counts every kept
    token, so the middle pool is P = T - N f and Eq. 2's middle share is S_h * P
    (R = P / (N M)).  Appendix A.1 (Algorithm 1) then caps each middle share at M and
    redistributes the excess.  mode 0: greedy redistribution (default reading);
    mode 1: proportional water filling; mode 2: "thr" variant of the appendix (scores below
    the mean set to zero first), then greedy; mode 3: "Reverse" row of the appendix's
    ablation (Table 3): the greedy allocation of T with every head's middle share m_h
    inverted to M - m_h (a head given 10 % of its middle keeps 90 %), floors kept, so the
    budgets sum to N (C + f) - T.
    """
    n = len(head_scores)
    C, T, f = int(context_len), int(total_budget), int(floor)
    if n <= 0 or f < 0 or f > C:
        raise ValueError("bad shape")
    if T < n * f or T > n * C:
        raise ValueError("infeasible budget")
    s = [float(x) for x in np.asarray(head_scores, dtype=np.float32).tolist()]
    if mode == THRESHOLD:
        mean = 0.0
        for x in s:
            mean += x
        mean = mean / n
        s = [x if x >= mean else 0.0 for x in s]
    S = normalise(np.asarray(s, dtype=np.float32))
    cap = C - f
    pool = T - n * f
    x = [S[h] * pool for h in range(n)]
    if mode in (GREEDY, THRESHOLD, REVERSE):
        xt = _greedy_redistribute(S, x, float(cap))
    elif mode == PROPORTIONAL:
        xt = _proportional_waterfill(S, float(pool), float(cap))
    else:
        raise ValueError("unknown mode")
    m = _largest_remainder(S, xt, pool, cap)
    if mode == REVERSE:
        m = [cap - v for v in m]
    return np.asarray([f + v for v in m], dtype=np.int64)


def mix_head_scores(a, b) -> np.ndarray:
    """Scores of the "SGD-KV + HeadKV" row of the appendix's ablation (Table 3): the two
    per-head score sets (summarization scores and the retrieval-reasoning scores of HeadKV)
    are each normalised to sum one over all heads and averaged: (a_h/sum a + b_h/sum b) / 2.
    float32 in, float32 out (the average formed in float64, rounded once)."""
    A, B = normalise(a), normalise(b)
    if len(A) != len(B):
        raise ValueError("score sets differ in length")
    return np.asarray([(A[h] + B[h]) / 2.0 for h in range(len(A))], dtype=np.float32)


# ----------------------------------------------------------------------------------------
# Window scoring (Section 3.3 / Section 5, SnapKV-style cumulative window attention)
# ----------------------------------------------------------------------------------------

def bf16_bits_to_f64(b) -> np.ndarray:
    """Exact value of bf16 bit patterns (uint16) as float64."""
    u = np.ascontiguousarray(b, dtype=np.uint16).astype(np.uint32) << 16
    return u.view(np.float32).astype(np.float64)


def window_scores(q_win, K, causal: bool = True) -> np.ndarray:
    """raw[h, j] = sum_{g < G} sum_{w < W} softmax_j(q[hG+g, w] . K[h, j] / sqrt(d)).

    q_win: [Hq, W, d], K: [Hkv, L, d] (bf16 bits or floats).  Window query w sits at
    position L - W + w and, with ``causal``, sees keys j <= L - W + w; masked keys take no
    part in its softmax.  Query head q belongs to KV head q // G.  Returns float32 [Hkv, L]
    (sums formed in float64, rounded once at the end).
    """
    q = bf16_bits_to_f64(q_win) if np.asarray(q_win).dtype == np.uint16 else np.asarray(q_win, np.float64)
    k = bf16_bits_to_f64(K) if np.asarray(K).dtype == np.uint16 else np.asarray(K, np.float64)
    Hq, W, d = q.shape
    Hkv, L, _ = k.shape
    G = Hq // Hkv
    raw = np.zeros((Hkv, L), dtype=np.float64)
    pos = np.arange(L)
    for h in range(Hkv):
        for g in range(G):
            logits = (q[h * G + g] @ k[h].T) / math.sqrt(d)          # [W, L]
            if causal:
                visible = pos[None, :] <= (L - W + np.arange(W))[:, None]
                logits = np.where(visible, logits, -np.inf)
            m = logits.max(axis=1, keepdims=True)
            e = np.exp(logits - m)
            p = e / e.sum(axis=1, keepdims=True)
            raw[h] += p.sum(axis=0)
    return raw.astype(np.float32)


def head_window_attention(q_win, K, causal: bool = True) -> np.ndarray:
    """A[q, j] = sum_{w < W} softmax_j(q[q, w] . K[q // G, j] / sqrt(d)) for every query head
    q (same softmax and mask as ``window_scores``); float64 [Hq, L]."""
    q = bf16_bits_to_f64(q_win) if np.asarray(q_win).dtype == np.uint16 else np.asarray(q_win, np.float64)
    k = bf16_bits_to_f64(K) if np.asarray(K).dtype == np.uint16 else np.asarray(K, np.float64)
    Hq, W, d = q.shape
    Hkv, L, _ = k.shape
    G = Hq // Hkv
    A = np.zeros((Hq, L), dtype=np.float64)
    pos = np.arange(L)
    for qh in range(Hq):
        logits = (q[qh] @ k[qh // G].T) / math.sqrt(d)            # [W, L]
        if causal:
            visible = pos[None, :] <= (L - W + np.arange(W))[:, None]
            logits = np.where(visible, logits, -np.inf)
        m = logits.max(axis=1, keepdims=True)
        e = np.exp(logits - m)
        A[qh] = (e / e.sum(axis=1, keepdims=True)).sum(axis=0)
    return A


def window_scores_ipt(q_win, K, head_weights, mode: int, causal: bool = True) -> np.ndarray:
    """Summarization-weighted GQA aggregation of the window attention (Appendix, head
    configuration variants).  head_weights: [Hq] non-negative summarization scores of the
    layer's query heads.  mode AGG_IPT_MAX: max_g w_g A_g; AGG_IPT_MEAN: mean_g w_g A_g;
    AGG_IPT_ONLY: A_{g*} with g* the group's highest-scoring head (lower index on ties);
    AGG_SUM: sum_g A_g (``window_scores``).  Returns float32 [Hkv, L]."""
    A = head_window_attention(q_win, K, causal)
    w = np.asarray(head_weights, dtype=np.float64)
    Hq, L = A.shape
    Hkv = np.asarray(K).shape[0]
    G = Hq // Hkv
    if w.shape != (Hq,) or not np.all(np.isfinite(w)) or np.any(w < 0):
        raise ValueError("head_weights must be Hq finite non-negative values")
    out = np.zeros((Hkv, L), dtype=np.float64)
    for h in range(Hkv):
        grp = slice(h * G, (h + 1) * G)
        if mode == AGG_SUM:
            out[h] = A[grp].sum(axis=0)
        elif mode == AGG_IPT_MAX:
            out[h] = (w[grp, None] * A[grp]).max(axis=0)
        elif mode == AGG_IPT_MEAN:
            out[h] = (w[grp, None] * A[grp]).mean(axis=0)
        elif mode == AGG_IPT_ONLY:
            out[h] = A[h * G + int(np.argmax(w[grp]))]
        else:
            raise ValueError("unknown aggregation mode")
    return out.astype(np.float32)


def max_pool(raw, kernel: int = 7) -> np.ndarray:
    """pooled[h, j] = max of raw[h, t] over t in [j - k//2, j + k//2] within [0, L)."""
    if kernel < 1 or kernel % 2 == 0:
        raise ValueError("pool kernel must be odd and positive")
    x = np.asarray(raw, dtype=np.float32)
    r = kernel // 2
    Hkv, L = x.shape
    padded = np.full((Hkv, L + 2 * r), -np.inf, dtype=np.float32)
    padded[:, r:r + L] = x
    out = padded[:, 0:L].copy()
    for t in range(1, kernel):
        out = np.maximum(out, padded[:, t:t + L])
    return out


# ----------------------------------------------------------------------------------------
# Selection and gather (Section 3.3)
# ----------------------------------------------------------------------------------------

def select_indices(pooled, budgets, n_sink: int, n_recent: int):
    """Kept positions per KV head and cu_seqlens.

    Positions [0, n_sink) and [L - n_recent, L) are always kept; of the middle
    [n_sink, L - n_recent) the first (b_h - n_sink - n_recent) in order of
    (pooled score descending, position ascending) are kept.  Returns (indices int32
    [sum b], cu_seqlens int32 [Hkv + 1]).
    """
    x = np.asarray(pooled, dtype=np.float32)
    Hkv, L = x.shape
    b = np.asarray(budgets, dtype=np.int64)
    if b.shape != (Hkv,) or n_sink < 0 or n_recent < 0 or n_sink + n_recent > L:
        raise ValueError("bad selection arguments")
    if np.any(b < n_sink + n_recent) or np.any(b > L):
        raise ValueError("budget outside [n_sink + n_recent, L]")
    out, cu = [], [0]
    middle = np.arange(n_sink, L - n_recent, dtype=np.int64)
    for h in range(Hkv):
        k = int(b[h]) - n_sink - n_recent
        order = np.lexsort((middle, -x[h, middle].astype(np.float64)))
        chosen = middle[order[:k]]
        keep = np.concatenate([np.arange(n_sink), chosen, np.arange(L - n_recent, L)])
        keep = np.sort(keep)
        out.append(keep)
        cu.append(cu[-1] + keep.size)
    idx = np.concatenate(out).astype(np.int32) if out else np.zeros(0, np.int32)
    return idx, np.asarray(cu, dtype=np.int32)


def gather(K, V, indices, cu_seqlens):
    """K_out[cu[h] + i] = K[h, indices[cu[h] + i]], likewise V (raw rows, bytes unchanged)."""
    K = np.asarray(K)
    V = np.asarray(V)
    Hkv = K.shape[0]
    ko, vo = [], []
    for h in range(Hkv):
        idx = np.asarray(indices[cu_seqlens[h]:cu_seqlens[h + 1]], dtype=np.int64)
        ko.append(K[h, idx])
        vo.append(V[h, idx])
    return np.concatenate(ko, axis=0), np.concatenate(vo, axis=0)


def decode_attention(q, K_out, V_out, cu_seqlens) -> np.ndarray:
    """out[qh, t] = sum_i softmax_i(q[qh, t] . K_out[c + i] / sqrt(d)) V_out[c + i].

    q: [Hq, n_tok, d]; K_out, V_out: [sum b_h, d] (bf16 bits or floats), the flat cache of
    ``gather``; cu_seqlens: [Hkv + 1].  Query head qh reads the rows of KV head qh // G,
    i in [0, cu[h+1] - cu[h]), c = cu[h].  Float64 throughout; returns float64
    [Hq, n_tok, d]; a head without rows gives zeros.
    """
    qf = bf16_bits_to_f64(q) if np.asarray(q).dtype == np.uint16 else np.asarray(q, np.float64)
    kf = bf16_bits_to_f64(K_out) if np.asarray(K_out).dtype == np.uint16 else np.asarray(K_out, np.float64)
    vf = bf16_bits_to_f64(V_out) if np.asarray(V_out).dtype == np.uint16 else np.asarray(V_out, np.float64)
    cu = np.asarray(cu_seqlens, dtype=np.int64)
    Hq, n_tok, d = qf.shape
    Hkv = cu.size - 1
    G = Hq // Hkv
    out = np.zeros((Hq, n_tok, d), dtype=np.float64)
    for qh in range(Hq):
        h = qh // G
        rows = slice(int(cu[h]), int(cu[h + 1]))
        if cu[h + 1] == cu[h]:
            continue
        logits = (qf[qh] @ kf[rows].T) / math.sqrt(d)          # [n_tok, rows]
        m = logits.max(axis=1, keepdims=True)
        e = np.exp(logits - m)
        p = e / e.sum(axis=1, keepdims=True)
        out[qh] = p @ vf[rows]
    return out


def compress_layer(q_win, K, V, budgets, n_sink, n_recent, pool=7, causal=True):
    """Whole per-layer step: window scores -> max pool -> top-b_h select -> gather."""
    raw = window_scores(q_win, K, causal=causal)
    pooled = max_pool(raw, pool) if pool > 1 else raw
    idx, cu = select_indices(pooled, budgets, n_sink, n_recent)
    ko, vo = gather(K, V, idx, cu)
    return dict(raw=raw, pooled=pooled, indices=idx, cu_seqlens=cu, K_out=ko, V_out=vo)
