"""Seeded synthetic inputs for the compression step.

This module only draws random inputs and holds none of the method's arithmetic; it is the
one piece shared by the tests, the oracle checks, ``bench.py`` and ``smoke()``.

Recipe (one prefilled layer of a cache, shaped like the paper's evaluation models):

* K, V ~ N(0, 1) in float32, rounded to bfloat16 (round to nearest even), layout
  ``[Hkv][L][d]``.  Window queries q_win ~ N(0, 1) bf16, layout ``[Hq][W][d]``; query head
  q belongs to KV head q // G.
* Planted structure per KV head h: the 4 sink positions 0..3 plus ``n_salient`` positions
  drawn uniformly without replacement from [4, L - W) get the key
  k = 4 * sqrt(d) * u_h, where u_h is the unit vector of the mean of the G*W window query
  rows of h's group (fp64, from the bf16 queries), rounded to bf16.  Its norm is 4x that
  of a typical N(0, I) key, so these keys carry clearly higher window attention.
* Per-(layer, KV head) summarization scores: U[0, 1) or Beta(0.5, 2) float32.
* Seeds: base 20260902; every stream gets splitmix64-chained seed
  (base, config id, layer, stream kind) and a NumPy PCG64 generator, so the bytes do not
  depend on the machine.  ``layer_inputs_device`` draws the bulk N(0,1) values with the
  torch CUDA generator instead (same recipe, different random bytes) for timing runs.
"""
from __future__ import annotations

import math

import numpy as np

from .configs import Workload, WORKLOADS, config_id

BASE_SEED = 20260902
_MASK64 = (1 << 64) - 1
_KINDS = {"q": 1, "k": 2, "v": 3, "positions": 4, "head_scores": 5, "device": 6}


def splitmix64(x: int) -> int:
    """One step of SplitMix64 (Steele, Lea, Flood 2014): returns the mixed output for state x."""
    z = (x + 0x9E3779B97F4A7C15) & _MASK64
    z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & _MASK64
    z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & _MASK64
    return z ^ (z >> 31)


def stream_seed(base: int, cfg: int, layer: int, kind: str) -> int:
    s = splitmix64(base & _MASK64)
    for v in (cfg, layer, _KINDS[kind]):
        s = splitmix64((s + v) & _MASK64)
    return s


def _rng(base, cfg, layer, kind) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(stream_seed(base, cfg, layer, kind)))


def bf16_round(x: np.ndarray) -> np.ndarray:
    """float32 -> bfloat16 bit patterns (uint16), round to nearest, ties to even (finite inputs)."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    u = (u + 0x7FFF + ((u >> 16) & 1)) >> 16
    return u.astype(np.uint16)


def bf16_to_f32(b: np.ndarray) -> np.ndarray:
    """bfloat16 bit patterns (uint16) -> exact float32 values."""
    return (np.ascontiguousarray(b, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


def _planted_positions(rng: np.random.Generator, L: int, W: int, n_salient: int, n_sinks: int):
    lo, hi = n_sinks, max(n_sinks, L - W)
    n = min(n_salient, hi - lo)
    pos = rng.choice(np.arange(lo, hi, dtype=np.int64), size=n, replace=False) if n > 0 \
        else np.zeros(0, np.int64)
    return np.sort(np.concatenate([np.arange(min(n_sinks, L), dtype=np.int64), pos]))


def _salient_key_bits(q_group_bits: np.ndarray, d: int) -> np.ndarray:
    qm = bf16_to_f32(q_group_bits).astype(np.float64).reshape(-1, d).mean(axis=0)
    nrm = np.linalg.norm(qm)
    u = qm / nrm if nrm > 0 else np.full(d, 1.0 / math.sqrt(d))
    return bf16_round((4.0 * math.sqrt(d) * u).astype(np.float32))


def layer_inputs_host(wl: Workload, layer: int = 0, base: int = BASE_SEED, cfg: int | None = None):
    """One layer's window queries and K/V cache as bf16 bit arrays (numpy uint16).

    Returns dict(q=[Hq,W,d], K=[Hkv,L,d], V=[Hkv,L,d], planted=list of int64 arrays per head).
    """
    cfg = config_id(wl) if cfg is None else cfg
    Hq, Hkv, d, L, W, G = wl.Hq, wl.Hkv, wl.d, wl.L, wl.W, wl.G
    q = bf16_round(_rng(base, cfg, layer, "q").standard_normal((Hq, W, d), dtype=np.float32))
    K = bf16_round(_rng(base, cfg, layer, "k").standard_normal((Hkv, L, d), dtype=np.float32))
    V = bf16_round(_rng(base, cfg, layer, "v").standard_normal((Hkv, L, d), dtype=np.float32))
    prng = _rng(base, cfg, layer, "positions")
    planted = []
    for h in range(Hkv):
        pos = _planted_positions(prng, L, W, wl.n_salient, wl.n_sinks_planted)
        K[h, pos, :] = _salient_key_bits(q[h * G:(h + 1) * G], d)
        planted.append(pos)
    return dict(q=q, K=K, V=V, planted=planted)


def head_scores(wl: Workload, base: int = BASE_SEED, cfg: int | None = None) -> np.ndarray:
    """Per-(layer, KV head) summarization scores, layer-major, float32 [n_layers * Hkv]."""
    cfg = config_id(wl) if cfg is None else cfg
    rng = _rng(base, cfg, 0, "head_scores")
    n = wl.n_heads_total
    if wl.score_dist == "uniform":
        s = rng.random(n)
    elif wl.score_dist == "beta":
        s = rng.beta(0.5, 2.0, n)
    else:
        raise ValueError(wl.score_dist)
    return s.astype(np.float32)


def to_torch_bf16(bits: np.ndarray, device="cpu"):
    import torch
    t = torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16)
    return t.to(device) if str(device) != "cpu" else t


def from_torch_bf16(t) -> np.ndarray:
    import torch
    return t.detach().to("cpu").contiguous().view(torch.int16).numpy().view(np.uint16)


def layer_inputs_device(wl: Workload, layer: int, device, base: int = BASE_SEED):
    """Same recipe as ``layer_inputs_host`` with the bulk N(0,1) draws made on the GPU.

    Used where the full model's caches are too large to draw on the host in reasonable time
    (timing runs).  Returns torch bf16 tensors q [Hq,W,d], K, V [Hkv,L,d] on ``device``.
    """
    import torch
    cfg = config_id(wl)
    g = torch.Generator(device=device)
    g.manual_seed(stream_seed(base, cfg, layer, "device") & ((1 << 63) - 1))
    Hq, Hkv, d, L, W, G = wl.Hq, wl.Hkv, wl.d, wl.L, wl.W, wl.G

    def normal_bf16(shape):
        out = torch.empty(shape, dtype=torch.bfloat16, device=device)
        flat = out.view(-1)
        step = 1 << 26
        for i in range(0, flat.numel(), step):
            n = min(step, flat.numel() - i)
            flat[i:i + n] = torch.randn(n, generator=g, device=device, dtype=torch.float32)
        return out

    q = normal_bf16((Hq, W, d))
    K = normal_bf16((Hkv, L, d))
    V = normal_bf16((Hkv, L, d))
    prng = _rng(base, cfg, layer, "positions")
    qh = from_torch_bf16(q)
    for h in range(Hkv):
        pos = _planted_positions(prng, L, W, wl.n_salient, wl.n_sinks_planted)
        key = to_torch_bf16(_salient_key_bits(qh[h * G:(h + 1) * G], d), device)
        K[h, torch.from_numpy(pos).to(device)] = key
    return dict(q=q, K=K, V=V)


def tiny_workload(Hq=4, Hkv=2, d=128, L=300, W=16, pool=7, n_salient=8, floor=32,
                  score_dist="uniform", n_layers=1) -> Workload:
    """A small custom shape for parity and edge-case tests (seeded like config id 100+)."""
    return Workload(f"tiny_{Hq}_{Hkv}_{d}_{L}_{W}", Hq=Hq, Hkv=Hkv, d=d, L=L, W=W, pool=pool,
                    n_layers=n_layers, n_salient=n_salient, score_dist=score_dist,
                    budget_fracs=(0.25,), floor=floor)


def tiny_inputs(wl: Workload, layer: int = 0, base: int = BASE_SEED, tag: int = 100):
    return layer_inputs_host(wl, layer, base, cfg=tag)


__all__ = ["BASE_SEED", "WORKLOADS", "splitmix64", "stream_seed", "bf16_round", "bf16_to_f32",
           "layer_inputs_host", "layer_inputs_device", "head_scores", "to_torch_bf16",
           "from_torch_bf16", "tiny_workload", "tiny_inputs"]
