"""Workload table: the five synthetic shapes the compression step is tested and timed on.

Each entry is one prefilled-cache shape taken from the paper's evaluation models
(Section 4: Qwen2.5-7B-Instruct-1M with 28 layers, 28 query / 4 KV heads; Qwen3-32B with
64 layers, 64 query / 8 KV heads; head_dim 128) at a given context length, window length,
pooling kernel and total budget.  The paper's benchmark caches (MRCR, ETHIC, BABILong)
and model weights are not available, so seeded synthetic K/V/Q of the same shapes stand
in for them (see ``synth.py``).

Budget convention (Section 3.3, Eq. 2): the total budget T counts every kept token of
every (layer, KV head), floors included; ``budget_frac`` is T / (n_layers * Hkv * L).
"""
from __future__ import annotations

from dataclasses import dataclass, field


@dataclass(frozen=True)
class Workload:
    name: str
    Hq: int
    Hkv: int
    d: int
    L: int
    W: int
    pool: int
    n_layers: int
    n_salient: int          # planted salient keys per KV head (besides the 4 sinks)
    score_dist: str         # "uniform" -> U[0,1); "beta" -> Beta(0.5, 2)
    budget_fracs: tuple = field(default=(0.25,))
    floor: int = 128
    n_sinks_planted: int = 4

    @property
    def G(self) -> int:
        return self.Hq // self.Hkv

    @property
    def n_heads_total(self) -> int:
        """Heads taking part in the allocation: every KV head of every layer."""
        return self.n_layers * self.Hkv

    def total_budget(self, frac: float) -> int:
        return int(round(frac * self.n_heads_total * self.L))


# index in this tuple == the config id used for seeding (synth.stream_seed)
WORKLOADS = (
    Workload("c1_single_layer_L4k", Hq=28, Hkv=4, d=128, L=4096, W=32, pool=7,
             n_layers=1, n_salient=64, score_dist="uniform", budget_fracs=(0.25,), floor=128),
    Workload("c2_qwen25_7b_L32k", Hq=28, Hkv=4, d=128, L=32768, W=32, pool=7,
             n_layers=28, n_salient=256, score_dist="beta", budget_fracs=(0.25,), floor=128),
    Workload("c3_qwen25_7b_L128k", Hq=28, Hkv=4, d=128, L=131072, W=64, pool=7,
             n_layers=28, n_salient=256, score_dist="beta", budget_fracs=(0.125, 0.25, 0.5),
             floor=256),
    Workload("c4_qwen3_32b_L128k", Hq=64, Hkv=8, d=128, L=131072, W=64, pool=7,
             n_layers=64, n_salient=256, score_dist="beta", budget_fracs=(0.25,), floor=256),
    Workload("c5_qwen25_7b_L1m", Hq=28, Hkv=4, d=128, L=1048576, W=64, pool=7,
             n_layers=28, n_salient=1024, score_dist="beta", budget_fracs=(0.25,), floor=512),
)

BY_NAME = {w.name: w for w in WORKLOADS}


def config_id(wl: Workload) -> int:
    return [w.name for w in WORKLOADS].index(wl.name)


def sink_recent_split(floor: int) -> tuple[int, int]:
    """Per-head floor f split into always-kept sink and recent tokens.

    Section 3.3 always keeps b_sink initial and b_window recent tokens and the appendix
    configuration uses equal sizes for both; the floor f = b_sink + b_window is split as
    n_sink = floor(f/2), n_recent = f - n_sink.
    """
    n_sink = floor // 2
    return n_sink, floor - n_sink
