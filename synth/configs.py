"""The five synthetic workloads of the routed-expert step (shapes and route-locality recipes).

Each stands in for one of the paper's model profiles / prompt suites, which are not
available: the shapes follow two real MoE families (~35B-total/3B-active with
hidden 2048, 128 experts, top-8, intermediate 768; ~26B-total/4B-active with hidden 2816,
128 experts, top-8, intermediate 1408) and the route classes give skewed, temporally
local routing.  Expert weights come from ``model_seed``; routes and activations from the
run seed.
"""
from __future__ import annotations

from dataclasses import dataclass, field

Q8_0 = 8
Q4_0 = 2


@dataclass(frozen=True)
class RouteClass:
    name: str
    zipf_s: float
    reuse: float


@dataclass(frozen=True)
class Config:
    name: str
    n_layers: int
    hidden: int
    n_experts: int
    top_k: int
    inter: int
    qtype: int
    n_tokens: int                 # decode tokens per run (per stream for batched decode)
    batch: int = 1                # concurrent decode streams (one token each per step)
    prefill: int = 0              # prefill chunk length before decode (0 = none)
    cache_pcts: tuple = ()        # cache fractions in percent; empty = explicit slots
    slots: int = 0                # explicit slot count (Tiny)
    route_classes: tuple = ()     # planted routing; empty = real routing from W_r
    seeds: tuple = (0,)
    model_seed: int = 0
    pool_cap_gib: float = 0.0     # slot-pool cap for static planning (0 = none)
    notes: str = field(default="", compare=False)


UNIFORM = RouteClass("uniform", 0.0, 0.0)
ZIPF08 = RouteClass("zipf0.8", 0.8, 0.0)
ZIPF12 = RouteClass("zipf1.2", 1.2, 0.0)
ZIPF12R = RouteClass("zipf1.2+reuse0.8", 1.2, 0.8)
ZIPF11R = RouteClass("zipf1.1+reuse0.6", 1.1, 0.6)
ZIPF10 = RouteClass("zipf1.0", 1.0, 0.0)

CONFIGS = {
    "tiny": Config("tiny", 1, 256, 8, 2, 512, Q8_0, n_tokens=64, slots=4,
                   notes="real routing from W_r ~ N(0,0.02), x ~ N(0,1), 4 slots, seed 0"),
    "l4e64": Config("l4e64", 4, 2048, 64, 8, 768, Q8_0, n_tokens=256, cache_pcts=(15.0, 35.0),
                    route_classes=(ZIPF11R,),
                    notes="4 layers, 256 decode tokens at batch 1, Zipf 1.1 + 0.6 reuse"),
    "l48e128": Config("l48e128", 48, 2048, 128, 8, 768, Q8_0, n_tokens=96,
                      cache_pcts=(15.0, 25.0, 35.0, 50.0, 65.0),
                      route_classes=(UNIFORM, ZIPF08, ZIPF12, ZIPF12R), seeds=(0, 1, 2, 3, 4),
                      notes="48 layers, ~35B-total/3B-active shape, 96 decode tokens x 5 seeds"),
    "l48e128q4": Config("l48e128q4", 48, 2048, 128, 8, 768, Q4_0, n_tokens=96, prefill=4096,
                        cache_pcts=(15.0, 35.0), route_classes=(ZIPF12,),
                        notes="Q4_0, 4096-token prefill then 96 decode tokens"),
    "l30e128b64": Config("l30e128b64", 30, 2816, 128, 8, 1408, Q8_0, n_tokens=64, batch=64,
                         cache_pcts=(15.0, 35.0, 50.0, 75.0), route_classes=(ZIPF10,),
                         pool_cap_gib=12.0,
                         notes="~26B-total/4B-active shape, 64 streams x 64 steps, 12 GiB slot-pool cap"),
}
