"""48 layers, hidden 2048, 128 experts, top-8, intermediate 768, Q8_0 (a ~35B-total/3B-active
MoE's expert shape): 96-token decodes at batch 1, 5 seeds x 4 route-locality classes x 5 cache
fractions, against the CPU oracle.  Exact: every routed index and every layer's counters.
Tolerance: sampled layer outputs.  One context (31 GB pinned pack, 83 slots per layer) serves
every cache fraction (mf_reset with fewer slots in use)."""
import numpy as np
import pytest

import oracle
import synth
from mfharness import (Ctx, Payloads, Shape, G_ATOL, assert_outputs_close, oracle_routes, oracle_stats,
                       oracle_trace, stats_tuple)

pytestmark = pytest.mark.gpu
CFG = synth.CONFIGS["l48e128"]
SHAPE = Shape.of(CFG)


def _slots(pct):
    return max(CFG.top_k, int(np.floor(pct * CFG.n_experts / 100 + 1e-9)))


@pytest.fixture(scope="module")
def ctx():
    import __graft_entry__
    __graft_entry__.build()
    c = Ctx(SHAPE, _slots(max(CFG.cache_pcts)), max_tokens=1)
    yield c
    c.close()


def _inputs(seed, klass):
    L, T, H, E, k = CFG.n_layers, CFG.n_tokens, CFG.hidden, CFG.n_experts, CFG.top_k
    xs = [synth.activations(seed, l, 0, 0, T, H) for l in range(L)]
    bs = [synth.plant_bias(synth.routes(seed, l, 0, E, k, T, klass.zipf_s, klass.reuse), E) for l in range(L)]
    return xs, bs


def _gpu_decode(ctx, xs, bs, slots):
    """Token-major decode of all layers; returns idx [L, T, k] and per-layer counters."""
    import torch
    mf, dev = ctx.mf, ctx.device
    L, T = len(xs), xs[0].shape[0]
    xd = torch.from_numpy(np.stack(xs, 1)).to(dev)   # [T, L, H]
    bd = torch.from_numpy(np.stack(bs, 1)).to(dev)   # [T, L, E]
    y = torch.empty(T, L, SHAPE.hidden, device=dev)
    idx = torch.empty(T, L, SHAPE.top_k, dtype=torch.int32, device=dev)
    mf.mf_reset(ctx.h, slots)
    for t in range(T):
        for l in range(L):
            mf.mf_moe_forward(ctx.h, l, xd[t, l], ctx.wr[l], bd[t, l], 1, y[t, l], idx[t, l], None)
    torch.cuda.synchronize()
    assert mf.mf_check(ctx.h) == 0
    return (idx.cpu().numpy().transpose(1, 0, 2), [mf.mf_stats(ctx.h, l) for l in range(L)],
            y.cpu().numpy().transpose(1, 0, 2))


def test_l48e128_traced_decode(ctx):
    """Seed 0, Zipf 1.2 + 0.8 reuse, 35 %: every access record, router weights, sampled outputs."""
    klass, slots = CFG.route_classes[3], _slots(35.0)
    xs, bs = _inputs(0, klass)
    L, T, k = CFG.n_layers, CFG.n_tokens, CFG.top_k
    ctx.mf.mf_reset(ctx.h, slots)
    lru = [oracle.LRU(CFG.n_experts, slots, synth.payload_bytes(CFG.hidden, CFG.inter, CFG.qtype)) for _ in range(L)]
    pays = Payloads(SHAPE)
    rng = np.random.default_rng(3)
    pick = set((int(rng.integers(L)), int(rng.integers(T))) for _ in range(12))
    for t in range(T):
        for l in range(L):
            y, idx, w, tr = ctx.forward(l, xs[l][t:t + 1], bs[l][t:t + 1], 1, trace=True)
            _, oidx, og = oracle.router(xs[l][t], ctx.wr_host[l], bs[l][t], k)
            assert np.array_equal(idx[0], oidx) and np.abs(w[0] - og).max() <= G_ATOL
            assert tr == oracle_trace(lru[l], idx), (l, t)
            if (l, t) in pick:
                yo, _, _ = oracle.layer(pays.for_layer(l, oidx), CFG.qtype, CFG.hidden, CFG.inter, k,
                                        ctx.wr_host[l], bs[l][t:t + 1], xs[l][t:t + 1])
                assert_outputs_close(y, yo, f"layer {l} token {t}")


@pytest.mark.parametrize("seed", CFG.seeds)
def test_l48e128_cache_sweep(ctx, seed):
    """Every class and cache fraction of one seed: routed indices and per-layer counters exact."""
    for klass in CFG.route_classes:
        xs, bs = _inputs(seed, klass)
        oidx = oracle_routes(SHAPE, ctx.wr_host, xs, bs)
        for pct in CFG.cache_pcts:
            slots = _slots(pct)
            idx, st, y = _gpu_decode(ctx, xs, bs, slots)
            assert np.array_equal(idx, oidx), (klass.name, pct)
            ost = oracle_stats(SHAPE, slots, [[oidx[l, t][None] for t in range(CFG.n_tokens)]
                                              for l in range(CFG.n_layers)])
            for l in range(CFG.n_layers):
                assert stats_tuple(st[l]) == stats_tuple(ost[l]), (klass.name, pct, l)
        # one sampled output per class (the last cache fraction's run)
        l, t = (seed * 7 + 5) % CFG.n_layers, (seed * 13 + 3) % CFG.n_tokens
        pays = Payloads(SHAPE)
        yo, _, _ = oracle.layer(pays.for_layer(l, oidx[l, t]), CFG.qtype, CFG.hidden, CFG.inter, CFG.top_k,
                                ctx.wr_host[l], bs[l][t:t + 1], xs[l][t:t + 1])
        assert_outputs_close(y[l, t][None], yo, f"{klass.name} layer {l} token {t}")
