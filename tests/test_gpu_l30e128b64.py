"""30 layers, hidden 2816, 128 experts, top-8, intermediate 1408, Q8_0 (a ~26B-total/4B-active
MoE's expert shape): 64 concurrent decode streams (one call of T = 64 per layer and step, ~107
distinct experts against 19 slots: waves) for 64 steps, with the slot pool capped at 12 GiB so
that the static plan accepts only the 15 % cache.  Exact: the plan decisions, every routed index,
every layer's counters, sampled access records.  Tolerance: sampled outputs."""
import numpy as np
import pytest

import oracle
import synth
from mfharness import (Ctx, Payloads, Shape, G_ATOL, assert_outputs_close, oracle_routes, oracle_stats,
                       oracle_trace, stats_tuple)

pytestmark = pytest.mark.gpu
CFG = synth.CONFIGS["l30e128b64"]
SHAPE = Shape.of(CFG)
CAP = int(CFG.pool_cap_gib * 2**30)
COMMON = CFG.n_layers * CFG.n_experts * CFG.hidden * 4  # router weights: the only common tensor here


def test_l30e128b64_static_plan():
    import paper_2607_09686_gb300 as mf
    model = mf.Model(CFG.n_layers, CFG.hidden, CFG.n_experts, CFG.top_k, CFG.inter, CFG.qtype)
    for pct in CFG.cache_pcts:
        p = mf.mf_plan(model, mf.PlanReq(pct, CAP, COMMON, 0, CFG.batch, 0))
        o = oracle.plan(CFG.n_layers, CFG.hidden, CFG.n_experts, CFG.top_k, CFG.inter, CFG.qtype, pct, CAP, COMMON, 0)
        assert (p.slots_per_layer, p.pool_bytes, p.lower_bound_bytes, bool(p.accepted)) == \
            (o["slots"], o["pool"], o["lower"], o["accepted"])
        assert bool(p.accepted) == (pct == 15.0)
        if not p.accepted:
            with pytest.raises(mf.MFError) as e:
                mf.mf_create(model, p, 0)
            assert e.value.status == mf.MF_E_BUDGET


@pytest.fixture(scope="module")
def ctx():
    import __graft_entry__
    __graft_entry__.build()
    c = Ctx(SHAPE, int(np.floor(15.0 * CFG.n_experts / 100 + 1e-9)), max_tokens=CFG.batch)
    yield c
    c.close()


def test_l30e128b64_batched_decode(ctx):
    import torch
    mf, dev = ctx.mf, ctx.device
    L, B, N, H, E, k = CFG.n_layers, CFG.batch, CFG.n_tokens, CFG.hidden, CFG.n_experts, CFG.top_k
    klass, seed, slots = CFG.route_classes[0], 0, ctx.plan.slots_per_layer
    mf.mf_reset(ctx.h)
    # routes [L][step][stream][k], activations per (layer, stream, step)
    routes = [np.stack([synth.routes(seed, l, s, E, k, N, klass.zipf_s, klass.reuse) for s in range(B)], 1)
              for l in range(L)]
    xs = [np.stack([synth.activations(seed, l, s, 0, N, H) for s in range(B)], 1) for l in range(L)]  # [N, B, H]
    idx_all = np.empty((L, N, B, k), np.int32)
    pays = Payloads(SHAPE)
    traced = {(0, 0), (7, 29), (63, 15)}
    lru_tr = {l: oracle.LRU(E, slots, synth.payload_bytes(H, CFG.inter, CFG.qtype)) for l in (0, 15, 29)}
    y_keep = {}
    for step in range(N):
        for l in range(L):
            b = synth.plant_bias(routes[l][step], E)
            xd, bd = torch.from_numpy(xs[l][step]).to(dev), torch.from_numpy(b).to(dev)
            y = torch.empty(B, H, device=dev)
            idx = torch.empty(B, k, dtype=torch.int32, device=dev)
            w = torch.empty(B, k, device=dev)
            mf.mf_moe_forward(ctx.h, l, xd, ctx.wr[l], bd, B, y, idx, w)
            if l in lru_tr or (step, l) in traced:
                torch.cuda.synchronize()
                tr = mf.mf_trace(ctx.h, l, cap=E)
                if l in lru_tr:
                    assert tr == oracle_trace(lru_tr[l], idx.cpu().numpy()), (step, l)
            idx_all[l, step] = idx.cpu().numpy()
            if (step, l) in traced:
                wg = w.cpu().numpy()
                y_keep[(step, l)] = (y.cpu().numpy(), b, wg)
    assert mf.mf_check(ctx.h) == 0
    # every routed index against the oracle router
    oidx = oracle_routes(SHAPE, ctx.wr_host, [xs[l].reshape(N * B, H) for l in range(L)],
                         [np.concatenate([synth.plant_bias(routes[l][s], E) for s in range(N)]) for l in range(L)])
    assert np.array_equal(idx_all.reshape(L, N * B, k), oidx)
    ost = oracle_stats(SHAPE, slots, [[oidx[l].reshape(N, B, k)[s] for s in range(N)] for l in range(L)])
    for l in range(L):
        assert stats_tuple(mf.mf_stats(ctx.h, l)) == stats_tuple(ost[l]), l
    for (step, l), (yg, b, wg) in y_keep.items():
        for t in (0, 33, 63):
            _, oi, og = oracle.router(xs[l][step][t], ctx.wr_host[l], b[t], k)
            assert np.abs(wg[t] - og).max() <= G_ATOL
            yo, _, _ = oracle.layer(pays.for_layer(l, oi), CFG.qtype, H, CFG.inter, k, ctx.wr_host[l], b[t:t + 1],
                                    xs[l][step][t:t + 1])
            assert_outputs_close(yg[t:t + 1], yo, f"step {step} layer {l} stream {t}")
