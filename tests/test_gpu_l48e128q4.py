"""48 layers, hidden 2048, 128 experts, top-8, intermediate 768, Q4_0: a 4096-token prefill chunk
per layer (one call of T = 4096: the step's ~128 distinct experts go through the cache in
waves of S) followed by 96 decode tokens at batch 1, cache 15 % and 35 %, against the oracle.
Exact: routed indices (all decode tokens; every prefill token of 3 layers), every layer's
counters.  Tolerance: sampled prefill and decode outputs."""
import numpy as np
import pytest

import oracle
import synth
from mfharness import Ctx, Payloads, Shape, assert_outputs_close, oracle_routes, oracle_stats, stats_tuple

pytestmark = pytest.mark.gpu
CFG = synth.CONFIGS["l48e128q4"]
SHAPE = Shape.of(CFG)
CHECK_PREFILL_LAYERS = (0, 17, 47)


def _slots(pct):
    return max(CFG.top_k, int(np.floor(pct * CFG.n_experts / 100 + 1e-9)))


@pytest.fixture(scope="module")
def ctx():
    import __graft_entry__
    __graft_entry__.build()
    c = Ctx(SHAPE, _slots(max(CFG.cache_pcts)), max_tokens=CFG.prefill)
    yield c
    c.close()


@pytest.mark.parametrize("pct", CFG.cache_pcts)
def test_l48e128q4_prefill_then_decode(ctx, pct):
    import torch
    mf, dev = ctx.mf, ctx.device
    L, P, T, H, E, k = CFG.n_layers, CFG.prefill, CFG.n_tokens, CFG.hidden, CFG.n_experts, CFG.top_k
    klass, seed, slots = CFG.route_classes[0], 0, _slots(pct)
    routes = [synth.routes(seed, l, 0, E, k, P + T, klass.zipf_s, klass.reuse) for l in range(L)]
    mf.mf_reset(ctx.h, slots)
    pays = Payloads(SHAPE)
    pre_idx = {}
    for l in range(L):  # prefill: one call per layer with all 4096 tokens
        x = synth.activations(seed, l, 0, 0, P, H)
        b = synth.plant_bias(routes[l][:P], E)
        xd, bd = torch.from_numpy(x).to(dev), torch.from_numpy(b).to(dev)
        y = torch.empty(P, H, device=dev)
        idx = torch.empty(P, k, dtype=torch.int32, device=dev)
        mf.mf_moe_forward(ctx.h, l, xd, ctx.wr[l], bd, P, y, idx, None)
        torch.cuda.synchronize()
        pre_idx[l] = idx.cpu().numpy()
        if l in CHECK_PREFILL_LAYERS:
            oidx = oracle_routes(SHAPE, [ctx.wr_host[l]], [x], [b])[0]
            assert np.array_equal(pre_idx[l], oidx), l
            yg = y.cpu().numpy()
            for t in (0, 1, P // 2, P - 1):
                yo, _, _ = oracle.layer(pays.for_layer(l, oidx[t]), CFG.qtype, H, CFG.inter, k, ctx.wr_host[l],
                                        b[t:t + 1], x[t:t + 1])
                assert_outputs_close(yg[t:t + 1], yo, f"prefill layer {l} token {t}")
    # decode: 96 tokens at batch 1, layers in order per token
    xs = [synth.activations(seed, l, 0, P, T, H) for l in range(L)]
    bs = [synth.plant_bias(routes[l][P:], E) for l in range(L)]
    xd = torch.from_numpy(np.stack(xs, 1)).to(dev)
    bd = torch.from_numpy(np.stack(bs, 1)).to(dev)
    yd = torch.empty(T, L, H, device=dev)
    idd = torch.empty(T, L, k, dtype=torch.int32, device=dev)
    for t in range(T):
        for l in range(L):
            mf.mf_moe_forward(ctx.h, l, xd[t, l], ctx.wr[l], bd[t, l], 1, yd[t, l], idd[t, l], None)
    torch.cuda.synchronize()
    assert mf.mf_check(ctx.h) == 0
    dec_idx = idd.cpu().numpy().transpose(1, 0, 2)
    assert np.array_equal(dec_idx, oracle_routes(SHAPE, ctx.wr_host, xs, bs))
    # counters: prefill step (the checked layers' oracle routes equal the GPU's) then decode steps
    ost = oracle_stats(SHAPE, slots, [[pre_idx[l]] + [dec_idx[l, t][None] for t in range(T)] for l in range(L)])
    for l in range(L):
        assert stats_tuple(mf.mf_stats(ctx.h, l)) == stats_tuple(ost[l]), l
    yg = yd.cpu().numpy()
    for (l, t) in ((3, 0), (20, 50), (47, 95)):
        yo, _, _ = oracle.layer(pays.for_layer(l, dec_idx[l, t]), CFG.qtype, H, CFG.inter, k, ctx.wr_host[l],
                                bs[l][t:t + 1], xs[l][t:t + 1])
        assert_outputs_close(yg[t, l][None], yo, f"decode layer {l} token {t}")
