"""The cache-size tuner and the verification-width accounting against the GPU path.

Tuner (section "Throughput Model": materialization_time(p) counts the misses at cache size p;
Discussion, "Cache Hit Rate Is an Incomplete Objective"): a route trace recorded on the GPU is
replayed by mf_tune_cache at three slot counts; its predicted misses must equal the misses the GPU
counts when it runs the same sequence with that many slots, for one-token and two-token steps and
both access orders.

Verification width (section "Throughput Model", extra_materialization; Discussion on
speculative decoding): a seeded speculative schedule (synth.verify_rows: the next token, the
accepted drafts, then rejected drafts with routes of an independent stream) runs as calls of
T = K + 1 rows; every routed index, every access record and the counters must equal the oracle
router and LRU fed the same rows, and the outputs the oracle layer's."""
import numpy as np
import pytest

import oracle
import synth
from mfharness import Ctx, Payloads, Shape, G_ATOL, assert_outputs_close, oracle_trace, stats_tuple

pytestmark = pytest.mark.gpu
SHAPE = Shape(2, 256, 16, 4, 256, synth.Q8_0, model_seed=21)


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()


def _sequence(n, seed=2):
    L, H, E, k = SHAPE.n_layers, SHAPE.hidden, SHAPE.n_experts, SHAPE.top_k
    xs = [synth.activations(seed, l, 0, 0, n, H) for l in range(L)]
    bs = [synth.plant_bias(synth.routes(seed, l, 0, E, k, n, 1.1, 0.5), E) for l in range(L)]
    return xs, bs


@pytest.mark.parametrize("T,order", [(1, 0), (2, 0), (2, 1)])
def test_tuner_predicts_the_gpu_misses(T, order):
    import torch
    n = 40
    L, E, k = SHAPE.n_layers, SHAPE.n_experts, SHAPE.top_k
    xs, bs = _sequence(n)
    ctx = Ctx(SHAPE, E, max_tokens=T)
    mf, dev = ctx.mf, ctx.device
    try:
        mf.mf_access_order(ctx.h, order)
        xd = [torch.from_numpy(x).to(dev) for x in xs]
        bd = [torch.from_numpy(b).to(dev) for b in bs]
        y = torch.empty(T, SHAPE.hidden, device=dev)
        idx = torch.empty(L, n, k, dtype=torch.int32, device=dev)

        def run(slots):
            mf.mf_reset(ctx.h, slots)
            for t0 in range(0, n, T):  # steps of T consecutive tokens, layers in order per step
                tt = min(T, n - t0)
                for l in range(L):
                    mf.mf_moe_forward(ctx.h, l, xd[l][t0:t0 + tt], ctx.wr[l], bd[l][t0:t0 + tt], tt, y[:tt],
                                      idx[l, t0:t0 + tt], None)
            torch.cuda.synchronize()
            assert mf.mf_check(ctx.h) == 0
            return mf.mf_stats(ctx.h, -1)

        run(E)
        trace = idx.cpu().numpy()  # [L][n][k], the router's rank order
        model = mf.Model(SHAPE.n_layers, SHAPE.hidden, E, k, SHAPE.inter, SHAPE.qtype)
        slot_counts = (4, 6, 10)
        pcts = [100.0 * s / E for s in slot_counts]
        pts, _ = mf.mf_tune_cache(model, mf.PlanReq(0.0, 1 << 62, 0, 0, T, 0), trace, T, 1e-3, 1e-4, pcts, order)
        for s, pt in zip(slot_counts, pts):
            assert pt["slots_per_layer"] == s
            st = run(s)
            assert (pt["accesses"], pt["hits"], pt["misses"]) == (st["accesses"], st["hits"], st["misses"]), s
            assert pt["bytes_materialized"] == st["bytes_materialized"]
            assert trace.tolist() == idx.cpu().numpy().tolist()  # routing does not depend on the cache
    finally:
        ctx.close()


def test_verify_schedule_against_the_oracle():
    import torch
    K, alpha, n = 4, 0.6, 24
    W = K + 1
    L, H, E, k = SHAPE.n_layers, SHAPE.hidden, SHAPE.n_experts, SHAPE.top_k
    rows = synth.verify_rows(3, n, K, alpha)  # [batches, W]
    nb, n_drafts = rows.shape[0], int((rows < 0).sum())
    assert n_drafts > 0 and nb < n  # some drafts accepted, some rejected
    xs, bs = _sequence(n, seed=3)
    slots = 6
    ctx = Ctx(SHAPE, slots, max_tokens=W)
    pays = Payloads(SHAPE)
    try:
        lru = [oracle.LRU(E, slots, synth.payload_bytes(H, SHAPE.inter, SHAPE.qtype)) for _ in range(L)]
        for l in range(L):
            xd = synth.activations(3, l, 1, 0, n_drafts, H)
            bd = synth.plant_bias(synth.routes(3, l, 1, E, k, n_drafts, 1.1, 0.0), E)
            xb = np.stack([[xs[l][v] if v >= 0 else xd[-1 - v] for v in r] for r in rows])  # [nb, W, H]
            bb = np.stack([[bs[l][v] if v >= 0 else bd[-1 - v] for v in r] for r in rows])
            for b in range(nb):
                y, idx, w, tr = ctx.forward(l, xb[b], bb[b], W, trace=True)
                yo, oidx, og = oracle.layer(pays.for_layer(l, range(E)), SHAPE.qtype, H, SHAPE.inter, k,
                                            ctx.wr_host[l], bb[b], xb[b])
                assert np.array_equal(idx, oidx), (l, b)
                assert np.abs(w - og).max() <= G_ATOL
                assert tr == oracle_trace(lru[l], idx), (l, b)
                committed = rows[b] >= 0
                assert_outputs_close(y[committed], yo[committed], f"layer {l} verify step {b}")
        assert ctx.mf.mf_check(ctx.h) == 0
        for l in range(L):
            assert stats_tuple(ctx.mf.mf_stats(ctx.h, l)) == stats_tuple(lru[l].stats()), l
    finally:
        ctx.close()
