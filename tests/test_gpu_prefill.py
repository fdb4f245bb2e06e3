"""Tensor-core grouped GEMM path (many tokens per expert) vs the CPU oracle, through the C ABI.

Calls with T >= the context's threshold run each wave's expert FFN as tcgen05 GEMMs over
(expert, 128-assignment block, 128-row block) units.  Checked here element by element on every
token: outputs within the stated tolerance, routed indices, the access sequence and the
counters exactly; assignment counts on the 128-column tile boundaries (127, 128, 129, 256),
several waves with misses and evictions, a warm second call, both quantisations, and the GEMM
path against the GEMV path on the same inputs."""
import numpy as np
import pytest

import oracle
import synth
from mfharness import Ctx, G_ATOL, Payloads, Shape, assert_outputs_close, compare_outputs, oracle_trace

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()


def _check_call(ctx, pays, lru, layer, x, bias, T):
    s = ctx.s
    y, idx, w, tr = ctx.forward(layer, x, bias, T, trace=True)
    yo, oidx, og = oracle.layer(pays.for_layer(layer, np.unique(idx)), s.qtype, s.hidden, s.inter, s.top_k,
                                ctx.wr_host[layer], bias, x)
    assert np.array_equal(idx, oidx)
    assert np.abs(w - og).max() <= G_ATOL
    assert tr == oracle_trace(lru, idx)
    assert_outputs_close(y, yo, f"layer {layer} T={T}")
    return y


def _boundary_routes(T, E, k, rng):
    """Routes whose per-expert assignment counts sit on the GEMM's 128-column tile edges."""
    want = [T, 129, 128, 127, 1]  # experts 0..4 (expert 0 in every token)
    r = np.full((T, k), -1, np.int32)
    r[:, 0] = 0
    for e, n in enumerate(want[1:], start=1):
        rows = [t for t in rng.permutation(T) if (r[t] == -1).any()][:n]
        for t in rows:
            r[t, np.flatnonzero(r[t] == -1)[0]] = e
    for t in range(T):  # remaining ranks: other experts, distinct within the token
        for j in range(k):
            if r[t, j] == -1:
                free = [e for e in range(5, E) if e not in r[t]]
                r[t, j] = free[rng.integers(len(free))]
    return r


@pytest.mark.parametrize("qtype", [synth.Q8_0, synth.Q4_0])
@pytest.mark.parametrize("H,I", [(256, 512), (384, 640)])
def test_gemm_tile_edges_tiny(qtype, H, I):
    """8 experts, top-4, 4 slots: 2 waves; counts 256/129/128/127/1.  hidden 384 and intermediate
    640 (K steps 12 and 20) end both GEMMs' reductions on a half scale group, and their 12 gate
    scales per row are padded to 16 bytes before the up scales."""
    shape = Shape(1, H, 8, 4, I, qtype, model_seed=3)
    T = 256
    ctx = Ctx(shape, slots=4, max_tokens=T)
    try:
        ctx.mf.mf_prefill_threshold(ctx.h, 2)
        pays = Payloads(shape)
        lru = oracle.LRU(shape.n_experts, 4, synth.payload_bytes(shape.hidden, shape.inter, qtype))
        rng = np.random.default_rng(7)
        r = _boundary_routes(T, shape.n_experts, shape.top_k, rng)
        counts = np.bincount(r.reshape(-1), minlength=shape.n_experts)
        assert list(counts[:5]) == [256, 129, 128, 127, 1]
        x = synth.activations(11, 0, 0, 0, T, shape.hidden)
        bias = synth.plant_bias(r, shape.n_experts)
        _check_call(ctx, pays, lru, 0, x, bias, T)
        # second call: a different token count (ragged, 2 tokens), warm cache
        _check_call(ctx, pays, lru, 0, x[:2], bias[:2], 2)
        assert ctx.mf.mf_check(ctx.h) == 0
        st, ost = ctx.mf.mf_stats(ctx.h, 0), lru.stats()
        assert (st["accesses"], st["hits"], st["misses"], st["evictions"], st["bytes_materialized"]) == \
            (ost["accesses"], ost["hits"], ost["misses"], ost["evictions"], ost["bytes"])
    finally:
        ctx.close()


@pytest.mark.parametrize("qtype", [synth.Q8_0, synth.Q4_0])
def test_gemm_l4e64_shape(qtype):
    """hidden 2048, 64 experts, top-8, intermediate 768 (the 4-layer workload's shape), 22 slots:
    3 waves per call; Zipf 1.1 + 0.6 reuse routing gives hot experts several 128-blocks and
    cold ones a ragged few; 320 tokens on layer 0, then 300 on layer 1, all outputs checked."""
    cfg = synth.CONFIGS["l4e64"]
    shape = Shape(2, cfg.hidden, cfg.n_experts, cfg.top_k, cfg.inter, qtype, model_seed=1)
    ctx = Ctx(shape, slots=22, max_tokens=320)
    try:
        assert ctx.mf.mf_prefill_threshold(ctx.h, 256) is None
        pays = Payloads(shape)
        pay = synth.payload_bytes(shape.hidden, shape.inter, qtype)
        for layer, T in ((0, 320), (1, 300)):
            lru = oracle.LRU(shape.n_experts, 22, pay)
            klass = cfg.route_classes[0]
            r = synth.routes(5, layer, 0, shape.n_experts, shape.top_k, T, klass.zipf_s, klass.reuse)
            assert np.bincount(r.reshape(-1)).max() > 256  # a hot expert spans three column blocks
            x = synth.activations(5, layer, 0, 0, T, shape.hidden)
            _check_call(ctx, pays, lru, layer, x, synth.plant_bias(r, shape.n_experts), T)
        assert ctx.mf.mf_check(ctx.h) == 0
    finally:
        ctx.close()


def test_gemm_resident_first_order():
    """The GEMM path with the resident-first order: 2 calls of 320 tokens on one layer (the second
    with most experts resident), every output, index, access record and counter against the
    oracle in that order."""
    cfg = synth.CONFIGS["l4e64"]
    shape = Shape(1, cfg.hidden, cfg.n_experts, cfg.top_k, cfg.inter, synth.Q4_0, model_seed=4)
    ctx = Ctx(shape, slots=22, max_tokens=320)
    try:
        ctx.mf.mf_access_order(ctx.h, 1)
        pays = Payloads(shape)
        lru = oracle.LRU(shape.n_experts, 22, synth.payload_bytes(shape.hidden, shape.inter, shape.qtype))
        for call in range(2):
            r = synth.routes(8, 0, call, shape.n_experts, shape.top_k, 320, 1.1, 0.0)
            x = synth.activations(8, 0, call, 0, 320, shape.hidden)
            bias = synth.plant_bias(r, shape.n_experts)
            y, idx, w, tr = ctx.forward(0, x, bias, 320, trace=True)
            yo, oidx, og = oracle.layer(pays.for_layer(0, np.unique(idx)), shape.qtype, shape.hidden, shape.inter,
                                        shape.top_k, ctx.wr_host[0], bias, x)
            assert np.array_equal(idx, oidx) and np.abs(w - og).max() <= G_ATOL
            assert tr == oracle_trace(lru, idx, 1), call
            assert_outputs_close(y, yo, f"call {call}")
        st, ost = ctx.mf.mf_stats(ctx.h, 0), lru.stats()
        assert (st["hits"], st["misses"], st["evictions"]) == (ost["hits"], ost["misses"], ost["evictions"])
        assert ctx.mf.mf_check(ctx.h) == 0
    finally:
        ctx.close()


def test_gemm_matches_gemv_path():
    """Same inputs through the GEMM path and the GEMV path: same routes, access sequence and
    counters; outputs agree within the oracle tolerance of each other."""
    shape = Shape(1, 1024, 32, 8, 768, synth.Q8_0, model_seed=2)
    T = 384
    x = synth.activations(9, 0, 0, 0, T, shape.hidden)
    r = synth.routes(9, 0, 0, shape.n_experts, shape.top_k, T, 1.2, 0.0)
    bias = synth.plant_bias(r, shape.n_experts)
    outs = []
    for thr in (2, 0):
        ctx = Ctx(shape, slots=12, max_tokens=T)
        try:
            ctx.mf.mf_prefill_threshold(ctx.h, thr)
            y, idx, w, tr = ctx.forward(0, x, bias, T, trace=True)
            assert ctx.mf.mf_check(ctx.h) == 0
            outs.append((y, idx, w, tr, ctx.mf.mf_stats(ctx.h, 0)))
        finally:
            ctx.close()
    (yg, ig, wg, tg, sg), (yv, iv, wv, tv, sv) = outs
    assert np.array_equal(ig, iv) and np.array_equal(wg, wv) and tg == tv and sg == sv
    r = compare_outputs(yg, yv)
    assert r["ratio"] <= 1.0, r


def test_threshold_arguments():
    import paper_2607_09686_gb300 as mf
    shape = Shape(1, 256, 8, 2, 512, synth.Q8_0)
    ctx = Ctx(shape, slots=4, max_tokens=8)
    try:
        for bad in (1, -1):
            with pytest.raises(mf.MFError):
                mf.mf_prefill_threshold(ctx.h, bad)
        mf.mf_prefill_threshold(ctx.h, 0)
        mf.mf_prefill_threshold(ctx.h, 2)
    finally:
        ctx.close()
    one = Ctx(shape, slots=4, max_tokens=1)  # no GEMM scratch for one-token contexts
    try:
        with pytest.raises(mf.MFError):
            mf.mf_prefill_threshold(one.h, 2)
        mf.mf_prefill_threshold(one.h, 0)
    finally:
        one.close()
    odd = Ctx(Shape(1, 192, 8, 2, 512, synth.Q8_0), slots=4, max_tokens=8)  # hidden not a multiple of 128
    try:
        with pytest.raises(mf.MFError):
            mf.mf_prefill_threshold(odd.h, 2)
    finally:
        odd.close()
