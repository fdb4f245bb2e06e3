"""GPU path vs the CPU oracle, element by element, through the C ABI.

Routed indices, the per-access hit/miss/slot sequence and the counters must match exactly;
layer outputs and router weights within the stated tolerances (tests/mfharness.py)."""
import numpy as np
import pytest

import oracle
import synth
from mfharness import Ctx, Payloads, Shape, G_ATOL, assert_outputs_close, oracle_trace

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()


def _decode_run(shape, slots, n_tokens, seed, route=None, layers=None, sample_y=None, rng_seed=0):
    """Token-major batch-1 decode over `layers`; checks idx, traces and counters exactly and
    outputs on every token (sample_y=None) or on `sample_y` random (layer, token) pairs."""
    layers = list(range(shape.n_layers)) if layers is None else layers
    ctx = Ctx(shape, slots, max_tokens=1)
    pays = Payloads(shape)
    try:
        L, H, E, k = shape.n_layers, shape.hidden, shape.n_experts, shape.top_k
        xs = {l: synth.activations(seed, l, 0, 0, n_tokens, H) for l in layers}
        bias = {}
        for l in layers:
            bias[l] = None if route is None else synth.plant_bias(
                synth.routes(seed, l, 0, E, k, n_tokens, route.zipf_s, route.reuse), E)
        lru = {l: oracle.LRU(E, slots, synth.payload_bytes(H, shape.inter, shape.qtype)) for l in layers}
        rng = np.random.default_rng(rng_seed)
        pick = None
        if sample_y is not None:
            pick = set((int(layers[rng.integers(len(layers))]), int(rng.integers(n_tokens))) for _ in range(sample_y))
        n_checked = 0
        for t in range(n_tokens):
            for l in layers:
                b = None if bias[l] is None else bias[l][t:t + 1]
                y, idx, w, tr = ctx.forward(l, xs[l][t:t + 1], b, 1, trace=True)
                z, oidx, og = oracle.router(xs[l][t], ctx.wr_host[l], None if b is None else b[0], k)
                assert np.array_equal(idx[0], oidx), (l, t, idx[0], oidx, z[oidx])
                assert np.abs(w[0] - og).max() <= G_ATOL
                assert tr == oracle_trace(lru[l], idx), (l, t)
                if pick is None or (l, t) in pick:
                    yo, _, _ = oracle.layer(pays.for_layer(l, oidx), shape.qtype, H, shape.inter, k,
                                            ctx.wr_host[l], b, xs[l][t:t + 1])
                    assert_outputs_close(y, yo, f"layer {l} token {t}")
                    n_checked += 1
        assert ctx.mf.mf_check(ctx.h) == 0
        for l in layers:
            st = ctx.mf.mf_stats(ctx.h, l)
            ost = lru[l].stats()
            assert (st["accesses"], st["hits"], st["misses"], st["evictions"], st["bytes_materialized"]) == \
                (ost["accesses"], ost["hits"], ost["misses"], ost["evictions"], ost["bytes"])
        return n_checked
    finally:
        ctx.close()


def test_tiny_decode_real_routing():
    cfg = synth.CONFIGS["tiny"]
    assert _decode_run(Shape.of(cfg), cfg.slots, cfg.n_tokens, seed=0) == cfg.n_tokens


@pytest.mark.parametrize("pct", [15.0, 35.0])
def test_l4e64_decode(pct):
    cfg = synth.CONFIGS["l4e64"]
    S = int(np.floor(pct * cfg.n_experts / 100 + 1e-9))
    _decode_run(Shape.of(cfg), S, cfg.n_tokens, seed=0, route=cfg.route_classes[0], sample_y=48)


@pytest.mark.parametrize("kernels", ["fused", "pipelined", "simple"])
@pytest.mark.parametrize("qtype", [synth.Q8_0, synth.Q4_0])
def test_ragged_shapes_decode(qtype, kernels, monkeypatch):
    """Rows of 6 / 10 (Q8_0) and 3 / 5 (Q4_0) 16-byte vectors: partially filled warps.  The fused
    one-launch batch-1 kernel, the two pipelined kernels it replaces, and the one-warp-per-row
    kernels (used for shapes the pipelined ones do not take) are checked."""
    if kernels == "simple":
        monkeypatch.setenv("MF_DECODE_SIMPLE", "1")
    if kernels == "pipelined":
        monkeypatch.setenv("MF_DECODE_UNFUSED", "1")
    shape = Shape(2, 96, 12, 3, 160, qtype, model_seed=5)
    _decode_run(shape, 4, 40, seed=3)


@pytest.mark.parametrize("hidden", [2048, 4096])
@pytest.mark.parametrize("qtype", [synth.Q8_0, synth.Q4_0])
def test_fused_decode_x_split_widths(qtype, hidden):
    """The fused kernel splits x four values per thread where x has at most 512 such words
    (hidden 2048: every consumer thread one word) and one group per thread above that (hidden
    4096); both against the oracle."""
    _decode_run(Shape(1, hidden, 16, 4, 256, qtype, model_seed=12), 6, 12, seed=4)


@pytest.mark.parametrize("inter", [640, 768])
def test_fused_decode_half_warp_down_rows(inter):
    """Q8_0 down rows of 40 and 48 16-byte vectors (inter 640, 768): the fused kernel gives each
    half-warp a row and each lane three vectors (idle lanes in the 40-vector rows)."""
    _decode_run(Shape(2, 512, 16, 8, inter, synth.Q8_0, model_seed=13), 9, 10, seed=5)


@pytest.mark.parametrize("kernels", ["fused", "pipelined"])
def test_q4_0_decode_full_width(kernels, monkeypatch):
    """Q4_0 at hidden 2048 / intermediate 768 (the 48-layer Q4_0 shape), one layer, batch 1."""
    if kernels == "pipelined":
        monkeypatch.setenv("MF_DECODE_UNFUSED", "1")
    shape = Shape(1, 2048, 128, 8, 768, synth.Q4_0, model_seed=0)
    _decode_run(shape, 19, 24, seed=2, route=synth.configs.ZIPF12, sample_y=12)


def _batch_run(shape, slots, T, n_steps, seed, zipf_s=1.0, layers=None, sample_tokens=None, order=0):
    layers = list(range(shape.n_layers)) if layers is None else layers
    ctx = Ctx(shape, slots, max_tokens=T)
    pays = Payloads(shape)
    try:
        ctx.mf.mf_access_order(ctx.h, order)
        H, E, k = shape.hidden, shape.n_experts, shape.top_k
        lru = {l: oracle.LRU(E, slots, synth.payload_bytes(H, shape.inter, shape.qtype)) for l in layers}
        routes = {l: np.stack([synth.routes(seed, l, s, E, k, n_steps, zipf_s, 0.0) for s in range(T)], 1)
                  for l in layers}  # [steps, T, k]
        for step in range(n_steps):
            for l in layers:
                x = np.concatenate([synth.activations(seed, l, s, step, 1, H) for s in range(T)])
                b = synth.plant_bias(routes[l][step], E)
                y, idx, w, tr = ctx.forward(l, x, b, T, trace=True)
                for t in range(T):
                    _, oidx, og = oracle.router(x[t], ctx.wr_host[l], b[t], k)
                    assert np.array_equal(idx[t], oidx)
                    assert np.abs(w[t] - og).max() <= G_ATOL
                assert tr == oracle_trace(lru[l], idx, order), (l, step)
                toks = range(T) if sample_tokens is None else sorted(
                    set(np.random.default_rng(step * 131 + l).integers(0, T, sample_tokens).tolist()))
                for t in toks:
                    yo, _, _ = oracle.layer(pays.for_layer(l, idx[t]), shape.qtype, H, shape.inter, k,
                                            ctx.wr_host[l], b[t:t + 1], x[t:t + 1])
                    assert_outputs_close(y[t:t + 1], yo, f"layer {l} step {step} token {t}")
        out = []
        for l in layers:
            st, ost = ctx.mf.mf_stats(ctx.h, l), lru[l].stats()
            assert (st["hits"], st["misses"], st["evictions"], st["bytes_materialized"]) == \
                (ost["hits"], ost["misses"], ost["evictions"], ost["bytes"])
            out.append(st)
        return out
    finally:
        ctx.close()


@pytest.mark.parametrize("qtype", [synth.Q8_0, synth.Q4_0])
def test_batched_steps_in_waves(qtype):
    """16 tokens x top-3 over 12 experts with 4 slots: up to 3 waves per step."""
    _batch_run(Shape(2, 96, 12, 3, 160, qtype, model_seed=9), 4, 16, 6, seed=1, zipf_s=0.5)


@pytest.mark.parametrize("qtype", [synth.Q8_0, synth.Q4_0])
def test_batched_steps_resident_first(qtype):
    """The same batched steps with the resident-first access order: routes, traces (access order,
    slots, hits), counters and outputs against the oracle in that order; never fewer hits than
    the first-occurrence order on these steps."""
    shape = Shape(2, 96, 12, 3, 160, qtype, model_seed=9)
    rf = _batch_run(shape, 4, 16, 6, seed=1, zipf_s=0.5, order=1)
    fo = _batch_run(shape, 4, 16, 6, seed=1, zipf_s=0.5, order=0)
    assert sum(s["hits"] for s in rf) >= sum(s["hits"] for s in fo)


def test_max_experts_and_many_waves():
    """1024 experts (the largest supported), top-8, 8 slots: a 64-token step touches up to 512 experts."""
    _batch_run(Shape(1, 64, 1024, 8, 64, synth.Q8_0, model_seed=2), 8, 64, 2, seed=4, zipf_s=0.3)


def test_host_buffer_entry_point_matches_device_entry_point():
    cfg = synth.CONFIGS["tiny"]
    shape = Shape.of(cfg)
    a, b = Ctx(shape, 4, max_tokens=8), Ctx(shape, 4, max_tokens=8)
    try:
        import paper_2607_09686_gb300 as mf
        for t in range(6):
            x = synth.activations(0, 0, 0, t * 8, 8, cfg.hidden)
            y1, i1, w1 = a.forward(0, x, None, 8)
            y2 = np.empty_like(y1)
            i2 = np.empty_like(i1)
            w2 = np.empty_like(w1)
            mf.mf_moe_forward_host(b.h, 0, x, b.wr[0], None, 8, y2, i2, w2)
            b.torch.cuda.synchronize()
            assert np.array_equal(y1, y2) and np.array_equal(i1, i2) and np.array_equal(w1, w2)
        assert mf.mf_stats(a.h) == mf.mf_stats(b.h)
    finally:
        a.close()
        b.close()


@pytest.mark.parametrize("pinned", [True, False])
def test_host_entry_point_one_token(pinned):
    """One token per call through the host-buffer entry point, with pinned buffers (the kernels
    read x and the bias and write y over the CPU-GPU link, no copy steps) and with pageable ones
    (staged copies): bit-identical to the device entry point, misses included."""
    shape = Shape(2, 1024, 32, 8, 512, synth.Q8_0, model_seed=6)
    a, b = Ctx(shape, 12, max_tokens=1), Ctx(shape, 12, max_tokens=1)
    try:
        import torch
        import paper_2607_09686_gb300 as mf
        T = 16
        for l in range(shape.n_layers):
            xs = synth.activations(2, l, 0, 0, T, shape.hidden)
            bs = synth.plant_bias(synth.routes(2, l, 0, shape.n_experts, shape.top_k, T, 1.1, 0.3), shape.n_experts)
            for t in range(T):
                y1, i1, w1 = a.forward(l, xs[t:t + 1], bs[t:t + 1], 1)
                if pinned:
                    xh = torch.from_numpy(xs[t:t + 1].copy()).pin_memory()
                    bh = torch.from_numpy(bs[t:t + 1].copy()).pin_memory()
                    yh = torch.empty(1, shape.hidden).pin_memory()
                    ih = torch.empty(1, shape.top_k, dtype=torch.int32).pin_memory()
                    wh = torch.empty(1, shape.top_k).pin_memory()
                    mf.mf_moe_forward_host(b.h, l, xh, b.wr[l], bh, 1, yh, ih, wh)
                    torch.cuda.synchronize()
                    y2, i2, w2 = yh.numpy(), ih.numpy(), wh.numpy()
                else:
                    y2 = np.empty_like(y1)
                    i2 = np.empty_like(i1)
                    w2 = np.empty_like(w1)
                    mf.mf_moe_forward_host(b.h, l, xs[t:t + 1].copy(), b.wr[l], bs[t:t + 1].copy(), 1, y2, i2, w2)
                    torch.cuda.synchronize()
                assert np.array_equal(y1, y2) and np.array_equal(i1, i2) and np.array_equal(w1, w2), (l, t)
        assert mf.mf_check(b.h) == 0
        assert mf.mf_stats(a.h) == mf.mf_stats(b.h) and mf.mf_stats(a.h)["misses"] > 0
    finally:
        a.close()
        b.close()


def test_reset_replays_and_empty_step():
    cfg = synth.CONFIGS["tiny"]
    ctx = Ctx(Shape.of(cfg), 4, max_tokens=4)
    try:
        mf = ctx.mf
        x = synth.activations(7, 0, 0, 0, 12, cfg.hidden)
        first = [ctx.forward(0, x[t:t + 1], None, 1, trace=True) for t in range(12)]
        s1 = mf.mf_stats(ctx.h, -1, reset=True)
        assert mf.mf_stats(ctx.h, -1)["accesses"] == 0
        mf.mf_reset(ctx.h)
        second = [ctx.forward(0, x[t:t + 1], None, 1, trace=True) for t in range(12)]
        for f, s in zip(first, second):
            assert all(np.array_equal(p, q) for p, q in zip(f[:3], s[:3])) and f[3] == s[3]
        assert mf.mf_stats(ctx.h, -1) == s1
        # T = 0 is a no-op: counters and the trace stay as they were
        ctx.forward(0, x[:0], None, 0)
        assert mf.mf_stats(ctx.h, -1) == s1
        # fewer slots in use after a reset
        mf.mf_reset(ctx.h, 2)
        lru = oracle.LRU(cfg.n_experts, 2, ctx.plan.payload_bytes)
        for t in range(12):
            _, idx, _, tr = ctx.forward(0, x[t:t + 1], None, 1, trace=True)
            assert tr == oracle_trace(lru, idx)
    finally:
        ctx.close()


def test_argument_and_state_errors():
    import torch
    import paper_2607_09686_gb300 as mf
    cfg = synth.CONFIGS["tiny"]
    model = mf.Model(1, cfg.hidden, cfg.n_experts, cfg.top_k, cfg.inter, cfg.qtype)
    rejected = mf.mf_plan(model, mf.PlanReq(50.0, 10, 0, 0, 1, 0))
    with pytest.raises(mf.MFError) as e:
        mf.mf_create(model, rejected, 0)
    assert e.value.status == mf.MF_E_BUDGET
    plan = mf.mf_plan(model, mf.PlanReq(50.0, 1 << 40, 0, 0, 2, 0))
    h = mf.mf_create(model, plan, 0)
    try:
        x = torch.zeros(2, cfg.hidden, device="cuda")
        wr = torch.zeros(cfg.n_experts, cfg.hidden, device="cuda")
        y = torch.empty(2, cfg.hidden, device="cuda")
        with pytest.raises(mf.MFError) as e:  # pack not filled yet
            mf.mf_moe_forward(h, 0, x, wr, None, 1, y)
        assert e.value.status == mf.MF_E_STATE
        pays = [synth.payload(0, 0, e_, cfg.hidden, cfg.inter, cfg.qtype) for e_ in range(cfg.n_experts)]
        for e_, p in enumerate(pays):
            mf.mf_pack_put(h, 0, e_, p)
        with pytest.raises(mf.MFError):
            mf.mf_pack_put(h, 0, 0, pays[0][:-1])  # wrong size
        for bad in (dict(layer=1), dict(T=3), dict(T=-1)):
            kw = dict(layer=0, T=1)
            kw.update(bad)
            with pytest.raises(mf.MFError) as e:
                mf.mf_moe_forward(h, kw["layer"], x, wr, None, kw["T"], y)
            assert e.value.status == mf.MF_E_INVAL
        with pytest.raises(mf.MFError):  # x not 16-byte aligned
            mf.mf_moe_forward(h, 0, x.data_ptr() + 4, wr, None, 1, y)
        mf.mf_moe_forward(h, 0, x, wr, None, 1, y)
        torch.cuda.synchronize()
        with pytest.raises(mf.MFError):
            mf.mf_reset(h, 1)  # fewer slots than top-k
        for bad in (-1, 2):
            with pytest.raises(mf.MFError) as e:
                mf.mf_access_order(h, bad)
            assert e.value.status == mf.MF_E_INVAL
        mf.mf_access_order(h, mf.MF_ORDER_RESIDENT_FIRST)
        mf.mf_access_order(h, mf.MF_ORDER_FIRST_OCCURRENCE)
    finally:
        mf.mf_destroy(h)
