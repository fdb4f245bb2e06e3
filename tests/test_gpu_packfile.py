"""The disk tier of the split-pack: mf_pack_save writes the payloads to a file (header, index,
records) and mf_create_from_file serves a context's misses from it (section "Split-Pack
Representation"; the Introduction's hierarchy of disk, memory and slots).

A file-backed context must compute exactly what a context with the pinned pack computes: the
same routed indices, access records, counters and (bit for bit) outputs, for one-token calls
through the fused kernel and through the separate kernels, for batched calls in waves, eagerly
and in a CUDA graph, and the same as the oracle.  Its reads are one record per miss."""
import os

import numpy as np
import pytest

import oracle
import synth
from mfharness import Ctx, Payloads, Shape, assert_outputs_close, oracle_trace

pytestmark = pytest.mark.gpu
SHAPE = Shape(2, 256, 16, 4, 256, synth.Q8_0, model_seed=31)


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()


def _call(mf, h, wr, layer, x, b, T, dev):
    import torch
    xd = torch.from_numpy(np.ascontiguousarray(x, np.float32)).to(dev)
    bd = torch.from_numpy(np.ascontiguousarray(b, np.float32)).to(dev)
    y = torch.empty(T, SHAPE.hidden, device=dev)
    idx = torch.empty(T, SHAPE.top_k, dtype=torch.int32, device=dev)
    mf.mf_moe_forward(h, layer, xd, wr, bd, T, y, idx, None)
    torch.cuda.synchronize()
    return y.cpu().numpy(), idx.cpu().numpy()


def _sequence(T, n_steps, seed):
    L, H, E, k = SHAPE.n_layers, SHAPE.hidden, SHAPE.n_experts, SHAPE.top_k
    out = []
    for l in range(L):
        r = np.stack([synth.routes(seed, l, s, E, k, n_steps, 1.1, 0.0) for s in range(T)], 1)  # [steps, T, k]
        x = [np.concatenate([synth.activations(seed, l, s, t, 1, H) for s in range(T)]) for t in range(n_steps)]
        out.append((x, [synth.plant_bias(r[t], E) for t in range(n_steps)]))
    return out


@pytest.mark.parametrize("T,kernels", [(1, "fused"), (1, "unfused"), (4, "batched")])
def test_file_backed_context_matches_the_pinned_pack(tmp_path, monkeypatch, T, kernels):
    if kernels == "unfused":
        monkeypatch.setenv("MF_DECODE_UNFUSED", "1")
    ctx = Ctx(SHAPE, 5, max_tokens=T)
    mf, dev = ctx.mf, ctx.device
    path = str(tmp_path / "experts.mfpack")
    fh = None
    try:
        mf.mf_pack_save(ctx.h, path)
        fh = mf.mf_create_from_file(ctx.model, ctx.plan, path, 0)
        seq = _sequence(T, 12, seed=4)
        pays = Payloads(SHAPE)
        lru = [oracle.LRU(SHAPE.n_experts, 5, synth.payload_bytes(SHAPE.hidden, SHAPE.inter, SHAPE.qtype))
               for _ in range(SHAPE.n_layers)]
        for step in range(12):
            for l in range(SHAPE.n_layers):
                x, b = seq[l][0][step], seq[l][1][step]
                y0, i0 = _call(mf, ctx.h, ctx.wr[l], l, x, b, T, dev)
                y1, i1 = _call(mf, fh, ctx.wr[l], l, x, b, T, dev)
                assert np.array_equal(i0, i1) and np.array_equal(y0, y1), (l, step)
                tr = mf.mf_trace(fh, l, cap=SHAPE.n_experts)
                assert tr == mf.mf_trace(ctx.h, l, cap=SHAPE.n_experts)
                assert tr == oracle_trace(lru[l], i1)
                if step % 4 == 0:
                    yo, oidx, _ = oracle.layer(pays.for_layer(l, range(SHAPE.n_experts)), SHAPE.qtype, SHAPE.hidden,
                                               SHAPE.inter, SHAPE.top_k, ctx.wr_host[l], b, x)
                    assert np.array_equal(i1, oidx)
                    assert_outputs_close(y1, yo, f"file-backed layer {l} step {step}")
        assert mf.mf_check(fh) == 0 and mf.mf_check(ctx.h) == 0
        st0, st1 = mf.mf_stats(ctx.h, -1), mf.mf_stats(fh, -1)
        assert st0 == st1 and st1["misses"] > 0
        fs = mf.mf_pack_file_stats(fh)
        assert fs["reads"] == st1["misses"]
        assert fs["bytes"] % fs["reads"] == 0 and fs["bytes"] // fs["reads"] % 4096 == 0
    finally:
        if fh:
            mf.mf_destroy(fh)
        ctx.close()


def test_file_backed_calls_in_a_graph(tmp_path):
    """Captured calls re-read their misses on every replay (the reads are host nodes)."""
    import torch
    ctx = Ctx(SHAPE, 4, max_tokens=1)
    mf, dev = ctx.mf, ctx.device
    path = str(tmp_path / "experts.mfpack")
    fh = None
    try:
        mf.mf_pack_save(ctx.h, path)
        fh = mf.mf_create_from_file(ctx.model, ctx.plan, path, 0)
        n = 10
        seq = _sequence(1, n, seed=9)
        xs = [torch.from_numpy(np.stack([seq[l][0][t][0] for t in range(n)])).to(dev) for l in range(SHAPE.n_layers)]
        bs = [torch.from_numpy(np.stack([seq[l][1][t][0] for t in range(n)])).to(dev) for l in range(SHAPE.n_layers)]
        y = torch.empty(n, SHAPE.n_layers, SHAPE.hidden, device=dev)
        s = torch.cuda.Stream()

        def calls(h):
            mf.mf_reset(h, 0, s)
            for t in range(n):
                for l in range(SHAPE.n_layers):
                    mf.mf_moe_forward(h, l, xs[l][t], ctx.wr[l], bs[l][t], 1, y[t, l], None, None, s)

        with torch.cuda.stream(s):
            calls(ctx.h)
        s.synchronize()
        ref = y.clone()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.stream(s):
            calls(fh)  # warm-up, eager
            s.synchronize()
            with torch.cuda.graph(g, stream=s):
                calls(fh)
        for _ in range(2):
            y.zero_()
            g.replay()
            torch.cuda.synchronize()
            assert torch.equal(y, ref)
        assert mf.mf_check(fh) == 0
        assert mf.mf_stats(fh, -1) == mf.mf_stats(ctx.h, -1)
        del g
    finally:
        if fh:
            mf.mf_destroy(fh)
        ctx.close()


def test_pack_file_errors(tmp_path):
    import paper_2607_09686_gb300 as mf
    ctx = Ctx(SHAPE, 4, max_tokens=1)
    path = str(tmp_path / "experts.mfpack")
    fh = None
    try:
        mf.mf_pack_save(ctx.h, path)
        with pytest.raises(mf.MFError) as e:  # a file that does not exist
            mf.mf_create_from_file(ctx.model, ctx.plan, str(tmp_path / "missing"), 0)
        assert e.value.status == mf.MF_E_INVAL
        other = mf.Model(SHAPE.n_layers, SHAPE.hidden, SHAPE.n_experts, SHAPE.top_k, SHAPE.inter + 32, SHAPE.qtype)
        oplan = mf.mf_plan(other, mf.PlanReq(25.0, 1 << 62, 0, 0, 1, 0))
        with pytest.raises(mf.MFError) as e:  # a file of another model
            mf.mf_create_from_file(other, oplan, path, 0)
        assert e.value.status == mf.MF_E_INVAL
        short = str(tmp_path / "short.mfpack")
        with open(path, "rb") as src, open(short, "wb") as dst:
            dst.write(src.read(os.path.getsize(path) - 4096))
        with pytest.raises(mf.MFError) as e:  # truncated
            mf.mf_create_from_file(ctx.model, ctx.plan, short, 0)
        assert e.value.status == mf.MF_E_INVAL
        bad = str(tmp_path / "bad.mfpack")
        with open(path, "rb") as src, open(bad, "wb") as dst:
            data = bytearray(src.read())
            data[0] ^= 0xFF
            dst.write(data)
        with pytest.raises(mf.MFError) as e:  # not a split-pack file
            mf.mf_create_from_file(ctx.model, ctx.plan, bad, 0)
        assert e.value.status == mf.MF_E_INVAL
        fh = mf.mf_create_from_file(ctx.model, ctx.plan, path, 0)
        with pytest.raises(mf.MFError) as e:  # the file-backed pack is read-only
            mf.mf_pack_put(fh, 0, 0, synth.payload(0, 0, 0, SHAPE.hidden, SHAPE.inter, SHAPE.qtype))
        assert e.value.status == mf.MF_E_STATE
        with pytest.raises(mf.MFError) as e:
            mf.mf_pack_save(fh, str(tmp_path / "again.mfpack"))
        assert e.value.status == mf.MF_E_STATE
        empty = mf.mf_create(ctx.model, ctx.plan, 0)
        try:
            with pytest.raises(mf.MFError) as e:  # payloads not put yet
                mf.mf_pack_save(empty, str(tmp_path / "empty.mfpack"))
            assert e.value.status == mf.MF_E_STATE
        finally:
            mf.mf_destroy(empty)
        assert mf.mf_pack_file_stats(fh)["reads"] == 0
        with pytest.raises(mf.MFError):
            mf.mf_pack_file_stats(ctx.h)
    finally:
        if fh:
            mf.mf_destroy(fh)
        ctx.close()
