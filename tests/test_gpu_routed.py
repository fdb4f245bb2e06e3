"""One-token calls routed inside the fused kernel: the router, the slot replacement and the expert
FFN (with the misses' materialisation) in one launch (Background section: per-token top-k
routing; section "Native Serving Path": least-recently-used slots, misses materialised into
them).

Every block of that launch computes some of the logits, then all of them rank the k largest and
replay the layer's replacement on their own copy of the cache state.  The launch must give the
router kernel's bits: the same routed indices, weights and outputs (bit for bit: the logits are
summed in the router's order), the same access records, counters and cache state, on
sequences where a miss evicts an expert that a later rank of the same call had found resident,
with E above the number of blocks (blocks that compute several logits), with x split in two
rounds (H = 4096), eagerly and in a CUDA graph; and the outputs must match the oracle."""
import numpy as np
import pytest

import oracle
import synth
from mfharness import Ctx, Payloads, Shape, assert_outputs_close, oracle_trace, stats_tuple

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()


def _pair(shape, slots, monkeypatch):
    """(routed context, router-kernel context) over the same payloads."""
    monkeypatch.setenv("MF_DECODE_ROUTER", "1")
    ref = Ctx(shape, slots, max_tokens=1)
    monkeypatch.delenv("MF_DECODE_ROUTER")
    return Ctx(shape, slots, max_tokens=1), ref


def _inputs(shape, n, seed, zipf=1.1, reuse=0.3):
    L, H, E, k = shape.n_layers, shape.hidden, shape.n_experts, shape.top_k
    xs = [synth.activations(seed, l, 0, 0, n, H) for l in range(L)]
    bs = [synth.plant_bias(synth.routes(seed, l, 0, E, k, n, zipf, reuse), E) for l in range(L)]
    return xs, bs


CASES = {
    # name: (shape, slots, calls per layer)
    "q8_tight": (Shape(3, 256, 16, 4, 256, synth.Q8_0, model_seed=41), 5, 24),
    "q4_tight": (Shape(2, 256, 16, 4, 512, synth.Q4_0, model_seed=42), 6, 20),
    "q8_e200": (Shape(1, 256, 200, 8, 256, synth.Q8_0, model_seed=43), 24, 16),
    "q8_h4096": (Shape(1, 4096, 16, 4, 256, synth.Q8_0, model_seed=44), 6, 10),
}


@pytest.mark.parametrize("case", list(CASES))
def test_routed_call_matches_the_router_kernel(case, monkeypatch):
    shape, slots, n = CASES[case]
    L, H, E, k = shape.n_layers, shape.hidden, shape.n_experts, shape.top_k
    routed, ref = _pair(shape, slots, monkeypatch)
    pays = Payloads(shape)
    try:
        xs, bs = _inputs(shape, n, seed=7)
        lru = [oracle.LRU(E, slots, synth.payload_bytes(H, shape.inter, shape.qtype)) for _ in range(L)]
        evicted_later = 0  # calls where a miss evicted an expert that a later rank found resident
        for t in range(n):
            for l in range(L):
                x, b = xs[l][t:t + 1], bs[l][t:t + 1]
                y1, i1, w1, tr1 = routed.forward(l, x, b, 1, trace=True)
                y0, i0, w0, tr0 = ref.forward(l, x, b, 1, trace=True)
                assert np.array_equal(i1, i0) and np.array_equal(w1, w0), (case, l, t)
                assert np.array_equal(y1, y0), (case, l, t)  # bit for bit
                assert tr1 == tr0, (case, l, t)
                before = set(int(e) for e in lru[l].slots() if e >= 0)
                assert tr1 == oracle_trace(lru[l], i1), (case, l, t)
                evicted_later += any(not h and e in before for e, h in zip(tr1[0], tr1[2]))
                if t % 5 == 0:
                    yo, oidx, _ = oracle.layer(pays.for_layer(l, range(E)), shape.qtype, H, shape.inter, k,
                                               routed.wr_host[l], b, x)
                    assert np.array_equal(i1, oidx)
                    assert_outputs_close(y1, yo, f"{case} layer {l} call {t}")
        assert routed.mf.mf_check(routed.h) == 0 and ref.mf.mf_check(ref.h) == 0
        for l in range(L):
            st = routed.mf.mf_stats(routed.h, l)
            assert st == ref.mf.mf_stats(ref.h, l)
            assert stats_tuple(st) == stats_tuple(lru[l].stats()), (case, l)
        if case.endswith("tight"):
            assert evicted_later > 0, "the sequence never evicted a later rank's resident expert"
    finally:
        routed.close()
        ref.close()


def test_routed_calls_in_a_graph(monkeypatch):
    """A captured sequence (cache reset included) replays to the eager router kernel's outputs,
    and leaves the same counters."""
    import torch
    shape, slots, n = CASES["q8_tight"]
    L, E = shape.n_layers, shape.n_experts
    routed, ref = _pair(shape, slots, monkeypatch)
    try:
        dev = routed.device
        xs, bs = _inputs(shape, n, seed=8)
        xd = [torch.from_numpy(x).to(dev) for x in xs]
        bd = [torch.from_numpy(b).to(dev) for b in bs]
        y = torch.empty(n, L, shape.hidden, device=dev)
        idx = torch.empty(n, L, shape.top_k, dtype=torch.int32, device=dev)
        s = torch.cuda.Stream()

        def calls(c):
            c.mf.mf_reset(c.h, 0, s)
            for t in range(n):
                for l in range(L):
                    c.mf.mf_moe_forward(c.h, l, xd[l][t], c.wr[l], bd[l][t], 1, y[t, l], idx[t, l], None, s)

        with torch.cuda.stream(s):
            calls(ref)
        s.synchronize()
        y_ref, idx_ref = y.clone(), idx.clone()
        st_ref = ref.mf.mf_stats(ref.h, -1)
        g = torch.cuda.CUDAGraph()
        with torch.cuda.stream(s):
            calls(routed)  # eager warm-up
            s.synchronize()
            with torch.cuda.graph(g, stream=s):
                calls(routed)
        for _ in range(2):
            y.zero_()
            idx.zero_()
            routed.mf.mf_stats(routed.h, -1, reset=True)
            g.replay()
            torch.cuda.synchronize()
            assert torch.equal(y, y_ref) and torch.equal(idx, idx_ref)
            assert routed.mf.mf_stats(routed.h, -1) == st_ref
        assert routed.mf.mf_check(routed.h) == 0
        del g
    finally:
        routed.close()
        ref.close()
