"""The cache-size tuner (mf_tune_cache, host code of the library) against the oracle: for every
candidate cache size its replay of a route trace must give the oracle LRU's accesses, hits and
misses exactly (both access orders, one and several tokens per step, steps wider than the
cache), its plan decisions must be the oracle planner's, and its prediction must follow the
throughput relation of section "Throughput Model" with the measured times it is given.  No GPU."""
import ctypes

import numpy as np
import pytest

import oracle
import synth
import __graft_entry__


@pytest.fixture(scope="module")
def mf():
    __graft_entry__.build()
    import paper_2607_09686_gb300 as pkg
    return pkg


def _oracle_replay(routes, E, S, T, order):
    """accesses, hits, misses of the oracle LRU over the trace, layer by layer, steps of T tokens."""
    acc = hits = misses = 0
    for l in range(routes.shape[0]):
        lru = oracle.LRU(E, S, 1)
        for t0 in range(0, routes.shape[1], T):
            lru.step(routes[l, t0:t0 + T], order=order)
        st = lru.stats()
        acc, hits, misses = acc + st["accesses"], hits + st["hits"], misses + st["misses"]
    return acc, hits, misses


def _trace(L, E, k, n, zipf_s, reuse, seed=3):
    return np.stack([synth.routes(seed, l, 0, E, k, n, zipf_s, reuse) for l in range(L)]).astype(np.int32)


@pytest.mark.parametrize("order", [0, 1])
@pytest.mark.parametrize("T,zipf_s,reuse", [(1, 1.1, 0.6), (1, 0.0, 0.0), (4, 1.0, 0.0), (7, 1.2, 0.3), (64, 0.8, 0.0),
                                            (199, 1.0, 0.0)])
def test_replay_matches_oracle_lru(mf, order, T, zipf_s, reuse):
    """2 layers, 32 experts, top-4, 200 tokens; T = 64 makes steps of up to 32 distinct experts
    against caches of 4..32 slots (several waves per step); T = 199 ends on a one-token step,
    which keeps first-occurrence order whatever the order."""
    L, E, k, n = 2, 32, 4, 200
    model = mf.Model(L, 256, E, k, 512, mf.Q8_0)
    routes = _trace(L, E, k, n, zipf_s, reuse)
    pcts = [0.0, 12.5, 15.0, 25.0, 40.0, 50.0, 75.0, 100.0]
    pts, best = mf.mf_tune_cache(model, mf.PlanReq(0.0, 1 << 62, 0, 0, 64, 0), routes, T, 1e-4, 1e-3, pcts, order)
    for p, pt in zip(pcts, pts):
        o = oracle.plan(L, 256, E, k, 512, mf.Q8_0, p, 1 << 62, 0, 0)
        assert (pt["slots_per_layer"], bool(pt["accepted"]), pt["pool_bytes"]) == (o["slots"], o["accepted"], o["pool"])
        assert (pt["accesses"], pt["hits"], pt["misses"]) == _oracle_replay(routes, E, o["slots"], T, order), p
        assert pt["bytes_materialized"] == pt["misses"] * o["payload"]
    assert best >= 0


def test_replay_of_the_decode_workload_in_router_order(mf):
    """The 4-layer decode workload (64 experts, top-8, 256 tokens, Zipf 1.1 + 0.6 reuse): the
    trace is the oracle router's output for the planted bias, in its rank order (the order the
    cache sees), replayed at 15, 25, 35, 50 and 100 %."""
    c = synth.CONFIGS["l4e64"]
    rc = c.route_classes[0]
    L, H, E, k = c.n_layers, c.hidden, c.n_experts, c.top_k
    routes = np.empty((L, c.n_tokens, k), np.int32)
    for l in range(L):
        b = synth.plant_bias(synth.routes(0, l, 0, E, k, c.n_tokens, rc.zipf_s, rc.reuse), E)
        x = synth.activations(0, l, 0, 0, c.n_tokens, H)
        wr = synth.router_weights(c.model_seed, l, E, H)
        for t in range(c.n_tokens):
            routes[l, t] = oracle.router(x[t], wr, b[t], k)[1]
    model = mf.Model(L, H, E, k, c.inter, c.qtype)
    pcts = [15.0, 25.0, 35.0, 50.0, 100.0]
    pts, _ = mf.mf_tune_cache(model, mf.PlanReq(0.0, 1 << 62, 0, 0, 1, 0), routes, 1, 1e-4, 1e-3, pcts)
    for pt in pts:
        S = pt["slots_per_layer"]
        assert (pt["accesses"], pt["hits"], pt["misses"]) == _oracle_replay(routes, E, S, 1, 0), pt["cache_pct"]


def test_prediction_closed_form(mf):
    """Full reuse at batch 1 (every token routes to the same k experts) with S >= k: only the
    first token of each layer misses, so misses = L k and the predicted time is
    n t_token + L k t_miss (section "Throughput Model", no pressure term)."""
    L, E, k, n = 3, 16, 4, 50
    routes = np.tile(np.array([5, 1, 9, 12], np.int32), (L, n, 1))
    model = mf.Model(L, 256, E, k, 512, mf.Q4_0)
    t_tok, t_miss = 2.5e-4, 7.5e-3
    pts, best = mf.mf_tune_cache(model, mf.PlanReq(0.0, 1 << 62, 0, 0, 1, 0), routes, 1, t_tok, t_miss,
                                 [25.0, 50.0, 100.0])
    for pt in pts:
        assert (pt["accesses"], pt["misses"]) == (L * n * k, L * k)
        assert pt["predicted_s"] == pytest.approx(n * t_tok + L * k * t_miss, rel=1e-15)
        assert pt["predicted_tokens_per_s"] == pytest.approx(n / (n * t_tok + L * k * t_miss), rel=1e-15)
    assert best == 0  # equal predictions: the smallest pool


def _is_choice(pts, best):
    """best has the fewest misses among the accepted candidates, and the smallest pool among those."""
    acc = [p for p in pts if p["accepted"]]
    fewest = min(p["misses"] for p in acc)
    return pts[best]["misses"] == fewest and pts[best]["pool_bytes"] == min(
        p["pool_bytes"] for p in acc if p["misses"] == fewest)


def test_choice_follows_budget_and_latency(mf):
    """Misses never increase with S (LRU inclusion), so with a positive miss time the choice is
    the accepted candidate with the fewest misses (the smallest pool among equals); a budget that
    rejects the large caches restricts it to the accepted ones; with a zero miss time every
    candidate predicts the same rate and the smallest pool wins; equal pools (same S) keep the
    earlier candidate."""
    L, E, k, n = 2, 32, 4, 300
    routes = _trace(L, E, k, n, 1.0, 0.2, seed=9)
    model = mf.Model(L, 256, E, k, 512, mf.Q8_0)
    pcts = [float(p) for p in range(0, 101, 5)]
    pts, best = mf.mf_tune_cache(model, mf.PlanReq(0.0, 1 << 62, 0, 0, 1, 0), routes, 1, 1e-4, 1e-3, pcts)
    misses = [pt["misses"] for pt in pts]
    assert all(a >= b for a, b in zip(misses, misses[1:]))
    assert _is_choice(pts, best)
    payload = oracle.payload_bytes(256, 512, mf.Q8_0)
    budget = L * 16 * payload  # pools of at most 16 slots per layer
    pts2, best2 = mf.mf_tune_cache(model, mf.PlanReq(0.0, budget, 0, 0, 1, 0), routes, 1, 1e-4, 1e-3, pcts)
    assert [bool(p["accepted"]) for p in pts2] == [p["slots_per_layer"] <= 16 for p in pts2]
    assert _is_choice(pts2, best2) and pts2[best2]["slots_per_layer"] <= 16
    _, best3 = mf.mf_tune_cache(model, mf.PlanReq(0.0, 1 << 62, 0, 0, 1, 0), routes, 1, 1e-4, 0.0, pcts)
    assert best3 == 0  # S = k for p = 0: the smallest pool
    _, best4 = mf.mf_tune_cache(model, mf.PlanReq(0.0, 1 << 62, 0, 0, 1, 0), routes, 1, 1e-4, 1e-3,
                                [100.0, 12.5, 100.0])
    assert best4 == 0


def test_none_accepted_and_bad_arguments(mf):
    lib = ctypes.CDLL(mf.LIB_PATH)
    L, E, k, n = 1, 8, 2, 10
    model = mf.Model(L, 256, E, k, 512, mf.Q8_0)
    routes = _trace(L, E, k, n, 0.0, 0.0)
    pts, best = mf.mf_tune_cache(model, mf.PlanReq(0.0, 10, 0, 0, 1, 0), routes, 1, 1e-4, 1e-3, [10.0, 50.0])
    assert best == -1 and not any(p["accepted"] for p in pts) and pts[1]["slots_per_layer"] == 4

    def call(routes=routes, n_tokens=n, T=1, order=0, t_tok=1e-4, t_miss=1e-3, pcts=(50.0,), model=model):
        r = np.ascontiguousarray(routes, np.int32)
        cand = (ctypes.c_double * max(1, len(pcts)))(*pcts)
        out = (mf.TunePoint * max(1, len(pcts)))()
        b = ctypes.c_int(7)
        rc = lib.mf_tune_cache(ctypes.byref(model), ctypes.byref(mf.PlanReq(0.0, 1 << 62, 0, 0, 1, 0)),
                               ctypes.c_void_p(r.ctypes.data), n_tokens, T, order, ctypes.c_double(t_tok),
                               ctypes.c_double(t_miss), cand, len(pcts), out, ctypes.byref(b))
        return rc, b.value

    lib.mf_tune_cache.restype = ctypes.c_int
    assert call() == (0, 0)
    bad = routes.copy()
    bad[0, 3, 1] = E
    assert call(routes=bad)[0] == -1
    bad[0, 3, 1] = -1
    assert call(routes=bad)[0] == -1
    assert call(n_tokens=0)[0] == -1
    assert call(T=0)[0] == -1
    assert call(order=2)[0] == -1
    assert call(t_tok=-1.0)[0] == -1
    assert call(t_miss=float("nan"))[0] == -1
    assert call(t_tok=float("inf"))[0] == -1
    assert call(pcts=())[0] == -1
    assert call(pcts=(101.0,))[0] == -1
    assert call(model=mf.Model(1, 200, E, k, 512, mf.Q8_0))[0] == -1


def test_batched_workload_under_its_pool_cap(mf):
    """The 30-layer, 64-stream workload (128 experts, top-8) under a 12 GiB slot-pool cap with
    the router weights resident: the static check accepts 15 % only, so the choice is 15 %
    whatever the rates; 64-token steps (about a hundred distinct experts each against 19 slots)
    replay like the oracle in both access orders (4 layers of the trace, 8 steps)."""
    c = synth.CONFIGS["l30e128b64"]
    L, E, k, B = 4, c.n_experts, c.top_k, c.batch
    common = c.n_layers * E * c.hidden * 4
    model = mf.Model(c.n_layers, c.hidden, E, k, c.inter, c.qtype)
    req = mf.PlanReq(0.0, 12 * 2**30, common, 0, B, 0)
    routes = np.zeros((c.n_layers, 8 * B, k), np.int32)
    for l in range(L):  # 64 independent streams per step, Zipf 1.0, stream-major within a step
        streams = [synth.routes(0, l, s, E, k, 8, 1.0, 0.0) for s in range(B)]
        for step in range(8):
            for s in range(B):
                routes[l, step * B + s] = streams[s][step]
    routes[L:] = routes[:1]  # layers 4..29 repeat layer 0's trace
    pcts = [15.0, 35.0, 50.0, 75.0]
    for order in (0, 1):
        pts, best = mf.mf_tune_cache(model, req, routes, B, 1e-4, 1e-3, pcts, order)
        assert [bool(p["accepted"]) for p in pts] == [True, False, False, False]
        assert best == 0 and pts[0]["slots_per_layer"] == 19
        for pt in pts:
            S = pt["slots_per_layer"]
            exp = _oracle_replay(routes, E, S, B, order)
            assert (pt["accesses"], pt["hits"], pt["misses"]) == exp, (order, pt["cache_pct"])
