"""Pins of the CPU oracle against things other than itself.

Each test checks one oracle function against a library routine, a hand-worked value
(``tests/golden``), exact rational arithmetic, a textbook data structure, brute force
or a closed form, chosen so that a dropped term, a wrong sign or index or a transposed
operand in the oracle fails somewhere here.
"""
import math
from collections import OrderedDict
from fractions import Fraction

import numpy as np
import pytest

import oracle
import synth
from conftest import golden_lines

Q8, Q4 = oracle.Q8_0, oracle.Q4_0


# ---------------------------------------------------------------- binary16 scale decode
def test_f16_matches_numpy_for_every_bit_pattern():
    bits = np.arange(65536, dtype=np.uint32).astype(np.uint16)
    ref = bits.view(np.float16).astype(np.float64)
    got = np.array([oracle.f16(int(b)) for b in bits])
    finite = np.isfinite(ref)
    assert np.array_equal(got[finite], ref[finite])
    assert np.array_equal(np.isnan(got), np.isnan(ref))
    assert np.array_equal(np.isinf(got) & (got > 0), np.isinf(ref) & (ref > 0))


def test_f16_hand_worked_values():
    for line in golden_lines("fp16_values.txt"):
        b, v = line.split()
        assert oracle.f16(int(b, 16)) == float(v), b


# ---------------------------------------------------------------- block dequantisation
def _d_bytes(d_hex):
    d = int(d_hex, 16)
    return [d & 0xFF, d >> 8]


def test_q8_0_blocks_hand_worked():
    for line in golden_lines("q8_0_blocks.txt"):
        d_hex, qs, ws = (s.strip() for s in line.split("|"))
        q = [int(v) for v in qs.split()]
        blk = np.array(_d_bytes(d_hex) + [v & 0xFF for v in q], dtype=np.uint8)
        got = oracle.dequant_row(Q8, blk, 32)
        assert np.array_equal(got, np.array([float(v) for v in ws.split()])), d_hex


def test_q4_0_block_hand_worked():
    for line in golden_lines("q4_0_block.txt"):
        d_hex, qs, ws = (s.strip() for s in line.split("|"))
        blk = np.array(_d_bytes(d_hex) + [int(v, 16) for v in qs.split()], dtype=np.uint8)
        got = oracle.dequant_row(Q4, blk, 32)
        assert np.array_equal(got, np.array([float(v) for v in ws.split()])), d_hex


def _numpy_dequant(qtype, raw, rows, cols):
    """Independent dequantisation through numpy's own binary16 decode."""
    nb = cols // 32
    if qtype == Q8:
        blk = raw.reshape(rows, nb, 34)
        d = blk[:, :, :2].copy().view(np.float16).astype(np.float64)  # [rows, nb, 1]
        q = blk[:, :, 2:].view(np.int8).astype(np.float64)
        return (d * q).reshape(rows, cols)
    blk = raw.reshape(rows, nb, 18)
    d = blk[:, :, :2].copy().view(np.float16).astype(np.float64)
    b = blk[:, :, 2:].astype(np.int64)
    n = np.concatenate([b & 0xF, b >> 4], axis=2).astype(np.float64)  # elements j, then j+16
    return (d * (n - 8.0)).reshape(rows, cols)


@pytest.mark.parametrize("qtype", [Q8, Q4])
def test_dequant_rows_match_numpy_decode(qtype):
    raw = synth.q_tensor(7, 0, 3, 1, 8, 256, qtype)
    ref = _numpy_dequant(qtype, raw, 8, 256)
    bb = 34 if qtype == Q8 else 18
    for r in range(8):
        got = oracle.dequant_row(qtype, raw[r * 8 * bb:(r + 1) * 8 * bb], 256)
        assert np.array_equal(got, ref[r])


# ---------------------------------------------------------------- router
def _f32_nearest(fr: Fraction) -> np.float32:
    """The binary32 value nearest to a rational (ties to even), by search over neighbours."""
    f = np.float32(float(fr))
    cands = [np.nextafter(f, np.float32(-np.inf)), f, np.nextafter(f, np.float32(np.inf))]
    best = min(cands, key=lambda c: (abs(Fraction(float(c)) - fr), int(np.array(c).view(np.uint32)) & 1))
    return np.float32(best)


def test_router_logits_are_correctly_rounded_exact_dot_products():
    rng = np.random.default_rng(11)
    E, H, k = 6, 40, 3
    wr = (rng.standard_normal((E, H)) * 0.02).astype(np.float32)
    for trial in range(20):
        x = rng.standard_normal(H).astype(np.float32)
        bias = (rng.standard_normal(E) * 0.5).astype(np.float32) if trial % 2 else None
        z, idx, g = oracle.router(x, wr, bias, k)
        for e in range(E):
            exact = sum(Fraction(float(wr[e, i])) * Fraction(float(x[i])) for i in range(H))
            ze = _f32_nearest(exact)
            if bias is not None:
                ze = np.float32(ze + bias[e])
            assert z[e] == ze
        order = sorted(range(E), key=lambda e: (-float(z[e]), e))[:k]
        assert list(idx) == order
        assert abs(g.sum() - 1.0) < 1e-12
        assert np.all(np.diff(g) <= 0)
        for j in range(1, k):  # softmax ratios are exponentials of logit gaps
            assert math.isclose(g[0] / g[j], math.exp(float(z[idx[0]]) - float(z[idx[j]])), rel_tol=1e-12)


def test_router_ties_go_to_lower_expert_and_equal_weights():
    E, H, k = 8, 32, 3
    z, idx, g = oracle.router(np.ones(H, np.float32), np.zeros((E, H), np.float32), None, k)
    assert list(idx) == [0, 1, 2]
    assert np.allclose(g, 1.0 / 3.0, rtol=0, atol=1e-15)
    bias = np.array([0, 5, 5, 1, 5, 0, 0, 9], np.float32)
    _, idx, _ = oracle.router(np.ones(H, np.float32), np.zeros((E, H), np.float32), bias, 4)
    assert list(idx) == [7, 1, 2, 4]


def test_router_weights_are_full_softmax_renormalised_over_the_selection():
    """Softmax over the k selected logits equals a library softmax over all E logits followed by
    renormalisation over the same k (the weights of the routed experts, section "Native Serving
    Path"); a gap of thousands between the first two logits gives weights (1, 0, ...) without
    overflow."""
    from scipy.special import softmax
    rng = np.random.default_rng(12)
    E, H, k = 16, 48, 4
    wr = (rng.standard_normal((E, H)) * 0.02).astype(np.float32)
    for trial in range(10):
        x = rng.standard_normal(H).astype(np.float32)
        bias = (rng.standard_normal(E) * 2.0).astype(np.float32)
        z, idx, g = oracle.router(x, wr, bias, k)
        full = softmax(z.astype(np.float64))
        ref = full[idx] / full[idx].sum()
        assert np.allclose(g, ref, rtol=1e-12, atol=0)
    bias = np.zeros(E, np.float32)
    bias[3], bias[9] = 4000.0, 1000.0
    z, idx, g = oracle.router(np.zeros(H, np.float32), wr, bias, 2)
    assert list(idx) == [3, 9]
    assert g[0] == 1.0 and g[1] == 0.0 and np.isfinite(g).all()


# ---------------------------------------------------------------- expert FFN and layer
def _silu(v):
    return v / (1.0 + np.exp(-v))


@pytest.mark.parametrize("qtype", [Q8, Q4])
def test_expert_ffn_matches_numpy_matmul(qtype):
    H, I = 256, 512
    p = synth.payload(0, 0, 5, H, I, qtype)
    x = synth.activations(0, 0, 0, 3, 1, H)[0]
    tb = synth.tensor_bytes(I, H, qtype)
    wg = _numpy_dequant(qtype, p[:tb], I, H)
    wu = _numpy_dequant(qtype, p[tb:2 * tb], I, H)
    wd = _numpy_dequant(qtype, p[2 * tb:], H, I)
    xd = x.astype(np.float64)
    h_ref = _silu(wg @ xd) * (wu @ xd)
    y_ref = wd @ h_ref
    y, h = oracle.expert_ffn(p, qtype, H, I, x)
    assert np.allclose(h, h_ref, rtol=1e-12, atol=1e-9 * np.abs(h_ref).max())
    assert np.allclose(y, y_ref, rtol=1e-12, atol=1e-11 * np.abs(y_ref).max())


def test_layer_is_router_weighted_sum_of_expert_outputs():
    cfg = synth.CONFIGS["tiny"]
    H, I, E, k = cfg.hidden, cfg.inter, cfg.n_experts, cfg.top_k
    pays = [synth.payload(0, 0, e, H, I, Q8) for e in range(E)]
    wr = synth.router_weights(0, 0, E, H)
    x = synth.activations(0, 0, 0, 0, 6, H)
    y, idx, g = oracle.layer(pays, Q8, H, I, k, wr, None, x)
    for t in range(6):
        z, it, gt = oracle.router(x[t], wr, None, k)
        assert np.array_equal(it, idx[t]) and np.array_equal(gt, g[t])
        acc = np.zeros(H)
        for j in range(k):
            acc += gt[j] * oracle.expert_ffn(pays[it[j]], Q8, H, I, x[t])[0]
        assert np.array_equal(y[t], acc.astype(np.float32))


def test_layer_with_one_expert_is_that_experts_output():
    H, I, E = 256, 512, 8
    pays = [synth.payload(1, 0, e, H, I, Q8) for e in range(E)]
    x = synth.activations(1, 0, 0, 0, 3, H)
    bias = np.zeros((3, E), np.float32)
    bias[:, 5] = 20.0
    y, idx, g = oracle.layer(pays, Q8, H, I, 1, synth.router_weights(1, 0, E, H), bias, x)
    assert np.all(idx == 5) and np.all(g == 1.0)
    for t in range(3):
        assert np.array_equal(y[t], oracle.expert_ffn(pays[5], Q8, H, I, x[t])[0].astype(np.float32))


def test_layer_with_equal_logits_is_mean_of_first_k_experts():
    H, I, E, k = 256, 512, 8, 4
    pays = [synth.payload(2, 0, e, H, I, Q4) for e in range(E)]
    x = synth.activations(2, 0, 0, 0, 1, H)
    y, idx, g = oracle.layer(pays, Q4, H, I, k, np.zeros((E, H), np.float32), None, x)
    assert list(idx[0]) == [0, 1, 2, 3]
    ref = sum(oracle.expert_ffn(pays[e], Q4, H, I, x[0])[0] for e in range(4)) / 4
    assert np.allclose(y[0], ref, rtol=1e-6, atol=1e-6 * np.abs(ref).max())


def test_layer_requires_every_routed_payload():
    H, I, E = 256, 512, 8
    bias = np.zeros((1, E), np.float32)
    bias[0, 2] = 30
    pays = [None] * E
    with pytest.raises(KeyError):
        oracle.layer(pays, Q8, H, I, 1, np.zeros((E, H), np.float32), bias, np.ones((1, H), np.float32))
    pays[2] = synth.payload(0, 0, 2, H, I, Q8)
    oracle.layer(pays, Q8, H, I, 1, np.zeros((E, H), np.float32), bias, np.ones((1, H), np.float32))


# ---------------------------------------------------------------- LRU slot cache
class TextbookLRU:
    """Least-recently-used cache on an OrderedDict; slots: lowest free first, else the victim's."""

    def __init__(self, S):
        self.S, self.d, self.free = S, OrderedDict(), list(range(S))

    def access(self, e):
        if e in self.d:
            self.d.move_to_end(e)
            return True, self.d[e]
        if self.free:
            s = self.free.pop(0)
        else:
            _, s = self.d.popitem(last=False)
        self.d[e] = s
        return False, s


def _steps_from_routes(r, T):
    return [r[i:i + T] for i in range(0, len(r), T)]


@pytest.mark.parametrize("S,T,s,rho", [(2, 1, 0.0, 0.0), (5, 1, 1.1, 0.6), (9, 1, 0.8, 0.0), (6, 4, 1.0, 0.0),
                                       (16, 3, 1.2, 0.3), (3, 2, 0.0, 0.0)])
def test_lru_matches_textbook(S, T, s, rho):
    E, k = 16, 2 if S < 4 else 3
    r = synth.routes(3, 0, 0, E, k, 120, s, rho)
    orc, ref = oracle.LRU(E, S, 1000), TextbookLRU(S)
    for step in _steps_from_routes(r, T):
        uniq, slot, hit = orc.step(step)
        seen = []
        for e in step.reshape(-1):
            if e not in seen:
                seen.append(int(e))
        assert list(uniq) == seen
        for u, e in enumerate(seen):
            h, sl = ref.access(e)
            assert (bool(hit[u]), int(slot[u])) == (h, sl)
        assert orc.occupancy() <= S
        res = orc.slots()
        assert sorted(int(e) for e in res if e >= 0) == sorted(ref.d.keys())
    st = orc.stats()
    assert st["accesses"] == st["hits"] + st["misses"]
    assert st["bytes"] == 1000 * st["misses"]
    assert st["evictions"] == st["misses"] - orc.occupancy()


def _run_hits(r, E, S):
    c = oracle.LRU(E, S, 1)
    for t in range(len(r)):
        c.step(r[t:t + 1])
    return c.stats()


@pytest.mark.parametrize("s,rho", [(0.0, 0.0), (0.8, 0.0), (1.2, 0.8), (1.1, 0.6)])
def test_lru_inclusion_property(s, rho):
    """Mattson et al. 1970: LRU is a stack algorithm, so hits never fall as capacity grows."""
    E, k = 32, 4
    r = synth.routes(5, 2, 0, E, k, 200, s, rho)
    hits = [_run_hits(r, E, S)["hits"] for S in range(k, E + 1)]
    assert all(a <= b for a, b in zip(hits, hits[1:]))
    distinct = len(set(r.reshape(-1).tolist()))
    full = _run_hits(r, E, E)
    assert full["misses"] == distinct and full["evictions"] == 0  # compulsory misses only


def test_lru_full_reuse_closed_form():
    E, k, T = 64, 8, 50
    r = synth.routes(9, 0, 0, E, k, T, 1.1, 1.0)  # every token repeats the first set
    st = _run_hits(r, E, k)
    assert st["hits"] == (T - 1) * k and st["misses"] == k


def test_lru_uniform_hit_rate_closed_form():
    """Uniform routing, k distinct experts per token, batch 1, S >= k.  At the j-th access of a
    token the cache holds that token's j earlier experts plus S - j others, and the access is
    uniform over the E - j experts not yet used by the token, so it hits with probability
    (S - j) / (E - j); the steady-state hit rate is the mean over j < k."""
    E, k, S, T = 128, 8, 32, 3000
    r = synth.routes(4, 0, 0, E, k, T, 0.0, 0.0)
    c = oracle.LRU(E, S, 1)
    for t in range(200):
        c.step(r[t:t + 1])
    before = c.stats()
    for t in range(200, T):
        c.step(r[t:t + 1])
    after = c.stats()
    rate = (after["hits"] - before["hits"]) / (after["accesses"] - before["accesses"])
    expect = sum((S - j) / (E - j) for j in range(k)) / k
    assert abs(rate - expect) < 0.012  # ~4 standard deviations of 22400 Bernoulli draws


def test_lru_resident_first_worked_example():
    """Two slots holding experts 0 and 1 (0 least recent); a step of two tokens routed [2, 3] then
    [0, 1].  First-occurrence order: 2 and 3 miss and evict 0 and 1, which then miss too (4
    misses).  Resident first: 0 and 1 hit, then 2 and 3 miss into their slots (2 misses)."""
    step = np.array([[2, 3], [0, 1]], np.int32)
    first, res = oracle.LRU(4, 2, 1), oracle.LRU(4, 2, 1)
    for c in (first, res):
        c.step(np.array([[0, 1]], np.int32))  # 0 then 1: 0 is least recent
    u, sl, h = first.step(step, order=0)
    assert (list(u), list(sl), list(h)) == ([2, 3, 0, 1], [0, 1, 0, 1], [False] * 4)
    u, sl, h = res.step(step, order=1)
    assert (list(u), list(sl), list(h)) == ([0, 1, 2, 3], [0, 1, 0, 1], [True, True, False, False])
    assert (first.stats()["misses"], res.stats()["misses"]) == (2 + 4, 2 + 2)


@pytest.mark.parametrize("S,T,s", [(4, 8, 0.8), (9, 16, 1.1), (19, 64, 1.0), (6, 2, 0.0)])
def test_lru_resident_first_against_textbook(S, T, s):
    """Resident-first steps on the textbook cache: the access list is the step's distinct
    experts resident at its start (first-occurrence order), then the rest; every one of the
    former hits; decisions and slots as the textbook LRU gives them for that sequence; and a
    step never has fewer hits than the residents it needs."""
    E, k = 32, 4
    r = synth.routes(11, 0, 0, E, k, 40 * T, s, 0.3)
    orc, ref = oracle.LRU(E, S, 1), TextbookLRU(S)
    for step in _steps_from_routes(r, T):
        seen = []
        for e in step.reshape(-1):
            if int(e) not in seen:
                seen.append(int(e))
        resident = [e for e in seen if e in ref.d] if T > 1 else []
        order = resident + [e for e in seen if e not in resident] if T > 1 else seen
        uniq, slot, hit = orc.step(step, order=1)
        assert list(uniq) == order
        for u, e in enumerate(order):
            h, sl = ref.access(e)
            assert (bool(hit[u]), int(slot[u])) == (h, sl)
        assert all(hit[:len(resident)])
        assert orc.occupancy() <= S


# ---------------------------------------------------------------- static budget check
def test_plan_closed_form_l30e128():
    for line in golden_lines("plan_l30e128b64.txt"):
        pct, S, pool, lower, acc = (int(v) for v in line.split())
        p = oracle.plan(30, 2816, 128, 8, 1408, Q8, pct, 12 * 2**30, common=30 * 128 * 2816 * 4, kv=0)
        assert (p["slots"], p["pool"], p["lower"], p["accepted"]) == (S, pool, lower, bool(acc))
        assert p["payload"] == 12638208


def test_plan_slot_floor_minimum_and_boundary():
    p = oracle.plan(4, 2048, 64, 8, 768, Q8, 1.0, 2**40)
    assert p["slots"] == 8  # at least top-k slots
    assert oracle.plan(4, 2048, 64, 8, 768, Q8, 35.0, 2**40)["slots"] == 22  # floor(22.4)
    assert oracle.plan(4, 2048, 64, 8, 768, Q8, 50.0, 2**40)["slots"] == 32  # exact product
    assert oracle.plan(4, 2048, 64, 8, 768, Q8, 100.0, 2**40)["slots"] == 64
    p = oracle.plan(4, 2048, 64, 8, 768, Q8, 15.0, 0, common=5, kv=7)
    assert p["payload"] == 3 * 768 * 64 * 34 and p["lower"] == 5 + 7 + 4 * 9 * 5013504
    assert oracle.plan(4, 2048, 64, 8, 768, Q8, 15.0, p["lower"], 5, 7)["accepted"]
    assert not oracle.plan(4, 2048, 64, 8, 768, Q8, 15.0, p["lower"] - 1, 5, 7)["accepted"]


def test_plan_lower_bound_is_linear_in_slots():
    """L = C + S * (layers * payload) + K: equal slot steps give equal L steps (the paper's
    rejected Gemma cells at 50% and 65% differ by the expert bytes of the extra slots only)."""
    ls = [oracle.plan(30, 2816, 128, 8, 1408, Q8, pct, 0, 11, 13) for pct in (25.0, 50.0, 75.0)]
    assert ls[1]["lower"] - ls[0]["lower"] == (ls[1]["slots"] - ls[0]["slots"]) * 30 * 12638208
    assert ls[2]["lower"] - ls[1]["lower"] == (ls[2]["slots"] - ls[1]["slots"]) * 30 * 12638208
