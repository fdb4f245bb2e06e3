"""The seeded input generator: determinism, value ranges and the route-locality recipe."""
import numpy as np
import pytest

import synth


def test_f64_to_f16_is_round_to_nearest_even():
    rng = np.random.default_rng(0)
    vals = np.concatenate([
        np.abs(rng.standard_normal(20000) * 0.02),
        rng.standard_normal(2000) * 1000,
        np.ldexp(rng.random(2000), -rng.integers(14, 26, 2000)),  # subnormal range
        [0.0, -0.0, 65504.0, 65519.0, 2.0**-25, 2.0**-24 * 1.5, 2.0**-24 * 2.5, 1.0 + 2.0**-11, 1.0 + 3 * 2.0**-11],
    ])
    for v in vals:
        ref = int(np.array([v]).astype(np.float16).view(np.uint16)[0])
        assert synth.f64_to_f16_bits(float(v)) == ref, v


def test_payload_deterministic_and_addressable():
    a = synth.payload(3, 2, 7, 256, 512, synth.Q8_0)
    b = synth.payload(3, 2, 7, 256, 512, synth.Q8_0)
    c = synth.payload(3, 2, 8, 256, 512, synth.Q8_0)
    assert np.array_equal(a, b) and not np.array_equal(a, c)
    tb = synth.tensor_bytes(512, 256, synth.Q8_0)
    assert np.array_equal(a[tb:2 * tb], synth.q_tensor(3, 2, 7, 1, 512, 256, synth.Q8_0))


@pytest.mark.parametrize("qtype", [synth.Q8_0, synth.Q4_0])
def test_block_value_distributions(qtype):
    raw = synth.q_tensor(1, 0, 0, 0, 256, 2048, qtype)
    bb = 34 if qtype == synth.Q8_0 else 18
    blk = raw.reshape(-1, bb)
    d = blk[:, :2].copy().view(np.float16).astype(np.float64)[:, 0]
    assert np.all(d >= 0) and abs(np.sqrt((d ** 2).mean()) - 0.02) < 0.001
    if qtype == synth.Q8_0:
        q = blk[:, 2:].view(np.int8).astype(np.int64)
        assert q.min() == -127 and q.max() == 127
        assert abs(q.mean()) < 0.2 and abs(q.std() - np.sqrt((255 ** 2 - 1) / 12)) < 0.3
    else:
        n = np.concatenate([blk[:, 2:] & 0xF, blk[:, 2:] >> 4]).astype(np.int64)
        assert n.min() == 0 and n.max() == 15 and abs(n.mean() - 7.5) < 0.02


def test_routes_valid_and_reuse_rate():
    E, k, T = 128, 8, 4000
    r = synth.routes(0, 3, 0, E, k, T, 1.2, 0.8)
    assert r.shape == (T, k) and r.min() >= 0 and r.max() < E
    assert all(len(set(row)) == k for row in r.tolist())
    same = np.mean([np.array_equal(r[t], r[t - 1]) for t in range(1, T)])
    assert abs(same - 0.8) < 0.03
    assert np.array_equal(r, synth.routes(0, 3, 0, E, k, T, 1.2, 0.8))
    assert not np.array_equal(r, synth.routes(0, 3, 1, E, k, T, 1.2, 0.8))


def test_routes_skew_follows_permutation():
    E, k = 128, 8
    r = synth.routes(0, 5, 0, E, k, 3000, 1.2, 0.0)
    perm = synth.permutation(0, 5, E)
    assert sorted(perm.tolist()) == list(range(E))
    counts = np.bincount(r.reshape(-1), minlength=E)
    assert counts[perm[0]] == counts.max()  # rank 0 is the most popular expert
    u = synth.routes(0, 5, 0, E, k, 3000, 0.0, 0.0)
    cu = np.bincount(u.reshape(-1), minlength=E)
    assert cu.max() / cu.mean() < 1.4  # uniform class


def test_plant_bias_orders_the_set():
    r = np.array([[5, 2, 7]], np.int32)
    b = synth.plant_bias(r, 8)
    assert b[0, 5] == 17.5 and b[0, 2] == 17.0 and b[0, 7] == 16.5 and b[0].sum() == 51.0


def test_acceptance_schedule_extremes_and_mean():
    """a_i counts the leading successes of K trials of probability alpha: 0 for alpha = 0, K for
    alpha = 1, and mean sum_{j=1..K} alpha^j (a truncated geometric count) over many steps."""
    assert (synth.accepts(1, 0, 500, 4, 0.0) == 0).all()
    assert (synth.accepts(1, 0, 500, 4, 1.0) == 4).all()
    assert (synth.accepts(1, 0, 50, 0, 0.7) == 0).all()
    n, K, alpha = 40000, 4, 0.6
    a = synth.accepts(7, 0, n, K, alpha)
    assert a.min() >= 0 and a.max() <= K
    mean = sum(alpha ** j for j in range(1, K + 1))
    var = sum((2 * j - 1) * alpha ** j for j in range(1, K + 1)) - mean ** 2  # E[a^2] = sum (2j-1) P(a >= j)
    assert abs(a.mean() - mean) < 4 * (var / n) ** 0.5
    assert np.array_equal(a, synth.accepts(7, 0, n, K, alpha))
    assert not np.array_equal(a[:100], synth.accepts(8, 0, 100, K, alpha))


@pytest.mark.parametrize("K,alpha", [(4, 0.6), (2, 0.0), (3, 1.0), (0, 0.5)])
def test_verify_rows_cover_the_sequence_once(K, alpha):
    """Every token appears once, in order, as a prefix of its batch (the target's token and the
    accepted drafts); the rest of each batch are rejected drafts numbered 0, 1, ... in order;
    K = 0 is plain decode."""
    n = 97
    rows = synth.verify_rows(3, n, K, alpha)
    assert rows.shape[1] == K + 1
    toks = [int(v) for v in rows.reshape(-1) if v >= 0]
    assert toks == list(range(n))
    drafts = [int(-1 - v) for v in rows.reshape(-1) if v < 0]
    assert drafts == list(range(len(drafts)))
    acc = synth.accepts(3, 0, n, K, alpha)
    for i, row in enumerate(rows):
        m = int((row >= 0).sum())
        assert (row[:m] >= 0).all() and (row[m:] < 0).all()
        assert m == min(int(acc[i]) + 1, n - int(row[0]))
    if K == 0:
        assert rows.reshape(-1).tolist() == list(range(n))
