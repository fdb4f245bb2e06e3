"""Router of many-token calls (the tiled path, T >= 16) vs the oracle router, through the C ABI.

Real routing (no planted bias) on seeded x and W_r, so the k-th and (k+1)-th logits are often
close: routed indices must equal the oracle's exactly, weights within G_ATOL.  The shapes cover
ragged token tiles (T not a multiple of 32), ragged expert tiles (E not a multiple of 64), one
and many K splits, the smallest and largest expert counts, exact ties at the selection boundary
(identical W_r rows and bias: the lower expert id first), and the switch between the
one-token-per-cluster router (T = 15) and the tiled one (T = 16) on the same tokens."""
import numpy as np
import pytest

import oracle
import synth
from mfharness import Ctx, G_ATOL, Shape

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()


def _check_routes(ctx, x, bias, T, k):
    _, idx, w = ctx.forward(0, x, bias, T)
    for t in range(T):
        _, oidx, og = oracle.router(x[t], ctx.wr_host[0], None if bias is None else bias[t], k)
        assert np.array_equal(idx[t], oidx), (t, idx[t], oidx)
        assert np.abs(w[t] - og).max() <= G_ATOL, t
    return idx


@pytest.mark.parametrize("H,E,k,T", [
    (2048, 100, 8, 300),   # ragged expert tile (64 + 36), 10 token tiles, 16 K splits
    (2048, 128, 8, 4096),  # the 48-layer prefill call: 256 tiles, no K split
    (256, 64, 4, 17),      # one token past a tile edge
    (96, 12, 3, 16),       # fewer experts than a tile, 3 K splits of one chunk
    (64, 1024, 8, 40),     # the largest expert count
    (2816, 128, 8, 64),    # the 30-layer batch-64 shape
])
def test_tiled_router_real_routing(H, E, k, T):
    shape = Shape(1, H, E, k, 64, synth.Q8_0, model_seed=5)
    ctx = Ctx(shape, slots=E, max_tokens=T)
    try:
        x = synth.activations(21, 0, 0, 0, T, H)
        _check_routes(ctx, x, None, T, k)
        assert ctx.mf.mf_check(ctx.h) == 0
    finally:
        ctx.close()


def test_tiled_router_exact_ties():
    """Rows 5 and 9 of W_r equal and both lifted by the same bias: they lead with equal logits
    (5 before 9); rows 3 and 20 equal with a smaller lift: they tie for the last place (3 wins)."""
    H, E, k, T = 256, 64, 3, 33
    shape = Shape(1, H, E, k, 64, synth.Q8_0, model_seed=6)
    ctx = Ctx(shape, slots=E, max_tokens=T)
    try:
        import torch
        wr = ctx.wr_host[0].copy()
        wr[9] = wr[5]
        wr[20] = wr[3]
        ctx.wr_host[0] = wr
        ctx.wr[0] = torch.from_numpy(wr).to(ctx.device)
        x = synth.activations(22, 0, 0, 0, T, H)
        bias = np.zeros((T, E), np.float32)
        bias[:, [5, 9]] = 1000.0
        bias[:, [3, 20]] = 500.0
        idx = _check_routes(ctx, x, bias, T, k)
        assert (idx[:, 0] == 5).all() and (idx[:, 1] == 9).all() and (idx[:, 2] == 3).all()
    finally:
        ctx.close()


def test_router_paths_agree_at_the_switch():
    """The same 15 tokens through the per-token router (T = 15) and, with one more token, the
    tiled router (T = 16): identical indices and weights for the 15."""
    H, E, k = 2048, 128, 8
    shape = Shape(1, H, E, k, 64, synth.Q8_0, model_seed=7)
    ctx = Ctx(shape, slots=E, max_tokens=16)
    try:
        x = synth.activations(23, 0, 0, 0, 16, H)
        i15 = _check_routes(ctx, x[:15], None, 15, k)
        _, w15 = ctx.forward(0, x[:15], None, 15)[1:]
        i16 = _check_routes(ctx, x, None, 16, k)
        _, w16 = ctx.forward(0, x, None, 16)[1:]
        assert np.array_equal(i15, i16[:15])
        assert np.array_equal(w15, w16[:15])
    finally:
        ctx.close()
