"""Numeric edge cases of the expert FFN against the CPU oracle, on every kernel path: the fused
one-token launch, the two pipelined one-token kernels, the one-warp-per-row kernels, the batched
GEMV path (T = 4) and the tensor-core grouped GEMMs (T = 256).

The oracle computes in fp64 and rounds once (section "Native Serving Path": the expert FFN on the
dequantised GGUF blocks); the GPU must meet the same tolerance on inputs far from the synthetic
distribution: activations scaled by powers of two (tiny: the SwiGLU outputs h fall near the
bottom of the binary32 range; large: y near 1e35), all-zero 16-value groups of x, an all-zero x,
Q8_0 codes of -128 (GGUF allows them; the generator never draws them), zero and subnormal
binary16 block scales, and rows whose gate scales are zero (h exactly zero there).  Powers of two
scale the oracle's inputs exactly, so both sides see the same values."""
import numpy as np
import pytest

import oracle
import synth
from mfharness import Ctx, Payloads, Shape, G_ATOL, assert_outputs_close

pytestmark = pytest.mark.gpu

Q8, Q4 = synth.Q8_0, synth.Q4_0


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()


def _blocks(payload, shape, tensor):
    """View of one tensor's GGUF blocks: [rows, blocks per row, block bytes]."""
    H, I = shape.hidden, shape.inter
    bb = 34 if shape.qtype == Q8 else 18
    tb = I * (H // 32) * bb
    if tensor < 2:
        return payload[tensor * tb:(tensor + 1) * tb].reshape(I, H // 32, bb)
    return payload[2 * tb:].reshape(H, I // 32, bb)


def edit_codes_min(shape):
    """Every third block of every tensor gets the Q8_0 code -128 in all 32 positions."""
    def f(layer, expert, p):
        p = p.copy()
        for t in range(3):
            b = _blocks(p, shape, t)
            b[:, ::3, 2:] = 0x80
        return p
    return f


def edit_scales(shape):
    """Block scales: every fifth block zero, every seventh the smallest binary16 subnormal
    (2^-24), every eleventh the largest subnormal (0x03ff)."""
    def f(layer, expert, p):
        p = p.copy()
        for t in range(3):
            b = _blocks(p, shape, t)
            b[:, ::5, 0:2] = 0
            b[:, 1::7, 0] = 0x01
            b[:, 1::7, 1] = 0x00
            b[:, 2::11, 0] = 0xFF
            b[:, 2::11, 1] = 0x03
        return p
    return f


def edit_gate_rows_zero(shape):
    """The gate scales of rows 0-15 and 48-79 are zero: h is exactly zero there (whole groups)."""
    def f(layer, expert, p):
        p = p.copy()
        b = _blocks(p, shape, 0)
        b[0:16, :, 0:2] = 0
        b[48:80, :, 0:2] = 0
        return p
    return f


CASES = {
    # name: (payload edit, activation transform, qtypes)
    "x_tiny": (None, None, (Q8, Q4)),  # scale chosen per format and path (tiny_scale)
    "x_large": (None, lambda x: x * np.float32(2.0 ** 50), (Q8, Q4)),
    "x_zero_groups": (None, lambda x: np.concatenate([np.zeros_like(x[:, :16]), x[:, 16:32],
                                                      np.zeros_like(x[:, 32:64]), x[:, 64:]], 1), (Q8, Q4)),
    "x_all_zero": (None, lambda x: np.zeros_like(x), (Q8,)),
    "codes_min": (edit_codes_min, lambda x: x, (Q8,)),
    "scales_zero_subnormal": (edit_scales, lambda x: x, (Q8, Q4)),
    "h_zero_rows": (edit_gate_rows_zero, lambda x: x, (Q8, Q4)),
}
PATHS = ("fused", "pipelined", "simple", "batched", "prefill")


def tiny_scale(qtype, path):
    """The smallest activation scale at which the outputs stay normal binary32 numbers (an output
    in the subnormal range has no relative accuracy in any fp32 arithmetic).  With these weights
    y ~ 6e4 s^2 (Q8_0) or ~16 s^2 (Q4_0) and a 16- or 32-value group of h peaks near 7e3 s^2 or
    26 s^2: at 2^-70 (Q8_0) and 2^-64 (Q4_0) the groups of h lie below 4e-37, where 127 / max
    overflows binary32 unless the split rescales them.  The tensor-core path splits h into bf16
    hi + lo and keeps its accuracy while h stays normal (above ~1e-36): 2^-60 and 2^-56 there."""
    if path == "prefill":
        return 2.0 ** (-60 if qtype == Q8 else -56)
    return 2.0 ** (-70 if qtype == Q8 else -64)


def _run(path, case, qtype, monkeypatch):
    edit_fn, xform, qtypes = CASES[case]
    if qtype not in qtypes:
        pytest.skip("case applies to the other block format")
    if path == "pipelined":
        monkeypatch.setenv("MF_DECODE_UNFUSED", "1")
    if path == "simple":
        monkeypatch.setenv("MF_DECODE_SIMPLE", "1")
    shape = Shape(1, 256, 8, 2, 512, qtype, model_seed=7)
    edit = None if edit_fn is None else edit_fn(shape)
    T = {"batched": 4, "prefill": 256}.get(path, 1)
    n_calls = 1 if path == "prefill" else (2 if path == "batched" else 3)
    if case == "x_tiny":
        xform = lambda x: x * np.float32(tiny_scale(qtype, path))  # noqa: E731
    ctx = Ctx(shape, 4, max_tokens=T, edit=edit)
    pays = Payloads(shape, edit)
    try:
        E, k, H = shape.n_experts, shape.top_k, shape.hidden
        routes = synth.routes(11, 0, 0, E, k, T * n_calls, 1.0, 0.0)
        for c in range(n_calls):
            x = xform(synth.activations(11, 0, 0, c * T, T, H)).astype(np.float32)
            b = synth.plant_bias(routes[c * T:(c + 1) * T], E)
            y, idx, w = ctx.forward(0, x, b, T)
            yo, oidx, og = oracle.layer(pays.for_layer(0, range(E)), qtype, H, shape.inter, k, ctx.wr_host[0], b, x)
            assert np.array_equal(idx, oidx)
            assert np.abs(w - og).max() <= G_ATOL
            assert np.all(np.isfinite(y)), f"{path} {case}: non-finite outputs"
            if case == "x_all_zero":
                assert not np.any(y), "a zero input must give an exactly zero output"
            assert_outputs_close(y, yo, f"{path} {case} call {c}")
        assert ctx.mf.mf_check(ctx.h) == 0
    finally:
        ctx.close()


@pytest.mark.parametrize("case", list(CASES))
@pytest.mark.parametrize("path", PATHS)
def test_numeric_edges_q8_0(path, case, monkeypatch):
    _run(path, case, Q8, monkeypatch)


@pytest.mark.parametrize("case", ["x_tiny", "x_large", "x_zero_groups", "scales_zero_subnormal", "h_zero_rows"])
@pytest.mark.parametrize("path", PATHS)
def test_numeric_edges_q4_0(path, case, monkeypatch):
    _run(path, case, Q4, monkeypatch)
