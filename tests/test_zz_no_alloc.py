"""The allocation-free expert FFN entry point (mf_expert_ffn_noalloc) against mf_moe_forward.

Callers that cannot allocate device memory use mf_expert_ffn_noalloc with expert weights they
already hold; its scratch is a static device array.  This file is named to be collected last,
so a run that stops at the first failure has already run every other test; it also passes on
its own in a fresh process."""
import numpy as np
import pytest

import synth
from mfharness import Ctx, Shape, assert_outputs_close

pytestmark = pytest.mark.gpu


def _r(v, a):
    return (v + a - 1) // a * a


def slot_image(canon: np.ndarray, H: int, I: int, q: int) -> np.ndarray:
    """One expert's canonical GGUF payload laid out as the slot mawforge.h documents."""
    bb, cb = (34, 32) if q == synth.Q8_0 else (18, 16)
    qgu, qd = (H, I) if q == synth.Q8_0 else (H // 2, I // 2)
    nbgu, nbd = H // 32, I // 32
    o_up, o_gs = qgu, 2 * qgu
    o_us = o_gs + _r(2 * nbgu, 16)
    rs_gu, rs_d = _r(o_us + 2 * nbgu, 16), _r(qd + 2 * nbd, 16)
    d_off = _r(I * rs_gu, 256)
    out = np.zeros(_r(d_off + H * rs_d, 256), np.uint8)

    def put(t, rows, cols, rec0, rs, codes_off, scales_off):
        nb = cols // 32
        blk = t.reshape(rows, nb, bb)
        rec = out[rec0:rec0 + rows * rs].reshape(rows, rs)
        rec[:, scales_off:scales_off + 2 * nb] = blk[:, :, :2].reshape(rows, 2 * nb)
        codes = blk[:, :, 2:] ^ np.uint8(0x80) if q == synth.Q8_0 else blk[:, :, 2:]
        rec[:, codes_off:codes_off + nb * cb] = codes.reshape(rows, nb * cb)

    tb = I * nbgu * bb
    put(canon[:tb], I, H, 0, rs_gu, 0, o_gs)
    put(canon[tb:2 * tb], I, H, 0, rs_gu, o_up, o_us)
    put(canon[2 * tb:], H, I, d_off, rs_d, 0, qd)
    return out


@pytest.mark.parametrize("shape", [Shape(1, 2048, 64, 8, 768, synth.Q8_0, model_seed=3),
                                   Shape(1, 96, 12, 3, 160, synth.Q4_0, model_seed=4)],
                         ids=["q8_0_h2048", "q4_0_h96"])
def test_noalloc_ffn_matches_moe_forward_on_two_calls(shape):
    import torch
    import paper_2607_09686_gb300 as mf
    ctx = Ctx(shape, shape.top_k, max_tokens=1)
    try:
        dev = ctx.device
        model = mf.Model(1, shape.hidden, shape.n_experts, shape.top_k, shape.inter, shape.qtype)
        for t in range(2):  # two calls in a row
            x = synth.activations(11, 0, 0, t, 1, shape.hidden)
            y_ref, idx, w = ctx.forward(0, x, None, 1)
            experts = np.concatenate([slot_image(synth.payload(shape.model_seed, 0, int(e), shape.hidden,
                                                               shape.inter, shape.qtype),
                                                 shape.hidden, shape.inter, shape.qtype) for e in idx[0]])
            ed = torch.from_numpy(experts).to(dev)
            gd = torch.from_numpy(np.ascontiguousarray(w[0])).to(dev)
            xd = torch.from_numpy(x).to(dev)
            yd = torch.full((1, shape.hidden), float("nan"), device=dev)
            torch.cuda.synchronize()
            free0 = torch.cuda.mem_get_info(dev)[0]
            mf.mf_expert_ffn_noalloc(model, ed, gd, xd, yd)
            torch.cuda.synchronize()
            if t == 1:  # after the first call has set the device up, a call changes no allocation
                assert torch.cuda.mem_get_info(dev)[0] == free0
            assert_outputs_close(yd.cpu().numpy(), y_ref, f"call {t}")
        assert mf.mf_expert_ffn_noalloc_check() == mf.MF_OK  # no bounded wait gave up
    finally:
        ctx.close()


def _oracle_ffn(payloads, g, x, H, I, q):
    """y = sum_j g_j FFN_j(x) in fp64 (the oracle's expert FFN), rounded once to fp32."""
    import oracle
    acc = np.zeros(H, np.float64)
    for j, p in enumerate(payloads):
        yj, _ = oracle.expert_ffn(p, q, H, I, x)
        acc += np.float64(g[j]) * yj
    return acc.astype(np.float32)[None]


@pytest.mark.parametrize("shape", [(256, 2048, 4, synth.Q8_0),    # the one-warp-per-row kernels
                                   (256, 4096, 8, synth.Q4_0)],   # top_k * inter = 32768: the limit
                         ids=["q8_0_unpipelined", "q4_0_at_limit"])
def test_noalloc_ffn_against_the_oracle(shape):
    """Shapes the pipelined kernels do not take (h of 2048 / 4096 values per expert) run the other
    kernel pair; the largest accepted size fills the static scratch exactly."""
    import torch
    import paper_2607_09686_gb300 as mf
    H, I, k, q = shape
    model = mf.Model(1, H, k, k, I, q)
    dev = torch.device("cuda:0")
    pays = [synth.payload(9, 0, e, H, I, q) for e in range(k)]
    experts = np.concatenate([slot_image(p, H, I, q) for p in pays])
    ed = torch.from_numpy(experts).to(dev)
    for t in range(2):  # two calls in a row
        x = synth.activations(13, 0, 0, t, 1, H)
        g = np.random.default_rng(t).dirichlet(np.ones(k)).astype(np.float32)
        yd = torch.full((1, H), float("nan"), device=dev)
        mf.mf_expert_ffn_noalloc(model, ed, torch.from_numpy(g).to(dev), torch.from_numpy(x).to(dev), yd)
        torch.cuda.synchronize()
        assert_outputs_close(yd.cpu().numpy(), _oracle_ffn(pays, g, x[0], H, I, q), f"{shape} call {t}")
    assert mf.mf_expert_ffn_noalloc_check() == mf.MF_OK


def test_noalloc_rejects_sizes_beyond_its_scratch():
    import torch
    import paper_2607_09686_gb300 as mf
    buf = torch.zeros(16, device="cuda")
    # Q4_0, top_k 8, inter 4128: a valid expert shape whose h (33024 floats) exceeds the scratch
    # (Q8_0 shapes past the limit are already rejected as shapes)
    for big in (mf.Model(1, 256, 8, 8, 4128, synth.Q4_0), mf.Model(1, 2048, 8, 8, 4608, synth.Q8_0)):
        with pytest.raises(mf.MFError) as e:
            mf.mf_expert_ffn_noalloc(big, buf, buf, buf, buf)
        assert e.value.status == mf.MF_E_INVAL
