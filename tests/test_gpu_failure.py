"""Failure detection without a GPU fault: a bounded device wait that runs out.

Every wait inside the kernels has a time limit (mf_wait_limit).  The context's test hold
(mf_test_hold) makes the one-token expert FFN's producer issue none of its copies, so the stages
the consumers wait for are never filled: their waits run out, the kernel records the failure and
returns with nothing in flight, and mf_check reports MF_E_TIMEOUT once.  The next call on the same
context is correct again.  The held call hits on every expert, so no slot is left half
materialised."""
import numpy as np
import pytest

import oracle
import synth
from mfharness import Ctx, Payloads, Shape, assert_outputs_close

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()


def test_wait_limit_arguments():
    import paper_2607_09686_gb300 as mf
    ctx = Ctx(Shape(1, 256, 8, 2, 512, synth.Q8_0, model_seed=3), 8, max_tokens=1)
    try:
        for bad in (0.0, -1.0, 61.0, float("nan")):
            with pytest.raises(mf.MFError) as e:
                mf.mf_wait_limit(ctx.h, bad)
            assert e.value.status == mf.MF_E_INVAL
        with pytest.raises(mf.MFError):
            mf.mf_test_hold(ctx.h, 2)
        mf.mf_wait_limit(ctx.h, 2.0)
        mf.mf_test_hold(ctx.h, 0)
    finally:
        ctx.close()


def test_bounded_wait_runs_out_and_the_context_recovers():
    import time
    import paper_2607_09686_gb300 as mf
    shape = Shape(1, 256, 8, 2, 512, synth.Q8_0, model_seed=3)
    ctx = Ctx(shape, 8, max_tokens=1)  # 8 slots: every expert stays resident once used
    pays = Payloads(shape)
    try:
        E, k, H = shape.n_experts, shape.top_k, shape.hidden
        x = synth.activations(5, 0, 0, 0, 8, H)
        # make every expert resident: token t plants experts 2t and 2t + 1
        warm = np.array([[2 * (t % 4), 2 * (t % 4) + 1] for t in range(4)], np.int32)
        for t in range(4):
            ctx.forward(0, x[t:t + 1], synth.plant_bias(warm[t:t + 1], E), 1)
        assert mf.mf_check(ctx.h) == 0
        before = mf.mf_stats(ctx.h, 0)
        b = synth.plant_bias(np.array([[5, 2]], np.int32), E)
        mf.mf_wait_limit(ctx.h, 0.005)
        mf.mf_test_hold(ctx.h, 1)
        t0 = time.perf_counter()
        ctx.forward(0, x[4:5], b, 1)  # synchronises
        held_s = time.perf_counter() - t0
        assert mf.mf_check(ctx.h) == mf.MF_E_TIMEOUT
        assert mf.mf_check(ctx.h) == 0  # the record is cleared
        assert held_s < 5.0, held_s
        after = mf.mf_stats(ctx.h, 0)
        assert after["misses"] == before["misses"] and after["hits"] == before["hits"] + 2  # all-hit call
        # the next calls on the same context are correct
        mf.mf_test_hold(ctx.h, 0)
        mf.mf_wait_limit(ctx.h, 1.0)
        for t in (4, 5, 6):
            bt = b if t == 4 else synth.plant_bias(np.array([[t % E, (t + 3) % E]], np.int32), E)
            y, idx, w = ctx.forward(0, x[t:t + 1], bt, 1)
            yo, oidx, _ = oracle.layer(pays.for_layer(0, range(E)), shape.qtype, H, shape.inter, k, ctx.wr_host[0],
                                       bt, x[t:t + 1])
            assert np.array_equal(idx, oidx)
            assert_outputs_close(y, yo, f"call after the timeout, token {t}")
        assert mf.mf_check(ctx.h) == 0
    finally:
        ctx.close()
