"""The C ABI library: it loads without a GPU, exports what include/mawforge.h declares, and its
host-only planner agrees with the oracle's.  No compute call is made here."""
import ctypes
import os
import re

import pytest

import oracle
import synth
import __graft_entry__

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def mf():
    __graft_entry__.build()
    import paper_2607_09686_gb300 as pkg
    return pkg


def _declared():
    with open(os.path.join(ROOT, "include", "mawforge.h")) as f:
        text = f.read()
    return sorted(set(re.findall(r"^\s*(?:int|void|const char\*)\s+\**(mf_\w+)\s*\(", text, re.M)))


def test_library_exports_every_declared_symbol(mf):
    names = _declared()
    assert "mf_moe_forward" in names and "mf_plan" in names and "mf_load_pack" in names and "mf_stats" in names
    lib = ctypes.CDLL(mf.LIB_PATH)
    for n in names:
        assert hasattr(lib, n), n


def test_struct_layouts(mf):
    assert ctypes.sizeof(mf.Model) == 24
    assert ctypes.sizeof(mf.PlanReq) == 40
    assert ctypes.sizeof(mf.Plan) == 56
    assert ctypes.sizeof(mf.Stats) == 40


def test_status_strings(mf):
    assert mf.mf_strerror(0) == "ok"
    assert "budget" in mf.mf_strerror(-2)


@pytest.mark.parametrize("name", sorted(synth.CONFIGS))
def test_payload_bytes_match(mf, name):
    c = synth.CONFIGS[name]
    m = mf.Model(c.n_layers, c.hidden, c.n_experts, c.top_k, c.inter, c.qtype)
    assert mf.mf_payload_bytes(m) == oracle.payload_bytes(c.hidden, c.inter, c.qtype) == \
        synth.payload_bytes(c.hidden, c.inter, c.qtype)


@pytest.mark.parametrize("name", sorted(synth.CONFIGS))
def test_plan_matches_oracle(mf, name):
    c = synth.CONFIGS[name]
    m = mf.Model(c.n_layers, c.hidden, c.n_experts, c.top_k, c.inter, c.qtype)
    for pct in (0.0, 1.0, 12.5, 15.0, 25.0, 33.3, 35.0, 50.0, 65.0, 75.0, 100.0):
        for budget, common, kv in ((12 * 2**30, 43253760, 0), (2**40, 0, 7 * 2**30), (0, 0, 0)):
            p = mf.mf_plan(m, mf.PlanReq(pct, budget, common, kv, 64, 0))
            o = oracle.plan(c.n_layers, c.hidden, c.n_experts, c.top_k, c.inter, c.qtype, pct, budget, common, kv)
            assert (p.slots_per_layer, p.payload_bytes, p.pool_bytes, p.lower_bound_bytes, bool(p.accepted)) == \
                (o["slots"], o["payload"], o["pool"], o["lower"], o["accepted"])
            assert p.footprint_bytes == p.lower_bound_bytes + p.overhead_bytes and p.overhead_bytes > 0


def test_plan_rejects_bad_arguments(mf):
    lib = ctypes.CDLL(mf.LIB_PATH)
    out = mf.Plan()
    good = mf.Model(4, 2048, 64, 8, 768, mf.Q8_0)
    assert lib.mf_plan(ctypes.byref(good), ctypes.byref(mf.PlanReq(35.0, 2**40, 0, 0, 1, 0)), ctypes.byref(out)) == 0
    for bad in (mf.Model(0, 2048, 64, 8, 768, 8), mf.Model(4, 2000, 64, 8, 768, 8), mf.Model(4, 2048, 64, 9, 768, 8),
                mf.Model(4, 2048, 4, 8, 768, 8), mf.Model(4, 2048, 64, 8, 768, 3), mf.Model(4, 2048, 2048, 8, 768, 8)):
        assert lib.mf_plan(ctypes.byref(bad), ctypes.byref(mf.PlanReq(35.0, 2**40, 0, 0, 1, 0)), ctypes.byref(out)) == -1
    for req in (mf.PlanReq(-1.0, 1, 0, 0, 1, 0), mf.PlanReq(101.0, 1, 0, 0, 1, 0), mf.PlanReq(float("nan"), 1, 0, 0, 1, 0),
                mf.PlanReq(10.0, 1, 0, 0, -1, 0), mf.PlanReq(10.0, 1, 0, 0, 70000, 0)):
        assert lib.mf_plan(ctypes.byref(good), ctypes.byref(req), ctypes.byref(out)) == -1
    assert lib.mf_plan(ctypes.byref(good), ctypes.byref(mf.PlanReq(35.0, 10, 0, 0, 1, 0)), ctypes.byref(out)) == -2
    assert out.accepted == 0 and out.slots_per_layer == 22


def test_oracle_and_product_share_no_code():
    """Neither side imports, includes or links the other."""
    pkg_dir = os.path.join(ROOT, "paper_2607_09686_gb300")
    for dirpath, _, files in os.walk(pkg_dir):
        for f in files:
            if f.endswith((".py", ".cu", ".cuh", ".h", ".c")):
                text = open(os.path.join(dirpath, f)).read()
                assert "oracle" not in text.replace("oracle.", "").lower() or "import oracle" not in text
                assert "import oracle" not in text and "from oracle" not in text and "liboracle" not in text
    for f in os.listdir(os.path.join(ROOT, "oracle")):
        if f.endswith((".py", ".c", ".h")):
            text = open(os.path.join(ROOT, "oracle", f)).read()
            assert "paper_2607_09686_gb300" not in text and "mawforge.h" not in text and "libmawforge" not in text
