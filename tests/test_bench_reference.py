"""bench.py's reference arm on CPU: it times the CPU oracle on a bounded sample of the headline
workload and prints one JSON line with the same metric, unit, direction and workload as the
GPU arm, a cpu_baseline object describing the run and an end-to-end object with no copies.
Two tokens through four of the 48 layers keep it to seconds."""
import argparse
import json

import bench


def test_reference_arm_json_line(monkeypatch, capsys):
    monkeypatch.setenv("WORLD_SIZE", "1")
    monkeypatch.setenv("RANK", "0")
    monkeypatch.setenv("LOCAL_RANK", "0")
    args = argparse.Namespace(steps=1, warmup=0, cpu_tokens=2, cache_pct=35.0)
    bench.run_reference(args)
    out = capsys.readouterr().out.strip().splitlines()
    assert len(out) == 1
    line = json.loads(out[0])
    assert line["impl"] == "reference"
    assert line["metric"] == bench.METRIC
    assert line["unit"] == "tokens/s" and line["higher_is_better"] is True
    assert line["n_gpus"] == 1 and line["steps"] == 1 and line["warmup"] == 0
    assert line["value"] > 0
    # value = layer-tokens / 48 per second: 2 tokens x 4 layers per step
    assert abs(line["ms_per_step"] - 1e3 * (2 * 4 / bench.N_LAYERS) / line["value"]) <= 1e-3 * line["ms_per_step"] + 1e-3
    assert line["config"]["workload"] == bench.workload_name(35.0)
    cb = line["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["value"] == line["value"] and cb["unit"] == line["unit"]
    assert cb["cores"] >= 1 and "2 tokens" in cb["sample"]
    assert line["e2e"] == {"value": line["value"], "unit": line["unit"], "h2d_bytes_per_step": 0,
                           "d2h_bytes_per_step": 0}


def test_cpu_baseline_cache_matches_the_planner():
    """The oracle's cache has as many slots per layer as the library's planner gives the GPU arm
    for the same cache share (the planner is host code: no GPU needed)."""
    import synth
    import paper_2607_09686_gb300 as mf
    cfg = synth.CONFIGS[bench.WORKLOAD]
    model = mf.Model(cfg.n_layers, cfg.hidden, cfg.n_experts, cfg.top_k, cfg.inter, cfg.qtype)
    for pct in (35.0, 15.0, 1.0):
        plan = mf.mf_plan(model, mf.PlanReq(pct, 1 << 62, 0, 0, 1, 0))
        r = bench.cpu_baseline(1, pct, 1)
        assert r["slots_per_layer"] == plan.slots_per_layer, pct
        assert r["value"] > 0 and r["kind"] == "oracle"


def test_oracle_samples_of_the_other_workloads():
    """The CPU-baseline leg also times the oracle on bounded samples of the prefill and 64-stream
    workloads (one layer each), beside the GPU's rates for them."""
    for fn in (bench.cpu_baseline_prefill, bench.cpu_baseline_batch64):
        r = fn(2)
        assert r["kind"] == "oracle" and r["value"] > 0 and r["unit"] == "tokens/s (one layer)"
        assert "first 2" in r["sample"]
