"""Benchmark of the routed-expert step: MoE-layer decode tokens/s at batch 1.

Workload (default): 4 MoE layers, hidden 2048, 64 experts, top-8, intermediate 768, Q8_0,
256 decode tokens at batch 1 per step, Zipf(1.1) routing with 0.6 reuse of the previous
token's set, expert cache 35% of each layer's experts (22 slots).  A step is the whole
256-token sequence through all 4 layers from a cold cache; `value` = tokens / s where a token
passes all 4 layers.  Inputs (activations, planted router bias, router weights) are resident
in HBM, the split-pack is in pinned host memory, misses are materialised inside the step.

Each step is one CUDA graph replay of the 1024 C-ABI calls (captured once); L2 is flushed
(a 512 MB write) between steps, outside the per-step CUDA events.  The kernel breakdown comes
from CUDA events the library records around every launch, on the launching stream; they are
captured into the graph, so they time the launches of the timed replays themselves.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--cache-pct P] [--impl mawforge|reference]
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

WORKLOAD = "l4e64"
N_TOKENS = 256
METRIC = "MoE-layer decode tokens/s at batch 1 (token = all 4 MoE layers)"  # both arms report it


def workload_name(cache_pct: float) -> str:
    """The headline workload, named the same way by both arms."""
    return (f"{WORKLOAD}: 4 MoE layers, hidden 2048, 64 experts, top-8, inter 768, Q8_0, "
            f"256 decode tokens batch 1, Zipf 1.1 + 0.6 reuse, cache {cache_pct:g}%")

# DRAM bytes (read + write) of one launch of the roofline kernel (the fused one-token FFN) from
# the ncu capture summarised under profiles/, valid while the kernel sources hash to `sha`
# (otherwise the line reports null: the counters no longer describe the kernel that ran).  The
# hash is re-recorded without a new capture only when the kernel's compiled device code is
# byte-identical to the captured build's.
KERNEL_TRAFFIC = {"sha": "07c0cef5dbf0b6c0", "bytes": 40199424,
                  "files": ("paper_2607_09686_gb300/csrc/mf_decode.cu", "paper_2607_09686_gb300/csrc/mf_dequant.cuh",
                            "paper_2607_09686_gb300/csrc/mf_internal.cuh")}


def _sources_sha():
    import hashlib
    h = hashlib.sha256()
    for f in KERNEL_TRAFFIC["files"]:
        with open(os.path.join(ROOT, f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def _captured_traffic():
    return KERNEL_TRAFFIC["bytes"] if KERNEL_TRAFFIC["sha"] == _sources_sha() else None


HBM_NOMINAL_GBS = 8000.0  # the GPU's nominal HBM3e bandwidth (~8 TB/s), reported beside the measured copy peak


def _peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


class ClockSampler:
    """nvidia-smi clock / throttle sampling during the timed region."""
    Q = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
         "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
         "clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index, self.proc = index, None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.index}", f"--query-gpu={self.Q}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None
        return self

    def __exit__(self, *a):
        self.lines = []
        if self.proc:
            self.proc.terminate()
            try:
                out, _ = self.proc.communicate(timeout=5)
                self.lines = [l for l in out.splitlines() if l.strip()]
            except Exception:
                self.proc.kill()

    def summary(self):
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in getattr(self, "lines", []):
            f = [v.strip() for v in line.split(",")]
            if len(f) < 7:
                continue
            try:
                sm.append(float(f[0]))
                mx = float(f[1])
            except ValueError:
                continue
            for n, v in zip(names, f[3:7]):
                if v.lower() == "active":
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(sm)}


def max_over_ranks(torch, v: float, device) -> float:
    """The largest of the ranks' values (a job ends with its slowest rank); v itself on one rank."""
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return v
    t = torch.tensor([v], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_rate(units_per_rank: float, ms_max: float, ws: int) -> float:
    """Whole-job throughput: every rank's units (weak scaling: the same on each) over the slowest
    rank's time."""
    return units_per_rank * ws / (ms_max * 1e-3)


def _dist():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def build_workload(torch, mf, synth, cache_pct, device):
    cfg = synth.CONFIGS[WORKLOAD]
    L, H, E, k, I, q = cfg.n_layers, cfg.hidden, cfg.n_experts, cfg.top_k, cfg.inter, cfg.qtype
    model = mf.Model(L, H, E, k, I, q)
    plan = mf.mf_plan(model, mf.PlanReq(cache_pct, 1 << 62, 0, 0, 1, 0))
    ctx = mf.mf_create(model, plan, device.index or 0)
    buf = np.empty(plan.payload_bytes, np.uint8)
    for l in range(L):
        for e in range(E):
            synth.payload(cfg.model_seed, l, e, H, I, q, out=buf)
            mf.mf_pack_put(ctx, l, e, buf)
    route = cfg.route_classes[0]
    x = np.stack([synth.activations(0, l, 0, 0, N_TOKENS, H) for l in range(L)], 1)  # [T, L, H]
    bias = np.stack([synth.plant_bias(synth.routes(0, l, 0, E, k, N_TOKENS, route.zipf_s, route.reuse), E)
                     for l in range(L)], 1)  # [T, L, E]
    wr = torch.from_numpy(np.stack([synth.router_weights(cfg.model_seed, l, E, H) for l in range(L)])).to(device)
    return cfg, model, plan, ctx, x, bias, wr


def run_mawforge(args):
    import torch
    import paper_2607_09686_gb300 as mf
    import synth

    ws, rank, local = _dist()
    if ws > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl" if torch.cuda.is_available() else "gloo")
    device = torch.device(f"cuda:{local}")
    torch.cuda.set_device(device)
    cfg, model, plan, ctx, x_np, bias_np, wr = build_workload(torch, mf, synth, args.cache_pct, device)
    L, H, E, k = cfg.n_layers, cfg.hidden, cfg.n_experts, cfg.top_k
    x = torch.from_numpy(x_np).to(device)
    bias = torch.from_numpy(bias_np).to(device)
    y = torch.empty(N_TOKENS, L, H, device=device)
    flush = torch.empty(512 * 1024 * 1024 // 4, dtype=torch.float32, device=device)
    stream = torch.cuda.Stream(device)

    def step_calls():
        mf.mf_reset(ctx, 0, stream)
        for t in range(N_TOKENS):
            for l in range(L):
                mf.mf_moe_forward(ctx, l, x[t, l], wr[l], bias[t, l], 1, y[t, l], None, None, stream)

    # one graph per step (the 1024 calls of a 256-token sequence), captured through the C ABI.  The
    # timed steps replay a graph without instrumentation; the per-kernel breakdown comes from the
    # same calls captured a second time with the library's CUDA-event records around each launch
    # (graph nodes, so they time the launches of those replays), replayed right after.
    timed = ["router", "resolve", "materialize", "ffn_fused", "gateup_swiglu", "down_combine"]
    graph, graph_k = torch.cuda.CUDAGraph(), torch.cuda.CUDAGraph()
    with torch.cuda.stream(stream):
        step_calls()  # untimed eager pass: warms the pool
        stream.synchronize()
        mf.mf_timing(ctx, [])
        with torch.cuda.graph(graph, stream=stream):
            step_calls()
        mf.mf_timing(ctx, timed)
        with torch.cuda.graph(graph_k, stream=stream):
            step_calls()
    torch.cuda.synchronize()

    def one_step(g, ev0, ev1):
        with torch.cuda.stream(stream):
            flush.zero_()
            ev0.record(stream)
            g.replay()
            ev1.record(stream)

    for _ in range(args.warmup):
        one_step(graph, torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
    torch.cuda.synchronize()

    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
    evk = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
    kt = {name: [0.0, 0] for name in mf.KERNEL_CLASSES}
    if ws > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    with ClockSampler(local) as clk:
        t0 = time.perf_counter()
        for i in range(args.steps):
            one_step(graph, *evs[i])
        torch.cuda.synchronize()
        wall = time.perf_counter() - t0
        for i in range(args.steps):  # instrumented replays: kernel breakdown
            one_step(graph_k, *evk[i])
            for name, (kms, n) in mf.mf_timing_read(ctx).items():  # waits for this replay (outside its events)
                kt[name][0] += kms
                kt[name][1] += n
        torch.cuda.synchronize()
    step_ms = [a.elapsed_time(b) for a, b in evs]
    ms = sum(step_ms) / len(step_ms)
    ms_instrumented = sum(a.elapsed_time(b) for a, b in evk) / len(evk)
    ms = max_over_ranks(torch, ms, device)
    st = mf.mf_stats(ctx, -1)  # every step starts cold (mf_reset), so these are one step's counters
    mf.mf_timing(ctx, [])

    # end to end through the host-buffer entry point: per token, pinned host x/bias in, y out
    xh = torch.from_numpy(x_np).pin_memory()
    bh = torch.from_numpy(bias_np).pin_memory()
    yh = torch.empty(N_TOKENS, L, H).pin_memory()
    e2e_graph = torch.cuda.CUDAGraph()

    def e2e_calls():
        mf.mf_reset(ctx, 0, stream)
        for t in range(N_TOKENS):
            for l in range(L):
                mf.mf_moe_forward_host(ctx, l, xh[t, l], wr[l], bh[t, l], 1, yh[t, l], None, None, stream)

    with torch.cuda.stream(stream):
        e2e_calls()
        stream.synchronize()
        with torch.cuda.graph(e2e_graph, stream=stream):
            e2e_calls()
    torch.cuda.synchronize()
    e2e_ms = []
    for i in range(args.warmup + args.steps):
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        with torch.cuda.stream(stream):
            flush.zero_()
            a.record(stream)
            e2e_graph.replay()
            b.record(stream)
        b.synchronize()
        if i >= args.warmup:
            e2e_ms.append(a.elapsed_time(b))
    y_dev = y.cpu()
    assert torch.equal(y_dev, yh), "host-buffer path disagrees with the device path"

    hbm, peak_kind = _peaks()
    steps_per_tok = L
    payload = plan.payload_bytes
    # algorithmic bytes of one gate/up launch (k experts' gate+up blocks) and one down launch
    gu_bytes = k * 2 * cfg.inter * (H // 32) * 34 + 4 * H + 4 * k * cfg.inter
    dn_bytes = k * H * (cfg.inter // 32) * 34 + 4 * k * cfg.inter + 4 * H
    ms_gu, n_gu = kt["gateup_swiglu"]
    ms_dn, n_dn = kt["down_combine"]
    ms_ff, n_ff = kt["ffn_fused"]
    ms_mat, n_mat = kt["materialize"]
    if n_ff:  # one launch per call: gate/up + SwiGLU + down + combine
        rf_kernel = "ffn_fused (grouped dequant-GEMV: k experts' gate/up rows, then their down rows, one launch)"
        rf_bytes = gu_bytes + dn_bytes
        rf_gbs = rf_bytes / (ms_ff / n_ff * 1e-3) / 1e9
    else:
        rf_kernel = "gateup_swiglu (grouped dequant-GEMV, k experts' gate+up rows)"
        rf_bytes = gu_bytes
        rf_gbs = gu_bytes / (ms_gu / n_gu * 1e-3) / 1e9
    gemv_ms = ms_ff + ms_gu + ms_dn
    gemv_gbs = (gu_bytes + dn_bytes) * (n_ff + n_gu) / (gemv_ms * 1e-3) / 1e9
    tokens = N_TOKENS * args.steps * ws
    value = job_rate(N_TOKENS, ms, ws)
    e2e_ms_max = max_over_ranks(torch, statistics.mean(e2e_ms), device)
    clocks = clk.summary()
    kernels = {name: {"ms_total": round(v[0], 4), "launches": v[1],
                      "us_per_launch": round(1e3 * v[0] / v[1], 3) if v[1] else None} for name, v in kt.items()}
    line = {
        "metric": METRIC,
        "value": round(value, 2),
        "unit": "tokens/s",
        "n_gpus": ws,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": round(ms, 4),
        "ms_per_step_instrumented": round(ms_instrumented, 4),
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "q8_0 weights, f32 activations and accumulation",
        "data": "synthetic (seeded; random-init Q8_0 experts; planted Zipf routing)",
        "config": {"workload": workload_name(args.cache_pct),
                   "cache_pct": args.cache_pct, "slots_per_layer": plan.slots_per_layer,
                   "tokens_per_step": N_TOKENS, "layers": L, "l2": "flushed between steps (512 MB write)",
                   "execution": "one CUDA graph per step of the 1024 C-ABI calls"},
        "cache": {"hit_rate": round(st["hits"] / max(1, st["accesses"]), 4),
                  "materialized_bytes_per_token": st["bytes_materialized"] / N_TOKENS,
                  "misses_per_token": st["misses"] / N_TOKENS, "accesses_per_step": st["accesses"]},
        "roofline": {"bound": "hbm", "kernel": rf_kernel,
                     "achieved": round(rf_gbs, 1), "peak": hbm, "unit": "GB/s",
                     "frac": round(rf_gbs / hbm, 4), "peak_kind": peak_kind, "traffic": _captured_traffic(),
                     "frac_of_nominal": round(rf_gbs / HBM_NOMINAL_GBS, 4),
                     "bytes_per_launch": rf_bytes,
                     "bytes_note": "every launch reads its resident experts' blocks from HBM and writes its missed "
                                   "experts' blocks to HBM: k payloads per launch; traffic is an all-resident "
                                   "launch's ncu DRAM bytes",
                     "timing": "CUDA events around each launch in instrumented replays of the step graph; "
                               "launches with misses wait on the host link"},
        "kernels": kernels,
        "copy": {"materialized_bytes_per_step": st["bytes_materialized"],
                 "materialize_gbs": round(args.steps * st["bytes_materialized"] / (ms_mat * 1e-3) / 1e9, 1)
                 if ms_mat else None,
                 "link_gbs_lower_bound": round(args.steps * st["bytes_materialized"] / (gemv_ms * 1e-3) / 1e9, 1)
                 if n_ff else None,
                 "note": "one-token calls materialise inside the fused FFN launch; the lower bound divides "
                         "the materialised bytes by all of that kernel's time"},
        "clocks": clocks,
        "e2e": {"value": round(job_rate(N_TOKENS, e2e_ms_max, ws), 2), "unit": "tokens/s",
                "h2d_bytes_per_step": N_TOKENS * L * (H + E) * 4, "d2h_bytes_per_step": N_TOKENS * L * H * 4},
        "gpu_launches": None,
        "wall_s": round(wall, 3),
    }
    # every kernel of the timed replays: the timed classes (counted in the instrumented replays of
    # the same calls) and one reset per step
    line["gpu_launches"] = int(sum(v[1] for v in kt.values())) + args.steps
    mf.mf_destroy(ctx)
    h2d = h2d_bandwidth(torch, device, stream)
    link_ms = st["bytes_materialized"] / (h2d * 1e9) * 1e3
    line["copy"].update({"h2d_gbs_measured": round(h2d, 1),
                         "link_ms_per_step_at_h2d": round(link_ms, 3),
                         "link_share_of_step": round(link_ms / ms, 4),
                         "h2d_how": "pinned host -> device cudaMemcpyAsync of 1 GiB, best of 10, this run"})
    if n_ff and not args.no_resident and rank == 0:
        line["roofline"]["resident"] = resident_measurement(torch, mf, synth, device, x, bias, wr, stream, flush,
                                                            args.steps, rf_bytes, hbm)
    if not args.no_prefill and rank == 0:
        line["prefill"] = prefill_measurement(torch, mf, synth, device)
    if not args.no_batch64 and rank == 0:
        line["batch64"] = batch64_measurement(torch, mf, synth, device)
    if not args.no_tuner and rank == 0:  # last of the GPU measurements: a failure here costs only this object
        try:
            line["tuner"] = tuner_measurement(torch, mf, synth, device, x, bias, wr, stream, flush, h2d)
        except Exception as e:
            line["tuner"] = {"error": f"{type(e).__name__}: {e}"}
    if not args.no_spec and rank == 0:
        try:
            line["speculative"] = spec_measurement(torch, mf, synth, device, x, bias, wr, stream, flush,
                                                   args.cache_pct)
        except Exception as e:
            line["speculative"] = {"error": f"{type(e).__name__}: {e}"}
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        runs = [cpu_baseline(args.cpu_tokens, args.cache_pct) for _ in range(args.cpu_passes)]
        line["cpu_baseline"] = dict(runs[0], value=round(statistics.mean(r["value"] for r in runs), 4),
                                    sample=runs[0]["sample"] + f", {args.cpu_passes} passes from a cold cache")
        others = {}  # the oracle beside the other measured workloads (bounded samples)
        for name, fn in (("prefill", cpu_baseline_prefill), ("batch64", cpu_baseline_batch64)):
            try:
                others[name] = fn()
            except Exception as e:
                others[name] = {"error": f"{type(e).__name__}: {e}"}
        line["cpu_baseline"]["other_workloads"] = others
    if rank == 0:
        print(json.dumps(line))
    if ws > 1:
        torch.distributed.destroy_process_group()


def resident_measurement(torch, mf, synth, device, x, bias, wr, stream, flush, steps, bytes_per_launch, hbm):
    """The same 1024 calls with every expert resident (a 100 % cache, warmed by one pass): the
    fused FFN launch is then HBM-bound; CUDA events around each launch in graph replays."""
    cfg = synth.CONFIGS[WORKLOAD]
    L, H, E, k, I, q = cfg.n_layers, cfg.hidden, cfg.n_experts, cfg.top_k, cfg.inter, cfg.qtype
    model = mf.Model(L, H, E, k, I, q)
    plan = mf.mf_plan(model, mf.PlanReq(100.0, 1 << 62, 0, 0, 1, 0))
    ctx = mf.mf_create(model, plan, device.index or 0)
    try:
        buf = np.empty(plan.payload_bytes, np.uint8)
        for l in range(L):
            for e in range(E):
                synth.payload(cfg.model_seed, l, e, H, I, q, out=buf)
                mf.mf_pack_put(ctx, l, e, buf)
        y = torch.empty(N_TOKENS, L, H, device=device)

        def calls():
            for t in range(N_TOKENS):
                for l in range(L):
                    mf.mf_moe_forward(ctx, l, x[t, l], wr[l], bias[t, l], 1, y[t, l], None, None, stream)

        with torch.cuda.stream(stream):
            for _ in range(2):  # every expert the sequence uses becomes resident
                calls()
            stream.synchronize()
            mf.mf_timing(ctx, ["ffn_fused"])
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=stream):
                calls()
        torch.cuda.synchronize()
        mf.mf_stats(ctx, -1, reset=True)
        ms, n = 0.0, 0
        for i in range(3 + steps):
            with torch.cuda.stream(stream):
                flush.zero_()
                g.replay()
            r = mf.mf_timing_read(ctx)["ffn_fused"]
            if i >= 3:
                ms += r[0]
                n += r[1]
        mf.mf_timing(ctx, [])
        st = mf.mf_stats(ctx, -1)
    finally:
        mf.mf_destroy(ctx)
    us = 1e3 * ms / n
    gbs = bytes_per_launch / (us * 1e-6) / 1e9
    return {"achieved": round(gbs, 1), "frac": round(gbs / hbm, 4), "frac_of_nominal": round(gbs / HBM_NOMINAL_GBS, 4),
            "us_per_launch": round(us, 3), "launches": n,
            "misses_in_timed_replays": st["misses"],
            "how": "same calls, 100 % cache warmed by two passes (every launch all-resident), L2 flushed per replay",
            "read_floor": read_floor(torch, device, stream, flush, bytes_per_launch, hbm)}


def tuner_measurement(torch, mf, synth, device, x, bias, wr, stream, flush, h2d_gbs: float,
                      pcts=(15.0, 25.0, 35.0, 50.0, 100.0), reps: int = 3) -> dict:
    """The cache-size tuner (mf_tune_cache) against measured steps of the same workload.  One
    context with a 100 % pool: a cold pass records the route trace (the router's output order),
    a warm pass makes every expert resident and its graph replays give the all-resident time per
    token; with the pinned link rate per payload these go into the tuner.  Each candidate size is
    then run (mf_reset to its slot count, graph replays that start cold) and its measured rate
    and miss count set beside the tuner's prediction."""
    cfg = synth.CONFIGS[WORKLOAD]
    L, H, E, k, I, q = cfg.n_layers, cfg.hidden, cfg.n_experts, cfg.top_k, cfg.inter, cfg.qtype
    model = mf.Model(L, H, E, k, I, q)
    plan = mf.mf_plan(model, mf.PlanReq(100.0, 1 << 62, 0, 0, 1, 0))
    ctx = mf.mf_create(model, plan, device.index or 0)
    try:
        buf = np.empty(plan.payload_bytes, np.uint8)
        for l in range(L):
            for e in range(E):
                synth.payload(cfg.model_seed, l, e, H, I, q, out=buf)
                mf.mf_pack_put(ctx, l, e, buf)
        y = torch.empty(N_TOKENS, L, H, device=device)
        idx = torch.empty(N_TOKENS, L, k, dtype=torch.int32, device=device)

        def calls(reset: bool, record: bool = False):
            if reset:
                mf.mf_reset(ctx, 0, stream)
            for t in range(N_TOKENS):
                for l in range(L):
                    mf.mf_moe_forward(ctx, l, x[t, l], wr[l], bias[t, l], 1, y[t, l], idx[t, l] if record else None,
                                      None, stream)

        def replay_ms(graph) -> float:  # one untimed replay, then the mean of `reps` (L2 flushed before each)
            ms = []
            for i in range(1 + reps):
                a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                with torch.cuda.stream(stream):
                    flush.zero_()
                    a.record(stream)
                    graph.replay()
                    b.record(stream)
                torch.cuda.synchronize()
                if i:
                    ms.append(a.elapsed_time(b))
            return statistics.mean(ms)

        with torch.cuda.stream(stream):
            calls(True, record=True)  # cold: the routes as the cache sees them
            calls(False)  # warm: every expert of the sequence resident
            stream.synchronize()
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=stream):
                calls(False)
        torch.cuda.synchronize()
        routes = idx.permute(1, 0, 2).contiguous().cpu().numpy()  # [L][tokens][k]
        resident_ms = replay_ms(g)
        del g
        t_token = resident_ms * 1e-3 / N_TOKENS
        t_miss = plan.payload_bytes / (h2d_gbs * 1e9)
        pts, best = mf.mf_tune_cache(model, mf.PlanReq(0.0, 1 << 62, 0, 0, 1, 0), routes, 1, t_token, t_miss,
                                     list(pcts))
        points = []
        for pt in pts:
            mf.mf_reset(ctx, pt["slots_per_layer"], stream)
            with torch.cuda.stream(stream):
                calls(True)
                stream.synchronize()
                g = torch.cuda.CUDAGraph()
                with torch.cuda.graph(g, stream=stream):
                    calls(True)
            torch.cuda.synchronize()
            ms = replay_ms(g)
            del g
            st = mf.mf_stats(ctx, -1)  # the last replay's counters: every replay starts with a reset
            points.append({"cache_pct": pt["cache_pct"], "slots_per_layer": pt["slots_per_layer"],
                           "misses_predicted": pt["misses"], "misses_measured": st["misses"],
                           "tokens_per_s_predicted": round(pt["predicted_tokens_per_s"], 1),
                           "tokens_per_s_measured": round(N_TOKENS / (ms * 1e-3), 1)})
        assert mf.mf_check(ctx) == 0
    finally:
        mf.mf_destroy(ctx)
    measured_best = max(range(len(points)), key=lambda i: points[i]["tokens_per_s_measured"])
    return {"how": "route trace of the 1024 calls (router order), all-resident time per token from graph replays "
                   "of a warm 100 % cache, link time per payload at the measured pinned copy rate; each candidate "
                   "run from a cold cache of its slot count (one context, mf_reset), L2 flushed per replay",
            "t_token_us": round(t_token * 1e6, 3), "t_miss_us": round(t_miss * 1e6, 3),
            "points": points, "best_predicted_pct": pts[best]["cache_pct"] if best >= 0 else None,
            "best_measured_pct": points[measured_best]["cache_pct"]}


def spec_measurement(torch, mf, synth, device, x, bias, wr, stream, flush, cache_pct: float, K: int = 4,
                     alpha: float = 0.6, reps: int = 2) -> dict:
    """Verification-width accounting of speculative decoding on the same 256 tokens (section
    "Throughput Model": extra_materialization; Discussion: record drafted and accepted tokens,
    verification width, misses and materialised bytes).  No draft model: a seeded schedule
    accepts the first a of K drafts per verify step (each with probability alpha), and rejected
    drafts carry routes and activations of an independent stream.  Each verify step is one call
    per layer with T = K + 1 (the union of its rows' experts is materialised); plain decode is
    one call per token and layer.  Both run eagerly on one context from a cold cache, CUDA
    events around the whole sequence; the cache-size tuner replays each recorded trace to
    predict its misses."""
    cfg = synth.CONFIGS[WORKLOAD]
    L, H, E, k, I, q = cfg.n_layers, cfg.hidden, cfg.n_experts, cfg.top_k, cfg.inter, cfg.qtype
    route = cfg.route_classes[0]
    W = K + 1
    rows = synth.verify_rows(0, N_TOKENS, K, alpha)  # [batches, W]
    nb, n_drafts = rows.shape[0], int((rows < 0).sum())
    xh, bh = x.cpu().numpy(), bias.cpu().numpy()  # [T, L, H], [T, L, E]
    xb = np.empty((nb, L, W, H), np.float32)
    bb = np.empty((nb, L, W, E), np.float32)
    for l in range(L):
        xd = synth.activations(0, l, 1, 0, n_drafts, H)
        bd = synth.plant_bias(synth.routes(0, l, 1, E, k, n_drafts, route.zipf_s, 0.0), E)
        for b in range(nb):
            for j in range(W):
                v = int(rows[b, j])
                xb[b, l, j] = xh[v, l] if v >= 0 else xd[-1 - v]
                bb[b, l, j] = bh[v, l] if v >= 0 else bd[-1 - v]
    xb, bb = torch.from_numpy(xb).to(device), torch.from_numpy(bb).to(device)
    model = mf.Model(L, H, E, k, I, q)
    plan = mf.mf_plan(model, mf.PlanReq(cache_pct, 1 << 62, 0, 0, W, 0))
    ctx = mf.mf_create(model, plan, device.index or 0)
    try:
        buf = np.empty(plan.payload_bytes, np.uint8)
        for l in range(L):
            for e in range(E):
                synth.payload(cfg.model_seed, l, e, H, I, q, out=buf)
                mf.mf_pack_put(ctx, l, e, buf)
        y1 = torch.empty(N_TOKENS, L, H, device=device)
        yb = torch.empty(nb, L, W, H, device=device)
        i1 = torch.empty(N_TOKENS, L, k, dtype=torch.int32, device=device)
        ib = torch.empty(nb, L, W, k, dtype=torch.int32, device=device)

        def decode():
            for t in range(N_TOKENS):
                for l in range(L):
                    mf.mf_moe_forward(ctx, l, x[t, l], wr[l], bias[t, l], 1, y1[t, l], i1[t, l], None, stream)

        def verify():
            for b in range(nb):
                for l in range(L):
                    mf.mf_moe_forward(ctx, l, xb[b, l], wr[l], bb[b, l], W, yb[b, l], ib[b, l], None, stream)

        def run(fn):  # one untimed pass, then the mean of `reps`; each from a cold cache
            ms = []
            for i in range(1 + reps):
                with torch.cuda.stream(stream):
                    flush.zero_()
                    mf.mf_reset(ctx, 0, stream)
                    a, z = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                    a.record(stream)
                    fn()
                    z.record(stream)
                z.synchronize()
                if i:
                    ms.append(a.elapsed_time(z))
            return statistics.mean(ms), mf.mf_stats(ctx, -1)

        ms1, st1 = run(decode)
        msv, stv = run(verify)
        assert mf.mf_check(ctx) == 0
        tr1 = i1.permute(1, 0, 2).contiguous().cpu().numpy()  # [L][tokens][k]
        trv = ib.permute(1, 0, 2, 3).reshape(L, nb * W, k).contiguous().cpu().numpy()  # [L][rows][k]
    finally:
        mf.mf_destroy(ctx)
    req = mf.PlanReq(0.0, 1 << 62, 0, 0, W, 0)
    p1 = mf.mf_tune_cache(model, req, tr1, 1, 0.0, 0.0, [cache_pct])[0][0]
    pv = mf.mf_tune_cache(model, req, trv, W, 0.0, 0.0, [cache_pct])[0][0]
    return {"how": "seeded acceptance schedule (no draft model), verify steps of K + 1 rows as one call per "
                   "layer, plain decode as one call per token and layer, eager calls on one context from a "
                   "cold cache, CUDA events around each whole sequence",
            "K": K, "alpha": alpha, "width": W, "cache_pct": cache_pct, "tokens": N_TOKENS, "verify_steps": nb,
            "accepted_drafts": N_TOKENS - nb, "rejected_drafts": n_drafts,
            "misses": {"decode": st1["misses"], "decode_predicted": p1["misses"],
                       "verify": stv["misses"], "verify_predicted": pv["misses"]},
            "extra_materialized_mb_per_token": round((stv["bytes_materialized"] - st1["bytes_materialized"])
                                                     / N_TOKENS / 1e6, 3),
            "tokens_per_s": {"decode": round(N_TOKENS / (ms1 * 1e-3), 1),
                             "speculative": round(N_TOKENS / (msv * 1e-3), 1)}}


def h2d_bandwidth(torch, device, stream, nbytes: int = 1 << 30, reps: int = 10) -> float:
    """GB/s of one pinned host -> device copy engine transfer (the CPU-GPU link's rate for a
    plain copy), best of `reps`."""
    src = torch.empty(nbytes, dtype=torch.uint8).pin_memory()
    dst = torch.empty(nbytes, dtype=torch.uint8, device=device)
    best = 0.0
    with torch.cuda.stream(stream):
        for _ in range(reps):
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(stream)
            dst.copy_(src, non_blocking=True)
            b.record(stream)
            b.synchronize()
            best = max(best, nbytes / (a.elapsed_time(b) * 1e-3) / 1e9)
    del src, dst
    return best


def read_floor(torch, device, stream, flush, nbytes, hbm, reps: int = 20) -> dict:
    """What one read-only launch of the same size achieves: a torch.sum over nbytes of fp32 from a
    cold L2, CUDA events around the launch (the launch and first-access latency that bound any
    single kernel of this size)."""
    buf = torch.ones(nbytes // 4, dtype=torch.float32, device=device)
    out = torch.empty((), dtype=torch.float32, device=device)
    times = []
    with torch.cuda.stream(stream):
        for i in range(3 + reps):
            flush.zero_()
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(stream)
            torch.sum(buf, 0, dtype=torch.float32, out=out)
            b.record(stream)
            b.synchronize()
            if i >= 3:
                times.append(a.elapsed_time(b) * 1e3)
    us = statistics.mean(times)
    gbs = nbytes / (us * 1e-6) / 1e9
    return {"us": round(us, 3), "achieved": round(gbs, 1), "frac": round(gbs / hbm, 4),
            "how": "one torch.sum launch over the same bytes after an L2 flush, CUDA events around it"}


def prefill_measurement(torch, mf, synth, device, calls: int = 4, cache_pct: float = 15.0) -> dict:
    """The tensor-core grouped GEMM path on one layer of the 48-layer Q4_0 workload: one
    4096-token prefill call (Zipf 1.2 routing) from a cold cache, `calls` times after one warm-up.
    Per call: the GEMM kernels' summed CUDA-event time (gate/up+SwiGLU and down, every wave) and the
    whole call.  FLOPs: useful = 2 * T * k * 3 * hidden * inter; issued on the tensor cores = 3x that
    (hi*hi + hi*lo + lo*hi bf16 products)."""
    cfg = synth.CONFIGS["l48e128q4"]
    H, E, k, I, q, T = cfg.hidden, cfg.n_experts, cfg.top_k, cfg.inter, cfg.qtype, cfg.prefill
    model = mf.Model(1, H, E, k, I, q)
    plan = mf.mf_plan(model, mf.PlanReq(cache_pct, 1 << 62, 0, 0, T, 0))
    ctx = mf.mf_create(model, plan, device.index or 0)
    try:
        buf = np.empty(plan.payload_bytes, np.uint8)
        for e in range(E):
            synth.payload(cfg.model_seed, 0, e, H, I, q, out=buf)
            mf.mf_pack_put(ctx, 0, e, buf)
        route = cfg.route_classes[0]
        x = torch.from_numpy(synth.activations(0, 0, 0, 0, T, H)).to(device)
        b = torch.from_numpy(synth.plant_bias(synth.routes(0, 0, 0, E, k, T, route.zipf_s, route.reuse), E)).to(device)
        wr = torch.from_numpy(synth.router_weights(cfg.model_seed, 0, E, H)).to(device)
        y = torch.empty(T, H, device=device)
        stream = torch.cuda.Stream(device)
        gemm_ms, call_ms, mat_ms, rt_ms, rs_ms, n_gemm = [], [], [], [], [], 0
        for i in range(calls + 1):
            mf.mf_reset(ctx, 0, stream)
            mf.mf_timing(ctx, ["router", "resolve", "materialize", "prefill_gemm"])
            a, z = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            with torch.cuda.stream(stream):
                a.record(stream)
                mf.mf_moe_forward(ctx, 0, x, wr, b, T, y, None, None, stream)
                z.record(stream)
            z.synchronize()
            tm = mf.mf_timing_read(ctx)
            if i > 0:
                gemm_ms.append(tm["prefill_gemm"][0])
                mat_ms.append(tm["materialize"][0])
                rt_ms.append(tm["router"][0])
                rs_ms.append(tm["resolve"][0])
                n_gemm = tm["prefill_gemm"][1]
                call_ms.append(a.elapsed_time(z))
        mf.mf_timing(ctx, [])
        assert mf.mf_check(ctx) == 0
        st = mf.mf_stats(ctx, -1)
    finally:
        mf.mf_destroy(ctx)
    g, c, m = statistics.mean(gemm_ms), statistics.mean(call_ms), statistics.mean(mat_ms)
    useful = 2.0 * T * k * 3 * H * I
    issued = 3 * useful
    peak = _bf16_peak()
    return {"workload": f"l48e128q4 layer 0: 4096-token prefill call, hidden {H}, {E} experts, top-{k}, inter {I}, "
                        f"Q4_0, Zipf 1.2, cache {cache_pct:g}% ({plan.slots_per_layer} slots), cold",
            "tokens_per_s": round(T / (c * 1e-3), 1), "call_ms": round(c, 4), "gemm_ms": round(g, 4),
            "gemm_waves": n_gemm, "materialize_ms": round(m, 4), "router_ms": round(statistics.mean(rt_ms), 4),
            "resolve_ms": round(statistics.mean(rs_ms), 4),
            "materialize_gbs": round(st["bytes_materialized"] / (m * 1e-3) / 1e9, 1),
            "useful_tflops": round(useful / (g * 1e-3) / 1e12, 2),
            "roofline": {"bound": "tensor", "kernel": "prefill grouped GEMMs (gate/up+SwiGLU, down)",
                         "achieved": round(issued / (g * 1e-3) / 1e12, 2), "peak": peak[0], "unit": "TFLOP/s",
                         "frac": round(issued / (g * 1e-3) / 1e12 / peak[0], 4), "peak_kind": peak[1],
                         "flops_per_call": {"useful": useful, "issued": issued}}}


def batch64_measurement(torch, mf, synth, device, steps: int = 8, warm: int = 2, cache_pct: float = 15.0) -> dict:
    """64 concurrent decode streams on one layer of the 30-layer workload (hidden 2816, 128
    experts, top-8, inter 1408, Q8_0, Zipf 1.0 per stream) at 15 % cache: one call of T = 64 per
    step (~107 distinct experts against 19 slots: 6 waves, their misses over the host link), for
    both access orders.  CUDA events around `steps` calls after `warm` calls."""
    cfg = synth.CONFIGS["l30e128b64"]
    H, E, k, I, q, B = cfg.hidden, cfg.n_experts, cfg.top_k, cfg.inter, cfg.qtype, cfg.batch
    model = mf.Model(1, H, E, k, I, q)
    plan = mf.mf_plan(model, mf.PlanReq(cache_pct, 1 << 62, 0, 0, B, 0))
    ctx = mf.mf_create(model, plan, device.index or 0)
    out = {"workload": f"l30e128b64 layer 0: {B} decode streams per call, hidden {H}, {E} experts, top-{k}, "
                       f"inter {I}, Q8_0, Zipf {cfg.route_classes[0].zipf_s:g} per stream, cache {cache_pct:g}% "
                       f"({plan.slots_per_layer} slots)"}
    try:
        buf = np.empty(plan.payload_bytes, np.uint8)
        for e in range(E):
            synth.payload(cfg.model_seed, 0, e, H, I, q, out=buf)
            mf.mf_pack_put(ctx, 0, e, buf)
        n = warm + steps
        klass = cfg.route_classes[0]
        routes = np.stack([synth.routes(0, 0, st, E, k, n, klass.zipf_s, klass.reuse) for st in range(B)], 1)
        wr = torch.from_numpy(synth.router_weights(cfg.model_seed, 0, E, H)).to(device)
        xs = [torch.from_numpy(np.concatenate([synth.activations(0, 0, st, i, 1, H) for st in range(B)])).to(device)
              for i in range(n)]
        bs = [torch.from_numpy(synth.plant_bias(routes[i], E)).to(device) for i in range(n)]
        y = torch.empty(B, H, device=device)
        for name, order in (("first_occurrence", mf.MF_ORDER_FIRST_OCCURRENCE),
                            ("resident_first", mf.MF_ORDER_RESIDENT_FIRST)):
            mf.mf_reset(ctx)
            mf.mf_access_order(ctx, order)
            for i in range(warm):
                mf.mf_moe_forward(ctx, 0, xs[i], wr, bs[i], B, y)
            torch.cuda.synchronize()
            mf.mf_stats(ctx, 0, reset=True)
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record()
            for i in range(warm, n):
                mf.mf_moe_forward(ctx, 0, xs[i], wr, bs[i], B, y)
            b.record()
            b.synchronize()
            ms = a.elapsed_time(b) / steps
            st = mf.mf_stats(ctx, 0)
            out[name] = {"tokens_per_s": round(B / (ms * 1e-3), 1), "ms_per_step": round(ms, 4),
                         "hit_rate": round(st["hits"] / st["accesses"], 4),
                         "materialized_mb_per_step": round(st["bytes_materialized"] / steps / 1e6, 2),
                         "link_gbs": round(st["bytes_materialized"] / steps / (ms * 1e-3) / 1e9, 1)}
        assert mf.mf_check(ctx) == 0
    finally:
        mf.mf_destroy(ctx)
    return out


def _bf16_peak():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return float(json.load(f)["bf16_tflops"]), "measured (burst)"
    except Exception:
        return 1900.0, "fallback"


def cpu_baseline(n_tokens: int, cache_pct: float = 35.0) -> dict:
    """The CPU oracle, as it stands, on the first tokens of the same workload (same cache share)."""
    import oracle
    import synth
    cfg = synth.CONFIGS[WORKLOAD]
    L, H, E, k, I, q = cfg.n_layers, cfg.hidden, cfg.n_experts, cfg.top_k, cfg.inter, cfg.qtype
    route = cfg.route_classes[0]
    pays = {}
    slots = max(k, int(np.floor(cache_pct * E / 100 + 1e-9)))  # the planner's slot count
    lru = [oracle.LRU(E, slots, synth.payload_bytes(H, I, q)) for _ in range(L)]
    xs = [synth.activations(0, l, 0, 0, n_tokens, H) for l in range(L)]
    bs = [synth.plant_bias(synth.routes(0, l, 0, E, k, n_tokens, route.zipf_s, route.reuse), E) for l in range(L)]
    wrs = [synth.router_weights(cfg.model_seed, l, E, H) for l in range(L)]
    for l in range(L):  # payload generation is input preparation, outside the timing
        for e in set(bs[l].nonzero()[1].tolist()):
            pays[(l, e)] = synth.payload(cfg.model_seed, l, e, H, I, q)
    t0 = time.perf_counter()
    for t in range(n_tokens):
        for l in range(L):
            _, idx, _ = oracle.router(xs[l][t], wrs[l], bs[l][t], k)
            lru[l].step(idx[None])
            oracle.layer([pays.get((l, e)) for e in range(E)], q, H, I, k, wrs[l], bs[l][t:t + 1], xs[l][t:t + 1])
    dt = time.perf_counter() - t0
    cores = int(os.environ.get("OMP_NUM_THREADS", os.cpu_count() or 1))
    return {"value": round(n_tokens / dt, 4), "unit": "tokens/s", "cores": cores, "kind": "oracle",
            "slots_per_layer": slots,
            "sample": f"first {n_tokens} tokens of the same sequence (256 = the whole step), all {L} layers "
                      f"(router + LRU with {slots} slots + fp64 layer)"}


def cpu_baseline_prefill(n_tokens: int = 8, cache_pct: float = 15.0) -> dict:
    """The CPU oracle on the first tokens of the prefill measurement's 4096-token call (layer 0 of
    the 48-layer Q4_0 workload, the same inputs): the fp64 layer with its routing, and the call's
    cache step; tokens/s of one layer, like the GPU's prefill rate."""
    import oracle
    import synth
    cfg = synth.CONFIGS["l48e128q4"]
    H, E, k, I, q, T = cfg.hidden, cfg.n_experts, cfg.top_k, cfg.inter, cfg.qtype, cfg.prefill
    route = cfg.route_classes[0]
    x = synth.activations(0, 0, 0, 0, n_tokens, H)
    b = synth.plant_bias(synth.routes(0, 0, 0, E, k, T, route.zipf_s, route.reuse)[:n_tokens], E)
    wr = synth.router_weights(cfg.model_seed, 0, E, H)
    pays = {e: synth.payload(cfg.model_seed, 0, e, H, I, q) for e in set(b.nonzero()[1].tolist())}
    lru = oracle.LRU(E, max(k, int(np.floor(cache_pct * E / 100 + 1e-9))), synth.payload_bytes(H, I, q))
    t0 = time.perf_counter()
    _, idx, _ = oracle.layer([pays.get(e) for e in range(E)], q, H, I, k, wr, b, x)
    lru.step(idx)
    dt = time.perf_counter() - t0
    return {"value": round(n_tokens / dt, 4), "unit": "tokens/s (one layer)", "kind": "oracle",
            "sample": f"the first {n_tokens} tokens of the 4096-token prefill call, layer 0 of l48e128q4"}


def cpu_baseline_batch64(n_streams: int = 8, cache_pct: float = 15.0) -> dict:
    """The CPU oracle on the first streams of the 64-stream measurement's first call (layer 0 of
    the 30-layer workload, the same inputs): the fp64 layer with its routing and the cache step;
    tokens/s of one layer, like the GPU's 64-stream rate."""
    import oracle
    import synth
    cfg = synth.CONFIGS["l30e128b64"]
    H, E, k, I, q = cfg.hidden, cfg.n_experts, cfg.top_k, cfg.inter, cfg.qtype
    klass = cfg.route_classes[0]
    routes = np.stack([synth.routes(0, 0, st, E, k, 1, klass.zipf_s, klass.reuse)[0] for st in range(n_streams)])
    x = np.concatenate([synth.activations(0, 0, st, 0, 1, H) for st in range(n_streams)])
    b = synth.plant_bias(routes, E)
    wr = synth.router_weights(cfg.model_seed, 0, E, H)
    pays = {e: synth.payload(cfg.model_seed, 0, e, H, I, q) for e in set(routes.reshape(-1).tolist())}
    lru = oracle.LRU(E, max(k, int(np.floor(cache_pct * E / 100 + 1e-9))), synth.payload_bytes(H, I, q))
    t0 = time.perf_counter()
    _, idx, _ = oracle.layer([pays.get(e) for e in range(E)], q, H, I, k, wr, b, x)
    lru.step(idx)
    dt = time.perf_counter() - t0
    return {"value": round(n_streams / dt, 4), "unit": "tokens/s (one layer)", "kind": "oracle",
            "sample": f"the first {n_streams} of the 64 streams of the first call, layer 0 of l30e128b64"}


def run_reference(args):
    ws, rank, _ = _dist()
    if rank != 0:
        return
    per_step = []
    for i in range(args.warmup + args.steps):
        r = cpu_baseline(args.cpu_tokens, getattr(args, "cache_pct", 35.0))
        if i >= args.warmup:
            per_step.append(r)
    value = statistics.mean(r["value"] for r in per_step)
    line = {"impl": "reference", "metric": METRIC,
            "value": round(value, 4), "unit": "tokens/s", "n_gpus": ws, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": round(1e3 * args.cpu_tokens / value, 3), "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64 (CPU oracle)", "data": "synthetic (seeded)",
            "config": {"workload": workload_name(getattr(args, "cache_pct", 35.0)),
                       "sample": f"the first {args.cpu_tokens} tokens of the 256-token step",
                       "tokens_per_step": args.cpu_tokens},
            "cpu_baseline": {"value": round(value, 4), "unit": "tokens/s", "kind": "oracle",
                             "cores": per_step[0]["cores"], "sample": per_step[0]["sample"]},
            "e2e": {"value": round(value, 4), "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line))


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--cache-pct", type=float, default=35.0)
    ap.add_argument("--impl", default="mawforge", choices=["mawforge", "reference"])
    ap.add_argument("--cpu-tokens", type=int, default=256, help="tokens of the sequence the CPU oracle runs per pass")
    ap.add_argument("--cpu-passes", type=int, default=3, help="passes of the CPU baseline leg (~3 s each)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-prefill", action="store_true", help="skip the 4096-token prefill measurement")
    ap.add_argument("--no-resident", action="store_true", help="skip the all-resident FFN measurement")
    ap.add_argument("--no-batch64", action="store_true", help="skip the 64-stream batched decode measurement")
    ap.add_argument("--no-tuner", action="store_true", help="skip the cache-size tuner against measured steps")
    ap.add_argument("--no-spec", action="store_true", help="skip the speculative verification-width accounting")
    args = ap.parse_args()
    if args.impl == "reference":
        import oracle
        oracle.build()
        run_reference(args)
        return
    import __graft_entry__
    __graft_entry__.build()
    run_mawforge(args)


if __name__ == "__main__":
    main()
