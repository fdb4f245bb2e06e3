"""Benchmark of the routed-expert step: MoE-layer decode tokens/s at batch 1.

Headline workload: 48 MoE layers shaped like a ~35B-total/3B-active MoE (hidden 2048, 128
experts, top-8, intermediate 768, Q8_0), a 96-token decode at batch 1 (seed 0), routing class
Zipf 1.2 with 0.8 reuse of the previous token's set, expert cache 35 % of each layer's experts
(44 slots).  A step is the whole 96-token sequence through all 48 layers from a cold cache (4608
calls); `value` = tokens / s where a token passes all 48 layers.  Inputs (activations, planted
router bias, router weights) are resident in HBM, the split-pack (31 GB) is in pinned host
memory, misses are materialised inside the step.

Each step is one CUDA graph replay of the 4608 C-ABI calls (captured once); L2 is flushed (a
512 MB write) between steps, outside the per-step CUDA events.  The kernel breakdown comes from
CUDA events the library records around every launch, on the launching stream; they are captured
into a second graph of the same calls, replayed after the timed steps.

Beside the headline the line carries: every route class x cache share of the workload (`sweep`),
the same calls with every expert resident (`roofline.resident`: per launch and sustained over the
step), the end-to-end rate through the host-buffer entry point (`e2e`), the pinned-pack placement
and link rates (`copy`), the cache-size tuner and the speculative verification accounting on the
headline sequence, the 48-layer Q4_0 workload (4096-token prefill call and the 96-token decode
that follows it), 64-stream batched decode, and the earlier 4-layer workload (`l4e64`).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl mawforge|reference]
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import time
from concurrent.futures import ThreadPoolExecutor

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

WORKLOAD = "l48e128"
HEAD_CLASS = "zipf1.2+reuse0.8"
HEAD_PCT = 35.0
HEAD_SEED = 0
N_TOKENS = 96
N_LAYERS = 48
METRIC = "MoE-layer decode tokens/s at batch 1 (token = all 48 MoE layers)"  # both arms report it


def workload_name(cache_pct: float = HEAD_PCT, klass: str = HEAD_CLASS) -> str:
    """The headline workload, named the same way by both arms."""
    return (f"{WORKLOAD}: 48 MoE layers, hidden 2048, 128 experts, top-8, inter 768, Q8_0, 96 decode tokens "
            f"batch 1 (seed {HEAD_SEED}), {klass}, cache {cache_pct:g}%")


# DRAM bytes (read + write) of one launch of the roofline kernel (the fused one-token FFN) from
# the ncu capture summarised under profiles/, valid while the kernel sources hash to `sha`
# (otherwise the line reports null: the counters no longer describe the kernel that ran).
KERNEL_TRAFFIC = {"sha": "66dcaba3a9f04fbd", "bytes": 40218368,
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


def _bf16_peak():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return float(json.load(f)["bf16_tflops"]), "measured (burst)"
    except Exception:
        return 1900.0, "fallback"


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


def slots_for(pct: float, n_experts: int, top_k: int) -> int:
    """The planner's slot count for a cache share (the same rule as mf_plan; used to name cells)."""
    return min(n_experts, max(top_k, int(np.floor(pct * n_experts / 100 + 1e-9))))


def _klass(cfg, name: str):
    return next(c for c in cfg.route_classes if c.name == name)


def fill_pack(mf, synth, ctx, cfg, workers: int = 16) -> None:
    """Every (layer, expert) payload of the model into the context's pinned pack."""
    L, H, E, I, q = cfg.n_layers, cfg.hidden, cfg.n_experts, cfg.inter, cfg.qtype
    n = synth.payload_bytes(H, I, q)

    def put(l):
        buf = np.empty(n, np.uint8)
        for e in range(E):
            synth.payload(cfg.model_seed, l, e, H, I, q, out=buf)
            mf.mf_pack_put(ctx, l, e, buf)

    with ThreadPoolExecutor(max_workers=workers) as ex:
        list(ex.map(put, range(L)))


def decode_inputs(synth, cfg, seed: int, klass, t0: int = 0, route_sets=None):
    """Activations [T, L, H] and planted bias [T, L, E] of a batch-1 decode (token-major)."""
    L, H, E, k, T = cfg.n_layers, cfg.hidden, cfg.n_experts, cfg.top_k, cfg.n_tokens
    x = np.stack([synth.activations(seed, l, 0, t0, T, H) for l in range(L)], 1)
    if route_sets is None:
        route_sets = [synth.routes(seed, l, 0, E, k, T, klass.zipf_s, klass.reuse) for l in range(L)]
    bias = np.stack([synth.plant_bias(route_sets[l], E) for l in range(L)], 1)
    return x, bias


class Decoder:
    """Graph captures of one decode sequence through a context: calls token-major, one per
    (token, layer); optionally a cache reset (to `slots` in use) at the start of the graph."""

    def __init__(self, torch, mf, ctx, x, bias, wr, stream):
        self.torch, self.mf, self.ctx, self.x, self.bias, self.wr, self.stream = torch, mf, ctx, x, bias, wr, stream
        self.T, self.L, self.H = x.shape[0], x.shape[1], x.shape[2]
        self.y = torch.empty_like(x)

    def calls(self, slots: int | None, idx=None):
        mf, ctx, s = self.mf, self.ctx, self.stream
        if slots is not None:
            mf.mf_reset(ctx, slots, s)
        for t in range(self.T):
            for l in range(self.L):
                mf.mf_moe_forward(ctx, l, self.x[t, l], self.wr[l], self.bias[t, l], 1, self.y[t, l],
                                  None if idx is None else idx[t, l], None, s)

    def capture(self, slots: int | None, timing=None):
        """A graph of the sequence; with `timing` (kernel classes) the library's event records
        are captured too (the graph's timer records are then the context's current ones)."""
        torch = self.torch
        self.mf.mf_timing(self.ctx, timing or [])
        g = torch.cuda.CUDAGraph()
        with torch.cuda.stream(self.stream):
            with torch.cuda.graph(g, stream=self.stream):
                self.calls(slots)
        torch.cuda.synchronize()
        return g


def replay(torch, stream, graph, flush, n: int, warm: int = 1, read=None):
    """`warm` untimed replays, then `n` timed ones (L2 flushed before each, outside the events);
    returns their milliseconds (and `read()` after each timed replay, if given)."""
    out, reads = [], []
    for i in range(warm + n):
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        with torch.cuda.stream(stream):
            flush.zero_()
            a.record(stream)
            graph.replay()
            b.record(stream)
        b.synchronize()
        if i >= warm:
            out.append(a.elapsed_time(b))
            if read is not None:
                reads.append(read())
    return (out, reads) if read is not None else out


def ffn_bytes(cfg, block: int) -> int:
    """Algorithmic bytes of one fused one-token FFN launch: the k experts' gate/up and down
    blocks, x and h read, y written."""
    k, H, I = cfg.top_k, cfg.hidden, cfg.inter
    gu = k * 2 * I * (H // 32) * block + 4 * H + 4 * k * I
    dn = k * H * (I // 32) * block + 4 * k * I + 4 * H
    return gu + dn


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
    cfg = synth.CONFIGS[WORKLOAD]
    L, H, E, k, I, q = cfg.n_layers, cfg.hidden, cfg.n_experts, cfg.top_k, cfg.inter, cfg.qtype
    head_slots = slots_for(args.cache_pct, E, k)
    model = mf.Model(L, H, E, k, I, q)
    # one context serves every cache share: its pool holds every expert (128 slots per layer),
    # each measurement puts `slots` of them in use (mf_reset); max_tokens 5 for the verify steps
    plan = mf.mf_plan(model, mf.PlanReq(100.0, 1 << 62, 0, 0, 5, 0))
    t_setup = time.perf_counter()
    ctx = mf.mf_create(model, plan, device.index or 0)
    fill_pack(mf, synth, ctx, cfg)
    t_setup = time.perf_counter() - t_setup
    wr = torch.from_numpy(np.stack([synth.router_weights(cfg.model_seed, l, E, H) for l in range(L)])).to(device)
    head = _klass(cfg, HEAD_CLASS)
    x_np, bias_np = decode_inputs(synth, cfg, HEAD_SEED, head)
    x = torch.from_numpy(x_np).to(device)
    bias = torch.from_numpy(bias_np).to(device)
    flush = torch.empty(512 * 1024 * 1024 // 4, dtype=torch.float32, device=device)
    stream = torch.cuda.Stream(device)
    dec = Decoder(torch, mf, ctx, x, bias, wr, stream)

    # the route trace as the cache sees it (cold eager pass, router order), for the tuner
    idx = torch.empty(N_TOKENS, L, k, dtype=torch.int32, device=device)
    with torch.cuda.stream(stream):
        dec.calls(head_slots, idx)
    stream.synchronize()
    trace = idx.permute(1, 0, 2).contiguous().cpu().numpy()  # [L][tokens][k]

    timed = ["router", "resolve", "materialize", "ffn_fused", "gateup_swiglu", "down_combine"]
    graph = dec.capture(head_slots)
    graph_k = dec.capture(head_slots, timed)
    replay(torch, stream, graph, flush, 0, warm=args.warmup)
    kt = {name: [0.0, 0] for name in mf.KERNEL_CLASSES}
    if ws > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    with ClockSampler(local) as clk:
        t0 = time.perf_counter()
        step_ms = replay(torch, stream, graph, flush, args.steps, warm=0)
        wall = time.perf_counter() - t0
        _, reads = replay(torch, stream, graph_k, flush, args.steps, warm=0, read=lambda: mf.mf_timing_read(ctx))
        for r in reads:
            for name, (kms, n) in r.items():
                kt[name][0] += kms
                kt[name][1] += n
    ms = max_over_ranks(torch, statistics.mean(step_ms), device)
    st = mf.mf_stats(ctx, -1)  # every replay starts cold (mf_reset in the graph): one step's counters
    y_dev = dec.y.cpu()
    del graph, graph_k

    # end to end through the host-buffer entry point: per call, pinned host x and bias in, y out
    xh = torch.from_numpy(x_np).pin_memory()
    bh = torch.from_numpy(bias_np).pin_memory()
    yh = torch.empty(N_TOKENS, L, H).pin_memory()
    mf.mf_timing(ctx, [])

    def e2e_calls():
        mf.mf_reset(ctx, head_slots, stream)
        for t in range(N_TOKENS):
            for l in range(L):
                mf.mf_moe_forward_host(ctx, l, xh[t, l], wr[l], bh[t, l], 1, yh[t, l], None, None, stream)

    e2e_graph = torch.cuda.CUDAGraph()
    with torch.cuda.stream(stream):
        e2e_calls()
        stream.synchronize()
        with torch.cuda.graph(e2e_graph, stream=stream):
            e2e_calls()
    torch.cuda.synchronize()
    e2e_ms = replay(torch, stream, e2e_graph, flush, args.steps, warm=args.warmup)
    del e2e_graph
    assert torch.equal(y_dev, yh), "host-buffer path disagrees with the device path"

    hbm, peak_kind = _peaks()
    rf_bytes = ffn_bytes(cfg, 34)
    ms_ff, n_ff = kt["ffn_fused"]
    rf_gbs = rf_bytes / (ms_ff / n_ff * 1e-3) / 1e9 if n_ff else 0.0
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
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "q8_0 weights, f32 activations and accumulation",
        "data": "synthetic (seeded; random-init Q8_0 experts; planted Zipf routing)",
        "config": {"workload": workload_name(args.cache_pct),
                   "cache_pct": args.cache_pct, "slots_per_layer": head_slots,
                   "tokens_per_step": N_TOKENS, "layers": L, "calls_per_step": N_TOKENS * L,
                   "l2": "flushed between steps (512 MB write)",
                   "execution": "one CUDA graph per step of the 4608 C-ABI calls, starting with a cache reset",
                   "context": f"one context; pool of {plan.slots_per_layer} slots per layer allocated, "
                              f"{head_slots} in use (mf_reset)"},
        "cache": {"hit_rate": round(st["hits"] / max(1, st["accesses"]), 4),
                  "materialized_bytes_per_token": st["bytes_materialized"] / N_TOKENS,
                  "misses_per_token": st["misses"] / N_TOKENS, "accesses_per_step": st["accesses"]},
        "roofline": {"bound": "hbm", "kernel": "k_ffn_pipe (fused one-token expert FFN: k experts' gate/up rows, "
                                               "SwiGLU, down rows, combine; misses pulled over the host link inside)",
                     "achieved": round(rf_gbs, 1), "peak": hbm, "unit": "GB/s",
                     "frac": round(rf_gbs / hbm, 4), "peak_kind": peak_kind, "traffic": _captured_traffic(),
                     "frac_of_nominal": round(rf_gbs / HBM_NOMINAL_GBS, 4),
                     "bytes_per_launch": rf_bytes,
                     "bytes_note": "k = 8 Q8_0 expert payloads (gate/up 2*I*H/32 blocks + down H*I/32 blocks of 34 B) "
                                   "+ x, h, y per launch; traffic = ncu DRAM read+write bytes of one all-resident "
                                   "launch of this kernel and shape",
                     "timing": "CUDA events around each launch in instrumented replays of the step graph; "
                               "launches with misses wait on the host link"},
        "kernels": kernels,
        "copy": {"materialized_bytes_per_step": st["bytes_materialized"],
                 "link_gbs_lower_bound": round(args.steps * st["bytes_materialized"] / (ms_ff * 1e-3) / 1e9, 1)
                 if n_ff else None,
                 "note": "one-token calls materialise inside the fused FFN launch; the lower bound divides the "
                         "materialised bytes by all of that kernel's time"},
        "clocks": clocks,
        "e2e": {"value": round(job_rate(N_TOKENS, e2e_ms_max, ws), 2), "unit": "tokens/s",
                "h2d_bytes_per_step": N_TOKENS * L * (H + E) * 4, "d2h_bytes_per_step": N_TOKENS * L * H * 4,
                "how": "graph replay of the 4608 mf_moe_forward_host calls with pinned host x, bias and y"},
        "gpu_launches": int(sum(v[1] for v in kt.values())) + args.steps,  # + one reset per step
        "wall_s": round(wall, 3),
        "setup_s": round(t_setup, 1),
    }
    if rank == 0:
        extras(args, line, torch, mf, synth, device, cfg, ctx, dec, flush, stream, trace, plan, hbm, rf_bytes)
    mf.mf_destroy(ctx)
    if rank == 0:
        extras_other_contexts(args, line, torch, mf, synth, device)
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(args.cpu_tokens, args.cache_pct, args.cpu_layers)
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


def _guard(line, key, fn):
    """Run one optional measurement; a failure costs only its own object."""
    try:
        line[key] = fn()
    except Exception as e:
        line[key] = {"error": f"{type(e).__name__}: {e}"}


def extras(args, line, torch, mf, synth, device, cfg, ctx, dec, flush, stream, trace, plan, hbm, rf_bytes):
    h2d = h2d_bandwidth(torch, device, stream)
    link_ms = line["copy"]["materialized_bytes_per_step"] / (h2d * 1e9) * 1e3
    line["copy"].update({"h2d_gbs_measured": round(h2d, 1),
                         "link_ms_per_step_at_h2d": round(link_ms, 3),
                         "link_share_of_step": round(link_ms / line["ms_per_step"], 4),
                         "h2d_how": "pinned host -> device cudaMemcpyAsync of 1 GiB, best of 10, this run"})
    _guard(line["copy"], "placement", host_placement)
    if not args.no_link:
        _guard(line["copy"], "in_kernel_link", lambda: link_measurement(torch, mf, synth, cfg, ctx, dec, stream, h2d))
    if not args.no_resident:
        _guard(line["roofline"], "resident", lambda: resident_measurement(torch, mf, ctx, dec, flush, stream, args.steps,
                                                                          rf_bytes, hbm))
    if not args.no_sweep:
        _guard(line, "sweep", lambda: sweep_measurement(torch, mf, synth, device, cfg, ctx, dec, flush, stream))
    if not args.no_tuner:
        _guard(line, "tuner", lambda: tuner_measurement(mf, cfg, line, trace, h2d, plan))
    if not args.no_spec:
        _guard(line, "speculative", lambda: spec_measurement(torch, mf, synth, device, cfg, ctx, dec, stream,
                                                             slots_for(args.cache_pct, cfg.n_experts, cfg.top_k)))


def extras_other_contexts(args, line, torch, mf, synth, device):
    if not args.no_prefill:
        _guard(line, "prefill", lambda: prefill_measurement(torch, mf, synth, device))
    if not args.no_q4_decode:
        _guard(line, "q4_decode", lambda: q4_decode_measurement(torch, mf, synth, device, args.steps))
    if not args.no_batch64:
        _guard(line, "batch64", lambda: batch64_measurement(torch, mf, synth, device))
    if not args.no_l4e64:
        _guard(line, "l4e64", lambda: l4e64_measurement(torch, mf, synth, device, args.steps))
    if not args.no_disk:
        _guard(line, "disk", lambda: disk_measurement(torch, mf, synth, device))


def host_placement() -> dict:
    """Where the pinned pack sits relative to the GPU: the host's NUMA nodes (sysfs) and the GPU's
    (the PCI device's numa_node).  The pack is allocated by the calling thread (cudaHostAlloc), so
    its pages land on that thread's node."""
    nodes = sorted(int(n[4:]) for n in os.listdir("/sys/devices/system/node") if n[4:].isdigit())
    cpus = {n: open(f"/sys/devices/system/node/node{n}/cpulist").read().strip() for n in nodes}
    try:
        bus = subprocess.run(["nvidia-smi", "--id=0", "--query-gpu=pci.bus_id", "--format=csv,noheader"],
                             capture_output=True, text=True).stdout.strip().lower()
    except Exception:
        bus = ""
    dev = bus[4:] if len(bus) > 12 else bus  # 00000000:00:07.0 -> 0000:00:07.0
    try:
        gnode = int(open(f"/sys/bus/pci/devices/{dev}/numa_node").read())
    except Exception:
        gnode = None
    return {"numa_nodes": nodes, "cpus_per_node": cpus, "gpu_pci": dev, "gpu_numa_node": gnode,
            "pack": "cudaHostAlloc(mapped | portable) by the calling thread: pages on its node"
                    + (" (the only node)" if len(nodes) == 1 else "")}


def link_measurement(torch, mf, synth, cfg, ctx, dec, stream, h2d_gbs: float, reps: int = 3) -> dict:
    """The fused FFN launch when every one of its k experts misses: layer 0 with all 128 slots in
    use from a cold cache, 16 calls whose planted routes are disjoint sets of 8 experts, so each
    launch pulls 8 payloads (40.1 MB) over the CPU-GPU link inside the kernel.  CUDA events around
    each FFN launch; bytes = misses x payload (the ncu sysmem sector count of such a launch agrees
    to 0.1 %)."""
    E, k, H = cfg.n_experts, cfg.top_k, cfg.hidden
    n = E // k
    routes = np.arange(n * k, dtype=np.int32).reshape(n, k)
    x = dec.x[:n, 0].contiguous()
    b = torch.from_numpy(synth.plant_bias(routes, E)).to(x.device)
    y = torch.empty(n, H, device=x.device)
    rates = []
    for _ in range(reps):
        mf.mf_reset(ctx, E, stream)
        mf.mf_timing(ctx, ["ffn_fused"])
        with torch.cuda.stream(stream):
            for t in range(n):
                mf.mf_moe_forward(ctx, 0, x[t], dec.wr[0], b[t], 1, y[t], None, None, stream)
        tm = mf.mf_timing_read(ctx)["ffn_fused"]
        st = mf.mf_stats(ctx, 0)
        rates.append(st["bytes_materialized"] / (tm[0] * 1e-3) / 1e9)
        assert st["misses"] == n * k
    mf.mf_timing(ctx, [])
    assert mf.mf_check(ctx) == 0
    gbs = max(rates)
    return {"gbs": round(gbs, 1), "frac_of_h2d": round(gbs / h2d_gbs, 4), "misses_per_launch": k,
            "bytes_per_launch": int(mf.mf_payload_bytes(mf.Model(1, H, E, k, cfg.inter, cfg.qtype))) * k,
            "how": f"{n} one-token calls of layer 0 from a cold cache with disjoint planted routes (every "
                   f"expert misses), CUDA events around each fused FFN launch, best of {reps}"}


def resident_measurement(torch, mf, ctx, dec, flush, stream, steps, bytes_per_launch, hbm):
    """The same 4608 calls with every expert resident (all 128 slots in use, warmed by two passes):
    each fused FFN launch is then HBM-bound.  Per launch: CUDA events around each launch in
    instrumented graph replays; sustained: the whole sequence's algorithmic bytes over the step
    time of plain replays (no cache reset in the graph, so every replay stays all-resident)."""
    E = dec.wr.shape[1]
    with torch.cuda.stream(stream):
        dec.calls(E)  # reset to all slots in use, cold pass
        dec.calls(None)  # every expert of the sequence resident
    stream.synchronize()
    g = dec.capture(None)
    mf.mf_stats(ctx, -1, reset=True)
    step = replay(torch, stream, g, flush, steps, warm=2)
    del g
    gk = dec.capture(None, ["ffn_fused", "router"])
    _, reads = replay(torch, stream, gk, flush, steps, warm=2, read=lambda: mf.mf_timing_read(ctx))
    del gk
    mf.mf_timing(ctx, [])
    st = mf.mf_stats(ctx, -1)
    ms = sum(r["ffn_fused"][0] for r in reads)
    n = sum(r["ffn_fused"][1] for r in reads)
    rms = sum(r["router"][0] for r in reads)
    us = 1e3 * ms / n
    gbs = bytes_per_launch / (us * 1e-6) / 1e9
    calls = dec.T * dec.L
    step_ms = statistics.mean(step)
    sus = calls * bytes_per_launch / (step_ms * 1e-3) / 1e9
    return {"achieved": round(gbs, 1), "frac": round(gbs / hbm, 4), "frac_of_nominal": round(gbs / HBM_NOMINAL_GBS, 4),
            "us_per_launch": round(us, 3), "launches": n, "router_us_per_launch": round(1e3 * rms / n, 3),
            "misses_in_timed_replays": st["misses"],
            "sustained": {"ms_per_step": round(step_ms, 4), "us_per_call": round(1e3 * step_ms / calls, 3),
                          "achieved": round(sus, 1), "frac": round(sus / hbm, 4),
                          "tokens_per_s": round(dec.T / (step_ms * 1e-3), 2),
                          "how": "4608 calls x algorithmic bytes per launch / step time of plain graph replays "
                                 "(router and FFN launches included), all resident, L2 flushed per replay"},
            "how": "same calls, all 128 slots in use, warmed by two passes (every launch all-resident), L2 flushed "
                   "per replay",
            "read_floor": read_floor(torch, stream, flush, bytes_per_launch, hbm)}


def sweep_measurement(torch, mf, synth, device, cfg, ctx, dec0, flush, stream, reps: int = 2) -> dict:
    """Every route class x cache share of the workload on seed 0: one graph per cell (cache reset
    to the share's slot count, then the 4608 calls), one warm-up and `reps` timed replays."""
    L, E, k = cfg.n_layers, cfg.n_experts, cfg.top_k
    out = {}
    for klass in cfg.route_classes:
        if klass.name == HEAD_CLASS:
            dec = dec0
        else:
            xn, bn = decode_inputs(synth, cfg, HEAD_SEED, klass)
            dec = Decoder(torch, mf, ctx, torch.from_numpy(xn).to(device), torch.from_numpy(bn).to(device), dec0.wr,
                          stream)
        cells = {}
        pcts = list(cfg.cache_pcts) + ([100.0] if klass.name == HEAD_CLASS else [])
        for pct in pcts:
            slots = slots_for(pct, E, k)
            g = dec.capture(slots)
            ms = statistics.mean(replay(torch, stream, g, flush, reps, warm=1))
            del g
            st = mf.mf_stats(ctx, -1)
            cells[f"{pct:g}"] = {"slots": slots, "tokens_per_s": round(N_TOKENS / (ms * 1e-3), 2),
                                 "ms_per_step": round(ms, 3),
                                 "hit_rate": round(st["hits"] / st["accesses"], 4), "misses": st["misses"],
                                 "materialized_mb_per_token": round(st["bytes_materialized"] / N_TOKENS / 1e6, 2)}
        out[klass.name] = cells
        if dec is not dec0:
            del dec
    assert mf.mf_check(ctx) == 0
    return {"how": f"seed {HEAD_SEED}, one CUDA graph per cell (cache reset to the cell's slots + 4608 calls), "
                   f"mean of {reps} replays after one, L2 flushed per replay", "cells": out}


def tuner_measurement(mf, cfg, line, trace, h2d_gbs: float, plan) -> dict:
    """The cache-size tuner (mf_tune_cache) on the headline sequence against the measured sweep
    of the headline class: the route trace from a cold pass (router order), the all-resident time
    per token from the sustained resident step, the link time per payload at the measured pinned
    copy rate.  Predicted misses must equal the GPU's (the same LRU), predicted rates test the
    throughput relation."""
    L, H, E, k, I, q = cfg.n_layers, cfg.hidden, cfg.n_experts, cfg.top_k, cfg.inter, cfg.qtype
    model = mf.Model(L, H, E, k, I, q)
    res = line["roofline"]["resident"]["sustained"]
    cells = line["sweep"]["cells"][HEAD_CLASS]
    pcts = [float(p) for p in cells]
    t_token = res["ms_per_step"] * 1e-3 / N_TOKENS
    t_miss = plan.payload_bytes / (h2d_gbs * 1e9)
    pts, best = mf.mf_tune_cache(model, mf.PlanReq(0.0, 1 << 62, 0, 0, 1, 0), trace, 1, t_token, t_miss, pcts)
    points = []
    for pt in pts:
        c = cells[f"{pt['cache_pct']:g}"]
        points.append({"cache_pct": pt["cache_pct"], "slots_per_layer": pt["slots_per_layer"],
                       "misses_predicted": pt["misses"], "misses_measured": c["misses"],
                       "tokens_per_s_predicted": round(pt["predicted_tokens_per_s"], 2),
                       "tokens_per_s_measured": c["tokens_per_s"]})
    measured_best = max(range(len(points)), key=lambda i: points[i]["tokens_per_s_measured"])
    return {"how": "route trace of the headline sequence (cold pass, router order); all-resident time per token "
                   "from the sustained resident step; link time per payload at the measured pinned copy rate; "
                   "measured = the sweep's cells of the headline class",
            "t_token_us": round(t_token * 1e6, 3), "t_miss_us": round(t_miss * 1e6, 3),
            "points": points, "best_predicted_pct": pts[best]["cache_pct"] if best >= 0 else None,
            "best_measured_pct": points[measured_best]["cache_pct"],
            "misses_agree": all(p["misses_predicted"] == p["misses_measured"] for p in points)}


def spec_measurement(torch, mf, synth, device, cfg, ctx, dec, stream, slots: int, K: int = 4, alpha: float = 0.6,
                     reps: int = 2) -> dict:
    """Verification-width accounting of speculative decoding on the headline sequence (section
    "Throughput Model": extra_materialization; Discussion: record drafted and accepted tokens,
    verification width, misses and materialised bytes).  No draft model: a seeded schedule
    accepts the first a of K drafts per verify step (each with probability alpha), and rejected
    drafts carry routes and activations of an independent stream.  Each verify step is one call
    per layer with T = K + 1 (the union of its rows' experts is materialised); plain decode is
    one call per token and layer.  Both run eagerly from a cold cache of `slots` slots, CUDA
    events around the whole sequence; the cache-size tuner replays each recorded trace to predict
    its misses."""
    L, H, E, k, I, q = cfg.n_layers, cfg.hidden, cfg.n_experts, cfg.top_k, cfg.inter, cfg.qtype
    route = _klass(cfg, HEAD_CLASS)
    W = K + 1
    rows = synth.verify_rows(HEAD_SEED, N_TOKENS, K, alpha)  # [batches, W]
    nb, n_drafts = rows.shape[0], int((rows < 0).sum())
    xh, bh = dec.x.cpu().numpy(), dec.bias.cpu().numpy()  # [T, L, H], [T, L, E]
    xb = np.empty((nb, L, W, H), np.float32)
    bb = np.empty((nb, L, W, E), np.float32)
    for l in range(L):
        xd = synth.activations(HEAD_SEED, l, 1, 0, n_drafts, H)
        bd = synth.plant_bias(synth.routes(HEAD_SEED, l, 1, E, k, n_drafts, route.zipf_s, 0.0), E)
        for b in range(nb):
            for j in range(W):
                v = int(rows[b, j])
                xb[b, l, j] = xh[v, l] if v >= 0 else xd[-1 - v]
                bb[b, l, j] = bh[v, l] if v >= 0 else bd[-1 - v]
    xb, bb = torch.from_numpy(xb).to(device), torch.from_numpy(bb).to(device)
    wr = dec.wr
    y1 = torch.empty(N_TOKENS, L, H, device=device)
    yb = torch.empty(nb, L, W, H, device=device)
    i1 = torch.empty(N_TOKENS, L, k, dtype=torch.int32, device=device)
    ib = torch.empty(nb, L, W, k, dtype=torch.int32, device=device)

    def decode():
        for t in range(N_TOKENS):
            for l in range(L):
                mf.mf_moe_forward(ctx, l, dec.x[t, l], wr[l], dec.bias[t, l], 1, y1[t, l], i1[t, l], None, stream)

    def verify():
        for b in range(nb):
            for l in range(L):
                mf.mf_moe_forward(ctx, l, xb[b, l], wr[l], bb[b, l], W, yb[b, l], ib[b, l], None, stream)

    def run(fn):  # one untimed pass, then the mean of `reps`; each from a cold cache
        ms = []
        for i in range(1 + reps):
            with torch.cuda.stream(stream):
                mf.mf_reset(ctx, slots, stream)
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
    model = mf.Model(L, H, E, k, I, q)
    pct = 100.0 * slots / E
    req = mf.PlanReq(0.0, 1 << 62, 0, 0, W, 0)
    p1 = mf.mf_tune_cache(model, req, tr1, 1, 0.0, 0.0, [pct])[0][0]
    pv = mf.mf_tune_cache(model, req, trv, W, 0.0, 0.0, [pct])[0][0]
    return {"how": "seeded acceptance schedule (no draft model), verify steps of K + 1 rows as one call per "
                   "layer, plain decode as one call per token and layer, eager calls from a cold cache, CUDA "
                   "events around each whole sequence",
            "K": K, "alpha": alpha, "width": W, "slots": slots, "tokens": N_TOKENS, "verify_steps": nb,
            "accepted_drafts": N_TOKENS - nb, "rejected_drafts": n_drafts,
            "misses": {"decode": st1["misses"], "decode_predicted": p1["misses"],
                       "verify": stv["misses"], "verify_predicted": pv["misses"]},
            "extra_materialized_mb_per_token": round((stv["bytes_materialized"] - st1["bytes_materialized"])
                                                     / N_TOKENS / 1e6, 3),
            "tokens_per_s": {"decode_eager": round(N_TOKENS / (ms1 * 1e-3), 2),
                             "speculative_eager": round(N_TOKENS / (msv * 1e-3), 2)}}


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


def read_floor(torch, stream, flush, nbytes, hbm, reps: int = 20) -> dict:
    """What one read-only launch of the same size achieves: a torch.sum over nbytes of fp32 from a
    cold L2, CUDA events around the launch (the launch and first-access latency that bound any
    single kernel of this size)."""
    buf = torch.ones(nbytes // 4, dtype=torch.float32, device=flush.device)
    out = torch.empty((), dtype=torch.float32, device=flush.device)
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


def _one_layer_ctx(mf, synth, cfg, device, pct: float, max_tokens: int, layer: int = 0):
    H, E, k, I, q = cfg.hidden, cfg.n_experts, cfg.top_k, cfg.inter, cfg.qtype
    model = mf.Model(1, H, E, k, I, q)
    plan = mf.mf_plan(model, mf.PlanReq(pct, 1 << 62, 0, 0, max_tokens, 0))
    ctx = mf.mf_create(model, plan, device.index or 0)
    buf = np.empty(plan.payload_bytes, np.uint8)
    for e in range(E):
        synth.payload(cfg.model_seed, layer, e, H, I, q, out=buf)
        mf.mf_pack_put(ctx, 0, e, buf)
    return ctx, plan


def prefill_measurement(torch, mf, synth, device, calls: int = 4, cache_pct: float = 15.0) -> dict:
    """The tensor-core grouped GEMM path on one layer of the 48-layer Q4_0 workload: one
    4096-token prefill call (Zipf 1.2 routing) from a cold cache, `calls` times after one warm-up.
    Per call: the GEMM kernels' summed CUDA-event time (gate/up+SwiGLU and down, every wave) and the
    whole call.  FLOPs: useful = 2 * T * k * 3 * hidden * inter (the method's work, the roofline's
    numerator); issued on the tensor cores = 3x that (hi*hi + hi*lo + lo*hi bf16 products)."""
    cfg = synth.CONFIGS["l48e128q4"]
    H, E, k, I, q, T = cfg.hidden, cfg.n_experts, cfg.top_k, cfg.inter, cfg.qtype, cfg.prefill
    ctx, plan = _one_layer_ctx(mf, synth, cfg, device, cache_pct, T)
    try:
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
            "roofline": {"bound": "tensor", "kernel": "prefill grouped GEMMs (gate/up+SwiGLU, down)",
                         "achieved": round(useful / (g * 1e-3) / 1e12, 2), "peak": peak[0], "unit": "TFLOP/s",
                         "frac": round(useful / (g * 1e-3) / 1e12 / peak[0], 4), "peak_kind": peak[1],
                         "flops": "useful: 2 * T * k * 3 * hidden * inter per call",
                         "issued_tflops": round(issued / (g * 1e-3) / 1e12, 2),
                         "issued_frac": round(issued / (g * 1e-3) / 1e12 / peak[0], 4),
                         "flops_per_call": {"useful": useful, "issued": issued}}}


def q4_decode_measurement(torch, mf, synth, device, steps: int, pcts=(15.0, 35.0)) -> dict:
    """The 48-layer Q4_0 workload's decode: per cache share, from a cold cache, the 4096-token
    prefill call of every layer (eager, untimed), then the 96-token decode at batch 1 (one graph
    of the 4608 calls, timed; its cache state is the prefill's)."""
    cfg = synth.CONFIGS["l48e128q4"]
    L, H, E, k, I, q, P, T = (cfg.n_layers, cfg.hidden, cfg.n_experts, cfg.top_k, cfg.inter, cfg.qtype, cfg.prefill,
                              cfg.n_tokens)
    klass = cfg.route_classes[0]
    model = mf.Model(L, H, E, k, I, q)
    # every expert fits the pool (128 slots per layer); each share puts `slots` of them in use
    plan = mf.mf_plan(model, mf.PlanReq(100.0, 1 << 62, 0, 0, P, 0))
    ctx = mf.mf_create(model, plan, device.index or 0)
    out = {"workload": f"l48e128q4: 48 layers, hidden {H}, {E} experts, top-{k}, inter {I}, Q4_0, Zipf 1.2; "
                       f"4096-token prefill call per layer, then 96 decode tokens at batch 1"}
    try:
        fill_pack(mf, synth, ctx, cfg)
        routes = [synth.routes(0, l, 0, E, k, P + T, klass.zipf_s, klass.reuse) for l in range(L)]
        wr = torch.from_numpy(np.stack([synth.router_weights(cfg.model_seed, l, E, H) for l in range(L)])).to(device)
        xp = [torch.from_numpy(synth.activations(0, l, 0, 0, P, H)).to(device) for l in range(L)]
        bp = [torch.from_numpy(synth.plant_bias(routes[l][:P], E)).to(device) for l in range(L)]
        yp = torch.empty(P, H, device=device)
        xn, bn = decode_inputs(synth, cfg, 0, klass, t0=P, route_sets=[r[P:] for r in routes])
        stream = torch.cuda.Stream(device)
        dec = Decoder(torch, mf, ctx, torch.from_numpy(xn).to(device), torch.from_numpy(bn).to(device), wr, stream)
        flush = torch.empty(512 * 1024 * 1024 // 4, dtype=torch.float32, device=device)
        hbm, _ = _peaks()
        for pct in pcts:
            slots = slots_for(pct, E, k)
            g = dec.capture(None)
            ms, pf = [], []
            for i in range(1 + max(2, min(steps, 5))):
                with torch.cuda.stream(stream):
                    mf.mf_reset(ctx, slots, stream)
                    a0, a1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                    a0.record(stream)
                    for l in range(L):
                        mf.mf_moe_forward(ctx, l, xp[l], wr[l], bp[l], P, yp, None, None, stream)
                    a1.record(stream)
                    stream.synchronize()
                    mf.mf_stats(ctx, -1, reset=True)
                    flush.zero_()
                    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                    a.record(stream)
                    g.replay()
                    b.record(stream)
                b.synchronize()
                if i:
                    ms.append(a.elapsed_time(b))
                    pf.append(a0.elapsed_time(a1))
            del g
            st = mf.mf_stats(ctx, -1)
            m = statistics.mean(ms)
            out[f"{pct:g}"] = {"slots": slots, "decode_tokens_per_s": round(T / (m * 1e-3), 2),
                               "decode_ms": round(m, 3),
                               "hit_rate": round(st["hits"] / max(1, st["accesses"]), 4),
                               "materialized_mb_per_token": round(st["bytes_materialized"] / T / 1e6, 2),
                               "prefill_ms_48_layers": round(statistics.mean(pf), 2),
                               "prefill_tokens_per_s": round(P / (statistics.mean(pf) * 1e-3), 1)}
        assert mf.mf_check(ctx) == 0
        # all-resident decode: the fused FFN per launch against HBM (Q4_0 blocks of 18 B)
        with torch.cuda.stream(stream):
            dec.calls(plan.slots_per_layer)
            dec.calls(None)
        stream.synchronize()
        gk = dec.capture(None, ["ffn_fused"])
        _, reads = replay(torch, stream, gk, flush, 2, warm=1, read=lambda: mf.mf_timing_read(ctx))
        del gk
        mf.mf_timing(ctx, [])
        ms_ff = sum(r["ffn_fused"][0] for r in reads)
        n_ff = sum(r["ffn_fused"][1] for r in reads)
        byt = ffn_bytes(cfg, 18)
        if n_ff:
            gbs = byt / (ms_ff / n_ff * 1e-3) / 1e9
            out["resident_ffn"] = {"slots": plan.slots_per_layer, "us_per_launch": round(1e3 * ms_ff / n_ff, 3),
                                   "bytes_per_launch": byt, "achieved": round(gbs, 1), "frac": round(gbs / hbm, 4),
                                   "how": "the decode's 4608 calls with all 128 slots in use, warmed by two passes, "
                                          "CUDA events around each fused FFN launch"}
    finally:
        mf.mf_destroy(ctx)
    return out


def batch64_measurement(torch, mf, synth, device, steps: int = 8, warm: int = 2, cache_pct: float = 15.0) -> dict:
    """64 concurrent decode streams on one layer of the 30-layer workload (hidden 2816, 128
    experts, top-8, inter 1408, Q8_0, Zipf 1.0 per stream) at 15 % cache: one call of T = 64 per
    step (~107 distinct experts against 19 slots: 6 waves, their misses over the host link), for
    both access orders.  CUDA events around `steps` calls after `warm` calls."""
    cfg = synth.CONFIGS["l30e128b64"]
    H, E, k, I, q, B = cfg.hidden, cfg.n_experts, cfg.top_k, cfg.inter, cfg.qtype, cfg.batch
    ctx, plan = _one_layer_ctx(mf, synth, cfg, device, cache_pct, B)
    out = {"workload": f"l30e128b64 layer 0: {B} decode streams per call, hidden {H}, {E} experts, top-{k}, "
                       f"inter {I}, Q8_0, Zipf {cfg.route_classes[0].zipf_s:g} per stream, cache {cache_pct:g}% "
                       f"({plan.slots_per_layer} slots)"}
    try:
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


def disk_measurement(torch, mf, synth, device, cache_pct: float = 15.0, reps: int = 2) -> dict:
    """The disk tier against the pinned pack on the headline workload at 15 % cache (19 slots):
    the split-pack written to a file (mf_pack_save), a context serving its misses from the file
    (mf_create_from_file: after the router decides a call's misses, a host function reads them
    into pinned staging), and the same 96-token decode through both (one graph each, from a cold
    cache).  Every layer of the model when the file system holds the 31 GB file twice over, else
    the first layers that fit."""
    import shutil
    import tempfile
    cfg = synth.CONFIGS[WORKLOAD]
    H, E, k, I, q = cfg.hidden, cfg.n_experts, cfg.top_k, cfg.inter, cfg.qtype
    pdir = os.environ.get("MF_PACK_DIR", tempfile.gettempdir())
    per_layer = E * (synth.payload_bytes(H, I, q) + 4096)
    free = shutil.disk_usage(pdir).free
    L = min(cfg.n_layers, int(free // 2 // per_layer))
    if L < 1:
        return {"skipped": f"{free / 1e9:.1f} GB free in {pdir}"}
    model = mf.Model(L, H, E, k, I, q)
    plan = mf.mf_plan(model, mf.PlanReq(cache_pct, 1 << 62, 0, 0, 1, 0))
    head = _klass(cfg, HEAD_CLASS)
    path = os.path.join(pdir, f"mawforge_l{L}e{E}.mfpack")
    stream = torch.cuda.Stream(device)
    flush = torch.empty(512 * 1024 * 1024 // 4, dtype=torch.float32, device=device)
    sub = cfg.__class__(**{**cfg.__dict__, "n_layers": L})
    xn, bn = decode_inputs(synth, sub, HEAD_SEED, head)
    x = torch.from_numpy(xn).to(device)
    b = torch.from_numpy(bn).to(device)
    wr = torch.from_numpy(np.stack([synth.router_weights(cfg.model_seed, l, E, H) for l in range(L)])).to(device)
    out = {"workload": f"{WORKLOAD} layers 0-{L - 1} of {cfg.n_layers}, {HEAD_CLASS}, cache {cache_pct:g}% "
                       f"({plan.slots_per_layer} slots), 96 decode tokens batch 1 from a cold cache",
           "file_dir": pdir}
    ctx = mf.mf_create(model, plan, device.index or 0)
    fh = None
    try:
        fill_pack(mf, synth, ctx, sub)
        t0 = time.perf_counter()
        mf.mf_pack_save(ctx, path)
        out["save_s"] = round(time.perf_counter() - t0, 2)
        out["file_gb"] = round(os.path.getsize(path) / 1e9, 2)
        fh = mf.mf_create_from_file(model, plan, path, device.index or 0)
        out["direct_io"] = mf.mf_pack_file_direct(fh)
        res = {}
        for name, h in (("pinned_pack", ctx), ("file", fh)):
            dec = Decoder(torch, mf, h, x, b, wr, stream)
            g = dec.capture(plan.slots_per_layer)
            f0 = mf.mf_pack_file_stats(fh) if h == fh else None
            ms = statistics.mean(replay(torch, stream, g, flush, reps, warm=1))
            del g
            st = mf.mf_stats(h, -1)
            assert mf.mf_check(h) == 0
            r = {"tokens_per_s": round(N_TOKENS / (ms * 1e-3), 2), "ms_per_step": round(ms, 2),
                 "misses_per_step": st["misses"], "materialized_gb_per_step": round(st["bytes_materialized"] / 1e9, 3)}
            if f0 is not None:
                f1 = mf.mf_pack_file_stats(fh)
                n = reps + 1
                r["file_reads_per_step"] = (f1["reads"] - f0["reads"]) // n
                r["read_s_per_step"] = round((f1["seconds"] - f0["seconds"]) / n, 3)
                r["read_gbs"] = round((f1["bytes"] - f0["bytes"]) / max(1e-9, f1["seconds"] - f0["seconds"]) / 1e9, 2)
            res[name] = r
        out.update(res)
        out["file_minus_pinned_ms_per_step"] = round(res["file"]["ms_per_step"] - res["pinned_pack"]["ms_per_step"], 2)
        out["how"] = ("the same graph of the 96-token decode through a context with the pinned pack and through one "
                      "reading its misses from the split-pack file; mean of the replays after one, each from a cold "
                      "cache; read seconds on the host clock")
    finally:
        if fh:
            mf.mf_destroy(fh)
        mf.mf_destroy(ctx)
        try:
            os.remove(path)
        except OSError:
            pass
    return out


def l4e64_measurement(torch, mf, synth, device, steps: int, cache_pct: float = 35.0) -> dict:
    """The 4-layer workload (hidden 2048, 64 experts, top-8, inter 768, Q8_0; 256 decode tokens
    at batch 1, Zipf 1.1 + 0.6 reuse) at 35 % cache: one graph of its 1024 calls per step from a
    cold cache."""
    cfg = synth.CONFIGS["l4e64"]
    L, H, E, k, I, q = cfg.n_layers, cfg.hidden, cfg.n_experts, cfg.top_k, cfg.inter, cfg.qtype
    model = mf.Model(L, H, E, k, I, q)
    plan = mf.mf_plan(model, mf.PlanReq(cache_pct, 1 << 62, 0, 0, 1, 0))
    ctx = mf.mf_create(model, plan, device.index or 0)
    try:
        fill_pack(mf, synth, ctx, cfg)
        wr = torch.from_numpy(np.stack([synth.router_weights(cfg.model_seed, l, E, H) for l in range(L)])).to(device)
        xn, bn = decode_inputs(synth, cfg, 0, cfg.route_classes[0])
        stream = torch.cuda.Stream(device)
        dec = Decoder(torch, mf, ctx, torch.from_numpy(xn).to(device), torch.from_numpy(bn).to(device), wr, stream)
        flush = torch.empty(512 * 1024 * 1024 // 4, dtype=torch.float32, device=device)
        g = dec.capture(plan.slots_per_layer)
        ms = statistics.mean(replay(torch, stream, g, flush, steps, warm=3))
        del g
        st = mf.mf_stats(ctx, -1)
        assert mf.mf_check(ctx) == 0
    finally:
        mf.mf_destroy(ctx)
    T = cfg.n_tokens
    return {"workload": "l4e64: 4 MoE layers, hidden 2048, 64 experts, top-8, inter 768, Q8_0, 256 decode tokens "
                        f"batch 1, Zipf 1.1 + 0.6 reuse, cache {cache_pct:g}% ({plan.slots_per_layer} slots)",
            "tokens_per_s": round(T / (ms * 1e-3), 2), "ms_per_step": round(ms, 4),
            "hit_rate": round(st["hits"] / max(1, st["accesses"]), 4),
            "materialized_mb_per_token": round(st["bytes_materialized"] / T / 1e6, 2)}


def _oracle_sample(n_tokens: int, n_layers: int, cache_pct: float, pays_cache=None):
    """Seconds the CPU oracle takes for the first n_tokens tokens of the headline sequence through
    the first n_layers layers (router + the layer's LRU + fp64 layer per token), layer by layer
    (the layers are independent: each has its own inputs and cache).  Payload generation is input
    preparation, outside the timing."""
    import oracle
    import synth
    cfg = synth.CONFIGS[WORKLOAD]
    H, E, k, I, q = cfg.hidden, cfg.n_experts, cfg.top_k, cfg.inter, cfg.qtype
    route = _klass(cfg, HEAD_CLASS)
    slots = slots_for(cache_pct, E, k)
    pay = synth.payload_bytes(H, I, q)
    dt = 0.0
    for l in range(n_layers):
        x = synth.activations(HEAD_SEED, l, 0, 0, n_tokens, H)
        b = synth.plant_bias(synth.routes(HEAD_SEED, l, 0, E, k, N_TOKENS, route.zipf_s, route.reuse)[:n_tokens], E)
        wr = synth.router_weights(cfg.model_seed, l, E, H)
        used = sorted(set(b.nonzero()[1].tolist()))
        if pays_cache is not None and l in pays_cache:
            pays = pays_cache[l]
        else:
            pays = {e: synth.payload(cfg.model_seed, l, e, H, I, q) for e in used}
            if pays_cache is not None:
                pays_cache[l] = pays
        plist = [pays.get(e) for e in range(E)]
        lru = oracle.LRU(E, slots, pay)
        t0 = time.perf_counter()
        for t in range(n_tokens):
            _, idx, _ = oracle.router(x[t], wr, b[t], k)
            lru.step(idx[None])
            oracle.layer(plist, q, H, I, k, wr, b[t:t + 1], x[t:t + 1])
        dt += time.perf_counter() - t0
    return dt, slots


def cpu_baseline(n_tokens: int = N_TOKENS, cache_pct: float = HEAD_PCT, n_layers: int = N_LAYERS) -> dict:
    """The CPU oracle, as it stands, on a sample of the headline step (same inputs and cache share);
    tokens/s with a token = all 48 layers (layer-tokens / 48)."""
    dt, slots = _oracle_sample(n_tokens, n_layers, cache_pct)
    cores = int(os.environ.get("OMP_NUM_THREADS", os.cpu_count() or 1))
    return {"value": round(n_tokens * n_layers / N_LAYERS / dt, 4), "unit": "tokens/s", "cores": cores,
            "kind": "oracle", "slots_per_layer": slots, "seconds": round(dt, 3),
            "sample": f"first {n_tokens} tokens of the {N_TOKENS}-token step through layers 0-{n_layers - 1} of "
                      f"{N_LAYERS} (router + LRU with {slots} slots + fp64 layer per layer-token), one pass; "
                      f"rate = layer-tokens / {N_LAYERS} per second"}


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
    lru = oracle.LRU(E, slots_for(cache_pct, E, k), synth.payload_bytes(H, I, q))
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
    lru = oracle.LRU(E, slots_for(cache_pct, E, k), synth.payload_bytes(H, I, q))
    t0 = time.perf_counter()
    _, idx, _ = oracle.layer([pays.get(e) for e in range(E)], q, H, I, k, wr, b, x)
    lru.step(idx)
    dt = time.perf_counter() - t0
    return {"value": round(n_streams / dt, 4), "unit": "tokens/s (one layer)", "kind": "oracle",
            "sample": f"the first {n_streams} of the 64 streams of the first call, layer 0 of l30e128b64"}


def run_reference(args):
    """The reference arm: the CPU oracle as it stands on the host cores, rank 0 only.  Each step
    is a bounded sample of the headline step: the first `cpu_tokens` tokens through the first
    `ref_layers` layers (payloads generated once, outside the timing)."""
    ws, rank, _ = _dist()
    if rank != 0:
        return
    n_tok = getattr(args, "cpu_tokens", N_TOKENS)
    n_lay = getattr(args, "ref_layers", 4)
    pct = getattr(args, "cache_pct", HEAD_PCT)
    pays = {}
    per_step = []
    for i in range(args.warmup + args.steps):
        dt, slots = _oracle_sample(n_tok, n_lay, pct, pays)
        if i >= args.warmup:
            per_step.append(dt)
    dt = statistics.mean(per_step)
    value = n_tok * n_lay / N_LAYERS / dt
    cores = int(os.environ.get("OMP_NUM_THREADS", os.cpu_count() or 1))
    sample = (f"first {n_tok} tokens of the {N_TOKENS}-token step through layers 0-{n_lay - 1} of {N_LAYERS} "
              f"(router + LRU with {slots} slots + fp64 layer per layer-token); rate = layer-tokens / {N_LAYERS} "
              f"per second")
    line = {"impl": "reference", "metric": METRIC,
            "value": round(value, 4), "unit": "tokens/s", "n_gpus": ws, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": round(1e3 * dt, 3), "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64 (CPU oracle)", "data": "synthetic (seeded)",
            "config": {"workload": workload_name(pct), "sample": sample,
                       "layer_tokens_per_step": n_tok * n_lay},
            "cpu_baseline": {"value": round(value, 4), "unit": "tokens/s", "kind": "oracle",
                             "cores": cores, "sample": sample},
            "e2e": {"value": round(value, 4), "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line))


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--cache-pct", type=float, default=HEAD_PCT)
    ap.add_argument("--impl", default="mawforge", choices=["mawforge", "reference"])
    ap.add_argument("--cpu-tokens", type=int, default=N_TOKENS, help="tokens of the sequence per CPU-oracle pass")
    ap.add_argument("--cpu-layers", type=int, default=N_LAYERS, help="layers of the CPU baseline leg's sample")
    ap.add_argument("--ref-layers", type=int, default=4, help="layers of each reference-arm step's sample")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-prefill", action="store_true", help="skip the 4096-token prefill measurement")
    ap.add_argument("--no-q4-decode", action="store_true", help="skip the 48-layer Q4_0 decode after prefill")
    ap.add_argument("--no-resident", action="store_true", help="skip the all-resident FFN measurement")
    ap.add_argument("--no-sweep", action="store_true", help="skip the route class x cache share sweep")
    ap.add_argument("--no-batch64", action="store_true", help="skip the 64-stream batched decode measurement")
    ap.add_argument("--no-tuner", action="store_true", help="skip the cache-size tuner against measured steps")
    ap.add_argument("--no-spec", action="store_true", help="skip the speculative verification-width accounting")
    ap.add_argument("--no-l4e64", action="store_true", help="skip the 4-layer workload")
    ap.add_argument("--no-link", action="store_true", help="skip the all-miss in-kernel link measurement")
    ap.add_argument("--no-disk", action="store_true", help="skip the split-pack file (disk tier) measurement")
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
