"""Helpers of the GPU parity tests: build a context from seeded inputs, run the CUDA path
through the C ABI, and compare with the CPU oracle on the same inputs."""
from __future__ import annotations

from concurrent.futures import ThreadPoolExecutor
from dataclasses import dataclass

import numpy as np

import oracle
import synth

# Output tolerance: |gpu - oracle| <= ATOL_RMS * rms(oracle row) + RTOL * |oracle| per element.
# The stated bound is max-abs 2e-3 / rel 1e-2 on fp32-accumulated outputs; with the specified
# weight distributions the outputs have rms ~1e4, so the absolute part is taken relative to
# the rms of the oracle's output row (the reading is argued in the design notes).
ATOL_RMS = 2e-3
RTOL = 1e-2
G_ATOL = 1e-5  # softmax weights, fp32 on the GPU vs fp64 in the oracle


def compare_outputs(got: np.ndarray, ref: np.ndarray) -> dict:
    got = np.asarray(got, np.float64).reshape(-1, ref.shape[-1])
    ref = np.asarray(ref, np.float64).reshape(-1, ref.shape[-1])
    rms = np.sqrt(np.mean(ref ** 2, axis=1, keepdims=True))
    err = np.abs(got - ref)
    bound = ATOL_RMS * rms + RTOL * np.abs(ref)
    # an all-zero reference row must be matched exactly (its bound is 0); NaN never passes
    ratio = np.where(err == 0, 0.0, err / np.where(bound > 0, bound, 1e-300))
    ratio = np.where(np.isfinite(got), ratio, np.inf)
    with np.errstate(divide="ignore", invalid="ignore"):
        rel_rms = np.where(rms > 0, err / np.where(rms > 0, rms, 1), np.where(err == 0, 0.0, np.inf))
    return dict(ratio=float(ratio.max()), max_abs=float(err.max()),
                max_abs_over_rms=float(rel_rms.max()),
                literal_fail_frac=float(np.mean(err > 2e-3 + 1e-2 * np.abs(ref))))


def assert_outputs_close(got, ref, what=""):
    r = compare_outputs(got, ref)
    assert r["ratio"] <= 1.0, f"{what}: outputs outside tolerance {r}"
    return r


@dataclass
class Shape:
    n_layers: int
    hidden: int
    n_experts: int
    top_k: int
    inter: int
    qtype: int
    model_seed: int = 0

    @staticmethod
    def of(cfg) -> "Shape":
        return Shape(cfg.n_layers, cfg.hidden, cfg.n_experts, cfg.top_k, cfg.inter, cfg.qtype, cfg.model_seed)


class Payloads:
    """Canonical payloads regenerated on demand (the oracle's view of the pack).  `edit`, if
    given, is applied to every generated payload (layer, expert, bytes) -> bytes: the same edited
    bytes go into the context's pack (Ctx(..., edit=...)) and to the oracle."""

    def __init__(self, shape: Shape, edit=None):
        self.s = shape
        self.edit = edit
        self._cache = {}

    def get(self, layer: int, expert: int) -> np.ndarray:
        key = (layer, expert)
        if key not in self._cache:
            s = self.s
            p = synth.payload(s.model_seed, layer, expert, s.hidden, s.inter, s.qtype)
            self._cache[key] = p if self.edit is None else self.edit(layer, expert, p)
        return self._cache[key]

    def for_layer(self, layer: int, experts) -> list:
        want = set(int(e) for e in np.asarray(experts).reshape(-1))
        return [self.get(layer, e) if e in want else None for e in range(self.s.n_experts)]


class Ctx:
    """A context of the CUDA library with its pack filled from the seeded generator."""

    def __init__(self, shape: Shape, slots: int, max_tokens: int, device: int = 0, workers: int = 8, edit=None):
        import torch
        import paper_2607_09686_gb300 as mf
        self.mf, self.torch, self.s = mf, torch, shape
        self.model = mf.Model(shape.n_layers, shape.hidden, shape.n_experts, shape.top_k, shape.inter, shape.qtype)
        self.plan = mf.mf_plan(self.model, mf.PlanReq(100.0 * slots / shape.n_experts, 1 << 62, 0, 0, max_tokens, 0))
        assert self.plan.accepted and self.plan.slots_per_layer == slots
        self.h = mf.mf_create(self.model, self.plan, device)
        self.device = torch.device(f"cuda:{device}")
        n = synth.payload_bytes(shape.hidden, shape.inter, shape.qtype)

        def put(le):
            buf = np.empty(n, np.uint8)
            synth.payload(shape.model_seed, le[0], le[1], shape.hidden, shape.inter, shape.qtype, out=buf)
            if edit is not None:
                buf = edit(le[0], le[1], buf)
            mf.mf_pack_put(self.h, le[0], le[1], buf)

        jobs = [(l, e) for l in range(shape.n_layers) for e in range(shape.n_experts)]
        with ThreadPoolExecutor(max_workers=workers) as ex:
            list(ex.map(put, jobs))
        self.wr_host = [synth.router_weights(shape.model_seed, l, shape.n_experts, shape.hidden)
                        for l in range(shape.n_layers)]
        self.wr = [torch.from_numpy(w).to(self.device) for w in self.wr_host]

    def close(self):
        if self.h:
            self.mf.mf_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def forward(self, layer, x, bias, T, trace=False):
        """Run one step; returns (y, idx, w[, trace]) as numpy arrays."""
        torch = self.torch
        s = self.s
        xd = torch.from_numpy(np.ascontiguousarray(x, np.float32)).to(self.device)
        bd = None if bias is None else torch.from_numpy(np.ascontiguousarray(bias, np.float32)).to(self.device)
        y = torch.empty(max(T, 1), s.hidden, device=self.device)
        idx = torch.empty(max(T, 1), s.top_k, dtype=torch.int32, device=self.device)
        w = torch.empty(max(T, 1), s.top_k, device=self.device)
        self.mf.mf_moe_forward(self.h, layer, xd, self.wr[layer], bd, T, y, idx, w)
        torch.cuda.synchronize()
        out = (y.cpu().numpy()[:T], idx.cpu().numpy()[:T], w.cpu().numpy()[:T])
        if trace:
            out = out + (self.mf.mf_trace(self.h, layer, cap=s.n_experts),)
        return out


def oracle_trace(lru: oracle.LRU, idx: np.ndarray, order: int = 0):
    u, sl, hit = lru.step(idx, order)
    return list(map(int, u)), list(map(int, sl)), list(map(bool, hit))


def oracle_routes(shape: Shape, wr_host, xs, biases, workers: int = 16) -> np.ndarray:
    """Oracle routing of many (layer, token) inputs, in a thread pool (the C oracle releases the
    GIL).  xs[l] is [T, H], biases[l] is [T, E] or None; returns idx [L, T, k]."""
    L = len(xs)
    T = xs[0].shape[0]
    out = np.empty((L, T, shape.top_k), np.int32)

    def one(lt):
        l, t = lt
        b = None if biases[l] is None else biases[l][t]
        out[l, t] = oracle.router(xs[l][t], wr_host[l], b, shape.top_k)[1]

    with ThreadPoolExecutor(max_workers=workers) as ex:
        list(ex.map(one, [(l, t) for l in range(L) for t in range(T)]))
    return out


def oracle_stats(shape: Shape, slots: int, idx_steps) -> list:
    """Per-layer oracle LRU counters after feeding idx_steps[l] = list of [T_step, k] arrays."""
    pay = synth.payload_bytes(shape.hidden, shape.inter, shape.qtype)
    res = []
    for steps in idx_steps:
        c = oracle.LRU(shape.n_experts, slots, pay)
        for st in steps:
            c.step(st)
        res.append(c.stats())
    return res


def stats_tuple(st: dict):
    return (st["accesses"], st["hits"], st["misses"], st["evictions"],
            st.get("bytes", st.get("bytes_materialized")))
