"""Seeded synthetic inputs for the routed-expert step (shared by the oracle and the CUDA path).

Holds no arithmetic of the method: it only produces the bytes and arrays both sides
consume (GGUF Q8_0/Q4_0 expert payloads, router weights, activations, route sets and
the logit bias that plants them).  The generator itself is ``synth.c`` (counter-based
SplitMix64), built into ``libsynth.so`` next to this file.
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

from .configs import CONFIGS, Config  # noqa: F401

Q8_0 = 8
Q4_0 = 2

_HERE = os.path.dirname(os.path.abspath(__file__))
_SO = os.path.join(_HERE, "libsynth.so")
_LIB = None


def build(force: bool = False) -> str:
    """Compile synth.c into libsynth.so (gcc, OpenMP, no FP contraction)."""
    src = os.path.join(_HERE, "synth.c")
    if force or not os.path.exists(_SO) or os.path.getmtime(_SO) < os.path.getmtime(src):
        tmp = _SO + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-fopenmp", "-ffp-contract=off", "-fPIC", "-shared",
                               "-std=c11", src, "-o", tmp, "-lm"])
        os.replace(tmp, _SO)
    return _SO


def _lib():
    global _LIB
    if _LIB is None:
        build()
        lib = ctypes.CDLL(_SO)
        u64, i32, dbl = ctypes.c_uint64, ctypes.c_int, ctypes.c_double
        vp = ctypes.c_void_p
        lib.syn_key.restype = u64
        lib.syn_key.argtypes = [u64, u64, u64, u64, u64]
        lib.syn_draw.restype = u64
        lib.syn_draw.argtypes = [u64, u64]
        lib.syn_f64_to_f16.restype = ctypes.c_uint16
        lib.syn_f64_to_f16.argtypes = [dbl]
        lib.syn_payload_bytes.restype = u64
        lib.syn_payload_bytes.argtypes = [i32, i32, i32]
        lib.syn_tensor_bytes.restype = u64
        lib.syn_tensor_bytes.argtypes = [i32, i32, i32]
        lib.syn_q_tensor.restype = i32
        lib.syn_q_tensor.argtypes = [u64, i32, i32, i32, i32, i32, i32, vp]
        lib.syn_payload.restype = i32
        lib.syn_payload.argtypes = [u64, i32, i32, i32, i32, i32, vp]
        lib.syn_router_weights.restype = None
        lib.syn_router_weights.argtypes = [u64, i32, i32, i32, vp]
        lib.syn_activations.restype = None
        lib.syn_activations.argtypes = [u64, i32, i32, ctypes.c_int64, i32, i32, vp]
        lib.syn_permutation.restype = None
        lib.syn_permutation.argtypes = [u64, i32, i32, vp]
        lib.syn_routes.restype = i32
        lib.syn_routes.argtypes = [u64, i32, i32, i32, i32, i32, dbl, dbl, vp]
        lib.syn_accepts.restype = i32
        lib.syn_accepts.argtypes = [u64, i32, i32, i32, dbl, vp]
        _LIB = lib
    return _LIB


def f64_to_f16_bits(v: float) -> int:
    return int(_lib().syn_f64_to_f16(float(v)))


def payload_bytes(hidden: int, inter: int, qtype: int) -> int:
    return int(_lib().syn_payload_bytes(hidden, inter, qtype))


def tensor_bytes(rows: int, cols: int, qtype: int) -> int:
    return int(_lib().syn_tensor_bytes(rows, cols, qtype))


def q_tensor(seed: int, layer: int, expert: int, tensor: int, rows: int, cols: int, qtype: int) -> np.ndarray:
    out = np.empty(tensor_bytes(rows, cols, qtype), dtype=np.uint8)
    if _lib().syn_q_tensor(seed, layer, expert, tensor, rows, cols, qtype, out.ctypes.data):
        raise ValueError("bad tensor shape or qtype")
    return out


def payload(seed: int, layer: int, expert: int, hidden: int, inter: int, qtype: int,
            out: np.ndarray | None = None) -> np.ndarray:
    """Canonical GGUF bytes of one expert: gate [I,H], up [I,H], down [H,I]."""
    n = payload_bytes(hidden, inter, qtype)
    if out is None:
        out = np.empty(n, dtype=np.uint8)
    assert out.dtype == np.uint8 and out.size >= n and out.flags.c_contiguous
    if _lib().syn_payload(seed, layer, expert, hidden, inter, qtype, out.ctypes.data):
        raise ValueError("bad payload shape or qtype")
    return out


def router_weights(seed: int, layer: int, n_experts: int, hidden: int) -> np.ndarray:
    out = np.empty((n_experts, hidden), dtype=np.float32)
    _lib().syn_router_weights(seed, layer, n_experts, hidden, out.ctypes.data)
    return out


def activations(seed: int, layer: int, stream: int, t0: int, n: int, hidden: int) -> np.ndarray:
    out = np.empty((n, hidden), dtype=np.float32)
    _lib().syn_activations(seed, layer, stream, t0, n, hidden, out.ctypes.data)
    return out


def permutation(seed: int, layer: int, n: int) -> np.ndarray:
    out = np.empty(n, dtype=np.int32)
    _lib().syn_permutation(seed, layer, n, out.ctypes.data)
    return out


def routes(seed: int, layer: int, stream: int, n_experts: int, top_k: int, n_tokens: int,
           zipf_s: float, reuse: float) -> np.ndarray:
    """[n_tokens, k] expert ids in draw order (draw order = planted rank)."""
    out = np.empty((n_tokens, top_k), dtype=np.int32)
    if _lib().syn_routes(seed, layer, stream, n_experts, top_k, n_tokens, float(zipf_s), float(reuse),
                         out.ctypes.data):
        raise ValueError("bad route parameters")
    return out


def plant_bias(route_sets: np.ndarray, n_experts: int) -> np.ndarray:
    """Logit bias that plants route sets: +16 + (k - rank) * 0.5 on the chosen experts, 0 elsewhere."""
    n, k = route_sets.shape
    bias = np.zeros((n, n_experts), dtype=np.float32)
    ranks = np.arange(k, dtype=np.float32)
    rows = np.repeat(np.arange(n), k)
    bias[rows, route_sets.reshape(-1)] = np.tile(16.0 + (k - ranks) * 0.5, n)
    return bias


def accepts(seed: int, stream: int, n_steps: int, K: int, alpha: float) -> np.ndarray:
    """[n_steps] drafted tokens accepted per verify step (leading successes, probability alpha each)."""
    out = np.empty(n_steps, dtype=np.int32)
    if _lib().syn_accepts(seed, stream, n_steps, K, float(alpha), out.ctypes.data):
        raise ValueError("bad schedule parameters")
    return out


def verify_rows(seed: int, n_tokens: int, K: int, alpha: float) -> np.ndarray:
    """Rows of the verify batches of a speculative run over n_tokens tokens: [n_batches, K + 1].
    Batch i starts at the first uncommitted token p_i and holds K + 1 rows: the tokens p_i ..
    p_i + a_i (the target's own token and the a_i accepted drafts) and then rejected drafts;
    p_{i+1} = p_i + a_i + 1.  Entry >= 0: that token of the sequence; entry < 0: rejected draft
    number -1 - entry (numbered from 0 across the run).  Rows past the sequence's end are drafts."""
    acc = accepts(seed, 0, n_tokens, K, alpha)  # every step commits at least one token
    rows, p, drafts, i = [], 0, 0, 0
    while p < n_tokens:
        a = int(acc[i])
        row = []
        for j in range(K + 1):
            if j <= a and p + j < n_tokens:
                row.append(p + j)
            else:
                row.append(-1 - drafts)
                drafts += 1
        rows.append(row)
        p += a + 1
        i += 1
    return np.array(rows, dtype=np.int32).reshape(-1, K + 1)
