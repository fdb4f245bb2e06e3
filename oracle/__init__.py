"""CPU oracle for the routed-expert step — TEST INFRASTRUCTURE.

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline leg (and its
``--impl reference`` arm) may import this package.  The product path (the CUDA library
and its binding) never does, and shares no code with it.

The arithmetic lives in ``oracle.c`` (plain C, fp64, one obvious loop per definition),
built into ``liboracle.so`` next to this file; this module only marshals arguments.
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

Q8_0 = 8
Q4_0 = 2

_HERE = os.path.dirname(os.path.abspath(__file__))
_SO = os.path.join(_HERE, "liboracle.so")
_LIB = None


def build(force: bool = False) -> str:
    """Compile oracle.c into liboracle.so (gcc, OpenMP over rows, no FP contraction)."""
    src = os.path.join(_HERE, "oracle.c")
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
        i32, u64, dbl, vp = ctypes.c_int, ctypes.c_uint64, ctypes.c_double, ctypes.c_void_p
        lib.orc_f16.restype = dbl
        lib.orc_f16.argtypes = [ctypes.c_uint16]
        lib.orc_dequant_row.restype = i32
        lib.orc_dequant_row.argtypes = [i32, vp, i32, vp]
        lib.orc_payload_bytes.restype = u64
        lib.orc_payload_bytes.argtypes = [i32, i32, i32]
        lib.orc_router.restype = i32
        lib.orc_router.argtypes = [vp, vp, vp, i32, i32, i32, vp, vp, vp]
        lib.orc_expert_ffn.restype = i32
        lib.orc_expert_ffn.argtypes = [vp, i32, i32, i32, vp, vp, vp]
        lib.orc_layer.restype = i32
        lib.orc_layer.argtypes = [vp, i32, i32, i32, i32, i32, vp, vp, vp, i32, vp, vp, vp]
        lib.orc_lru_new.restype = vp
        lib.orc_lru_new.argtypes = [i32, i32, u64]
        lib.orc_lru_free.restype = None
        lib.orc_lru_free.argtypes = [vp]
        lib.orc_lru_step.restype = i32
        lib.orc_lru_step.argtypes = [vp, vp, i32, i32, i32, vp, vp, vp]
        lib.orc_lru_stats.restype = None
        lib.orc_lru_stats.argtypes = [vp, vp]
        lib.orc_lru_occupancy.restype = i32
        lib.orc_lru_occupancy.argtypes = [vp]
        lib.orc_lru_slots.restype = None
        lib.orc_lru_slots.argtypes = [vp, vp]
        lib.orc_plan.restype = i32
        lib.orc_plan.argtypes = [i32, i32, i32, i32, i32, i32, dbl, u64, u64, u64, vp]
        _LIB = lib
    return _LIB


def _ptr(a: np.ndarray | None):
    return None if a is None else a.ctypes.data


def f16(bits: int) -> float:
    return float(_lib().orc_f16(int(bits)))


def dequant_row(qtype: int, blocks: np.ndarray, cols: int) -> np.ndarray:
    blocks = np.ascontiguousarray(blocks, dtype=np.uint8)
    out = np.empty(cols, dtype=np.float64)
    if _lib().orc_dequant_row(qtype, _ptr(blocks), cols, _ptr(out)):
        raise ValueError("bad qtype or cols")
    return out


def payload_bytes(hidden: int, inter: int, qtype: int) -> int:
    return int(_lib().orc_payload_bytes(hidden, inter, qtype))


def router(x: np.ndarray, wr: np.ndarray, bias: np.ndarray | None, k: int):
    """(z float32 [E], idx int32 [k], g float64 [k]) for one token."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    wr = np.ascontiguousarray(wr, dtype=np.float32)
    E, H = wr.shape
    b = None if bias is None else np.ascontiguousarray(bias, dtype=np.float32)
    z = np.empty(E, np.float32)
    idx = np.empty(k, np.int32)
    g = np.empty(k, np.float64)
    if _lib().orc_router(_ptr(x), _ptr(wr), _ptr(b), E, H, k, _ptr(z), _ptr(idx), _ptr(g)):
        raise ValueError("bad router arguments")
    return z, idx, g


def expert_ffn(payload: np.ndarray, qtype: int, hidden: int, inter: int, x: np.ndarray):
    """(y float64 [H], h float64 [I]) of one expert on one token."""
    payload = np.ascontiguousarray(payload, dtype=np.uint8)
    x = np.ascontiguousarray(x, dtype=np.float32)
    y = np.empty(hidden, np.float64)
    h = np.empty(inter, np.float64)
    if _lib().orc_expert_ffn(_ptr(payload), qtype, hidden, inter, _ptr(x), _ptr(y), _ptr(h)):
        raise ValueError("bad expert arguments")
    return y, h


def layer(payloads, qtype: int, hidden: int, inter: int, top_k: int, wr: np.ndarray,
          bias: np.ndarray | None, x: np.ndarray):
    """(y float32 [T,H], idx int32 [T,k], g float64 [T,k]).

    ``payloads`` is a sequence of length E of uint8 arrays (None where no token routes)."""
    E = len(payloads)
    keep = [None if p is None else np.ascontiguousarray(p, dtype=np.uint8) for p in payloads]
    arr = (ctypes.c_void_p * E)(*[None if p is None else p.ctypes.data for p in keep])
    x = np.ascontiguousarray(x, dtype=np.float32).reshape(-1, hidden)
    T = x.shape[0]
    wr = np.ascontiguousarray(wr, dtype=np.float32)
    b = None if bias is None else np.ascontiguousarray(bias, dtype=np.float32).reshape(T, E)
    y = np.empty((T, hidden), np.float32)
    idx = np.empty((T, top_k), np.int32)
    g = np.empty((T, top_k), np.float64)
    rc = _lib().orc_layer(ctypes.cast(arr, ctypes.c_void_p), qtype, E, hidden, inter, top_k, _ptr(wr), _ptr(b),
                          _ptr(x), T, _ptr(y), _ptr(idx), _ptr(g))
    if rc == -3:
        raise KeyError("a routed expert's payload was not supplied")
    if rc:
        raise ValueError(f"orc_layer failed ({rc})")
    return y, idx, g


class LRU:
    """One layer's bounded slot cache (least-recently-used replacement)."""

    def __init__(self, n_experts: int, slots: int, payload: int):
        self._h = _lib().orc_lru_new(n_experts, slots, payload)
        if not self._h:
            raise ValueError("bad cache shape")
        self.E, self.S = n_experts, slots

    def __del__(self):
        h = getattr(self, "_h", None)
        if h:
            _lib().orc_lru_free(h)
            self._h = None

    def step(self, idx: np.ndarray, order: int = 0):
        """Process one step's routes [T,k]: returns (experts, slots, hits) of its accesses.
        order 0: first-occurrence order; 1: for T > 1, the experts resident at the start first."""
        idx = np.ascontiguousarray(idx, dtype=np.int32)
        T, k = idx.reshape(-1, idx.shape[-1]).shape
        n = T * k
        uniq = np.empty(n, np.int32)
        slot = np.empty(n, np.int32)
        hit = np.empty(n, np.uint8)
        U = _lib().orc_lru_step(self._h, _ptr(idx), T, k, int(order), _ptr(uniq), _ptr(slot), _ptr(hit))
        if U < 0:
            raise ValueError("expert id out of range" if U == -1 else "out of memory")
        return uniq[:U].copy(), slot[:U].copy(), hit[:U].astype(bool)

    def stats(self) -> dict:
        out = np.empty(5, np.uint64)
        _lib().orc_lru_stats(self._h, _ptr(out))
        return dict(zip(("accesses", "hits", "misses", "evictions", "bytes"), (int(v) for v in out)))

    def occupancy(self) -> int:
        return int(_lib().orc_lru_occupancy(self._h))

    def slots(self) -> np.ndarray:
        out = np.empty(self.S, np.int32)
        _lib().orc_lru_slots(self._h, _ptr(out))
        return out


def plan(n_layers, hidden, n_experts, top_k, inter, qtype, cache_pct, budget, common=0, kv=0) -> dict:
    out = np.empty(5, np.uint64)
    if _lib().orc_plan(n_layers, hidden, n_experts, top_k, inter, qtype, float(cache_pct), int(budget), int(common),
                       int(kv), _ptr(out)):
        raise ValueError("bad plan arguments")
    return dict(slots=int(out[0]), payload=int(out[1]), pool=int(out[2]), lower=int(out[3]), accepted=bool(out[4]))
