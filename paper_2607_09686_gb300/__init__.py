"""GB300 routed-expert step of one MoE decoder layer (MawForge, arXiv 2607.09686).

Thin ctypes binding of ``libmawforge.so`` (declared in ``include/mawforge.h``).  Every
step of the path runs in the library's CUDA kernels; this module only marshals
arguments.  Device buffers may be given as torch CUDA tensors (anything with
``data_ptr()``) or as raw integer addresses; streams as ``torch.cuda.Stream`` objects,
raw handles, or ``None`` for torch's current stream.

There is no CPU fallback: importing this package fails if the library has not been built
(``python -c "import __graft_entry__ as g; g.build()"``).
"""
from __future__ import annotations

import ctypes
import os

__all__ = [
    "MFError", "Model", "PlanReq", "Plan", "Stats", "TunePoint", "Q8_0", "Q4_0", "LIB_PATH", "KERNEL_CLASSES",
    "mf_payload_bytes", "mf_plan", "mf_tune_cache", "mf_create", "mf_pack_put", "mf_load_pack", "mf_moe_forward",
    "mf_moe_forward_host", "mf_prefill_threshold", "mf_access_order", "mf_stats", "mf_reset", "mf_trace", "mf_timing", "mf_timing_read", "mf_check", "mf_wait_limit", "mf_test_hold", "mf_expert_ffn_noalloc",
    "mf_expert_ffn_noalloc_check", "mf_pack_save", "mf_create_from_file", "mf_pack_file_stats",
    "mf_pack_file_direct", "mf_destroy",
    "mf_strerror", "mf_last_cuda_error",
]

Q4_0 = 2
Q8_0 = 8
MF_OK, MF_E_INVAL, MF_E_BUDGET, MF_E_OOM, MF_E_CUDA, MF_E_STATE, MF_E_TIMEOUT, MF_E_IO = 0, -1, -2, -3, -4, -5, -6, -7
KERNEL_CLASSES = ("router", "resolve", "materialize", "gateup_swiglu", "down_combine", "prefill_gemm", "ffn_fused")

LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "libmawforge.so")
if not os.path.exists(LIB_PATH):
    raise ImportError(f"{LIB_PATH} is missing: build the CUDA library first "
                      "(python -c 'import __graft_entry__ as g; g.build()')")
_lib = ctypes.CDLL(LIB_PATH)


class Model(ctypes.Structure):
    _fields_ = [("n_layers", ctypes.c_int32), ("hidden", ctypes.c_int32), ("n_experts", ctypes.c_int32),
                ("top_k", ctypes.c_int32), ("inter", ctypes.c_int32), ("qtype", ctypes.c_int32)]


class PlanReq(ctypes.Structure):
    _fields_ = [("cache_pct", ctypes.c_double), ("budget_bytes", ctypes.c_uint64), ("common_bytes", ctypes.c_uint64),
                ("kv_bytes", ctypes.c_uint64), ("max_tokens", ctypes.c_int32), ("reserved", ctypes.c_int32)]


class Plan(ctypes.Structure):
    _fields_ = [("accepted", ctypes.c_int32), ("slots_per_layer", ctypes.c_int32),
                ("payload_bytes", ctypes.c_uint64), ("pool_bytes", ctypes.c_uint64),
                ("lower_bound_bytes", ctypes.c_uint64), ("overhead_bytes", ctypes.c_uint64),
                ("footprint_bytes", ctypes.c_uint64), ("max_tokens", ctypes.c_int32), ("reserved", ctypes.c_int32)]

    def as_dict(self) -> dict:
        return {name: getattr(self, name) for name, _ in self._fields_ if name != "reserved"}


class Stats(ctypes.Structure):
    _fields_ = [("accesses", ctypes.c_uint64), ("hits", ctypes.c_uint64), ("misses", ctypes.c_uint64),
                ("evictions", ctypes.c_uint64), ("bytes_materialized", ctypes.c_uint64)]

    def as_dict(self) -> dict:
        return {name: int(getattr(self, name)) for name, _ in self._fields_}


class TunePoint(ctypes.Structure):
    _fields_ = [("cache_pct", ctypes.c_double), ("accepted", ctypes.c_int32), ("slots_per_layer", ctypes.c_int32),
                ("pool_bytes", ctypes.c_uint64), ("footprint_bytes", ctypes.c_uint64), ("accesses", ctypes.c_uint64),
                ("hits", ctypes.c_uint64), ("misses", ctypes.c_uint64), ("bytes_materialized", ctypes.c_uint64),
                ("predicted_s", ctypes.c_double), ("predicted_tokens_per_s", ctypes.c_double)]

    def as_dict(self) -> dict:
        return {name: getattr(self, name) for name, _ in self._fields_}


_vp, _i32, _u64 = ctypes.c_void_p, ctypes.c_int, ctypes.c_uint64
_sig = {
    "mf_payload_bytes": (_i32, [ctypes.POINTER(Model), ctypes.POINTER(_u64)]),
    "mf_plan": (_i32, [ctypes.POINTER(Model), ctypes.POINTER(PlanReq), ctypes.POINTER(Plan)]),
    "mf_tune_cache": (_i32, [ctypes.POINTER(Model), ctypes.POINTER(PlanReq), _vp, _i32, _i32, _i32, ctypes.c_double,
                             ctypes.c_double, _vp, _i32, ctypes.POINTER(TunePoint), ctypes.POINTER(_i32)]),
    "mf_create": (_i32, [ctypes.POINTER(_vp), ctypes.POINTER(Model), ctypes.POINTER(Plan), _i32]),
    "mf_pack_put": (_i32, [_vp, _i32, _i32, _vp, _u64]),
    "mf_load_pack": (_i32, [ctypes.POINTER(_vp), ctypes.POINTER(Model), ctypes.POINTER(Plan), _vp, _i32]),
    "mf_moe_forward": (_i32, [_vp, _i32, _vp, _vp, _vp, _i32, _vp, _vp, _vp, _vp]),
    "mf_moe_forward_host": (_i32, [_vp, _i32, _vp, _vp, _vp, _i32, _vp, _vp, _vp, _vp]),
    "mf_prefill_threshold": (_i32, [_vp, _i32]),
    "mf_access_order": (_i32, [_vp, _i32]),
    "mf_stats": (_i32, [_vp, _i32, ctypes.POINTER(Stats), _i32]),
    "mf_reset": (_i32, [_vp, _i32, _vp]),
    "mf_trace": (_i32, [_vp, _i32, _vp, _vp, _vp, _i32, ctypes.POINTER(_i32)]),
    "mf_timing": (_i32, [_vp, ctypes.c_uint]),
    "mf_timing_read": (_i32, [_vp, _vp, _vp]),
    "mf_check": (_i32, [_vp]),
    "mf_wait_limit": (_i32, [_vp, ctypes.c_double]),
    "mf_test_hold": (_i32, [_vp, _i32]),
    "mf_expert_ffn_noalloc": (_i32, [ctypes.POINTER(Model), _vp, _vp, _vp, _vp, _vp]),
    "mf_expert_ffn_noalloc_check": (_i32, []),
    "mf_pack_save": (_i32, [_vp, ctypes.c_char_p]),
    "mf_create_from_file": (_i32, [ctypes.POINTER(_vp), ctypes.POINTER(Model), ctypes.POINTER(Plan), ctypes.c_char_p,
                                   _i32]),
    "mf_pack_file_stats": (_i32, [_vp, ctypes.POINTER(_u64), ctypes.POINTER(_u64), ctypes.POINTER(ctypes.c_double)]),
    "mf_pack_file_direct": (_i32, [_vp]),
    "mf_destroy": (None, [_vp]),
    "mf_strerror": (ctypes.c_char_p, [_i32]),
    "mf_last_cuda_error": (ctypes.c_char_p, []),
}
for _name, (_res, _args) in _sig.items():
    _f = getattr(_lib, _name)
    _f.restype, _f.argtypes = _res, _args


class MFError(RuntimeError):
    def __init__(self, status: int, where: str):
        msg = _lib.mf_strerror(status).decode()
        if status == MF_E_CUDA:
            msg += f" ({_lib.mf_last_cuda_error().decode()})"
        super().__init__(f"{where}: {msg} [{status}]")
        self.status = status


def _check(status: int, where: str) -> None:
    if status != MF_OK:
        raise MFError(status, where)


def _addr(buf):
    """Address of a buffer: None, an int, a torch tensor, or a numpy array."""
    if buf is None:
        return None
    if isinstance(buf, int):
        return buf
    if hasattr(buf, "data_ptr"):
        return buf.data_ptr()
    if hasattr(buf, "ctypes"):
        return buf.ctypes.data
    raise TypeError(f"cannot take the address of {type(buf).__name__}")


def _stream(stream):
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def mf_strerror(status: int) -> str:
    return _lib.mf_strerror(status).decode()


def mf_last_cuda_error() -> str:
    return _lib.mf_last_cuda_error().decode()


def mf_payload_bytes(model: Model) -> int:
    out = _u64()
    _check(_lib.mf_payload_bytes(ctypes.byref(model), ctypes.byref(out)), "mf_payload_bytes")
    return int(out.value)


def mf_plan(model: Model, req: PlanReq) -> Plan:
    """Static plan; a rejected plan is returned too (plan.accepted == 0), not raised."""
    out = Plan()
    rc = _lib.mf_plan(ctypes.byref(model), ctypes.byref(req), ctypes.byref(out))
    if rc not in (MF_OK, MF_E_BUDGET):
        _check(rc, "mf_plan")
    return out


def mf_tune_cache(model: Model, req: PlanReq, routes, T: int, t_token_s: float, t_miss_s: float, pcts,
                  order: int = 0):
    """Cache-size tuner (host only).  routes: int32 array [n_layers][n_tokens][top_k] (C order).
    Returns (list of per-candidate dicts, index of the best accepted candidate or -1)."""
    import numpy as np
    r = np.ascontiguousarray(routes, dtype=np.int32)
    if r.ndim != 3:
        raise ValueError("routes must be [n_layers][n_tokens][top_k]")
    n = len(pcts)
    cand = (ctypes.c_double * max(1, n))(*[float(p) for p in pcts])
    out = (TunePoint * max(1, n))()
    best = _i32(-1)
    rc = _lib.mf_tune_cache(ctypes.byref(model), ctypes.byref(req), r.ctypes.data, r.shape[1], T, order,
                            float(t_token_s), float(t_miss_s), cand, n, out, ctypes.byref(best))
    if rc not in (MF_OK, MF_E_BUDGET):
        _check(rc, "mf_tune_cache")
    return [out[i].as_dict() for i in range(n)], best.value


def mf_create(model: Model, plan: Plan, device: int = 0) -> int:
    h = _vp()
    _check(_lib.mf_create(ctypes.byref(h), ctypes.byref(model), ctypes.byref(plan), device), "mf_create")
    return h.value


def mf_pack_put(ctx: int, layer: int, expert: int, payload) -> None:
    n = payload.nbytes if hasattr(payload, "nbytes") else len(payload)
    _check(_lib.mf_pack_put(ctx, layer, expert, _addr(payload), n), "mf_pack_put")


def mf_pack_save(ctx: int, path: str) -> None:
    """Write the context's split-pack to a file (header, index, one record per payload)."""
    _check(_lib.mf_pack_save(ctx, os.fsencode(path)), "mf_pack_save")


def mf_create_from_file(model: Model, plan: Plan, path: str, device: int = 0) -> int:
    """A context whose split-pack is the file written by mf_pack_save (misses read from it)."""
    h = _vp()
    _check(_lib.mf_create_from_file(ctypes.byref(h), ctypes.byref(model), ctypes.byref(plan), os.fsencode(path),
                                    device), "mf_create_from_file")
    return h.value


def mf_pack_file_stats(ctx: int) -> dict:
    """{reads, bytes, seconds} of a file-backed context's reads so far."""
    r, b, t = _u64(), _u64(), ctypes.c_double()
    _check(_lib.mf_pack_file_stats(ctx, ctypes.byref(r), ctypes.byref(b), ctypes.byref(t)), "mf_pack_file_stats")
    return {"reads": int(r.value), "bytes": int(b.value), "seconds": float(t.value)}


def mf_pack_file_direct(ctx: int) -> bool:
    """True if the file-backed context reads its file unbuffered (O_DIRECT)."""
    rc = _lib.mf_pack_file_direct(ctx)
    if rc < 0:
        _check(rc, "mf_pack_file_direct")
    return rc == 1


def mf_load_pack(model: Model, plan: Plan, payloads, device: int = 0) -> int:
    """payloads: sequence of L*E host buffers (numpy uint8), layer-major."""
    arr = (_vp * len(payloads))(*[_addr(p) for p in payloads])
    h = _vp()
    _check(_lib.mf_load_pack(ctypes.byref(h), ctypes.byref(model), ctypes.byref(plan),
                             ctypes.cast(arr, _vp), device), "mf_load_pack")
    return h.value


def mf_moe_forward(ctx: int, layer: int, x, router_w, logit_bias, T: int, y, idx_out=None, w_out=None,
                   stream=None) -> None:
    _check(_lib.mf_moe_forward(ctx, layer, _addr(x), _addr(router_w), _addr(logit_bias), T, _addr(y),
                               _addr(idx_out), _addr(w_out), _stream(stream)), "mf_moe_forward")


def mf_moe_forward_host(ctx: int, layer: int, x, router_w, logit_bias, T: int, y, idx_out=None, w_out=None,
                        stream=None) -> None:
    _check(_lib.mf_moe_forward_host(ctx, layer, _addr(x), _addr(router_w), _addr(logit_bias), T, _addr(y),
                                    _addr(idx_out), _addr(w_out), _stream(stream)), "mf_moe_forward_host")


def mf_prefill_threshold(ctx: int, min_tokens: int) -> None:
    """Calls with T >= min_tokens use the tensor-core grouped GEMMs (0 = never)."""
    _check(_lib.mf_prefill_threshold(ctx, min_tokens), "mf_prefill_threshold")


MF_ORDER_FIRST_OCCURRENCE = 0
MF_ORDER_RESIDENT_FIRST = 1


def mf_access_order(ctx: int, order: int) -> None:
    """Order of a many-token call's accesses to the cache (MF_ORDER_*)."""
    _check(_lib.mf_access_order(ctx, order), "mf_access_order")


def mf_stats(ctx: int, layer: int = -1, reset: bool = False) -> dict:
    out = Stats()
    _check(_lib.mf_stats(ctx, layer, ctypes.byref(out), 1 if reset else 0), "mf_stats")
    return out.as_dict()


def mf_reset(ctx: int, slots_per_layer: int = 0, stream=None) -> None:
    _check(_lib.mf_reset(ctx, slots_per_layer, _stream(stream)), "mf_reset")


def mf_trace(ctx: int, layer: int, cap: int = 1024):
    """(experts, slots, hits) of the latest call of `layer`, as Python lists."""
    exp = (ctypes.c_int32 * cap)()
    slo = (ctypes.c_int32 * cap)()
    hit = (ctypes.c_uint8 * cap)()
    n = _i32()
    _check(_lib.mf_trace(ctx, layer, exp, slo, hit, cap, ctypes.byref(n)), "mf_trace")
    return list(exp[:n.value]), list(slo[:n.value]), [bool(v) for v in hit[:n.value]]


def mf_timing(ctx: int, classes=None) -> None:
    """Time the kernel classes named in `classes` (names from KERNEL_CLASSES; None = all, [] = off)."""
    if classes is None:
        mask = (1 << len(KERNEL_CLASSES)) - 1
    elif classes is False:
        mask = 0
    else:
        mask = 0
        for c in classes:
            mask |= 1 << KERNEL_CLASSES.index(c)
    _check(_lib.mf_timing(ctx, mask), "mf_timing")


def mf_timing_read(ctx: int) -> dict:
    """{kernel class: (summed ms, launches)} from the CUDA events of each launch."""
    ms = (ctypes.c_double * len(KERNEL_CLASSES))()
    n = (ctypes.c_int64 * len(KERNEL_CLASSES))()
    _check(_lib.mf_timing_read(ctx, ms, n), "mf_timing_read")
    return {KERNEL_CLASSES[i]: (float(ms[i]), int(n[i])) for i in range(len(KERNEL_CLASSES))}


def mf_check(ctx: int) -> int:
    """0, MF_E_TIMEOUT if a kernel of this context gave up a bounded wait, or MF_E_IO if a read of
    its split-pack file failed (returned, not raised)."""
    rc = _lib.mf_check(ctx)
    if rc not in (MF_OK, MF_E_TIMEOUT, MF_E_IO):
        _check(rc, "mf_check")
    return rc


def mf_wait_limit(ctx: int, seconds: float) -> None:
    """Time limit of every bounded wait inside the context's kernels."""
    _check(_lib.mf_wait_limit(ctx, float(seconds)), "mf_wait_limit")


def mf_test_hold(ctx: int, hold: int) -> None:
    """Test hold of the failure path: 1 = the one-token FFN's producer issues no copies."""
    _check(_lib.mf_test_hold(ctx, int(hold)), "mf_test_hold")


def mf_expert_ffn_noalloc_check() -> int:
    """0, or MF_E_TIMEOUT if a no-allocation call on the current device gave up a bounded wait since
    the last check (returned, not raised)."""
    rc = _lib.mf_expert_ffn_noalloc_check()
    if rc not in (MF_OK, MF_E_TIMEOUT):
        _check(rc, "mf_expert_ffn_noalloc_check")
    return rc


def mf_expert_ffn_noalloc(model: Model, experts, g, x, y, stream=None) -> None:
    """One-token expert FFN from caller-held expert slots, allocating nothing (see mawforge.h)."""
    _check(_lib.mf_expert_ffn_noalloc(ctypes.byref(model), _addr(experts), _addr(g), _addr(x), _addr(y),
                                      _stream(stream)), "mf_expert_ffn_noalloc")


def mf_destroy(ctx: int) -> None:
    if ctx:
        _lib.mf_destroy(ctx)
