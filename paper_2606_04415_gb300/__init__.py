"""GB300 mixed prefill/decode paged attention: Python binding of the C ABI.

Thin ctypes marshalling over ``_build/libfnpu.so`` (declared in
``include/fnpu.h``); every step of the computation runs in the library's CUDA
kernels. Functions carry the C names without the ``fnpu_`` prefix:

    kv_append(desc, k_new, v_new, slot_mapping, k_cache, v_cache, stream=None)
    mixed_attn_plan(desc, query_len, context_len, phase, block_table, opts=None, stream=None)
    mixed_attn_replan(plan, query_len, context_len, phase, block_table, opts=None, stream=None)
    mixed_attn_run(plan, q, k_cache, v_cache, out, lse, stream=None)
    check(stream=None), plan_check(plan, stream=None), status_str(code)

Device arguments are CUDA torch tensors (torch supplies device memory and
streams only) or raw integer device addresses; host metadata are numpy arrays.
There is no CPU fallback: if the library is missing, importing the binding's
entry points raises.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional

import numpy as np

from . import build as _build

FNPU_OK = 0
FNPU_EINVAL = -1
FNPU_EUNSUPPORTED = -2
FNPU_ECUDA = -3
FNPU_EDEVICE_TIMEOUT = -4
FNPU_ENOMEM = -5
FNPU_EDEVICE_RANGE = -6

PLAN_SEPARATE_LAUNCHES = 1
PLAN_NO_TCGEN05 = 2
PLAN_GREEN_CONTEXTS = 4
PLAN_FUSED_APPEND = 8

EXPORTED = (
    "fnpu_kv_append", "fnpu_mixed_attn_plan", "fnpu_mixed_attn_plan_ex", "fnpu_mixed_attn_run",
    "fnpu_plan_check", "fnpu_check", "fnpu_plan_destroy", "fnpu_plan_info", "fnpu_status_str",
    "fnpu_version", "fnpu_decode_attn_noalloc", "fnpu_last_cuda_error", "fnpu_plan_phase_ms",
    "fnpu_dispatch_next_share", "fnpu_mla_expand", "fnpu_mixed_attn_replan",
    "fnpu_plan_decode_share", "fnpu_mixed_step",
)


class FnpuError(RuntimeError):
    def __init__(self, code: int, what: str):
        msg = f"{what}: {status_str(code)} ({code})"
        if code == FNPU_ECUDA:
            msg += f" [{last_cuda_error()}]"
        super().__init__(msg)
        self.code = code


class AttnDesc(ctypes.Structure):
    _fields_ = [("num_q_heads", ctypes.c_int32), ("num_kv_heads", ctypes.c_int32),
                ("head_dim_qk", ctypes.c_int32), ("head_dim_v", ctypes.c_int32),
                ("block_size", ctypes.c_int32), ("num_blocks", ctypes.c_int32),
                ("v_in_k_latent", ctypes.c_int32), ("softmax_scale", ctypes.c_float),
                ("kv_fp8", ctypes.c_int32)]


class PlanOpts(ctypes.Structure):
    _fields_ = [("decode_split_keys", ctypes.c_int32), ("decode_share_pct", ctypes.c_int32),
                ("num_sms", ctypes.c_int32), ("flags", ctypes.c_int32)]


_lib = None


def lib_path() -> str:
    return _build.LIB


def load(build_if_missing: bool = True):
    """Load the CUDA library (building it first if it is absent or stale)."""
    global _lib
    if _lib is not None:
        return _lib
    if build_if_missing:
        _build.build()
    if not os.path.exists(_build.LIB):
        raise ImportError(f"CUDA library {_build.LIB} is missing; run __graft_entry__.build()")
    lib = ctypes.CDLL(_build.LIB)
    P, i32, i64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64
    lib.fnpu_kv_append.argtypes = [ctypes.POINTER(AttnDesc), P, P, P, i32, P, P, P]
    lib.fnpu_mixed_attn_plan.argtypes = [ctypes.POINTER(AttnDesc), i32, P, P, P, P, i32, P,
                                         ctypes.POINTER(P)]
    lib.fnpu_mixed_attn_plan_ex.argtypes = [ctypes.POINTER(AttnDesc), i32, P, P, P, P, i32,
                                            ctypes.POINTER(PlanOpts), P, ctypes.POINTER(P)]
    lib.fnpu_mixed_attn_replan.argtypes = [P, i32, P, P, P, P, i32, ctypes.POINTER(PlanOpts), P]
    lib.fnpu_mixed_attn_run.argtypes = [P, P, P, P, P, P, P]
    lib.fnpu_mixed_step.argtypes = [P, P, P, P, P, P, P, P, P, P]
    lib.fnpu_plan_decode_share.argtypes = [P, ctypes.POINTER(i32)]
    lib.fnpu_mla_expand.argtypes = [ctypes.POINTER(AttnDesc), P, P, i32, P, P, P, P, P, P]
    lib.fnpu_plan_check.argtypes = [P, P]
    lib.fnpu_check.argtypes = [P]
    lib.fnpu_plan_destroy.argtypes = [P]
    lib.fnpu_plan_destroy.restype = None
    lib.fnpu_plan_info.argtypes = [P, ctypes.POINTER(i32), ctypes.POINTER(i32), ctypes.POINTER(i32),
                                   ctypes.POINTER(i64)]
    lib.fnpu_decode_attn_noalloc.argtypes = [ctypes.POINTER(AttnDesc), i32, P, P, i32, i32, i32,
                                             P, P, P, P, P, P]
    lib.fnpu_last_cuda_error.argtypes = []
    lib.fnpu_last_cuda_error.restype = ctypes.c_char_p
    lib.fnpu_status_str.argtypes = [ctypes.c_int]
    lib.fnpu_status_str.restype = ctypes.c_char_p
    lib.fnpu_plan_phase_ms.argtypes = [P, ctypes.POINTER(ctypes.c_float), ctypes.POINTER(ctypes.c_float)]
    lib.fnpu_dispatch_next_share.argtypes = [i32, ctypes.c_float, ctypes.c_float, ctypes.c_float,
                                             ctypes.POINTER(i32)]
    for name in ("fnpu_kv_append", "fnpu_mixed_attn_plan", "fnpu_mixed_attn_plan_ex",
                 "fnpu_mixed_attn_run", "fnpu_plan_check", "fnpu_check", "fnpu_plan_info",
                 "fnpu_version", "fnpu_decode_attn_noalloc", "fnpu_plan_phase_ms",
                 "fnpu_dispatch_next_share", "fnpu_mla_expand", "fnpu_mixed_attn_replan",
                 "fnpu_plan_decode_share"):
        getattr(lib, name).restype = ctypes.c_int
    _lib = lib
    return lib


def last_cuda_error() -> str:
    return load().fnpu_last_cuda_error().decode()


def status_str(code: int) -> str:
    return load().fnpu_status_str(int(code)).decode()


def _dptr(x) -> Optional[int]:
    """Device address of a CUDA tensor / raw int / None."""
    if x is None:
        return None
    if isinstance(x, int):
        return x
    if hasattr(x, "data_ptr"):
        if not x.is_cuda:
            raise ValueError("expected a CUDA tensor")
        if not x.is_contiguous():
            raise ValueError("expected a contiguous tensor")
        return x.data_ptr()
    raise TypeError(f"cannot take a device address of {type(x)!r}")


def _stream(stream) -> Optional[int]:
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _np(a, dtype) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(a), dtype=dtype)


# bytes of one block of the FP8 cache format (16 slots, 4 kv heads, d = 128):
# K or V codes [16 * 4 * 128] then fp32 scales [16 * 4]
FP8_BLOCK_BYTES = 16 * 4 * 128 + 16 * 4 * 4


def mla_expand(desc: AttnDesc, latent_cache, slots, w_uk, w_uv, workspace, k_out, v_out, stream=None,
               num_rows: Optional[int] = None) -> None:
    """Per-head keys [n, Hq, 192] and values [n, Hq, 128] of latent rows
    (``fnpu_mla_expand``): MLA prefill without absorption."""
    if num_rows is None:
        num_rows = int(slots.shape[0])
    rc = load().fnpu_mla_expand(ctypes.byref(desc), _dptr(latent_cache), _dptr(slots), int(num_rows), _dptr(w_uk),
                                _dptr(w_uv), _dptr(workspace), _dptr(k_out), _dptr(v_out), _stream(stream))
    if rc != FNPU_OK:
        raise FnpuError(rc, "fnpu_mla_expand")


def make_desc(num_q_heads, num_kv_heads, head_dim_qk, head_dim_v, block_size, num_blocks,
              latent=False, softmax_scale=0.0, kv_fp8=False) -> AttnDesc:
    return AttnDesc(num_q_heads, num_kv_heads, head_dim_qk, head_dim_v, block_size, num_blocks,
                    int(bool(latent)), float(softmax_scale), int(bool(kv_fp8)))


def kv_append(desc: AttnDesc, k_new, v_new, slot_mapping, k_cache, v_cache, stream=None,
              num_tokens: Optional[int] = None) -> None:
    """Store new K/V rows into their paged slots (``fnpu_kv_append``)."""
    if num_tokens is None:
        num_tokens = int(slot_mapping.shape[0])
    rc = load().fnpu_kv_append(ctypes.byref(desc), _dptr(k_new), _dptr(v_new), _dptr(slot_mapping),
                               int(num_tokens), _dptr(k_cache), _dptr(v_cache), _stream(stream))
    if rc != FNPU_OK:
        raise FnpuError(rc, "fnpu_kv_append")


class Plan:
    """Owner of an ``fnpu_plan*``; destroyed with the object."""

    def __init__(self, handle: int, desc: AttnDesc, num_tokens: int):
        self.handle = handle
        self.desc = desc
        self.num_tokens = num_tokens

    def info(self) -> dict:
        pi, di, la = ctypes.c_int32(), ctypes.c_int32(), ctypes.c_int32()
        ws = ctypes.c_int64()
        rc = load().fnpu_plan_info(self.handle, ctypes.byref(pi), ctypes.byref(di), ctypes.byref(la),
                                   ctypes.byref(ws))
        if rc != FNPU_OK:
            raise FnpuError(rc, "fnpu_plan_info")
        return {"prefill_items": pi.value, "decode_items": di.value, "launches_per_run": la.value,
                "workspace_bytes": ws.value}

    def destroy(self) -> None:
        if self.handle:
            load().fnpu_plan_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.destroy()
        except Exception:
            pass


def mixed_attn_plan(desc: AttnDesc, query_len, context_len, phase, block_table,
                    opts: Optional[PlanOpts] = None, stream=None) -> Plan:
    """Build the phase-aware work list of one step (``fnpu_mixed_attn_plan_ex``)."""
    ql = _np(query_len, np.int32)
    cl = _np(context_len, np.int32)
    ph = _np(phase, np.uint8)
    bt = _np(block_table, np.int32)
    if bt.ndim != 2 or not (ql.shape == cl.shape == ph.shape) or bt.shape[0] != ql.shape[0]:
        raise ValueError("metadata shapes disagree")
    out = ctypes.c_void_p()
    rc = load().fnpu_mixed_attn_plan_ex(ctypes.byref(desc), int(ql.shape[0]), ql.ctypes.data,
                                        cl.ctypes.data, ph.ctypes.data, bt.ctypes.data,
                                        int(bt.shape[1]), None if opts is None else ctypes.byref(opts),
                                        _stream(stream), ctypes.byref(out))
    if rc != FNPU_OK:
        raise FnpuError(rc, "fnpu_mixed_attn_plan")
    return Plan(out.value, desc, int(ql.sum()))


def mixed_attn_replan(plan: Plan, query_len, context_len, phase, block_table,
                      opts: Optional[PlanOpts] = None, stream=None) -> None:
    """Rebuild ``plan`` for a new step's metadata, reusing its streams, events,
    staging and workspace (``fnpu_mixed_attn_replan``)."""
    ql = _np(query_len, np.int32)
    cl = _np(context_len, np.int32)
    ph = _np(phase, np.uint8)
    bt = _np(block_table, np.int32)
    if bt.ndim != 2 or not (ql.shape == cl.shape == ph.shape) or bt.shape[0] != ql.shape[0]:
        raise ValueError("metadata shapes disagree")
    rc = load().fnpu_mixed_attn_replan(plan.handle, int(ql.shape[0]), ql.ctypes.data, cl.ctypes.data,
                                       ph.ctypes.data, bt.ctypes.data, int(bt.shape[1]),
                                       None if opts is None else ctypes.byref(opts), _stream(stream))
    if rc != FNPU_OK:
        raise FnpuError(rc, "fnpu_mixed_attn_replan")
    plan.num_tokens = int(ql.sum())


def mixed_attn_run(plan: Plan, q, k_cache, v_cache, out, lse, stream=None) -> None:
    """Attention of every planned query (``fnpu_mixed_attn_run``)."""
    rc = load().fnpu_mixed_attn_run(plan.handle, _dptr(q), _dptr(k_cache), _dptr(v_cache),
                                    _dptr(out), _dptr(lse), _stream(stream))
    if rc != FNPU_OK:
        raise FnpuError(rc, "fnpu_mixed_attn_run")


def mixed_step(plan: Plan, k_new, v_new, slot_mapping, q, k_cache, v_cache, out, lse, stream=None) -> None:
    """Append of the step's new rows and attention of every planned query in
    one call (``fnpu_mixed_step``; the same results as ``kv_append`` then
    ``mixed_attn_run``)."""
    rc = load().fnpu_mixed_step(plan.handle, _dptr(k_new), _dptr(v_new), _dptr(slot_mapping), _dptr(q),
                                _dptr(k_cache), _dptr(v_cache), _dptr(out), _dptr(lse), _stream(stream))
    if rc != FNPU_OK:
        raise FnpuError(rc, "fnpu_mixed_step")


def decode_attn_noalloc(desc: AttnDesc, context_len, block_table, max_context_len: int, q,
                        k_cache, v_cache, out, lse, split_keys: int = 0, stream=None) -> None:
    """Decode attention with the library's fixed scratch and no allocation
    (``fnpu_decode_attn_noalloc``); context_len and block_table are device
    int32 tensors."""
    rc = load().fnpu_decode_attn_noalloc(ctypes.byref(desc), int(context_len.shape[0]),
                                         _dptr(context_len), _dptr(block_table),
                                         int(block_table.shape[1]), int(max_context_len),
                                         int(split_keys), _dptr(q), _dptr(k_cache), _dptr(v_cache),
                                         _dptr(out), _dptr(lse), _stream(stream))
    if rc != FNPU_OK:
        raise FnpuError(rc, "fnpu_decode_attn_noalloc")


def plan_check(plan: Plan, stream=None) -> int:
    return int(load().fnpu_plan_check(plan.handle, _stream(stream)))


def check(stream=None) -> int:
    return int(load().fnpu_check(_stream(stream)))


def version() -> int:
    return int(load().fnpu_version())


def plan_phase_ms(plan: Plan) -> tuple:
    """(prefill_ms, decode_ms) of the last co-located run of `plan`."""
    a, b = ctypes.c_float(), ctypes.c_float()
    rc = load().fnpu_plan_phase_ms(plan.handle, ctypes.byref(a), ctypes.byref(b))
    if rc != FNPU_OK:
        raise FnpuError(rc, "fnpu_plan_phase_ms")
    return a.value, b.value


def plan_decode_share(plan: Plan) -> int:
    """Decode share (percent of SMs) a co-located plan uses."""
    out = ctypes.c_int32()
    rc = load().fnpu_plan_decode_share(plan.handle, ctypes.byref(out))
    if rc != FNPU_OK:
        raise FnpuError(rc, "fnpu_plan_decode_share")
    return out.value


def dispatch_next_share(share_pct: int, prefill_ms: float, decode_ms: float, tolerance: float = 0.05) -> int:
    """Decode share (percent of SMs) for the next step of a serving loop."""
    out = ctypes.c_int32()
    rc = load().fnpu_dispatch_next_share(int(share_pct), float(prefill_ms), float(decode_ms), float(tolerance),
                                         ctypes.byref(out))
    if rc != FNPU_OK:
        raise FnpuError(rc, "fnpu_dispatch_next_share")
    return out.value
