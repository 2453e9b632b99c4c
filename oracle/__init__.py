"""fp64 CPU oracle for the mixed prefill/decode paged-attention step.

TEST INFRASTRUCTURE. Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU
baseline legs of ``bench.py`` may import this package. It shares no code with
the CUDA path and never imports it.

The arithmetic lives in ``fnpu_oracle.c`` (plain C, double precision, OpenMP
over output rows); this module compiles it with gcc on first use and wraps it
with ctypes. What it computes is the textbook causal scaled-dot-product
attention over keys gathered through a block table, with the phase semantics of
the paper (prefill chunks with an optional cached prefix and one-token decodes
sharing one KV pool; Sec. 1, Sec. 2.3, Sec. 3.4). The paper prints no attention
formula; every reading taken where it is silent is listed in the C file's
header and in the design notes.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading
from typing import Optional

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "fnpu_oracle.c")
_BUILD_DIR = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD_DIR, "libfnpu_oracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (-O2, OpenMP). Returns the library path."""
    os.makedirs(_BUILD_DIR, exist_ok=True)
    if force or not os.path.exists(_LIB_PATH) or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC):
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fopenmp",
                               _SRC, "-o", tmp, "-lm"])
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is None:
            # FNPU_ORACLE_LIB lets the mutation tests load a deliberately broken copy
            lib = ctypes.CDLL(os.environ.get("FNPU_ORACLE_LIB") or build())
            P = ctypes.c_void_p
            i32, i64, f64 = ctypes.c_int32, ctypes.c_int64, ctypes.c_double
            lib.oracle_kv_append.argtypes = [P, P, i64, i64, P, i64]
            lib.oracle_kv_append.restype = ctypes.c_int
            lib.oracle_attention.argtypes = [i32, P, P, P, i32, i32, i32, i32, i32, i32, i32, f64,
                                             P, P, P, P, i64, P, P, i32]
            lib.oracle_attention.restype = ctypes.c_int
            lib.oracle_softmax_weights.argtypes = [i32, P, P, P, i32, i32, i32, i32, i32, i32, i32,
                                                   f64, P, P, P, i64, i32, P]
            lib.oracle_softmax_weights.restype = ctypes.c_int64
            lib.oracle_max_threads.restype = ctypes.c_int
            _lib = lib
    return _lib


def _ptr(a: Optional[np.ndarray]):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _c(a, dtype):
    return None if a is None else np.ascontiguousarray(a, dtype=dtype)


def max_threads() -> int:
    return int(_load().oracle_max_threads())


def kv_append(cache: np.ndarray, rows: np.ndarray, slot_mapping: np.ndarray) -> np.ndarray:
    """Return a copy of ``cache`` (bf16 bits, [num_blocks, bs, ...]) with row t
    of ``rows`` stored at slot ``slot_mapping[t]`` (skipped when negative)."""
    out = np.array(cache, dtype=np.uint16, copy=True, order="C")
    num_slots = out.shape[0] * out.shape[1]
    row_elems = int(np.prod(out.shape[2:]))
    rows = _c(rows, np.uint16)
    slots = _c(slot_mapping, np.int64)
    if rows.size != slots.shape[0] * row_elems:
        raise ValueError("rows do not match the cache's slot width")
    rc = _load().oracle_kv_append(_ptr(rows), _ptr(slots), slots.shape[0], row_elems,
                                  _ptr(out), num_slots)
    if rc != 0:
        raise ValueError("slot out of range")
    return out


def attention(query_len, context_len, block_table, q, k_cache, v_cache, *,
              num_q_heads: int, num_kv_heads: int, head_dim_qk: int, head_dim_v: int,
              block_size: int, latent: bool = False, scale: float = 0.0,
              tokens: Optional[np.ndarray] = None, threads: int = 0):
    """Attention output (float64 [rows, Hq, d_v]) and LSE (float64 [rows, Hq]).

    ``q``, ``k_cache``, ``v_cache`` are bf16 bit arrays (uint16); ``v_cache`` is
    ignored for the latent layout. ``tokens`` selects output rows (default all).
    ``scale <= 0`` means 1/sqrt(head_dim_qk).
    """
    ql = _c(query_len, np.int32)
    cl = _c(context_len, np.int32)
    bt = _c(block_table, np.int32)
    if bt.ndim != 2:
        raise ValueError("block_table must be 2-D")
    qa = _c(q, np.uint16)
    kc = _c(k_cache, np.uint16)
    vc = None if latent else _c(v_cache, np.uint16)
    T = int(ql.sum())
    tok = None if tokens is None else _c(tokens, np.int64)
    rows = T if tok is None else tok.shape[0]
    out = np.empty((rows, num_q_heads, head_dim_v), np.float64)
    lse = np.empty((rows, num_q_heads), np.float64)
    rc = _load().oracle_attention(ql.shape[0], _ptr(ql), _ptr(cl), _ptr(bt), bt.shape[1],
                                  num_q_heads, num_kv_heads, head_dim_qk, head_dim_v, block_size,
                                  int(bool(latent)), float(scale), _ptr(qa), _ptr(kc), _ptr(vc),
                                  _ptr(tok), 0 if tok is None else tok.shape[0],
                                  _ptr(out), _ptr(lse), int(threads))
    if rc != 0:
        raise ValueError("oracle_attention rejected its arguments")
    return out, lse


def softmax_weights(query_len, context_len, block_table, q, k_cache, v_cache, token: int,
                    head: int, *, num_q_heads: int, num_kv_heads: int, head_dim_qk: int,
                    head_dim_v: int, block_size: int, latent: bool = False,
                    scale: float = 0.0) -> np.ndarray:
    """Softmax weights exp(s_j - LSE) over the visible keys of one output row."""
    ql = _c(query_len, np.int32)
    cl = _c(context_len, np.int32)
    bt = _c(block_table, np.int32)
    qa = _c(q, np.uint16)
    kc = _c(k_cache, np.uint16)
    vc = None if latent else _c(v_cache, np.uint16)
    w = np.empty(int(cl.max()), np.float64)
    n = _load().oracle_softmax_weights(ql.shape[0], _ptr(ql), _ptr(cl), _ptr(bt), bt.shape[1],
                                       num_q_heads, num_kv_heads, head_dim_qk, head_dim_v,
                                       block_size, int(bool(latent)), float(scale), _ptr(qa),
                                       _ptr(kc), _ptr(vc), int(token), int(head), _ptr(w))
    if n < 0:
        raise ValueError("bad row")
    return w[:n]


def run_step(batch, tokens: Optional[np.ndarray] = None, threads: int = 0):
    """One whole step of a ``workloads.Batch``: append, then attention.

    Returns (out float64, lse float64, k_cache after append, v_cache after append).
    """
    sh = batch.shape
    kc = kv_append(batch.k_cache, batch.k_new, batch.slot_mapping)
    vc = None if sh.latent else kv_append(batch.v_cache, batch.v_new, batch.slot_mapping)
    out, lse = attention(batch.query_len, batch.context_len, batch.block_table, batch.q, kc, vc,
                         num_q_heads=sh.num_q_heads, num_kv_heads=sh.num_kv_heads,
                         head_dim_qk=sh.head_dim_qk, head_dim_v=sh.head_dim_v,
                         block_size=sh.block_size, latent=sh.latent, tokens=tokens,
                         threads=threads)
    return out, lse, kc, vc
