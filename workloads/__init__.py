"""Seeded synthetic mixed prefill/decode batches over a paged KV cache.

This module only draws inputs. It holds none of the attention arithmetic, so
both the fp64 oracle (``oracle/``) and the CUDA path can be fed from it.

A batch is one serving step in which prefill chunks (phase 0) and decode
queries (phase 1) share the device and the KV pool (the co-location setting of
Sec. 3.4; prefill is compute-heavy, decode is bound by KV-cache reads, Sec. 1
and Sec. 3.3). The paper prints no attention shapes or lengths; the five named
workloads below stand in for its serving mixes (Sec. 4.1: DeepSeek-R1 1K/1K and
1K/4K, Qwen2.5-7B with 256/1024-token prompts) with the models' attention
shapes. No dataset item is used or reproduced.

Conventions (fixed by the C ABI in ``include/fnpu.h``):

* ``context_len`` counts this step's new tokens, so the queries of a sequence
  sit at absolute positions ``ctx - q .. ctx - 1``.
* Queries are packed sequence by sequence (varlen order).
* K/V cache: ``[num_blocks, block_size, Hkv, d]`` bf16, one array each; the
  latent (MLA) cache is one ``[num_blocks, block_size, d_qk]`` array whose first
  ``d_v`` columns are V.
* The prefix tokens (positions ``< ctx - q``) are already in the cache; the
  step's new tokens reach it through ``slot_mapping`` (KV append).
* Every slot that holds no token is filled with a bf16 NaN canary, and the
  unused block-table columns point at random in-range blocks, so a kernel that
  reads a key it must not see produces a wrong (non-finite) result instead of
  a silently right one.

Values are float32 N(0, 1) from ``numpy.random.default_rng(seed)`` (PCG64),
rounded to bf16 with round-to-nearest-even; both sides receive identical bf16
bits.
"""
from __future__ import annotations

import dataclasses
import math
from typing import Optional

import numpy as np

BF16_CANARY = np.uint16(0x7FC1)  # a quiet NaN with a distinct payload

CONFIG_NAMES = ("tiny", "qwen_decode", "qwen_prefill", "qwen_coloc", "mla_coloc", "mla_coloc_small", "mla_prefill")


@dataclasses.dataclass(frozen=True)
class Shape:
    num_q_heads: int
    num_kv_heads: int
    head_dim_qk: int
    head_dim_v: int
    block_size: int
    latent: bool  # MLA: one latent head, V = first head_dim_v columns of K

    @property
    def group(self) -> int:
        return self.num_q_heads // self.num_kv_heads


SHAPES = {
    # 4 q heads / 2 kv heads / d 64: a small GQA shape for exhaustive checks
    "tiny": Shape(4, 2, 64, 64, 16, False),
    # Qwen2.5-7B attention: 28 q heads, 4 kv heads (GQA 7:1), head_dim 128
    "qwen": Shape(28, 4, 128, 128, 16, False),
    # DeepSeek-R1 absorbed MLA: 128 q heads over one 576-wide latent (512 + 64 rope)
    "mla": Shape(128, 1, 576, 512, 64, True),
}


@dataclasses.dataclass
class Batch:
    name: str
    shape: Shape
    seed: int
    query_len: np.ndarray      # int32 [S]
    context_len: np.ndarray    # int32 [S]
    phase: np.ndarray          # uint8 [S], 0 = prefill, 1 = decode
    block_table: np.ndarray    # int32 [S, W]
    num_blocks: int
    q: np.ndarray              # uint16 (bf16 bits) [T, Hq, d_qk]
    k_new: np.ndarray          # uint16 [T, Hkv, d_qk]   (latent: [T, d_qk])
    v_new: Optional[np.ndarray]  # uint16 [T, Hkv, d_v] (latent: None)
    slot_mapping: np.ndarray   # int64 [T]
    k_cache: np.ndarray        # uint16 [num_blocks, bs, Hkv, d_qk] (latent: [num_blocks, bs, d_qk])
    v_cache: Optional[np.ndarray]  # uint16 [num_blocks, bs, Hkv, d_v] (latent: None)

    @property
    def num_seqs(self) -> int:
        return int(self.query_len.shape[0])

    @property
    def num_tokens(self) -> int:
        return int(self.query_len.sum())

    @property
    def query_start(self) -> np.ndarray:
        return np.concatenate([[0], np.cumsum(self.query_len)]).astype(np.int64)


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float32 to bf16 (round to nearest, ties to even); finite inputs."""
    u = np.array(x, dtype=np.float32, copy=True, order="C").view(np.uint32)
    lsb = u >> np.uint32(16)
    lsb &= np.uint32(1)
    lsb += np.uint32(0x7FFF)
    u += lsb
    u >>= np.uint32(16)
    return u.astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    return (np.asarray(b, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def _normal_bf16(rng: np.random.Generator, shape) -> np.ndarray:
    x = rng.standard_normal(size=shape, dtype=np.float32)
    u = x.view(np.uint32)
    lsb = u >> np.uint32(16)
    lsb &= np.uint32(1)
    lsb += np.uint32(0x7FFF)
    u += lsb
    u >>= np.uint32(16)
    return u.astype(np.uint16)


def draw_lengths(name: str, rng: np.random.Generator):
    """Per-sequence (query_len, context_len, phase) of a named workload."""
    if name == "tiny":
        # 2 prefill prompts of 128 tokens (no prefix) + 6 decodes, ctx ~ U[64, 512]
        dec = rng.integers(64, 512, endpoint=True, size=6)
        q = [128, 128] + [1] * 6
        ctx = [128, 128] + dec.tolist()
        ph = [0, 0] + [1] * 6
    elif name == "qwen_decode":
        # 64 decodes, ctx ~ U[512, 4096]
        ctx = rng.integers(512, 4096, endpoint=True, size=64).tolist()
        q = [1] * 64
        ph = [1] * 64
    elif name == "qwen_prefill":
        # one 2048-token prompt as four 512-token chunks on prefixes 0/512/1024/1536
        q = [512] * 4
        ctx = [512, 1024, 1536, 2048]
        ph = [0] * 4
    elif name == "qwen_coloc":
        # one 2048-token chunk on a prefix ~ U[0, 8192] + 128 decodes whose ctx is
        # log-normal, median 1024 (sigma 1), clipped to [128, 8192]
        prefix = int(rng.integers(0, 8192, endpoint=True))
        z = rng.standard_normal(128)
        dec = np.clip(np.rint(np.exp(math.log(1024.0) + z)), 128, 8192).astype(np.int64)
        q = [2048] + [1] * 128
        ctx = [prefix + 2048] + dec.tolist()
        ph = [0] + [1] * 128
    elif name == "mla_coloc":
        # one 1024-token prompt (no prefix) + 256 decodes, ctx ~ U[1024, 16384]
        dec = rng.integers(1024, 16384, endpoint=True, size=256)
        q = [1024] + [1] * 256
        ctx = [1024] + dec.tolist()
        ph = [0] + [1] * 256
    elif name == "mla_coloc_small":
        # the MLA co-located mix at about a quarter of the size (for profiler
        # captures, which replay a kernel many times): one 256-token prompt
        # (no prefix) + 48 decodes, ctx ~ U[4096, 16384]
        dec = rng.integers(4096, 16384, endpoint=True, size=48)
        q = [256] + [1] * 48
        ctx = [256] + dec.tolist()
        ph = [0] + [1] * 48
    elif name == "mla_prefill":
        # the prefill chunk of the MLA co-located mix alone: one 1024-token
        # prompt, no prefix (for the expanded, non-absorbed prefill path)
        q, ctx, ph = [1024], [1024], [0]
    else:
        raise ValueError(f"unknown workload {name!r}")
    return (np.asarray(q, np.int32), np.asarray(ctx, np.int32), np.asarray(ph, np.uint8))


def shape_of(name: str) -> Shape:
    if name == "tiny":
        return SHAPES["tiny"]
    if name.startswith("qwen"):
        return SHAPES["qwen"]
    if name.startswith("mla"):
        return SHAPES["mla"]
    raise ValueError(f"unknown workload {name!r}")


def build_batch(shape: Shape, query_len, context_len, phase, rng: np.random.Generator,
                name: str = "custom", seed: int = -1, num_blocks: Optional[int] = None,
                pool_slack: float = 1.25, extra_bt_cols: int = 1,
                shuffle_pool: bool = True) -> Batch:
    """Lay a batch out in a shuffled paged pool and draw its values.

    Draw order: block permutation, padding block ids, q, new K, new V, prefix K,
    prefix V.
    """
    query_len = np.asarray(query_len, np.int32)
    context_len = np.asarray(context_len, np.int32)
    phase = np.asarray(phase, np.uint8)
    if np.any(context_len < query_len) or np.any(query_len < 1):
        raise ValueError("need 1 <= query_len <= context_len")
    bs = shape.block_size
    nblk = (context_len.astype(np.int64) + bs - 1) // bs
    need = int(nblk.sum())
    if num_blocks is None:
        num_blocks = int(math.ceil(pool_slack * need))
    if num_blocks < need:
        raise ValueError("pool too small")
    perm = rng.permutation(num_blocks) if shuffle_pool else np.arange(num_blocks)
    width = int(nblk.max()) + extra_bt_cols
    S = len(query_len)
    bt = rng.integers(0, num_blocks, size=(S, width)).astype(np.int32)  # padding: in-range junk
    off = 0
    for s in range(S):
        n = int(nblk[s])
        bt[s, :n] = perm[off:off + n]
        off += n

    T = int(query_len.sum())
    H, Hk, dq, dv = shape.num_q_heads, shape.num_kv_heads, shape.head_dim_qk, shape.head_dim_v
    q = _normal_bf16(rng, (T, H, dq))
    if shape.latent:
        k_new = _normal_bf16(rng, (T, dq))
        v_new = None
    else:
        k_new = _normal_bf16(rng, (T, Hk, dq))
        v_new = _normal_bf16(rng, (T, Hk, dv))

    # slots: prefix positions (already cached) and the new tokens' positions
    pre_slots, new_slots = [], []
    for s in range(S):
        p = int(context_len[s] - query_len[s])
        pos = np.arange(int(context_len[s]), dtype=np.int64)
        slots = bt[s, pos // bs].astype(np.int64) * bs + pos % bs
        pre_slots.append(slots[:p])
        new_slots.append(slots[p:])
    pre_slots = np.concatenate(pre_slots) if S else np.zeros(0, np.int64)
    slot_mapping = np.concatenate(new_slots).astype(np.int64) if S else np.zeros(0, np.int64)

    nslot = num_blocks * bs
    if shape.latent:
        k_cache = np.full((nslot, dq), BF16_CANARY, np.uint16)
        k_cache[pre_slots] = _normal_bf16(rng, (len(pre_slots), dq))
        k_cache = k_cache.reshape(num_blocks, bs, dq)
        v_cache = None
    else:
        k_cache = np.full((nslot, Hk, dq), BF16_CANARY, np.uint16)
        v_cache = np.full((nslot, Hk, dv), BF16_CANARY, np.uint16)
        k_cache[pre_slots] = _normal_bf16(rng, (len(pre_slots), Hk, dq))
        v_cache[pre_slots] = _normal_bf16(rng, (len(pre_slots), Hk, dv))
        k_cache = k_cache.reshape(num_blocks, bs, Hk, dq)
        v_cache = v_cache.reshape(num_blocks, bs, Hk, dv)

    return Batch(name=name, shape=shape, seed=seed, query_len=query_len,
                 context_len=context_len, phase=phase, block_table=bt,
                 num_blocks=num_blocks, q=q, k_new=k_new, v_new=v_new,
                 slot_mapping=slot_mapping, k_cache=k_cache, v_cache=v_cache)


def make_batch(name: str, seed: int = 0) -> Batch:
    """One of the five named workloads, drawn from ``default_rng(seed)``."""
    rng = np.random.default_rng(seed)
    q, ctx, ph = draw_lengths(name, rng)
    shape = shape_of(name)
    nb = 256 if name == "tiny" else None
    return build_batch(shape, q, ctx, ph, rng, name=name, seed=seed, num_blocks=nb)


def prefix_slots(batch: Batch) -> np.ndarray:
    """Slots of every sequence's prefix positions (< ctx - q), sequence by
    sequence: the rows that are in the cache before the step."""
    bs = batch.shape.block_size
    out = []
    for s in range(batch.num_seqs):
        pos = np.arange(int(batch.context_len[s] - batch.query_len[s]), dtype=np.int64)
        out.append(batch.block_table[s, pos // bs].astype(np.int64) * bs + pos % bs)
    return np.concatenate(out) if out else np.zeros(0, np.int64)


def prefix_rows(batch: Batch) -> tuple:
    """(k_rows, v_rows, slots): the bf16 bits of the prefix rows of the pool,
    for filling a cache of another storage format through its own append."""
    sl = prefix_slots(batch)
    sh = batch.shape
    k = batch.k_cache.reshape(-1, sh.num_kv_heads, sh.head_dim_qk)[sl]
    v = batch.v_cache.reshape(-1, sh.num_kv_heads, sh.head_dim_v)[sl]
    return np.ascontiguousarray(k), np.ascontiguousarray(v), sl


def stale_pool_bytes(nbytes: int, seed: int) -> tuple:
    """Seeded random bytes for the K and V pools of a byte-format cache before
    any append: every byte value occurs, NaN codes and NaN scales included, so a
    kernel that reads a slot it must not see goes wrong visibly."""
    rng = np.random.default_rng([seed, 0xF8])
    return (rng.integers(0, 256, nbytes, dtype=np.uint8), rng.integers(0, 256, nbytes, dtype=np.uint8))


def mla_expand_inputs(batch: Batch, seed: int = 0) -> dict:
    """Inputs of MLA prefill without absorption on a latent batch: the per-head
    up-projections W_UK, W_UV (bf16 [Hq, 512, 128], N(0, 1/512) so that the
    expanded keys and values are about N(0, 1)) and the decompressed queries
    [T, Hq, 192] (N(0, 1)), all seeded."""
    sh = batch.shape
    if not sh.latent:
        raise ValueError("a latent batch is needed")
    rng = np.random.default_rng([seed, 0x3A])
    H = sh.num_q_heads
    w_uk = f32_to_bf16_bits((rng.standard_normal((H, 512, 128)) / math.sqrt(512)).astype(np.float32))
    w_uv = f32_to_bf16_bits((rng.standard_normal((H, 512, 128)) / math.sqrt(512)).astype(np.float32))
    q = _normal_bf16(rng, (batch.num_tokens, H, 192))
    return {"w_uk": w_uk, "w_uv": w_uv, "q": q}


def expanded_layout(batch: Batch, block_size: int = 16) -> tuple:
    """Rows of the expanded cache of a latent batch: every sequence's positions
    0..ctx-1 in order, each sequence starting on a block boundary (padding rows
    have slot -1). Returns (slots int64 [n], block_table int32 [S, width],
    num_blocks): block_table[s][j] is the expanded block of position 16 j."""
    bs_l = batch.shape.block_size
    S = batch.num_seqs
    nblk = [(int(c) + block_size - 1) // block_size for c in batch.context_len]
    width = max(nblk) if nblk else 1
    bt = np.zeros((S, width), np.int32)
    slots = []
    first = 0
    for s in range(S):
        c = int(batch.context_len[s])
        pos = np.arange(c, dtype=np.int64)
        sl = batch.block_table[s, pos // bs_l].astype(np.int64) * bs_l + pos % bs_l
        pad = nblk[s] * block_size - c
        slots.append(np.concatenate([sl, np.full(pad, -1, np.int64)]))
        bt[s, :nblk[s]] = np.arange(first, first + nblk[s])
        first += nblk[s]
    return (np.concatenate(slots) if slots else np.zeros(0, np.int64)), bt, max(first, 1)


def pairs(batch: Batch) -> int:
    """Visible (query, key) pairs: sum over seqs of q*p + q(q+1)/2."""
    q = batch.query_len.astype(np.int64)
    p = batch.context_len.astype(np.int64) - q
    return int((q * p + q * (q + 1) // 2).sum())


def prefill_path_flops(batch: Batch) -> int:
    """FLOPs of the rows that take the prefill path (sequences with more than
    one query token: chunks and multi-token decodes): 2*Hq*pairs*(d_qk + d_v)
    over those sequences only."""
    sh = batch.shape
    q = batch.query_len.astype(np.int64)
    p = batch.context_len.astype(np.int64) - q
    sel = q > 1
    pr = int((q[sel] * p[sel] + q[sel] * (q[sel] + 1) // 2).sum())
    return int(2 * sh.num_q_heads * pr * (sh.head_dim_qk + sh.head_dim_v))


def algorithmic_work(batch: Batch, kv_fp8: bool = False) -> dict:
    """Algorithmic FLOPs and HBM bytes of one step (append + attention).

    With kv_fp8 the cache rows are one-byte codes plus one fp32 scale per
    (slot, kv head) row of K and of V; the append reads bf16 rows and writes
    that format.

    FLOPs count QK^T and PV over visible pairs only: 2*Hq*pairs*(d_qk + d_v).
    Bytes count each cache row of every sequence read once, Q read, O (bf16)
    and LSE (fp32) written, the append (new rows read and written), 8 B per
    slot_mapping entry and 4 B per used block-table entry. Split-KV scratch
    traffic is not algorithmic and is not counted.
    """
    sh = batch.shape
    T = batch.num_tokens
    ctx = batch.context_len.astype(np.int64)
    flops = 2 * sh.num_q_heads * pairs(batch) * (sh.head_dim_qk + sh.head_dim_v)
    row_bytes = 2 * (sh.head_dim_qk if sh.latent else sh.num_kv_heads * (sh.head_dim_qk + sh.head_dim_v))
    cache_row = row_bytes
    if kv_fp8:
        cache_row = sh.num_kv_heads * (sh.head_dim_qk + 4 + sh.head_dim_v + 4)
    kv_read = int(ctx.sum()) * cache_row
    q_read = T * sh.num_q_heads * sh.head_dim_qk * 2
    o_write = T * sh.num_q_heads * sh.head_dim_v * 2
    lse_write = T * sh.num_q_heads * 4
    append = T * (row_bytes + cache_row)
    meta = 8 * T + 4 * int(((ctx + sh.block_size - 1) // sh.block_size).sum())
    return {
        "flops": int(flops),
        "bytes": int(kv_read + q_read + o_write + lse_write + append + meta),
        "kv_read_bytes": int(kv_read),
        "append_bytes": int(append),
        "pairs": pairs(batch),
    }
