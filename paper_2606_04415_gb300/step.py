"""Convenience driver for one mixed step held in device memory.

``DeviceStep`` takes a batch description (any object with the attributes of
``workloads.Batch``: shape, lengths, phase, block table, q / new K/V bits,
slot mapping and the cache pool), uploads it once as CUDA tensors, builds the
plan, and runs KV append + attention through the C ABI. Torch provides the
device memory and the stream; all compute is in the library's kernels.

With ``kv_fp8=True`` the pools hold the library's FP8 (e4m3) cache format
(byte arrays of ``FP8_BLOCK_BYTES`` per block): they start from the given
bytes (zeros by default) and the batch's prefix rows enter them through the
library's quantising append, before the step's own append.
"""
from __future__ import annotations

from typing import Optional

import numpy as np

from . import (FP8_BLOCK_BYTES, PlanOpts, kv_append, make_desc, mixed_attn_plan, mixed_attn_replan,
               mixed_attn_run, mixed_step)


def _to_dev(a: Optional[np.ndarray], torch, dtype, device):
    if a is None:
        return None
    t = torch.from_numpy(np.ascontiguousarray(a))
    if dtype is not None:
        t = t.view(dtype)
    return t.to(device)


class DeviceStep:
    def __init__(self, batch, opts: Optional[PlanOpts] = None, device: str = "cuda",
                 softmax_scale: float = 0.0, kv_fp8: bool = False, pool_init=None):
        import torch
        self.torch = torch
        self.batch = batch
        self.kv_fp8 = bool(kv_fp8)
        sh = batch.shape
        self.desc = make_desc(sh.num_q_heads, sh.num_kv_heads, sh.head_dim_qk, sh.head_dim_v,
                              sh.block_size, batch.num_blocks, sh.latent, softmax_scale, kv_fp8)
        bf = torch.bfloat16
        self.q = _to_dev(batch.q, torch, bf, device)
        self.k_new = _to_dev(batch.k_new, torch, bf, device)
        self.v_new = _to_dev(batch.v_new, torch, bf, device)
        self.slot_mapping = _to_dev(batch.slot_mapping, torch, None, device)
        if self.kv_fp8:
            nbytes = batch.num_blocks * FP8_BLOCK_BYTES
            if pool_init is None:
                pool_init = (np.zeros(nbytes, np.uint8), np.zeros(nbytes, np.uint8))
            if pool_init[0].size != nbytes or pool_init[1].size != nbytes:
                raise ValueError("FP8 pools need num_blocks * FP8_BLOCK_BYTES bytes each")
            self.k_cache = _to_dev(pool_init[0], torch, None, device)
            self.v_cache = _to_dev(pool_init[1], torch, None, device)
            self._fill_prefix(device)
        else:
            self.k_cache = _to_dev(batch.k_cache, torch, bf, device)
            self.v_cache = _to_dev(batch.v_cache, torch, bf, device)
        T = batch.num_tokens
        self.out = torch.empty((T, sh.num_q_heads, sh.head_dim_v), dtype=bf, device=device)
        self.lse = torch.empty((T, sh.num_q_heads), dtype=torch.float32, device=device)
        self.plan = mixed_attn_plan(self.desc, batch.query_len, batch.context_len, batch.phase,
                                    batch.block_table, opts=opts)

    def _fill_prefix(self, device):
        """Store the batch's prefix rows (its bf16 pool at the prefix slots)
        through the library's append."""
        b, sh, torch = self.batch, self.batch.shape, self.torch
        bs = sh.block_size
        sl = []
        for s in range(len(b.query_len)):
            pos = np.arange(int(b.context_len[s] - b.query_len[s]), dtype=np.int64)
            sl.append(b.block_table[s, pos // bs].astype(np.int64) * bs + pos % bs)
        sl = np.concatenate(sl) if sl else np.zeros(0, np.int64)
        if sl.size == 0:
            return
        k = b.k_cache.reshape(-1, sh.num_kv_heads, sh.head_dim_qk)[sl]
        v = b.v_cache.reshape(-1, sh.num_kv_heads, sh.head_dim_v)[sl]
        kv_append(self.desc, _to_dev(k, torch, torch.bfloat16, device), _to_dev(v, torch, torch.bfloat16, device),
                  _to_dev(sl, torch, None, device), self.k_cache, self.v_cache)

    def replan(self, opts: Optional[PlanOpts] = None, stream=None):
        """Plan the same batch again with other options (for instance the
        decode share a dispatch controller chose for the next step), reusing
        the plan's resources (``fnpu_mixed_attn_replan``)."""
        b = self.batch
        mixed_attn_replan(self.plan, b.query_len, b.context_len, b.phase, b.block_table, opts=opts, stream=stream)

    def append(self, stream=None):
        kv_append(self.desc, self.k_new, self.v_new, self.slot_mapping, self.k_cache, self.v_cache,
                  stream=stream)

    def attend(self, stream=None):
        mixed_attn_run(self.plan, self.q, self.k_cache, self.v_cache, self.out, self.lse,
                       stream=stream)

    def run(self, stream=None):
        """One step: the append of the new tokens and the attention, in one
        call (``fnpu_mixed_step``; the same results as ``append`` then
        ``attend``)."""
        mixed_step(self.plan, self.k_new, self.v_new, self.slot_mapping, self.q, self.k_cache, self.v_cache,
                   self.out, self.lse, stream=stream)

    def results(self):
        """(out float32 numpy, lse float32 numpy) after synchronising."""
        self.torch.cuda.synchronize()
        return (self.out.float().cpu().numpy(), self.lse.cpu().numpy())

    def cache_bits(self):
        t = self.torch
        if self.kv_fp8:  # byte pools
            return self.k_cache.cpu().numpy(), self.v_cache.cpu().numpy()
        kc = self.k_cache.view(t.int16).cpu().numpy().view(np.uint16)
        vc = None if self.v_cache is None else self.v_cache.view(t.int16).cpu().numpy().view(np.uint16)
        return kc, vc


class ExpandedMlaPrefill:
    """MLA prefill without absorption, on device: the chunk's new latent rows
    are appended (``fnpu_kv_append``), the latent rows of every sequence's
    context are expanded (``fnpu_mla_expand``) into a paged cache of
    per-head keys [n, Hq, 192] and values [n, Hq, 128] (each sequence from a
    block boundary, blocks of 16), and the chunk runs as multi-head attention
    over it through the ordinary plan / run.

    ``batch``: a latent batch (its latent cache, block table and lengths; all
    sequences are prefill chunks). ``slots``, ``block_table`` and
    ``num_blocks`` give the expanded layout (host arrays, see
    ``workloads.expanded_layout``); ``w_uk``, ``w_uv``, ``q`` are bf16 bits.
    """

    def __init__(self, batch, w_uk, w_uv, q, slots, block_table, num_blocks, device: str = "cuda",
                 opts: Optional[PlanOpts] = None):
        import torch
        from . import mla_expand
        self.torch = torch
        self._expand = mla_expand
        sh = batch.shape
        H = sh.num_q_heads
        bf = torch.bfloat16
        self.latent_desc = make_desc(H, 1, sh.head_dim_qk, sh.head_dim_v, sh.block_size, batch.num_blocks, True)
        self.desc = make_desc(H, H, 192, 128, 16, int(num_blocks))
        self.latent = _to_dev(batch.k_cache, torch, bf, device)
        self.k_new = _to_dev(batch.k_new, torch, bf, device)
        self.slot_mapping = _to_dev(batch.slot_mapping, torch, None, device)
        self.w_uk = _to_dev(w_uk, torch, bf, device)
        self.w_uv = _to_dev(w_uv, torch, bf, device)
        self.q = _to_dev(q, torch, bf, device)
        self.slots = _to_dev(np.asarray(slots, np.int64), torch, None, device)
        n = int(len(slots))
        self.n = n
        self.workspace = torch.empty((max(n, 1), 512), dtype=bf, device=device)
        self.k = torch.empty((int(num_blocks) * 16, H, 192), dtype=bf, device=device)
        self.v = torch.empty((int(num_blocks) * 16, H, 128), dtype=bf, device=device)
        T = batch.num_tokens
        self.out = torch.empty((T, H, 128), dtype=bf, device=device)
        self.lse = torch.empty((T, H), dtype=torch.float32, device=device)
        self.plan = mixed_attn_plan(self.desc, batch.query_len, batch.context_len, np.zeros(batch.num_seqs, np.uint8),
                                    block_table, opts=opts)

    def append(self, stream=None):
        kv_append(self.latent_desc, self.k_new, None, self.slot_mapping, self.latent, None, stream=stream)

    def expand(self, stream=None):
        self._expand(self.latent_desc, self.latent, self.slots, self.w_uk, self.w_uv, self.workspace, self.k, self.v,
                     stream=stream, num_rows=self.n)

    def attend(self, stream=None):
        mixed_attn_run(self.plan, self.q, self.k, self.v, self.out, self.lse, stream=stream)

    def run(self, stream=None):
        """One step: append the chunk's latent rows, expand, attention."""
        self.append(stream)
        self.expand(stream)
        self.attend(stream)

    def results(self):
        self.torch.cuda.synchronize()
        return (self.out.float().cpu().numpy(), self.lse.cpu().numpy())

    def expanded_bits(self):
        t = self.torch
        t.cuda.synchronize()
        return (self.k[:self.n].view(t.int16).cpu().numpy().view(np.uint16),
                self.v[:self.n].view(t.int16).cpu().numpy().view(np.uint16))
