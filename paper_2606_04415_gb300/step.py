"""Convenience driver for one mixed step held in device memory.

``DeviceStep`` takes a batch description (any object with the attributes of
``workloads.Batch``: shape, lengths, phase, block table, q / new K/V bits,
slot mapping and the cache pool), uploads it once as CUDA tensors, builds the
plan, and runs KV append + attention through the C ABI. Torch provides the
device memory and the stream; all compute is in the library's kernels.
"""
from __future__ import annotations

from typing import Optional

import numpy as np

from . import (PlanOpts, kv_append, make_desc, mixed_attn_plan, mixed_attn_run)


def _to_dev(a: Optional[np.ndarray], torch, dtype, device):
    if a is None:
        return None
    t = torch.from_numpy(np.ascontiguousarray(a))
    if dtype is not None:
        t = t.view(dtype)
    return t.to(device)


class DeviceStep:
    def __init__(self, batch, opts: Optional[PlanOpts] = None, device: str = "cuda",
                 softmax_scale: float = 0.0):
        import torch
        self.torch = torch
        self.batch = batch
        sh = batch.shape
        self.desc = make_desc(sh.num_q_heads, sh.num_kv_heads, sh.head_dim_qk, sh.head_dim_v,
                              sh.block_size, batch.num_blocks, sh.latent, softmax_scale)
        bf = torch.bfloat16
        self.q = _to_dev(batch.q, torch, bf, device)
        self.k_new = _to_dev(batch.k_new, torch, bf, device)
        self.v_new = _to_dev(batch.v_new, torch, bf, device)
        self.slot_mapping = _to_dev(batch.slot_mapping, torch, None, device)
        self.k_cache = _to_dev(batch.k_cache, torch, bf, device)
        self.v_cache = _to_dev(batch.v_cache, torch, bf, device)
        T = batch.num_tokens
        self.out = torch.empty((T, sh.num_q_heads, sh.head_dim_v), dtype=bf, device=device)
        self.lse = torch.empty((T, sh.num_q_heads), dtype=torch.float32, device=device)
        self.plan = mixed_attn_plan(self.desc, batch.query_len, batch.context_len, batch.phase,
                                    batch.block_table, opts=opts)

    def replan(self, opts: Optional[PlanOpts] = None):
        """Plan the same batch again with other options (for instance the
        decode share a dispatch controller chose for the next step)."""
        self.plan.destroy()
        b = self.batch
        self.plan = mixed_attn_plan(self.desc, b.query_len, b.context_len, b.phase, b.block_table, opts=opts)

    def append(self, stream=None):
        kv_append(self.desc, self.k_new, self.v_new, self.slot_mapping, self.k_cache, self.v_cache,
                  stream=stream)

    def attend(self, stream=None):
        mixed_attn_run(self.plan, self.q, self.k_cache, self.v_cache, self.out, self.lse,
                       stream=stream)

    def run(self, stream=None):
        """One step: append the new tokens, then attention."""
        self.append(stream)
        self.attend(stream)

    def results(self):
        """(out float32 numpy, lse float32 numpy) after synchronising."""
        self.torch.cuda.synchronize()
        return (self.out.float().cpu().numpy(), self.lse.cpu().numpy())

    def cache_bits(self):
        t = self.torch
        kc = self.k_cache.view(t.int16).cpu().numpy().view(np.uint16)
        vc = None if self.v_cache is None else self.v_cache.view(t.int16).cpu().numpy().view(np.uint16)
        return kc, vc
