"""fp64 reference for MLA prefill without absorption: expansion of latent
cache rows into per-head keys and values.

TEST INFRASTRUCTURE, like the rest of ``oracle``: only ``tests/`` and the
bench's CPU legs may import it. It shares no code with the CUDA path.

DeepSeek-R1's attention (the paper's W8A8 deployment, Sec. 4.1) caches one
latent row per token: c (512 columns) and a rotary key r (64 columns) shared by
all heads. Decompressed, query head h attends with the key [c W_UK[h], r] and
the value c W_UV[h] (128 columns each); the query is [q_nope (128), q_rope (64)].
The paper prints none of this; the shapes are the model's.

The expanded keys and values are materialised in bf16 (the dtype the attention
then reads): each product is computed in fp64 and rounded once to bf16,
nearest with ties to even. The attention over them is the C oracle's
(``oracle.attention``) with d_qk = 192, d_v = 128 and one kv head per head.
"""
from __future__ import annotations

import numpy as np

C, R, DN = 512, 64, 128
DK = DN + R


def bf16_bits_to_f64(bits) -> np.ndarray:
    return (np.asarray(bits, np.uint16).astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def f64_to_bf16_bits(x) -> np.ndarray:
    """Round fp64 values to bf16 once (nearest, ties to even): the 8-bit
    significand of each value's binade, rounded by np.rint (half to even).
    Finite normal magnitudes only (no overflow or bf16 subnormals expected)."""
    x = np.asarray(x, np.float64)
    m, e = np.frexp(x)                       # x = m 2^e, |m| in [0.5, 1)
    q = np.ldexp(np.rint(np.ldexp(m, 8)), e - 8)
    return (q.astype(np.float32).view(np.uint32) >> 16).astype(np.uint16)


def latent_rows(latent_cache_bits, slots) -> np.ndarray:
    """fp64 latent rows [n, 576] at `slots` (a negative slot gives zeros)."""
    lat = np.asarray(latent_cache_bits, np.uint16).reshape(-1, C + R)
    s = np.asarray(slots, np.int64)
    rows = bf16_bits_to_f64(lat[np.maximum(s, 0)])
    rows[s < 0] = 0.0
    return rows


def expand_exact(latent_cache_bits, slots, w_uk_bits, w_uv_bits) -> tuple:
    """fp64 keys [n, H, 192] and values [n, H, 128], not rounded."""
    rows = latent_rows(latent_cache_bits, slots)
    c, r = rows[:, :C], rows[:, C:]
    wk = bf16_bits_to_f64(w_uk_bits)          # [H, 512, 128]
    wv = bf16_bits_to_f64(w_uv_bits)
    H = wk.shape[0]
    k = np.empty((rows.shape[0], H, DK))
    v = np.empty((rows.shape[0], H, DN))
    for h in range(H):
        k[:, h, :DN] = c @ wk[h]
        k[:, h, DN:] = r
        v[:, h, :] = c @ wv[h]
    return k, v


def expand(latent_cache_bits, slots, w_uk_bits, w_uv_bits) -> tuple:
    """bf16 bits of the expanded keys [n, H, 192] and values [n, H, 128]."""
    k, v = expand_exact(latent_cache_bits, slots, w_uk_bits, w_uv_bits)
    return f64_to_bf16_bits(k), f64_to_bf16_bits(v)
