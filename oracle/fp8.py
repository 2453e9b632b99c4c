"""fp64 reference for the FP8 (e4m3) KV-cache format of the decode path.

TEST INFRASTRUCTURE, like the rest of ``oracle``: only ``tests/`` may import
it. It shares no code with the CUDA path.

The paper's DeepSeek-R1 deployment quantises weights and activations to
8 bits (Sec. 4.1); it prints no KV-cache format. The format here is this
library's:

* Quantisation, per stored row (one slot, one kv head, d values): amax =
  max |x| over the row (the bf16 inputs, exact in fp32); scale = amax / 448
  in fp32 (1 when amax is 0); code = e4m3(x / scale), the fp32 quotient
  rounded to the nearest e4m3 value, ties to the even code, magnitudes above
  448 saturating to 448. e4m3 (OCP FP8): 1 sign bit, 4 exponent bits (bias 7),
  3 mantissa bits; exponent field 0 holds the subnormals m/8 * 2^-6; field 15
  with mantissa 7 is NaN, so 448 = 1.75 * 2^8 is the largest finite value.
  The dequantised value of a code is value(code) * scale.
* Layout of a pool of `num_blocks` blocks of bs = 16 slots, Hkv kv heads and
  d = 128 (all little endian):

    K block: codes [bs][Hkv][128], column j of a row at byte position
             kpos(j) (below), then fp32 scales [bs][Hkv]
    V block: codes [Hkv][128][bs] (transposed), slot s of a column at byte
             position vpos(s), then fp32 scales [bs][Hkv]

  kpos(16 k + j) = 32 c + 4 k + r and vpos(j) = 4 c + r for j in 0..15, with
  c = (j mod 8) // 2 and r = (j mod 2) + 2 (j // 8): the four values a lane
  of a 16x8x16 matrix product multiplies together (j = 2c, 2c+1, 2c+8, 2c+9)
  sit in four consecutive bytes.
"""
from __future__ import annotations

import numpy as np

E4M3_MAX = 448.0
BS = 16
D = 128


def e4m3_value(code: int) -> float:
    """Value of an e4m3 code (0..255) from the format definition."""
    s = -1.0 if code & 0x80 else 1.0
    e = (code >> 3) & 0xF
    m = code & 0x7
    if e == 0xF and m == 0x7:
        return float("nan")
    if e == 0:
        return s * (m / 8.0) * 2.0 ** -6
    return s * (1.0 + m / 8.0) * 2.0 ** (e - 7)


# the 127 non-negative finite values, ascending (codes 0..126)
_POS = np.array([e4m3_value(c) for c in range(127)], np.float64)


def e4m3_round(x) -> np.ndarray:
    """Codes of float32 values: nearest e4m3 value, ties to the even code,
    magnitudes above 448 saturating to 448 (NaN inputs are not expected).

    Per binade: a magnitude a in [2^E, 2^(E+1)) (E >= -6; every a below 2^-6,
    the subnormals, counts as E = -6) sits on the grid of spacing 2^(E-3)
    there, so m = a / 2^(E-3) (exact: a power-of-two scaling) rounded half to
    even is the nearest grid point; it is 8(E+6) + m as a code (code parity =
    mantissa parity = parity of m, so ties go to the even code, and m = 16
    carries into the next binade's first code). Equal to the table search
    ``e4m3_round_by_search`` (a test checks both)."""
    x = np.asarray(x, np.float32)
    shape = x.shape
    x = x.reshape(-1)
    a = np.minimum(np.abs(x), np.float32(E4M3_MAX))  # every step below is exact in fp32
    _, e = np.frexp(a)                               # a = f 2^e, f in [0.5, 1); frexp(0) = (0, 0)
    E = np.maximum(e - 1, -6)
    E[a < 2.0 ** -6] = -6                            # the subnormals and zero
    m = np.rint(np.ldexp(a, 3 - E))                  # rint: half to even
    code = (8 * (E + 6) + m.astype(np.int32)).astype(np.uint8)
    code[np.signbit(x) & (code != 0)] |= np.uint8(0x80)
    return code.reshape(shape)


def e4m3_round_by_search(x) -> np.ndarray:
    """The same rounding by search in the table of the 127 finite values."""
    a = np.abs(np.asarray(x, np.float32).astype(np.float64))
    neg = np.signbit(np.asarray(x, np.float32))
    a = np.minimum(a, E4M3_MAX)
    hi = np.searchsorted(_POS, a, side="left")        # first value >= a
    hi = np.minimum(hi, 126)
    lo = np.maximum(hi - 1, 0)
    d_hi = _POS[hi] - a
    d_lo = a - _POS[lo]
    pick_hi = (d_hi < d_lo) | ((d_hi == d_lo) & (hi % 2 == 0))
    code = np.where(_POS[hi] == a, hi, np.where(pick_hi, hi, lo)).astype(np.uint8)
    return np.where(neg & (code != 0), code | np.uint8(0x80), code).astype(np.uint8)


def e4m3_decode(codes) -> np.ndarray:
    c = np.asarray(codes, np.uint8)
    return np.array([e4m3_value(int(v)) for v in range(256)], np.float64)[c]


def bf16_bits_to_f32(bits) -> np.ndarray:
    return (np.asarray(bits, np.uint16).astype(np.uint32) << 16).view(np.float32)


def quantize_rows(rows_bf16) -> tuple:
    """Codes (uint8 [..., d]) and scales (float32 [...]) of rows of bf16 bits."""
    x = bf16_bits_to_f32(rows_bf16)
    amax = np.max(np.abs(x), axis=-1)
    scale = np.where(amax > 0, amax / np.float32(E4M3_MAX), np.float32(1.0)).astype(np.float32)
    q = (x / scale[..., None]).astype(np.float32)
    return e4m3_round(q), scale


def _cr(j):
    j = np.asarray(j)
    return (j % 8) // 2, (j % 2) + 2 * (j // 8)


def kpos(col):
    """Byte position of K column `col` (0..127) inside a stored row."""
    col = np.asarray(col)
    k, j = col // 16, col % 16
    c, r = _cr(j)
    return 32 * c + 4 * k + r


def vpos(slot):
    """Byte position of slot `slot` (0..15) inside a stored V column."""
    c, r = _cr(np.asarray(slot))
    return 4 * c + r


def block_bytes(hkv: int) -> int:
    return BS * hkv * D + BS * hkv * 4


def pack_pools(k_codes, k_scales, v_codes, v_scales) -> tuple:
    """Byte pools (uint8 [num_blocks * block_bytes]) from logical codes
    [num_blocks, bs, Hkv, d] and scales [num_blocks, bs, Hkv]."""
    nb, bs, hkv, d = k_codes.shape
    assert bs == BS and d == D
    cols, slots = np.arange(D), np.arange(BS)
    kb = np.zeros((nb, bs, hkv, d), np.uint8)
    kb[..., kpos(cols)] = k_codes
    vb = np.zeros((nb, hkv, d, bs), np.uint8)
    vb[..., vpos(slots)] = np.transpose(v_codes, (0, 2, 3, 1))
    k_pool = np.concatenate([kb.reshape(nb, -1), np.ascontiguousarray(k_scales, np.float32).view(np.uint8).reshape(nb, -1)], 1)
    v_pool = np.concatenate([vb.reshape(nb, -1), np.ascontiguousarray(v_scales, np.float32).view(np.uint8).reshape(nb, -1)], 1)
    return k_pool.reshape(-1), v_pool.reshape(-1)


def unpack_pools(k_pool, v_pool, hkv: int) -> tuple:
    """Inverse of pack_pools: logical (k_codes, k_scales, v_codes, v_scales)."""
    bb = block_bytes(hkv)
    nb = np.asarray(k_pool).size // bb
    kp = np.asarray(k_pool, np.uint8).reshape(nb, bb)
    vp = np.asarray(v_pool, np.uint8).reshape(nb, bb)
    ncode = BS * hkv * D
    cols, slots = np.arange(D), np.arange(BS)
    kb = kp[:, :ncode].reshape(nb, BS, hkv, D)
    k_codes = kb[..., kpos(cols)]
    vb = vp[:, :ncode].reshape(nb, hkv, D, BS)
    v_codes = np.transpose(vb[..., vpos(slots)], (0, 3, 1, 2))
    k_scales = np.ascontiguousarray(kp[:, ncode:]).view(np.float32).reshape(nb, BS, hkv)
    v_scales = np.ascontiguousarray(vp[:, ncode:]).view(np.float32).reshape(nb, BS, hkv)
    return k_codes, k_scales, v_codes, v_scales


def kv_append(k_pool, v_pool, k_new, v_new, slot_mapping, hkv: int) -> tuple:
    """The fp8 KV append: quantise each new (token, kv head) row and store it
    (codes and scale) at its slot; negative slots are skipped."""
    k_codes, k_scales, v_codes, v_scales = unpack_pools(k_pool, v_pool, hkv)
    kc, ks = quantize_rows(k_new)
    vc, vs = quantize_rows(v_new)
    for t, s in enumerate(np.asarray(slot_mapping, np.int64)):
        if s < 0:
            continue
        b, o = divmod(int(s), BS)
        k_codes[b, o], k_scales[b, o] = kc[t], ks[t]
        v_codes[b, o], v_scales[b, o] = vc[t], vs[t]
    return pack_pools(k_codes, k_scales, v_codes, v_scales)


def decode_attention(context_len, block_table, q_bf16, k_pool, v_pool, *, num_q_heads: int, num_kv_heads: int,
                     scale: float = 0.0) -> tuple:
    """Output (float64 [S, Hq, d]) and LSE (float64 [S, Hq]) of one-token
    decodes (token s = sequence s at position ctx_s - 1) over the dequantised
    cache: softmax(q k^T * scale) v with k, v = code value * row scale."""
    k_codes, k_scales, v_codes, v_scales = unpack_pools(k_pool, v_pool, num_kv_heads)
    g = num_q_heads // num_kv_heads
    sc = scale if scale > 0 else 1.0 / np.sqrt(D)
    qf = bf16_bits_to_f32(q_bf16).astype(np.float64).reshape(-1, num_q_heads, D)
    S = len(context_len)
    out = np.zeros((S, num_q_heads, D))
    lse = np.zeros((S, num_q_heads))
    for s in range(S):
        c = int(context_len[s])
        idx = np.arange(c)
        blk = np.asarray(block_table)[s, idx // BS]
        # the sequence's keys and values, dequantised: [c, Hkv, d]
        keys = e4m3_decode(k_codes[blk, idx % BS]) * k_scales[blk, idx % BS][..., None].astype(np.float64)
        vals = e4m3_decode(v_codes[blk, idx % BS]) * v_scales[blk, idx % BS][..., None].astype(np.float64)
        for h in range(num_q_heads):
            kvh = h // g
            x = keys[:, kvh, :] @ qf[s, h] * sc
            m = x.max()
            w = np.exp(x - m)
            l = w.sum()
            out[s, h] = (w[:, None] * vals[:, kvh, :]).sum(0) / l
            lse[s, h] = m + np.log(l)
    return out, lse


def attention(query_len, context_len, block_table, q_bf16, k_pool, v_pool, *, num_q_heads: int, num_kv_heads: int,
              scale: float = 0.0, tokens=None) -> tuple:
    """Output (float64 [rows, Hq, d]) and LSE (float64 [rows, Hq]) of a mixed
    step over the dequantised cache: sequence s's query i sits at position
    ctx_s - q_s + i and attends causally to keys 0..pos (keys of sequence s
    at block_table[s][j / 16], offset j % 16); softmax(q k^T * scale) v with
    k, v = code value * row scale. Queries are packed sequence by sequence;
    `tokens` selects output rows (default all)."""
    k_codes, k_scales, v_codes, v_scales = unpack_pools(k_pool, v_pool, num_kv_heads)
    g = num_q_heads // num_kv_heads
    sc = scale if scale > 0 else 1.0 / np.sqrt(D)
    qf = bf16_bits_to_f32(q_bf16).astype(np.float64).reshape(-1, num_q_heads, D)
    ql = np.asarray(query_len, np.int64)
    cl = np.asarray(context_len, np.int64)
    starts = np.concatenate([[0], np.cumsum(ql)])
    T = int(starts[-1])
    rows = np.arange(T) if tokens is None else np.asarray(tokens, np.int64)
    out = np.zeros((rows.size, num_q_heads, D))
    lse = np.zeros((rows.size, num_q_heads))
    seq_of = np.searchsorted(starts, rows, side="right") - 1
    for s in np.unique(seq_of):
        c = int(cl[s])
        idx = np.arange(c)
        blk = np.asarray(block_table)[s, idx // BS]
        keys = e4m3_decode(k_codes[blk, idx % BS]) * k_scales[blk, idx % BS][..., None].astype(np.float64)
        vals = e4m3_decode(v_codes[blk, idx % BS]) * v_scales[blk, idx % BS][..., None].astype(np.float64)
        for ri in np.flatnonzero(seq_of == s):
            t = int(rows[ri])
            pos = c - int(ql[s]) + (t - int(starts[s]))
            for h in range(num_q_heads):
                kvh = h // g
                x = keys[:pos + 1, kvh, :] @ qf[t, h] * sc
                m = x.max()
                w = np.exp(x - m)
                out[ri, h] = (w[:, None] * vals[:pos + 1, kvh, :]).sum(0) / w.sum()
                lse[ri, h] = m + np.log(w.sum())
    return out, lse
