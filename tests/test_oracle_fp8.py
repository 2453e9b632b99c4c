"""Pins of the fp8 (e4m3) KV-cache reference against the format definition and
the bf16 oracle. No GPU."""
import numpy as np
import pytest

import oracle
from oracle import fp8


def test_e4m3_values_of_known_codes():
    assert fp8.e4m3_value(0x00) == 0.0
    assert fp8.e4m3_value(0x01) == 2.0 ** -9          # smallest subnormal
    assert fp8.e4m3_value(0x07) == 7 * 2.0 ** -9       # largest subnormal
    assert fp8.e4m3_value(0x08) == 2.0 ** -6           # smallest normal
    assert fp8.e4m3_value(0x38) == 1.0
    assert fp8.e4m3_value(0x44) == 3.0
    assert fp8.e4m3_value(0x7E) == 448.0               # largest finite
    assert np.isnan(fp8.e4m3_value(0x7F))
    assert fp8.e4m3_value(0xB8) == -1.0
    assert fp8.e4m3_value(0xFE) == -448.0


def test_every_finite_value_rounds_to_its_own_code():
    codes = np.arange(127, dtype=np.uint8)
    vals = np.array([fp8.e4m3_value(int(c)) for c in codes], np.float32)
    assert np.array_equal(fp8.e4m3_round(vals), codes)
    assert np.array_equal(fp8.e4m3_round(-vals[1:]), codes[1:] | 0x80)


def test_ties_go_to_the_even_code_and_large_values_saturate():
    # 1.0625 lies halfway between 1.0 (code 56) and 1.125 (57); 1.1875 between 57 and 58
    assert fp8.e4m3_round(np.float32(1.0625)) == 56
    assert fp8.e4m3_round(np.float32(1.1875)) == 58
    assert fp8.e4m3_round(np.float32(1.07)) == 57
    # subnormal range: 2^-10 halfway between 0 and 2^-9, 3*2^-10 between codes 1 and 2
    assert fp8.e4m3_round(np.float32(2.0 ** -10)) == 0
    assert fp8.e4m3_round(np.float32(3 * 2.0 ** -10)) == 2
    for big in (448.5, 463.9, 500.0, 1e30):
        assert fp8.e4m3_round(np.float32(big)) == 0x7E
        assert fp8.e4m3_round(np.float32(-big)) == 0xFE


def _bf16(x):
    return (np.asarray(x, np.float32).view(np.uint32) >> 16).astype(np.uint16)


def test_row_quantisation_maps_amax_to_448_and_bounds_the_error():
    rng = np.random.default_rng(3)
    x = rng.standard_normal((64, 4, 128)).astype(np.float32) * 3
    bits = _bf16(x)
    xf = fp8.bf16_bits_to_f32(bits).astype(np.float64)
    codes, scale = fp8.quantize_rows(bits)
    amax = np.abs(xf).max(-1)
    assert np.allclose(scale, amax / 448, rtol=1e-7)
    argmax = np.abs(xf).argmax(-1)
    top = np.take_along_axis(codes, argmax[..., None], -1)[..., 0]
    assert np.all((top & 0x7F) == 0x7E)
    deq = fp8.e4m3_decode(codes) * scale[..., None]
    # half a step of the e4m3 grid: 2^-4 relative for normals, 2^-10 * scale absolute below
    err = np.abs(deq - xf)
    assert np.all(err <= np.maximum(np.abs(xf) * 2.0 ** -4, scale[..., None] * 2.0 ** -10) * 1.0001)
    zero = fp8.quantize_rows(np.zeros((1, 128), np.uint16))
    assert zero[1][0] == 1.0 and not zero[0].any()


def test_layout_permutations_are_bijections_and_group_lane_operands():
    assert sorted(fp8.kpos(np.arange(128)).tolist()) == list(range(128))
    assert sorted(fp8.vpos(np.arange(16)).tolist()) == list(range(16))
    for k in range(8):
        for c in range(4):
            cols = [16 * k + 2 * c, 16 * k + 2 * c + 1, 16 * k + 2 * c + 8, 16 * k + 2 * c + 9]
            assert fp8.kpos(cols).tolist() == [32 * c + 4 * k + r for r in range(4)]
    for c in range(4):
        assert fp8.vpos([2 * c, 2 * c + 1, 2 * c + 8, 2 * c + 9]).tolist() == [4 * c + r for r in range(4)]


def test_pack_unpack_round_trip_and_append():
    rng = np.random.default_rng(4)
    nb, hkv = 5, 4
    kc = rng.integers(0, 256, (nb, 16, hkv, 128), dtype=np.uint8)
    vc = rng.integers(0, 256, (nb, 16, hkv, 128), dtype=np.uint8)
    ks = rng.random((nb, 16, hkv)).astype(np.float32)
    vs = rng.random((nb, 16, hkv)).astype(np.float32)
    kp, vp = fp8.pack_pools(kc, ks, vc, vs)
    assert kp.size == nb * fp8.block_bytes(hkv)
    back = fp8.unpack_pools(kp, vp, hkv)
    for a, b in zip(back, (kc, ks, vc, vs)):
        assert np.array_equal(a, b)
    new_k = _bf16(rng.standard_normal((4, hkv, 128)))
    new_v = _bf16(rng.standard_normal((4, hkv, 128)))
    slots = np.array([17, -1, 79, 0], np.int64)
    kp2, vp2 = fp8.kv_append(kp, vp, new_k, new_v, slots, hkv)
    k2, ks2, v2, vs2 = fp8.unpack_pools(kp2, vp2, hkv)
    qk, sk = fp8.quantize_rows(new_k)
    qv, sv = fp8.quantize_rows(new_v)
    assert np.array_equal(k2[1, 1], qk[0]) and np.array_equal(ks2[4, 15], sk[2])
    assert np.array_equal(k2[0, 0], qk[3]) and np.array_equal(v2[0, 0], qv[3]) and vs2[0, 0, 1] == sv[3, 1]
    assert np.array_equal(k2[3], kc[3]) and np.array_equal(v2[2], vc[2])   # untouched blocks


def test_decode_attention_closed_forms():
    rng = np.random.default_rng(5)
    hkv, hq = 4, 8
    kc = rng.integers(0, 120, (2, 16, hkv, 128), dtype=np.uint8)
    vc = rng.integers(0, 120, (2, 16, hkv, 128), dtype=np.uint8)
    ks = np.full((2, 16, hkv), 0.5, np.float32)
    vs = np.full((2, 16, hkv), 0.25, np.float32)
    kp, vp = fp8.pack_pools(kc, ks, vc, vs)
    q = _bf16(rng.standard_normal((1, hq, 128)))
    out, lse = fp8.decode_attention([1], np.array([[1, 0]]), q, kp, vp, num_q_heads=hq, num_kv_heads=hkv)
    k0 = fp8.e4m3_decode(kc[1, 0]) * 0.5
    v0 = fp8.e4m3_decode(vc[1, 0]) * 0.25
    qf = fp8.bf16_bits_to_f32(q)[0].astype(np.float64)
    for h in range(hq):   # one key: the output is its value, the LSE its score
        assert np.allclose(out[0, h], v0[h // 2])
        assert np.isclose(lse[0, h], k0[h // 2] @ qf[h] / np.sqrt(128))


def test_matches_the_bf16_oracle_when_every_scale_is_one():
    """Rows whose amax is exactly 448 have scale 1, and e4m3 values are exact
    in bf16: the fp8 reference must then equal the bf16 oracle on the
    dequantised cache."""
    rng = np.random.default_rng(6)
    hkv, hq, nb = 4, 28, 6
    vals = np.array([fp8.e4m3_value(c) for c in range(127)], np.float32)
    def rows(n):
        x = rng.choice(np.concatenate([vals, -vals[1:]]), size=(n, 16, hkv, 128)).astype(np.float32) / 64
        x[..., 0] = 448.0
        return x
    kx, vx = rows(nb), rows(nb)
    kc, ks = fp8.quantize_rows(_bf16(kx))
    vc, vs = fp8.quantize_rows(_bf16(vx))
    assert np.all(ks == 1.0) and np.all(vs == 1.0)
    kp, vp = fp8.pack_pools(kc, ks, vc, vs)
    ctx = np.array([37, 90, 5])
    bt = np.array([[2, 4, 0, 0, 0, 0], [1, 3, 5, 0, 2, 4], [5, 0, 0, 0, 0, 0]], np.int32)
    q = _bf16(rng.standard_normal((3, hq, 128)))
    out, lse = fp8.decode_attention(ctx, bt, q, kp, vp, num_q_heads=hq, num_kv_heads=hkv)
    kdq = _bf16(fp8.e4m3_decode(kc).astype(np.float32))
    vdq = _bf16(fp8.e4m3_decode(vc).astype(np.float32))
    ref_o, ref_l = oracle.attention(np.ones(3, np.int32), ctx, bt, q, kdq, vdq, num_q_heads=hq,
                                    num_kv_heads=hkv, head_dim_qk=128, head_dim_v=128, block_size=16)
    assert np.abs(out - ref_o).max() < 1e-12 and np.abs(lse - ref_l).max() < 1e-12


def test_binade_rounding_equals_the_table_search():
    """The per-binade rounding and the table search agree on random
    magnitudes over the whole range, on every value, and on every midpoint
    between neighbouring values (the ties)."""
    rng = np.random.default_rng(7)
    x = (rng.standard_normal(200000) * np.exp2(rng.uniform(-14, 10, 200000))).astype(np.float32)
    vals = np.array([fp8.e4m3_value(c) for c in range(127)])
    mids = ((vals[1:] + vals[:-1]) / 2).astype(np.float32)
    near = np.concatenate([np.nextafter(mids, np.float32(0)), np.nextafter(mids, np.float32(1e9))])
    for arr in (x, vals.astype(np.float32), mids, -mids, near, np.array([0, -0.0, 448, 449, 470, 1e38], np.float32)):
        assert np.array_equal(fp8.e4m3_round(arr), fp8.e4m3_round_by_search(arr))


def test_mixed_step_matches_the_bf16_oracle_when_every_scale_is_one():
    """Prefill chunks on prefixes, a multi-token decode and decodes: with every
    scale 1 the fp8 reference equals the bf16 C oracle on the dequantised cache
    (causal rows at absolute positions, sampled and whole)."""
    rng = np.random.default_rng(8)
    hkv, hq, nb = 4, 28, 12
    vals = np.array([fp8.e4m3_value(c) for c in range(127)], np.float32)
    def rows(n):
        x = rng.choice(np.concatenate([vals, -vals[1:]]), size=(n, 16, hkv, 128)).astype(np.float32) / 64
        x[..., 0] = 448.0
        return x
    kc, ks = fp8.quantize_rows(_bf16(rows(nb)))
    vc, vs = fp8.quantize_rows(_bf16(rows(nb)))
    kp, vp = fp8.pack_pools(kc, ks, vc, vs)
    ql = np.array([20, 1, 3, 1], np.int32)
    cl = np.array([50, 77, 40, 1], np.int32)
    bt = rng.integers(0, nb, size=(4, 5)).astype(np.int32)  # blocks may repeat: both sides read the same
    q = _bf16(rng.standard_normal((int(ql.sum()), hq, 128)))
    kdq = _bf16(fp8.e4m3_decode(kc).astype(np.float32))
    vdq = _bf16(fp8.e4m3_decode(vc).astype(np.float32))
    ref_o, ref_l = oracle.attention(ql, cl, bt, q, kdq, vdq, num_q_heads=hq, num_kv_heads=hkv, head_dim_qk=128,
                                    head_dim_v=128, block_size=16)
    out, lse = fp8.attention(ql, cl, bt, q, kp, vp, num_q_heads=hq, num_kv_heads=hkv)
    assert np.abs(out - ref_o).max() < 1e-12 and np.abs(lse - ref_l).max() < 1e-12
    tok = np.array([0, 19, 21, 23, 24])
    o2, l2 = fp8.attention(ql, cl, bt, q, kp, vp, num_q_heads=hq, num_kv_heads=hkv, tokens=tok)
    assert np.array_equal(o2, out[tok]) and np.array_equal(l2, lse[tok])


def test_worked_example_from_the_golden_file():
    """tests/golden/fp8_row_example.txt: a row quantised by hand."""
    import os
    path = os.path.join(os.path.dirname(__file__), "golden", "fp8_row_example.txt")
    lines = [l.split() for l in open(path) if l.strip() and not l.startswith("#")]
    want_scale = float(lines[0][1])
    want_codes = [int(c) for c in lines[1][1:]]
    x = np.zeros(128, np.float32)
    x[:5] = [3.5, -1.75, 0.0078125, 5.25, 0.001]
    codes, scale = fp8.quantize_rows(_bf16(x)[None])
    assert scale[0] == np.float32(want_scale)
    assert codes[0, :5].tolist() == want_codes and not codes[0, 5:].any()


def test_zero_keys_give_the_mean_of_the_dequantised_values():
    """K codes all zero: every score is 0, the weights are uniform, so O is the
    mean of the visible dequantised values (each row with its own V scale) and
    LSE = ln(pos + 1); for decodes and for causal prefill rows."""
    rng = np.random.default_rng(12)
    hkv, hq, nb = 4, 8, 6
    kc = np.zeros((nb, 16, hkv, 128), np.uint8)
    vc = rng.integers(0, 120, (nb, 16, hkv, 128), dtype=np.uint8)
    ks = rng.random((nb, 16, hkv)).astype(np.float32) + 0.5
    vs = rng.random((nb, 16, hkv)).astype(np.float32) + 0.5
    kp, vp = fp8.pack_pools(kc, ks, vc, vs)
    bt = np.array([[3, 1, 4, 0], [5, 2, 0, 0]], np.int32)
    ql, cl = np.array([5, 1]), np.array([50, 20])
    q = _bf16(rng.standard_normal((6, hq, 128)))
    out, lse = fp8.attention(ql, cl, bt, q, kp, vp, num_q_heads=hq, num_kv_heads=hkv)
    vd = fp8.e4m3_decode(vc) * vs[..., None].astype(np.float64)
    rows = [(0, 0, 45 + i, i) for i in range(5)] + [(1, 0, 19, 5)]
    for s, _, pos, t in rows:
        idx = np.arange(pos + 1)
        vals = vd[bt[s, idx // 16], idx % 16]          # [pos + 1, Hkv, d]
        for h in range(hq):
            assert np.allclose(out[t, h], vals[:, h // 2].mean(0), atol=1e-12)
            assert np.isclose(lse[t, h], np.log(pos + 1), atol=1e-12)
