"""Pins of the reference for MLA prefill without absorption (latent rows
expanded into per-head keys and values), against the absorbed form of the same
attention, closed forms and the bf16 rounding definition. No GPU."""
import numpy as np

import oracle
import workloads as W
from oracle import mla_expand as X


def test_bf16_rounding_matches_the_fp32_rounding_on_fp32_values_and_breaks_ties_to_even():
    rng = np.random.default_rng(0)
    x = (rng.standard_normal(100000) * np.exp2(rng.uniform(-20, 20, 100000))).astype(np.float32)
    assert np.array_equal(X.f64_to_bf16_bits(x.astype(np.float64)), W.f32_to_bf16_bits(x))
    one = 1.0
    assert X.f64_to_bf16_bits(one) == 0x3F80
    assert X.f64_to_bf16_bits(one + 2.0 ** -8) == 0x3F80          # tie -> even (1.0)
    assert X.f64_to_bf16_bits(one + 3 * 2.0 ** -8) == 0x3F82      # tie -> even (1 + 2^-6)
    assert X.f64_to_bf16_bits(one + 2.0 ** -8 + 2.0 ** -40) == 0x3F81  # past the tie, no double rounding
    assert X.f64_to_bf16_bits(-(one + 2.0 ** -8)) == 0xBF80
    assert X.f64_to_bf16_bits(0.0) == 0


def _small_latent(rng, S_ctx, H=4, bs=16):
    nb = sum((c + bs - 1) // bs for c in S_ctx) + 2
    lat = W.f32_to_bf16_bits(rng.standard_normal((nb, bs, 576)).astype(np.float32))
    perm = rng.permutation(nb)
    bt = np.zeros((len(S_ctx), max((c + bs - 1) // bs for c in S_ctx)), np.int32)
    o = 0
    for s, c in enumerate(S_ctx):
        k = (c + bs - 1) // bs
        bt[s, :k] = perm[o:o + k]
        o += k
    wk = W.f32_to_bf16_bits((rng.standard_normal((H, 512, 128)) / np.sqrt(512)).astype(np.float32))
    wv = W.f32_to_bf16_bits((rng.standard_normal((H, 512, 128)) / np.sqrt(512)).astype(np.float32))
    return lat, bt, wk, wv


def _slots(bt, s, c, bs=16):
    pos = np.arange(c)
    return bt[s, pos // bs].astype(np.int64) * bs + pos % bs


def test_expanded_attention_equals_the_absorbed_form():
    """q_nope . (c W_UK[h]) = (W_UK[h] q_nope) . c: attention over the expanded
    keys and values (not rounded) equals attention over the latent rows with
    the absorbed query [W_UK[h] q_nope, q_rope], its latent output projected by
    W_UV[h]; checked for causal rows of a chunk on a prefix."""
    rng = np.random.default_rng(1)
    H, c, q_len = 4, 70, 9
    lat, bt, wk, wv = _small_latent(rng, [c], H)
    sl = _slots(bt, 0, c)
    k, v = X.expand_exact(lat, sl, wk, wv)
    q = X.bf16_bits_to_f64(W.f32_to_bf16_bits(rng.standard_normal((q_len, H, 192)).astype(np.float32)))
    rows = X.latent_rows(lat, sl)
    wkf, wvf = X.bf16_bits_to_f64(wk), X.bf16_bits_to_f64(wv)
    scale = 1 / np.sqrt(192)
    for i in range(q_len):
        pos = c - q_len + i
        for h in range(H):
            s_exp = k[:pos + 1, h] @ q[i, h] * scale
            p = np.exp(s_exp - s_exp.max())
            o_exp = p @ v[:pos + 1, h] / p.sum()
            q_abs = np.concatenate([wkf[h] @ q[i, h, :128], q[i, h, 128:]])
            s_abs = rows[:pos + 1] @ q_abs * scale
            pa = np.exp(s_abs - s_abs.max())
            o_abs = (pa @ rows[:pos + 1, :512] / pa.sum()) @ wvf[h]
            assert np.allclose(s_exp, s_abs, rtol=0, atol=1e-10)
            assert np.allclose(o_exp, o_abs, rtol=0, atol=1e-10)


def test_selection_weights_give_latent_columns_exactly():
    """W_UK[h] selecting latent columns 0..127 and W_UV[h] columns 128 + h ..:
    the expanded rows are those columns (bf16-exact), r is copied to every head,
    and negative slots give zero rows."""
    rng = np.random.default_rng(2)
    H = 3
    lat, bt, _, _ = _small_latent(rng, [40], H)
    wk = np.zeros((H, 512, 128), np.float32)
    wv = np.zeros((H, 512, 128), np.float32)
    for h in range(H):
        wk[h, np.arange(128), np.arange(128)] = 1.0
        wv[h, 128 + h + np.arange(128), np.arange(128)] = 1.0
    wk, wv = W.f32_to_bf16_bits(wk), W.f32_to_bf16_bits(wv)
    sl = np.concatenate([_slots(bt, 0, 40), [-1, -7]])
    kb, vb = X.expand(lat, sl, wk, wv)
    latr = lat.reshape(-1, 576)
    for h in range(H):
        assert np.array_equal(kb[:40, h, :128], latr[sl[:40], :128])
        assert np.array_equal(kb[:40, h, 128:], latr[sl[:40], 512:])
        assert np.array_equal(vb[:40, h], latr[sl[:40], 128 + h:256 + h])
    assert not kb[40:].any() and not vb[40:].any()


def test_attention_oracle_on_expanded_rows_matches_brute_force():
    """The C oracle with d_qk 192, d_v 128, one kv head per head, over the
    rounded expanded cache laid out by workloads.expanded_layout, equals a
    direct fp64 softmax over the same values."""
    rng = np.random.default_rng(3)
    sh = W.Shape(4, 1, 576, 512, 64, True)
    batch = W.build_batch(sh, [5, 33], [40, 100], [0, 0], rng, name="mla_exp")
    ins = W.mla_expand_inputs(batch, seed=3)
    slots, bt, nb = W.expanded_layout(batch)
    lat = oracle.kv_append(batch.k_cache, batch.k_new, batch.slot_mapping)  # the chunk's own rows
    kb, vb = X.expand(lat, slots, ins["w_uk"], ins["w_uv"])
    out, lse = oracle.attention(batch.query_len, batch.context_len, bt, ins["q"], kb, vb, num_q_heads=4,
                                num_kv_heads=4, head_dim_qk=192, head_dim_v=128, block_size=16)
    kf, vf = X.bf16_bits_to_f64(kb), X.bf16_bits_to_f64(vb)
    qf = X.bf16_bits_to_f64(ins["q"])
    t = 0
    for s in range(2):
        base = int(bt[s, 0]) * 16
        c, ql = int(batch.context_len[s]), int(batch.query_len[s])
        for i in range(ql):
            pos = c - ql + i
            for h in range(4):
                x = kf[base:base + pos + 1, h] @ qf[t, h] / np.sqrt(192)
                p = np.exp(x - x.max())
                assert np.allclose(out[t, h], p @ vf[base:base + pos + 1, h] / p.sum(), atol=1e-12)
                assert np.isclose(lse[t, h], x.max() + np.log(p.sum()), atol=1e-12)
            t += 1


def test_expanded_path_equals_the_c_latent_oracle_with_selection_weights():
    """With W_UK[h] selecting latent columns 64h .. 64h + 127 and W_UV[h]
    columns 128 + 32h .. 255 + 32h, every expanded value and the absorbed
    query [W_UK[h] q_nope, q_rope] are exact in bf16, so the expanded
    reference (this module + the C oracle at 192 / 128, one kv head per head)
    must equal the C oracle's latent attention (576 / 512, one latent head) with
    that query, its output columns selected by W_UV[h]: two independent paths."""
    rng = np.random.default_rng(9)
    H = 4
    sh = W.Shape(H, 1, 576, 512, 64, True)
    batch = W.build_batch(sh, [7, 1, 20], [30, 90, 20], [0, 0, 0], rng, name="mla_sel")
    wk = np.zeros((H, 512, 128), np.float32)
    wv = np.zeros((H, 512, 128), np.float32)
    for h in range(H):
        wk[h, 64 * h + np.arange(128), np.arange(128)] = 1.0
        wv[h, 128 + 32 * h + np.arange(128), np.arange(128)] = 1.0
    wk, wv = W.f32_to_bf16_bits(wk), W.f32_to_bf16_bits(wv)
    q = W.f32_to_bf16_bits(rng.standard_normal((batch.num_tokens, H, 192)).astype(np.float32))
    lat = oracle.kv_append(batch.k_cache, batch.k_new, batch.slot_mapping)
    slots, bt, _ = W.expanded_layout(batch)
    kb, vb = X.expand(lat, slots, wk, wv)
    scale = 1.0 / np.sqrt(192)
    out_e, lse_e = oracle.attention(batch.query_len, batch.context_len, bt, q, kb, vb, num_q_heads=H,
                                    num_kv_heads=H, head_dim_qk=192, head_dim_v=128, block_size=16, scale=scale)
    q_abs = np.zeros((batch.num_tokens, H, 576), np.uint16)
    for h in range(H):
        q_abs[:, h, 64 * h:64 * h + 128] = q[:, h, :128]
        q_abs[:, h, 512:] = q[:, h, 128:]
    out_l, lse_l = oracle.attention(batch.query_len, batch.context_len, batch.block_table, q_abs, lat, None,
                                    num_q_heads=H, num_kv_heads=1, head_dim_qk=576, head_dim_v=512, block_size=64,
                                    latent=True, scale=scale)
    for h in range(H):
        assert np.abs(out_e[:, h] - out_l[:, h, 128 + 32 * h:256 + 32 * h]).max() < 1e-12
    assert np.abs(lse_e - lse_l).max() < 1e-12
