"""Pins of the fp64 oracle against facts that do not come from the oracle.

The paper prints no worked attention example (it is a runtime-systems paper;
Sec. 3.4 only fixes that prefill chunks and decode queries share one KV pool),
so each pin below comes from the mathematics of causal softmax attention:
brute force over unpaged K/V, a library cross-check (torch SDPA in float64),
closed forms, and invariants. Each is chosen so that a plausible slip in the
oracle (a dropped scale, a wrong sign, an off-by-one in the mask or the query
position, swapped block index/offset, a wrong GQA head map, log2 in place of
ln) fails at least one of them.
"""
import math

import numpy as np
import pytest
import torch

import oracle
import workloads as W


def _oracle(batch, kc=None, vc=None, scale=0.0, tokens=None):
    sh = batch.shape
    return oracle.attention(batch.query_len, batch.context_len, batch.block_table, batch.q,
                            batch.k_cache if kc is None else kc,
                            batch.v_cache if vc is None else vc,
                            num_q_heads=sh.num_q_heads, num_kv_heads=sh.num_kv_heads,
                            head_dim_qk=sh.head_dim_qk, head_dim_v=sh.head_dim_v,
                            block_size=sh.block_size, latent=sh.latent, scale=scale,
                            tokens=tokens)


def _dense_batch(shape, qlens, ctxs, seed, *, transform=None, scale_pool=2.0):
    """Draw per-sequence dense K/V ([ctx, Hkv, d]) in the test, then copy them
    block by block into a shuffled pool. Returns (batch, dense_k, dense_v)."""
    rng = np.random.default_rng(seed)
    qlens = np.asarray(qlens, np.int32)
    ctxs = np.asarray(ctxs, np.int32)
    bs = shape.block_size
    nblk = [(c + bs - 1) // bs for c in ctxs]
    num_blocks = int(scale_pool * sum(nblk)) + 1
    perm = rng.permutation(num_blocks)
    width = max(nblk) + 2
    bt = np.zeros((len(qlens), width), np.int32)
    o = 0
    for s, n in enumerate(nblk):
        bt[s, :n] = perm[o:o + n]
        bt[s, n:] = perm[-1]  # unused columns point at a canary block
        o += n
    H, Hk, dq, dv = shape.num_q_heads, shape.num_kv_heads, shape.head_dim_qk, shape.head_dim_v
    T = int(qlens.sum())
    q = W.f32_to_bf16_bits(rng.standard_normal((T, H, dq), dtype=np.float32))
    dk, dvv = [], []
    for c in ctxs:
        if shape.latent:
            lat = W.f32_to_bf16_bits(rng.standard_normal((c, dq), dtype=np.float32))
            dk.append(lat)
            dvv.append(None)
        else:
            dk.append(W.f32_to_bf16_bits(rng.standard_normal((c, Hk, dq), dtype=np.float32)))
            dvv.append(W.f32_to_bf16_bits(rng.standard_normal((c, Hk, dv), dtype=np.float32)))
    if transform is not None:
        q, dk, dvv = transform(q, dk, dvv)
    if shape.latent:
        kc = np.full((num_blocks, bs, dq), W.BF16_CANARY, np.uint16)
        vc = None
    else:
        kc = np.full((num_blocks, bs, Hk, dq), W.BF16_CANARY, np.uint16)
        vc = np.full((num_blocks, bs, Hk, dv), W.BF16_CANARY, np.uint16)
    for s, c in enumerate(ctxs):
        for b in range(nblk[s]):
            lo, hi = b * bs, min(c, (b + 1) * bs)
            kc[bt[s, b], :hi - lo] = dk[s][lo:hi]
            if vc is not None:
                vc[bt[s, b], :hi - lo] = dvv[s][lo:hi]
    batch = W.Batch(name="dense", shape=shape, seed=seed, query_len=qlens, context_len=ctxs,
                    phase=(qlens == 1).astype(np.uint8), block_table=bt, num_blocks=num_blocks,
                    q=q, k_new=None, v_new=None, slot_mapping=np.zeros(0, np.int64),
                    k_cache=kc, v_cache=vc)
    return batch, dk, dvv


def _f64(bits):
    return W.bf16_bits_to_f32(bits).astype(np.float64)


def _brute_force(batch, dk, dv, scale):
    """Triple loop over unpaged K/V: sequence, query, head, then keys."""
    sh = batch.shape
    g = sh.num_q_heads // sh.num_kv_heads
    T = batch.num_tokens
    out = np.zeros((T, sh.num_q_heads, sh.head_dim_v))
    lse = np.zeros((T, sh.num_q_heads))
    t = 0
    for s in range(batch.num_seqs):
        ql, cl = int(batch.query_len[s]), int(batch.context_len[s])
        K = _f64(dk[s])
        V = _f64(dv[s]) if dv[s] is not None else _f64(dk[s])[..., :sh.head_dim_v]
        for i in range(ql):
            pos = cl - ql + i
            for h in range(sh.num_q_heads):
                qv = _f64(batch.q[t, h])
                if sh.latent:
                    kk, vv = K[:pos + 1], V[:pos + 1]
                else:
                    kk, vv = K[:pos + 1, h // g], V[:pos + 1, h // g]
                sc = scale * (kk @ qv)
                m = sc.max()
                e = np.exp(sc - m)
                out[t, h] = (e[:, None] * vv).sum(0) / e.sum()
                lse[t, h] = m + math.log(e.sum())
            t += 1
    return out, lse


TINY = W.SHAPES["tiny"]
SMALL_MLA = W.Shape(8, 1, 96, 64, 8, True)


@pytest.mark.parametrize("shape", [TINY, W.Shape(6, 3, 32, 48, 4, False), SMALL_MLA])
def test_brute_force_matches_paged_oracle(shape):
    qlens = [5, 1, 17, 1, 3]
    ctxs = [5, 9, 40, 33, 20]
    batch, dk, dv = _dense_batch(shape, qlens, ctxs, seed=11)
    scale = 0.29
    o_ref, l_ref = _brute_force(batch, dk, dv, scale)
    o, l = _oracle(batch, scale=scale)
    assert np.abs(o - o_ref).max() < 1e-12
    assert np.abs(l - l_ref).max() < 1e-12


@pytest.mark.parametrize("shape", [W.Shape(6, 3, 32, 48, 4, False), SMALL_MLA])
def test_default_scale_is_inverse_sqrt_dqk(shape):
    batch, dk, dv = _dense_batch(shape, [3, 1], [7, 19], seed=3)
    o_ref, l_ref = _brute_force(batch, dk, dv, 1.0 / math.sqrt(shape.head_dim_qk))
    o, l = _oracle(batch)  # scale <= 0 selects the default
    assert np.abs(o - o_ref).max() < 1e-12 and np.abs(l - l_ref).max() < 1e-12


def test_torch_sdpa_float64_crosscheck():
    """Library cross-check: torch SDPA (float64, explicit bool mask, GQA by
    repeat_interleave) and torch.logsumexp on the same dense tensors."""
    sh = W.Shape(6, 2, 32, 32, 8, False)
    qlens, ctxs = [12, 1, 4], [30, 17, 4]
    batch, dk, dv = _dense_batch(sh, qlens, ctxs, seed=5)
    o, l = _oracle(batch)
    g = sh.num_q_heads // sh.num_kv_heads
    scale = 1.0 / math.sqrt(sh.head_dim_qk)
    t = 0
    for s in range(batch.num_seqs):
        ql, cl = qlens[s], ctxs[s]
        Q = torch.from_numpy(_f64(batch.q[t:t + ql])).permute(1, 0, 2)          # [H, ql, d]
        K = torch.from_numpy(_f64(dk[s])).permute(1, 0, 2).repeat_interleave(g, 0)  # [H, cl, d]
        V = torch.from_numpy(_f64(dv[s])).permute(1, 0, 2).repeat_interleave(g, 0)
        pos = torch.arange(cl - ql, cl)[:, None]
        mask = torch.arange(cl)[None, :] <= pos                                 # [ql, cl]
        ref = torch.nn.functional.scaled_dot_product_attention(Q, K, V, attn_mask=mask)
        sc = (Q @ K.transpose(1, 2)) * scale
        lse_ref = torch.logsumexp(sc.masked_fill(~mask, float("-inf")), dim=-1)
        assert np.abs(o[t:t + ql] - ref.permute(1, 0, 2).numpy()).max() < 1e-12
        assert np.abs(l[t:t + ql] - lse_ref.T.numpy()).max() < 1e-12
        t += ql


def test_closed_form_single_key():
    """ctx = 1: the only key is the query's own, so O = v0, LSE = scale*<q,k0>."""
    batch, dk, dv = _dense_batch(TINY, [1, 1], [1, 1], seed=7)
    scale = 0.37
    o, l = _oracle(batch, scale=scale)
    g = TINY.group
    for s in range(2):
        for h in range(TINY.num_q_heads):
            k0 = _f64(dk[s][0, h // g])
            v0 = _f64(dv[s][0, h // g])
            assert np.array_equal(o[s, h], v0)
            assert abs(l[s, h] - scale * float(_f64(batch.q[s, h]) @ k0)) < 1e-12


def test_closed_form_zero_keys():
    """K = 0: all scores 0, O = mean of the visible V rows, LSE = ln(pos + 1)."""
    def zero_k(q, dk, dv):
        return q, [np.zeros_like(k) for k in dk], dv
    qlens, ctxs = [6, 1], [10, 37]
    batch, dk, dv = _dense_batch(TINY, qlens, ctxs, seed=8, transform=zero_k)
    o, l = _oracle(batch)
    g = TINY.group
    t = 0
    for s in range(2):
        for i in range(qlens[s]):
            pos = ctxs[s] - qlens[s] + i
            for h in range(TINY.num_q_heads):
                assert abs(l[t, h] - math.log(pos + 1)) < 1e-12
                mean = _f64(dv[s][:pos + 1, h // g]).mean(0)
                assert np.abs(o[t, h] - mean).max() < 1e-12
            t += 1


def test_closed_form_ones_values_and_equal_keys():
    """V = 1 gives O = 1 (weights sum to 1). All keys equal to k gives uniform
    weights: LSE = scale*<q,k> + ln(pos + 1)."""
    def const(q, dk, dv):
        k1 = dk[0][0:1]
        return q, [np.repeat(k1, len(k), 0) for k in dk], [np.full_like(v, 0x3F80) for v in dv]
    qlens, ctxs = [4, 1, 1], [4, 50, 129]
    batch, dk, dv = _dense_batch(TINY, qlens, ctxs, seed=9, transform=const)
    o, l = _oracle(batch)
    assert np.abs(o - 1.0).max() < 1e-12
    g = TINY.group
    t = 0
    scale = 1.0 / math.sqrt(TINY.head_dim_qk)
    for s in range(3):
        for i in range(qlens[s]):
            pos = ctxs[s] - qlens[s] + i
            for h in range(TINY.num_q_heads):
                ref = scale * float(_f64(batch.q[t, h]) @ _f64(dk[s][0, h // g])) + math.log(pos + 1)
                assert abs(l[t, h] - ref) < 1e-12
            t += 1


def test_block_permutation_invariance_bit_exact():
    """Moving physical blocks and rewriting the block table changes nothing."""
    batch = W.make_batch("tiny", seed=4)
    sh = batch.shape
    kc0 = oracle.kv_append(batch.k_cache, batch.k_new, batch.slot_mapping)
    vc0 = oracle.kv_append(batch.v_cache, batch.v_new, batch.slot_mapping)
    o, l = _oracle(batch, kc0, vc0)
    perm = np.random.default_rng(99).permutation(batch.num_blocks)  # new id of block b
    kc1 = np.empty_like(kc0)
    vc1 = np.empty_like(vc0)
    kc1[perm] = kc0
    vc1[perm] = vc0
    bt = perm[batch.block_table].astype(np.int32)
    o2, l2 = oracle.attention(batch.query_len, batch.context_len, bt, batch.q, kc1, vc1,
                              num_q_heads=sh.num_q_heads, num_kv_heads=sh.num_kv_heads,
                              head_dim_qk=sh.head_dim_qk, head_dim_v=sh.head_dim_v,
                              block_size=sh.block_size)
    assert np.isfinite(o).all() and np.isfinite(l).all()
    assert np.array_equal(o, o2) and np.array_equal(l, l2)


def test_decode_row_equals_prefill_row():
    """Decode at position t of a sequence = row t of a full prefill of it."""
    L = 70
    batch, dk, dv = _dense_batch(TINY, [L], [L], seed=12)
    o_full, l_full = _oracle(batch)
    positions = [0, 1, 15, 16, 17, 44, 69]
    # the same pool and block table, now as decodes of contexts t + 1
    qlens = np.ones(len(positions), np.int32)
    ctxs = np.asarray([p + 1 for p in positions], np.int32)
    bt = np.repeat(batch.block_table, len(positions), 0)
    qd = batch.q[positions]
    sh = TINY
    o_dec, l_dec = oracle.attention(qlens, ctxs, bt, qd, batch.k_cache, batch.v_cache,
                                    num_q_heads=sh.num_q_heads, num_kv_heads=sh.num_kv_heads,
                                    head_dim_qk=sh.head_dim_qk, head_dim_v=sh.head_dim_v,
                                    block_size=sh.block_size)
    assert np.array_equal(o_dec, o_full[positions]) and np.array_equal(l_dec, l_full[positions])


def test_chunked_prefill_equals_one_shot():
    """Four 32-token chunks on growing prefixes = one 128-token prefill."""
    L = 128
    batch, dk, dv = _dense_batch(TINY, [L], [L], seed=13)
    o_full, l_full = _oracle(batch)
    qlens = np.full(4, 32, np.int32)
    ctxs = np.asarray([32, 64, 96, 128], np.int32)
    bt = np.repeat(batch.block_table, 4, 0)
    sh = TINY
    o_ch, l_ch = oracle.attention(qlens, ctxs, bt, batch.q, batch.k_cache, batch.v_cache,
                                  num_q_heads=sh.num_q_heads, num_kv_heads=sh.num_kv_heads,
                                  head_dim_qk=sh.head_dim_qk, head_dim_v=sh.head_dim_v,
                                  block_size=sh.block_size)
    assert np.array_equal(o_ch, o_full) and np.array_equal(l_ch, l_full)


def test_softmax_weights_sum_to_one_and_reproduce_output():
    batch, dk, dv = _dense_batch(TINY, [9, 1], [40, 300], seed=14)
    o, l = _oracle(batch)
    sh = TINY
    for t, h in [(0, 0), (8, 3), (9, 2)]:
        w = oracle.softmax_weights(batch.query_len, batch.context_len, batch.block_table,
                                   batch.q, batch.k_cache, batch.v_cache, t, h,
                                   num_q_heads=sh.num_q_heads, num_kv_heads=sh.num_kv_heads,
                                   head_dim_qk=sh.head_dim_qk, head_dim_v=sh.head_dim_v,
                                   block_size=sh.block_size)
        assert abs(w.sum() - 1.0) < 1e-12
        s = 0 if t < 9 else 1
        V = _f64(dv[s])[:len(w), h // sh.group]
        assert np.abs(w @ V - o[t, h]).max() < 1e-12


def test_split_merge_identity():
    """Attention over keys [0, a) and [a, pos] merged by LSE equals the whole:
    lse = ln(e^lse1 + e^lse2), O = e^(lse1-lse) O1 + e^(lse2-lse) O2."""
    L, a = 90, 37
    batch, dk, dv = _dense_batch(TINY, [1], [L], seed=15)
    o, l = _oracle(batch)
    sh = TINY

    def part(lo, hi):
        def take(q, kk, vv):
            return batch.q, [dk[0][lo:hi]], [dv[0][lo:hi]]
        b2, _, _ = _dense_batch(TINY, [1], [hi - lo], seed=16, transform=take)
        return _oracle(b2)
    o1, l1 = part(0, a)
    o2, l2 = part(a, L)
    lm = np.logaddexp(l1, l2)
    om = np.exp(l1 - lm)[..., None] * o1 + np.exp(l2 - lm)[..., None] * o2
    assert np.abs(lm - l).max() < 1e-12 and np.abs(om - o).max() < 1e-12


def test_kv_append_copies_exactly():
    rng = np.random.default_rng(3)
    cache = rng.integers(0, 65535, size=(8, 4, 2, 8), dtype=np.uint16)
    rows = rng.integers(0, 65535, size=(6, 2, 8), dtype=np.uint16)
    slots = np.array([3, -1, 31, 0, -5, 17], np.int64)
    out = oracle.kv_append(cache, rows, slots)
    ref = cache.reshape(32, 2, 8).copy()
    for t, s in enumerate(slots):
        if s >= 0:
            ref[s] = rows[t]
    assert np.array_equal(out.reshape(32, 2, 8), ref)
    with pytest.raises(ValueError):
        oracle.kv_append(cache, rows, np.array([0, 1, 2, 3, 4, 32], np.int64))


def test_pairs_and_work_count():
    batch = W.make_batch("tiny", seed=0)
    n = 0
    for s in range(batch.num_seqs):
        ql, cl = int(batch.query_len[s]), int(batch.context_len[s])
        for i in range(ql):
            n += cl - ql + i + 1
    assert W.pairs(batch) == n


def test_bf16_rounding_matches_torch():
    x = np.random.default_rng(1).standard_normal(100000).astype(np.float32) * 37
    ref = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(W.f32_to_bf16_bits(x), ref)


def test_workloads_shapes_and_canaries():
    b = W.make_batch("tiny", seed=0)
    assert b.num_tokens == 262 and b.num_blocks == 256
    assert list(b.query_len[:2]) == [128, 128] and (b.query_len[2:] == 1).all()
    assert ((b.context_len[2:] >= 64) & (b.context_len[2:] <= 512)).all()
    # every new token's slot held a canary before the append
    kc = b.k_cache.reshape(-1, *b.k_cache.shape[2:])
    assert (kc[b.slot_mapping] == W.BF16_CANARY).all()


def _read_golden(name):
    vals = {}
    with open(__import__("os").path.join(__import__("os").path.dirname(__file__), "golden", name)) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            k, v = (x.strip() for x in line.split("=", 1))
            vals[k] = v
    return vals


def test_golden_worked_example():
    g = _read_golden("worked_example_2tok.txt")
    ev = lambda e: float(eval(e, {"exp": math.exp, "log": math.log}))  # noqa: E731
    num = lambda s: [float(x) for x in s.split()]  # noqa: E731
    bt = np.asarray([num(g["block_table"])], np.int32)
    kc = np.full((4, 1, 1, 2), W.BF16_CANARY, np.uint16)
    vc = np.full((4, 1, 1, 2), W.BF16_CANARY, np.uint16)
    for j in range(2):
        kc[bt[0, j], 0, 0] = W.f32_to_bf16_bits(np.asarray(num(g[f"k{j}"]), np.float32))
        vc[bt[0, j], 0, 0] = W.f32_to_bf16_bits(np.asarray(num(g[f"v{j}"]), np.float32))
    q = W.f32_to_bf16_bits(np.asarray([[num(g["q0"])], [num(g["q1"])]], np.float32))
    o, l = oracle.attention([2], [2], bt, q, kc, vc, num_q_heads=1, num_kv_heads=1,
                            head_dim_qk=2, head_dim_v=2, block_size=1, scale=1.0)
    for r in range(2):
        exp_o = [ev(x) for x in g[f"O{r}"].split(";")]
        assert np.abs(o[r, 0] - exp_o).max() < 1e-15
        assert abs(l[r, 0] - ev(g[f"LSE{r}"])) < 1e-15
