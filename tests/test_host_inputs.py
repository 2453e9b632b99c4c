"""Host-side input helpers used by the FP8 and expanded-MLA paths (no GPU):
prefix rows, stale pool bytes, the expanded cache layout, the FP8 byte counts."""
import numpy as np

import workloads as W


def _batch(seed=0, latent=False):
    rng = np.random.default_rng(seed)
    sh = W.Shape(8, 1, 576, 512, 64, True) if latent else W.Shape(28, 4, 128, 128, 16, False)
    return W.build_batch(sh, [5, 1, 40], [37, 300, 40], [0, 1, 0], rng, name="host")


def test_prefix_rows_are_the_cached_positions_in_order():
    b = _batch()
    k, v, sl = W.prefix_rows(b)
    bs = b.shape.block_size
    want = []
    for s in range(b.num_seqs):
        for pos in range(int(b.context_len[s] - b.query_len[s])):
            want.append(int(b.block_table[s, pos // bs]) * bs + pos % bs)
    assert sl.tolist() == want
    assert np.array_equal(k, b.k_cache.reshape(-1, 4, 128)[sl])
    assert np.array_equal(v, b.v_cache.reshape(-1, 4, 128)[sl])
    assert not np.isnan(W.bf16_bits_to_f32(k)).any()   # prefix slots hold values, not canaries


def test_stale_pool_bytes_are_seeded_and_cover_every_byte_value():
    a = W.stale_pool_bytes(1 << 16, 3)
    b = W.stale_pool_bytes(1 << 16, 3)
    c = W.stale_pool_bytes(1 << 16, 4)
    assert np.array_equal(a[0], b[0]) and np.array_equal(a[1], b[1])
    assert not np.array_equal(a[0], c[0]) and not np.array_equal(a[0], a[1])
    assert len(np.unique(a[0])) == 256


def test_expanded_layout_starts_each_sequence_on_a_block():
    b = _batch(latent=True)
    slots, bt, nb = W.expanded_layout(b)
    assert slots.size == nb * 16
    bsl = b.shape.block_size
    first = 0
    for s in range(b.num_seqs):
        c = int(b.context_len[s])
        n = (c + 15) // 16
        assert bt[s, :n].tolist() == list(range(first, first + n))
        rows = slots[first * 16:first * 16 + n * 16]
        pos = np.arange(c)
        assert np.array_equal(rows[:c], b.block_table[s, pos // bsl].astype(np.int64) * bsl + pos % bsl)
        assert np.all(rows[c:] == -1)
        first += n
    assert first == nb


def test_fp8_algorithmic_bytes_count_codes_and_scales():
    b = _batch()
    w16 = W.algorithmic_work(b)
    w8 = W.algorithmic_work(b, kv_fp8=True)
    ctx = int(b.context_len.sum())
    assert w16["kv_read_bytes"] == ctx * 4 * 256 * 2
    assert w8["kv_read_bytes"] == ctx * 4 * (128 + 4) * 2
    T = b.num_tokens
    assert w8["append_bytes"] == T * (4 * 256 * 2 + 4 * (128 + 4) * 2)
    assert w8["flops"] == w16["flops"]
