"""Parity of the FP8 (e4m3) KV-cache path with the fp64 FP8 reference.

The append must be bit-exact over the whole byte pools (stale random bytes in
every slot that no token reaches, NaN codes and NaN scales among them). The
decode must match the reference's attention over the dequantised cache within
the bf16 path's tolerances (|O - O_ref| <= 2e-2, |LSE - LSE_ref| <= 1e-3): the
codes are exact in the kernel's f16 operands, so the only extra rounding is the
f16 query, f16 probabilities and fp32 accumulation.
"""
import dataclasses

import numpy as np
import pytest

import workloads as W
from oracle import fp8 as F8

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

O_TOL = 2e-2
LSE_TOL = 1e-3


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2606_04415_gb300 as fnpu
    fnpu.load()


def _batch(ctx, hq=28, seed=0, slack=1.25, ql=None, phase=None):
    rng = np.random.default_rng(seed)
    S = len(ctx)
    shape = W.Shape(hq, 4, 128, 128, 16, False)
    ql = np.ones(S, np.int32) if ql is None else np.asarray(ql, np.int32)
    phase = np.ones(S, np.uint8) if phase is None else np.asarray(phase, np.uint8)
    return W.build_batch(shape, ql, np.asarray(ctx, np.int32), phase, rng, name="fp8", seed=seed, pool_slack=slack)


def _reference_pools(batch, init, seqs=None):
    """The reference's pools after the prefix fill and the step's append (of
    the sequences `seqs` only, default all)."""
    kp, vp = init
    k, v, sl = W.prefix_rows(batch)
    kn, vn, sm = batch.k_new, batch.v_new, batch.slot_mapping
    if seqs is not None:
        pre = (batch.context_len - batch.query_len).astype(np.int64)
        p0 = np.concatenate([[0], np.cumsum(pre)])
        q0 = batch.query_start
        pi = np.concatenate([np.arange(p0[s], p0[s + 1]) for s in seqs])
        qi = np.concatenate([np.arange(q0[s], q0[s] + batch.query_len[s]) for s in seqs])
        k, v, sl = k[pi], v[pi], sl[pi]
        kn, vn, sm = kn[qi], vn[qi], sm[qi]
    kp, vp = F8.kv_append(kp, vp, k, v, sl, 4)
    return F8.kv_append(kp, vp, kn, vn, sm, 4)


def _run(batch, seed=0, split=0, check_pools=True, flags=0, share=0):
    import paper_2606_04415_gb300 as fnpu
    from paper_2606_04415_gb300.step import DeviceStep
    init = W.stale_pool_bytes(batch.num_blocks * F8.block_bytes(4), seed)
    st = DeviceStep(batch, opts=fnpu.PlanOpts(split, share, 0, flags), kv_fp8=True, pool_init=init)
    st.run()
    assert fnpu.plan_check(st.plan) == fnpu.FNPU_OK and fnpu.check() == fnpu.FNPU_OK
    out, lse = st.results()
    kp, vp = _reference_pools(batch, init)
    if check_pools:
        gk, gv = st.cache_bits()
        assert np.array_equal(gk, kp), f"K pool differs at {np.flatnonzero(gk != kp)[:8]}"
        assert np.array_equal(gv, vp), f"V pool differs at {np.flatnonzero(gv != vp)[:8]}"
    return st, out, lse, kp, vp


def _compare(batch, out, lse, kp, vp, tokens=None):
    if np.all(batch.query_len == 1) and tokens is None:
        ref_o, ref_l = F8.decode_attention(batch.context_len, batch.block_table, batch.q, kp, vp,
                                           num_q_heads=batch.shape.num_q_heads, num_kv_heads=4)
    else:
        ref_o, ref_l = F8.attention(batch.query_len, batch.context_len, batch.block_table, batch.q, kp, vp,
                                    num_q_heads=batch.shape.num_q_heads, num_kv_heads=4, tokens=tokens)
        if tokens is not None:
            out, lse = out[tokens], lse[tokens]
    assert np.isfinite(out).all() and np.isfinite(lse).all()
    eo, el = np.abs(out - ref_o).max(), np.abs(lse - ref_l).max()
    assert eo <= O_TOL, f"max |dO| = {eo}"
    assert el <= LSE_TOL, f"max |dLSE| = {el}"
    return eo, el


RAGGED = [1, 2, 15, 16, 17, 33, 64, 65, 300, 1000, 2049]


def test_fp8_append_bit_exact_with_special_rows():
    """Zero rows (scale 1), a lone huge value (other codes underflow to
    subnormals and zero), tiny rows and negative zeros, on top of a ragged
    batch, all bit-exact."""
    batch = _batch(RAGGED, seed=1)
    k = batch.k_new.copy()
    v = batch.v_new.copy()
    k[0] = 0
    v[0, 1] = 0x8000                      # negative zeros
    k[1, 2, :] = W.f32_to_bf16_bits(np.full(128, 1e-3, np.float32))
    k[1, 2, 7] = W.f32_to_bf16_bits(np.float32(30000.0))
    v[2] = W.f32_to_bf16_bits((np.arange(4 * 128, dtype=np.float32).reshape(4, 128) - 256) * 1e-30)
    k[3, 3] = W.f32_to_bf16_bits(np.full(128, -7.0, np.float32))   # amax on every column
    batch = dataclasses.replace(batch, k_new=k, v_new=v)
    _, out, lse, kp, vp = _run(batch, seed=1)
    _compare(batch, out, lse, kp, vp)


def test_fp8_append_skips_padding_and_flags_out_of_range():
    import paper_2606_04415_gb300 as fnpu
    from paper_2606_04415_gb300.step import DeviceStep
    batch = _batch([40, 7, 100], seed=2)
    init = W.stale_pool_bytes(batch.num_blocks * F8.block_bytes(4), 2)
    st = DeviceStep(batch, kv_fp8=True, pool_init=init)
    torch.cuda.synchronize()
    before = st.cache_bits()
    slots = torch.tensor([-1, batch.num_blocks * 16 + 3, -5], dtype=torch.int64, device="cuda")
    fnpu.kv_append(st.desc, st.k_new, st.v_new, slots, st.k_cache, st.v_cache)
    assert fnpu.check() == fnpu.FNPU_EDEVICE_RANGE
    assert fnpu.check() == fnpu.FNPU_OK  # the flag was cleared
    after = st.cache_bits()
    assert np.array_equal(before[0], after[0]) and np.array_equal(before[1], after[1])


@pytest.mark.parametrize("hq", [4, 16, 28, 32])
@pytest.mark.parametrize("split", [0, 64, 192])
def test_fp8_decode_ragged_groups_and_splits(hq, split):
    batch = _batch(RAGGED, hq=hq, seed=3 + hq)
    _, out, lse, kp, vp = _run(batch, seed=3, split=split)
    _compare(batch, out, lse, kp, vp)


def test_fp8_decode_qwen_full_size_sampled_sequences():
    """The 64-decode Qwen2.5-7B workload (ctx ~ U[512, 4096]) at full size and
    in the bench's launch configuration; the reference recomputes the blocks
    and outputs of 8 sequences (the longest, the shortest and 6 at random)."""
    import paper_2606_04415_gb300 as fnpu
    from paper_2606_04415_gb300.step import DeviceStep
    batch = W.make_batch("qwen_decode", seed=0)
    init = W.stale_pool_bytes(batch.num_blocks * F8.block_bytes(4), 0)
    st = DeviceStep(batch, kv_fp8=True, pool_init=init)
    st.run()
    assert fnpu.plan_check(st.plan) == fnpu.FNPU_OK and fnpu.check() == fnpu.FNPU_OK
    out, lse = st.results()
    gk, gv = st.cache_bits()
    rng = np.random.default_rng(11)
    ctx = batch.context_len
    seqs = sorted({int(ctx.argmax()), int(ctx.argmin())} | set(rng.choice(64, 6, replace=False).tolist()))
    kp, vp = _reference_pools(batch, init, seqs)
    bb = F8.block_bytes(4)
    for s in seqs:
        blocks = batch.block_table[s, :(int(ctx[s]) + 15) // 16]
        for b in blocks:
            assert np.array_equal(gk[b * bb:(b + 1) * bb], kp[b * bb:(b + 1) * bb]), (s, b)
            assert np.array_equal(gv[b * bb:(b + 1) * bb], vp[b * bb:(b + 1) * bb]), (s, b)
    ref_o, ref_l = F8.decode_attention(ctx[seqs], batch.block_table[seqs], batch.q[seqs], kp, vp,
                                       num_q_heads=28, num_kv_heads=4)
    eo, el = np.abs(out[seqs] - ref_o).max(), np.abs(lse[seqs] - ref_l).max()
    assert eo <= O_TOL and el <= LSE_TOL, (eo, el)


def test_fp8_decode_long_context_split_cap():
    """A 40000-key sequence: 64-key splits would exceed the 256-split cap, so
    the planner lengthens them; plus short neighbours."""
    batch = _batch([40000, 1, 513], seed=4, slack=1.0)
    _, out, lse, kp, vp = _run(batch, seed=4, split=64)
    _compare(batch, out, lse, kp, vp)


def test_fp8_plan_reuse_runs_repeatedly():
    batch = _batch([300, 77, 1500], seed=5)
    st, out, lse, kp, vp = _run(batch, seed=5, check_pools=False)
    for _ in range(3):
        st.attend()
    o2, l2 = st.results()
    assert np.array_equal(out, o2) and np.array_equal(lse, l2)
    _compare(batch, o2, l2, kp, vp)


@pytest.mark.parametrize("flags", [0, 2])
@pytest.mark.parametrize("hq", [28, 32])
def test_fp8_mixed_step_prefill_and_decode(hq, flags):
    """Prefill chunks on prefixes (64 rows on none, 130 on 170), a 3-token
    decode (the prefill queue) and one-token decodes (one of 2049 keys) over
    the FP8 cache: the prefill rows on the tcgen05 kernel over f16-staged blocks
    (flags 0) or on the f16 mma.sync FP8 kernel (FNPU_PLAN_NO_TCGEN05), the
    decodes on the FP8 decode kernel; all rows against the reference."""
    batch = _batch([64, 500, 300, 200, 2049], hq=hq, seed=7, ql=[64, 1, 130, 3, 1], phase=[0, 1, 0, 1, 1])
    _, out, lse, kp, vp = _run(batch, seed=7, flags=flags)
    _compare(batch, out, lse, kp, vp)


@pytest.mark.parametrize("share", [0, 20])
def test_fp8_colocated_and_separate_launches_agree(share):
    """A co-located FP8 step (prefill on tcgen05 over the staged blocks beside
    the FP8 decode kernel) at the planner's and a fixed decode share, and the
    same step as separate launches: parity against the reference, and the two
    launch modes within rounding of each other."""
    import paper_2606_04415_gb300 as fnpu
    batch = _batch([1000, 700, 64, 3000, 129, 900], hq=28, seed=9, ql=[300, 1, 64, 1, 1, 1],
                   phase=[0, 1, 0, 1, 1, 1])
    st, out, lse, kp, vp = _run(batch, seed=9, share=share)
    _compare(batch, out, lse, kp, vp)
    st2, out2, lse2, _, _ = _run(batch, seed=9, flags=fnpu.PLAN_SEPARATE_LAUNCHES, check_pools=False)
    assert np.abs(out - out2).max() <= 1e-2 and np.abs(lse - lse2).max() <= 1e-3


def test_fp8_colocated_workload_sampled_rows():
    """The co-located Qwen workload over the FP8 cache (one 2048-token chunk on
    a prefix of 6969 + 128 decodes, seed 0) at full size; the reference fills
    the blocks of the chunk's sequence and of 6 decodes and recomputes rows at
    tile boundaries of the chunk, random rows and those decodes."""
    import paper_2606_04415_gb300 as fnpu
    from paper_2606_04415_gb300.step import DeviceStep
    batch = W.make_batch("qwen_coloc", seed=0)
    init = W.stale_pool_bytes(batch.num_blocks * F8.block_bytes(4), 0)
    st = DeviceStep(batch, kv_fp8=True, pool_init=init)
    st.run()
    assert fnpu.plan_check(st.plan) == fnpu.FNPU_OK and fnpu.check() == fnpu.FNPU_OK
    out, lse = st.results()
    rng = np.random.default_rng(12)
    dec = sorted(rng.choice(np.arange(1, batch.num_seqs), 6, replace=False).tolist())
    seqs = [0] + dec
    kp, vp = _reference_pools(batch, init, seqs)
    rows = sorted({0, 1, 63, 64, 65, 127, 1023, 1024, 2047} | set(rng.integers(0, 2048, 10).tolist()))
    tokens = np.asarray(rows + [int(batch.query_start[s]) for s in dec], np.int64)
    _compare(batch, out, lse, kp, vp, tokens=tokens)


def test_fp8_colocated_in_green_context_partitions():
    """A co-located FP8 step with the SM split enforced by green contexts (the
    staging kernels and the tcgen05 prefill in the prefill partition, the FP8
    decode in the decode partition): parity against the reference."""
    import paper_2606_04415_gb300 as fnpu
    batch = _batch([1000, 700, 64, 3000, 129, 900], hq=28, seed=10, ql=[300, 1, 64, 1, 1, 1],
                   phase=[0, 1, 0, 1, 1, 1])
    st, out, lse, kp, vp = _run(batch, seed=10, flags=fnpu.PLAN_GREEN_CONTEXTS, share=20)
    _compare(batch, out, lse, kp, vp)
    pre, dec = fnpu.plan_phase_ms(st.plan)
    assert pre > 0 and dec > 0


@pytest.mark.parametrize("case", range(10))
def test_fp8_random_mixed_step_all_rows(case):
    """Randomised mixes over the FP8 cache (Hkv = 4, d = 128, 16-slot blocks;
    2 to 8 query heads per kv head): one-token and multi-token decodes,
    chunks with and without a prefix, under random decode shares, key-split
    lengths and launch modes. The pools must equal the reference's bit for
    bit and every row must match the FP8 oracle."""
    rng = np.random.default_rng(5000 + case)
    hq = int(rng.choice([8, 12, 16, 28, 32]))
    S = int(rng.integers(2, 11))
    ql, ctx, ph = [], [], []
    for _ in range(S):
        kind = rng.choice(["decode", "decode", "multi", "chunk", "chunk_prefix"])
        if kind == "decode":
            ql.append(1), ctx.append(int(rng.integers(1, 3000))), ph.append(1)
        elif kind == "multi":
            q = int(rng.integers(2, 8))
            ql.append(q), ctx.append(q + int(rng.integers(0, 2000))), ph.append(1)
        elif kind == "chunk":
            q = int(rng.integers(1, 300))
            ql.append(q), ctx.append(q), ph.append(0)
        else:
            q = int(rng.integers(2, 300))
            ql.append(q), ctx.append(q + int(rng.integers(1, 2500))), ph.append(0)
    batch = _batch(ctx, hq=hq, seed=70 + case, ql=ql, phase=ph)
    share = int(rng.choice([0, 0, 3, 20, 45]))
    split = int(rng.choice([0, 0, 64, 256]))
    flags = int(rng.choice([0, 0, 0, 1, 2]))  # separate launches / the mma.sync prefill
    _, out, lse, kp, vp = _run(batch, seed=70 + case, split=split, flags=flags, share=share)
    _compare(batch, out, lse, kp, vp)
