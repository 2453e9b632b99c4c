"""Parity of the CUDA path (through the C ABI) with the fp64 oracle.

Tolerances: |O - O_ref| <= 2e-2 and |LSE - LSE_ref| <= 1e-3 (bf16 inputs,
fp32 scores and accumulation, bf16 output); KV append bit-exact over the
whole pool, untouched (canary) slots included.
"""
import numpy as np
import pytest

import oracle
import workloads as W

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


def _step(batch, **opts):
    import paper_2606_04415_gb300 as fnpu
    from paper_2606_04415_gb300.step import DeviceStep
    o = fnpu.PlanOpts(opts.get("split", 0), opts.get("share", 0), opts.get("sms", 0),
                      opts.get("flags", 0))
    st = DeviceStep(batch, opts=o)
    st.run()
    assert fnpu.plan_check(st.plan) == fnpu.FNPU_OK, "device error flag raised"
    return st


def _compare(batch, out, lse, tokens=None, kc=None, vc=None):
    if kc is None:
        ref_o, ref_l, _, _ = oracle.run_step(batch, tokens=tokens)
    else:
        sh = batch.shape
        ref_o, ref_l = oracle.attention(batch.query_len, batch.context_len, batch.block_table,
                                        batch.q, kc, vc, num_q_heads=sh.num_q_heads,
                                        num_kv_heads=sh.num_kv_heads, head_dim_qk=sh.head_dim_qk,
                                        head_dim_v=sh.head_dim_v, block_size=sh.block_size,
                                        latent=sh.latent, tokens=tokens)
    if tokens is not None:
        out, lse = out[tokens], lse[tokens]
    assert np.isfinite(out).all() and np.isfinite(lse).all()
    eo = np.abs(out - ref_o).max()
    el = np.abs(lse - ref_l).max()
    assert eo <= O_TOL, f"max |dO| = {eo}"
    assert el <= LSE_TOL, f"max |dLSE| = {el}"
    return eo, el


def _sample_tokens(batch, per_seq_rows=6, seed=0):
    """Rows the oracle recomputes at full size: every decode row, and for each
    prefill chunk its first/last rows, tile boundaries and random rows."""
    rng = np.random.default_rng(seed)
    qs = batch.query_start
    toks = []
    for s in range(batch.num_seqs):
        q = int(batch.query_len[s])
        if q == 1:
            toks.append(qs[s])
            continue
        rows = {0, q - 1, min(63, q - 1), min(64, q - 1), min(127, q - 1), min(128, q - 1)}
        rows |= set(rng.integers(0, q, size=per_seq_rows).tolist())
        toks += [qs[s] + r for r in sorted(rows)]
    return np.asarray(sorted(set(toks)), np.int64)


def test_kv_append_bit_exact_whole_pool():
    batch = W.make_batch("tiny", seed=1)
    st = _step(batch)
    kc, vc = st.cache_bits()
    ref_k = oracle.kv_append(batch.k_cache, batch.k_new, batch.slot_mapping)
    ref_v = oracle.kv_append(batch.v_cache, batch.v_new, batch.slot_mapping)
    assert np.array_equal(kc, ref_k) and np.array_equal(vc, ref_v)


def test_kv_append_padding_and_range_flag():
    import paper_2606_04415_gb300 as fnpu
    batch = W.make_batch("tiny", seed=2)
    st = _step(batch)
    assert fnpu.check() == fnpu.FNPU_OK
    # padding slots (-1) are skipped; an out-of-range slot is skipped and flagged
    slots = batch.slot_mapping.copy()
    slots[::7] = -1
    nslot = batch.num_blocks * batch.shape.block_size
    slots[5] = nslot + 3
    k0 = st.k_cache.clone()
    v0 = st.v_cache.clone()
    sm = torch.from_numpy(slots).cuda()
    fnpu.kv_append(st.desc, st.k_new, st.v_new, sm, st.k_cache, st.v_cache)
    assert fnpu.check() == fnpu.FNPU_EDEVICE_RANGE
    assert fnpu.check() == fnpu.FNPU_OK  # cleared
    good = slots.copy()
    good[5] = -1
    ref_k = oracle.kv_append(k0.view(torch.int16).cpu().numpy().view(np.uint16), batch.k_new, good)
    ref_v = oracle.kv_append(v0.view(torch.int16).cpu().numpy().view(np.uint16), batch.v_new, good)
    kc, vc = st.cache_bits()
    assert np.array_equal(kc, ref_k) and np.array_equal(vc, ref_v)


def test_kv_append_full_size_bit_exact():
    batch = W.make_batch("qwen_coloc", seed=0)
    st = _step(batch)
    kc, vc = st.cache_bits()
    assert np.array_equal(kc, oracle.kv_append(batch.k_cache, batch.k_new, batch.slot_mapping))
    assert np.array_equal(vc, oracle.kv_append(batch.v_cache, batch.v_new, batch.slot_mapping))


NO_TC = 2  # FNPU_PLAN_NO_TCGEN05: prefill on the mma.sync path


@pytest.mark.parametrize("flags", [0, NO_TC])
@pytest.mark.parametrize("seed", [0, 1, 2])
def test_tiny_mixed_batch_all_rows(seed, flags):
    batch = W.make_batch("tiny", seed=seed)
    st = _step(batch, flags=flags)
    out, lse = st.results()
    _compare(batch, out, lse)


@pytest.mark.parametrize("split", [64, 128, 4096])
def test_decode_split_counts_agree(split):
    batch = W.make_batch("tiny", seed=5)
    st = _step(batch, split=split)
    out, lse = st.results()
    _compare(batch, out, lse)


def test_plan_reuse_runs_repeatedly():
    batch = W.make_batch("tiny", seed=6)
    st = _step(batch, split=64)
    out1, lse1 = st.results()
    for _ in range(3):
        st.run()
    out2, lse2 = st.results()
    assert np.array_equal(out1, out2) and np.array_equal(lse1, lse2)


def test_qwen_decode_full_size_all_rows():
    batch = W.make_batch("qwen_decode", seed=0)
    st = _step(batch)
    out, lse = st.results()
    _compare(batch, out, lse)


@pytest.mark.parametrize("flags", [0, NO_TC])
def test_qwen_prefill_full_size_sampled_rows(flags):
    batch = W.make_batch("qwen_prefill", seed=0)
    st = _step(batch, flags=flags)
    out, lse = st.results()
    _compare(batch, out, lse, tokens=_sample_tokens(batch))


def test_qwen_coloc_full_size_sampled_rows():
    batch = W.make_batch("qwen_coloc", seed=0)
    st = _step(batch)
    out, lse = st.results()
    _compare(batch, out, lse, tokens=_sample_tokens(batch, per_seq_rows=10))


@pytest.mark.parametrize("flags", [0, NO_TC])
@pytest.mark.parametrize("bs", [1, 16, 32, 64])
@pytest.mark.parametrize("dim", [64, 128])
def test_ragged_edges(bs, dim, flags):
    """ctx = 1 prefill, 1-row and ragged chunks, prefixes not on block edges."""
    sh = W.Shape(8, 2, dim, dim, bs, False)
    ql = [1, 1, 63, 65, 130, 1, 1, 7]
    ctx = [1, 37, 63, 100, 131, 1, 2, 7 + 91]
    ph = [0, 1, 0, 0, 0, 1, 1, 0]
    rng = np.random.default_rng(bs * 1000 + dim)
    batch = W.build_batch(sh, ql, ctx, ph, rng, name="ragged")
    st = _step(batch, flags=flags)
    out, lse = st.results()
    _compare(batch, out, lse)


def test_block_permutation_invariance_gpu():
    batch = W.make_batch("tiny", seed=7)
    st = _step(batch)
    out, lse = st.results()
    perm = np.random.default_rng(3).permutation(batch.num_blocks)
    kc = np.empty_like(batch.k_cache)
    vc = np.empty_like(batch.v_cache)
    kc[perm] = batch.k_cache
    vc[perm] = batch.v_cache
    b2 = W.Batch(**{**batch.__dict__, "k_cache": kc, "v_cache": vc,
                    "block_table": perm[batch.block_table].astype(np.int32),
                    "slot_mapping": (perm[batch.slot_mapping // 16] * 16 + batch.slot_mapping % 16)})
    st2 = _step(b2)
    out2, lse2 = st2.results()
    assert np.array_equal(out, out2) and np.array_equal(lse, lse2)


def test_decode_row_matches_prefill_row_gpu():
    """Decode of position t (decode kernel) vs row t of a prefill (prefill kernel)."""
    sh = W.SHAPES["qwen"]
    L = 300
    rng = np.random.default_rng(21)
    pre = W.build_batch(sh, [L], [L], [0], rng, name="pre", extra_bt_cols=0)
    st = _step(pre)
    out_p, lse_p = st.results()
    kc, vc = st.cache_bits()
    positions = [0, 15, 16, 150, 299]
    dec = W.Batch(name="dec", shape=sh, seed=0, query_len=np.ones(len(positions), np.int32),
                  context_len=np.asarray([p + 1 for p in positions], np.int32),
                  phase=np.ones(len(positions), np.uint8),
                  block_table=np.repeat(pre.block_table, len(positions), 0), num_blocks=pre.num_blocks,
                  q=pre.q[positions], k_new=pre.k_new[positions], v_new=pre.v_new[positions],
                  slot_mapping=pre.slot_mapping[positions], k_cache=kc, v_cache=vc)
    st2 = _step(dec)
    out_d, lse_d = st2.results()
    assert np.abs(out_d - out_p[positions]).max() <= O_TOL
    assert np.abs(lse_d - lse_p[positions]).max() <= LSE_TOL


def test_empty_batch_is_a_noop():
    import paper_2606_04415_gb300 as fnpu
    desc = fnpu.make_desc(4, 2, 64, 64, 16, 8)
    plan = fnpu.mixed_attn_plan(desc, np.zeros(0, np.int32), np.zeros(0, np.int32),
                                np.zeros(0, np.uint8), np.zeros((0, 1), np.int32))
    dummy = torch.zeros(16, dtype=torch.bfloat16, device="cuda")
    fnpu.mixed_attn_run(plan, dummy, dummy, dummy, dummy, dummy.float())
    assert fnpu.plan_check(plan) == fnpu.FNPU_OK
    assert plan.info()["prefill_items"] == 0 and plan.info()["decode_items"] == 0


@pytest.mark.parametrize("group", [1, 3, 7, 8])
def test_prefill_gqa_packing_groups(group):
    """tcgen05 tiles pack floor(128 / G) positions x G heads; sweep G."""
    sh = W.Shape(2 * group, 2, 128, 128, 16, False)
    rng = np.random.default_rng(100 + group)
    batch = W.build_batch(sh, [200, 37, 1], [200, 300, 50], [0, 0, 1], rng, name="gqa")
    st = _step(batch)
    out, lse = st.results()
    _compare(batch, out, lse)


def test_tc_and_mma_prefill_agree_on_coloc():
    batch = W.make_batch("qwen_coloc", seed=2)
    a = _step(batch).results()
    b = _step(batch, flags=NO_TC).results()
    assert np.abs(a[0] - b[0]).max() <= O_TOL and np.abs(a[1] - b[1]).max() <= LSE_TOL


@pytest.mark.parametrize("split", [0, 64, 192])
@pytest.mark.parametrize("bs", [16, 32, 64])
def test_decode_four_kv_heads_edges(bs, split):
    """Hkv = 4 decodes (the TMA-fed decode kernel): contexts shorter than a
    stage, not on stage or block edges, and several split lengths."""
    sh = W.Shape(28, 4, 128, 128, bs, False)
    ctx = [1, 2, 15, 16, 17, 63, 64, 65, 300, 1000, 2049]
    rng = np.random.default_rng(7 * bs + split)
    batch = W.build_batch(sh, [1] * len(ctx), ctx, [1] * len(ctx), rng, name="dec4")
    st = _step(batch, split=split)
    out, lse = st.results()
    _compare(batch, out, lse)


@pytest.mark.parametrize("bs", [16, 64])
@pytest.mark.parametrize("dim", [64, 128])
def test_prefill_key_splits(bs, dim):
    """Few prefill tiles over long cached prefixes: the planner splits their
    keys across CTAs and the last split merges the partial results. Chunks of
    one row, ragged chunks and prefixes off block edges, beside decodes."""
    sh = W.Shape(8, 2, dim, dim, bs, False)
    ql = [40, 1, 200, 1, 77]
    ctx = [3040, 5000, 2500, 900, 77 + 1999]
    ph = [0, 0, 0, 1, 0]
    rng = np.random.default_rng(31 * bs + dim)
    batch = W.build_batch(sh, ql, ctx, ph, rng, name="ksplit")
    st = _step(batch)
    units = sum((q + 63) // 64 * 2 for q, p in zip(ql, ph) if p == 0)  # tile pairs x kv heads
    assert st.plan.info()["prefill_items"] > units, "expected the planner to split prefill keys"
    out, lse = st.results()
    _compare(batch, out, lse)
    for _ in range(2):  # the merge counters are back at zero after a run
        st.run()
    out2, lse2 = st.results()
    assert np.array_equal(out, out2) and np.array_equal(lse, lse2)


SEPARATE = 1  # FNPU_PLAN_SEPARATE_LAUNCHES


@pytest.mark.parametrize("share", [0, 2, 50])
def test_colocated_launch_matches_separate_launches(share):
    """Prefill and decode launched together on split SMs (any decode share)
    give the results of the two phases launched one after the other."""
    sh = W.SHAPES["qwen"]
    rng = np.random.default_rng(77)
    ql = [300, 1, 1, 129, 1] + [1] * 12
    ctx = [300 + 2000, 700, 1500, 129 + 40, 33] + list(rng.integers(20, 3000, size=12))
    ph = [0, 1, 1, 0, 1] + [1] * 12
    batch = W.build_batch(sh, ql, ctx, ph, rng, name="coloc_small")
    a_out, a_lse = _step(batch, share=share).results()
    b_out, b_lse = _step(batch, flags=SEPARATE).results()
    _compare(batch, a_out, a_lse)
    assert np.abs(a_out - b_out).max() <= O_TOL and np.abs(a_lse - b_lse).max() <= LSE_TOL


@pytest.mark.parametrize("flags", [0, NO_TC])
@pytest.mark.parametrize("bs", [16, 32, 64])
def test_mla_small_mixed_batch_all_rows(bs, flags):
    """Absorbed MLA (128 heads on one 576-wide latent, V = its first 512
    columns): prefill chunks with and without prefix, decodes long enough to
    be split and merged, ragged lengths (tiles past a sequence's last block,
    pieces ending inside a block); every row against the oracle, on the
    tcgen05 kernel (d_v halves, merge kernel) and on the mma.sync kernel. The
    latent KV append is bit-exact."""
    sh = W.Shape(128, 1, 576, 512, bs, True)
    ql = [7, 1, 1, 33, 1, 1]
    ctx = [7, 2500, 1, 33 + 450, 777, 3100]
    ph = [0, 1, 1, 0, 1, 1]
    rng = np.random.default_rng(500 + bs)
    batch = W.build_batch(sh, ql, ctx, ph, rng, name="mla_small")
    st = _step(batch, flags=flags)
    kc, _ = st.cache_bits()
    assert np.array_equal(kc, oracle.kv_append(batch.k_cache, batch.k_new, batch.slot_mapping))
    out, lse = st.results()
    _compare(batch, out, lse)
    st.run()  # merge counters back at zero: a second run is identical
    out2, lse2 = st.results()
    assert np.array_equal(out, out2) and np.array_equal(lse, lse2)


def test_mla_coloc_full_size_sampled_rows():
    """The DeepSeek-R1-shaped co-located step at full size (1024-token
    prefill + 256 decodes up to 16K keys); the oracle recomputes a sample of
    decode rows and prefill rows."""
    batch = W.make_batch("mla_coloc", seed=0)
    st = _step(batch)
    out, lse = st.results()
    rng = np.random.default_rng(1)
    qs = batch.query_start
    dec = [int(qs[s]) for s in np.flatnonzero(batch.phase == 1)]
    pre = [s for s in range(batch.num_seqs) if batch.phase[s] == 0]
    toks = sorted(rng.choice(dec, size=12, replace=False).tolist())
    for s in pre:
        q = int(batch.query_len[s])
        toks += [int(qs[s]) + r for r in sorted({0, 1, 63, 64, q - 1, int(rng.integers(0, q))})]
    _compare(batch, out, lse, tokens=np.asarray(sorted(set(toks)), np.int64))


@pytest.mark.parametrize("heads", [64, 256])
def test_mla_other_head_counts(heads):
    """Latent attention with 64 or 256 query heads (the mma.sync kernel: the
    tcgen05 one takes exactly 128 rows per token); a split decode and a
    prefill chunk on a prefix; every row against the oracle."""
    sh = W.Shape(heads, 1, 576, 512, 64, True)
    ql, ctx, ph = [1, 20, 1], [2200, 20 + 70, 300], [1, 0, 1]
    rng = np.random.default_rng(900 + heads)
    batch = W.build_batch(sh, ql, ctx, ph, rng, name="mla_heads")
    out, lse = _step(batch).results()
    _compare(batch, out, lse)


def test_mla_long_decode_many_pieces():
    """One 40000-key latent decode beside a short one: the planner cuts it into
    about 40 pieces of 16 tiles, so the d_v = 512 merge runs more than one
    32-split chunk (running maximum across chunks)."""
    sh = W.Shape(128, 1, 576, 512, 64, True)
    ql, ctx, ph = [1, 1], [40000, 77], [1, 1]
    rng = np.random.default_rng(910)
    batch = W.build_batch(sh, ql, ctx, ph, rng, name="mla_long")
    st = _step(batch)
    assert st.plan.info()["prefill_items"] > 2 * 32
    out, lse = st.results()
    _compare(batch, out, lse)


@pytest.mark.parametrize("split", [0, 128])
def test_decode_long_token_many_splits(split):
    """A lone 8192-key decode on the TMA decode kernel: 128-key items (chosen
    by the planner for so few keys, or asked for) give it 64 splits, two
    32-split chunks in the merge kernel."""
    sh = W.SHAPES["qwen"]
    ql, ctx, ph = [1, 1], [8192, 300], [1, 1]
    rng = np.random.default_rng(920)
    batch = W.build_batch(sh, ql, ctx, ph, rng, name="long_decode")
    st = _step(batch, split=split)
    assert st.plan.info()["decode_items"] >= 64
    out, lse = st.results()
    _compare(batch, out, lse)


@pytest.mark.parametrize("seed", [0, 1])
def test_decode_many_short_sequences(seed):
    """300 decodes of 1..700 keys: more items than resident CTAs, so CTAs
    take several items from the queue; also planned for 64 SMs."""
    sh = W.SHAPES["qwen"]
    rng = np.random.default_rng(950 + seed)
    ctx = rng.integers(1, 701, size=300).tolist()
    batch = W.build_batch(sh, [1] * 300, ctx, [1] * 300, rng, name="short_decodes")
    for sms in (0, 64):
        st = _step(batch, sms=sms)
        out, lse = st.results()
        _compare(batch, out, lse)


def test_decode_longest_context_split_cap():
    """A 100000-key decode beside short ones: items of 448 keys (the planner
    keeps a token to at most 256 splits), about 224 partials merged in seven
    32-split chunks."""
    sh = W.SHAPES["qwen"]
    ql, ctx, ph = [1, 1, 1], [100000, 1000, 17], [1, 1, 1]
    rng = np.random.default_rng(930)
    batch = W.build_batch(sh, ql, ctx, ph, rng, name="longest_decode")
    st = _step(batch)
    assert st.plan.info()["decode_items"] > 200
    out, lse = st.results()
    _compare(batch, out, lse)


def test_mla_longest_context():
    """A 131072-key latent decode and a short prefill: about 128 pieces of
    16 tiles, merged in four 32-split chunks at d_v 512."""
    sh = W.Shape(128, 1, 576, 512, 64, True)
    ql, ctx, ph = [1, 9], [131072, 9], [1, 0]
    rng = np.random.default_rng(940)
    batch = W.build_batch(sh, ql, ctx, ph, rng, name="mla_longest")
    st = _step(batch)
    assert st.plan.info()["prefill_items"] > 2 * 96
    out, lse = st.results()
    _compare(batch, out, lse)


def test_dispatch_feedback_loop_on_colocated_steps():
    """Phase times of co-located runs feed the decode-share controller for a
    few steps (the dispatch ratio of Sec. 3.4); each step's plan uses the
    share the last one chose, and the output stays correct."""
    import paper_2606_04415_gb300 as fnpu
    sh = W.SHAPES["qwen"]
    rng = np.random.default_rng(950)
    ql = [512] + [1] * 48
    ctx = [512 + 3000] + rng.integers(200, 6000, size=48).tolist()
    ph = [0] + [1] * 48
    batch = W.build_batch(sh, ql, ctx, ph, rng, name="dispatch_loop")
    share = 24
    st = _step(batch, share=share)
    shares = [share]
    for _ in range(4):
        pre, dec = fnpu.plan_phase_ms(st.plan)
        assert 0 < pre < 1000 and 0 < dec < 1000
        share = fnpu.dispatch_next_share(share, pre, dec)
        assert 1 <= share <= 50
        shares.append(share)
        st.replan(fnpu.PlanOpts(0, share, 0, 0))
        st.attend()
        assert fnpu.plan_check(st.plan) == fnpu.FNPU_OK
    out, lse = st.results()
    _compare(batch, out, lse)


def test_phase_times_need_a_colocated_plan_that_ran():
    import paper_2606_04415_gb300 as fnpu
    from paper_2606_04415_gb300.step import DeviceStep
    sh = W.SHAPES["qwen"]
    rng = np.random.default_rng(960)
    dec_only = W.build_batch(sh, [1, 1], [700, 90], [1, 1], rng, name="dec_only")
    st = _step(dec_only)
    with pytest.raises(fnpu.FnpuError) as e:
        fnpu.plan_phase_ms(st.plan)
    assert e.value.code == fnpu.FNPU_EUNSUPPORTED
    mixed = W.build_batch(sh, [300, 1], [300, 900], [0, 1], rng, name="mixed_unrun")
    fresh = DeviceStep(mixed)  # planned, never run
    with pytest.raises(fnpu.FnpuError) as e:
        fnpu.plan_phase_ms(fresh.plan)
    assert e.value.code == fnpu.FNPU_EINVAL


@pytest.mark.parametrize("flags", [0, NO_TC])
def test_multi_token_decode(flags):
    """Decode steps of several tokens (speculative verification of 2, 4 and 7
    draft tokens) beside one-token decodes and a prefill chunk: the
    multi-token rows take the prefill path with their causal mask; every row
    against the oracle."""
    sh = W.SHAPES["qwen"]
    ql = [2, 4, 7, 1, 1, 300]
    ctx = [2000, 513, 4096 + 7, 1000, 77, 300 + 900]
    ph = [1, 1, 1, 1, 1, 0]
    rng = np.random.default_rng(970)
    batch = W.build_batch(sh, ql, ctx, ph, rng, name="multi_token_decode")
    out, lse = _step(batch, flags=flags).results()
    _compare(batch, out, lse)


def test_mla_multi_token_decode():
    """A three-token latent decode (speculative verification) beside a
    one-token one."""
    sh = W.Shape(128, 1, 576, 512, 64, True)
    ql, ctx, ph = [3, 1], [1500, 700], [1, 1]
    rng = np.random.default_rng(980)
    batch = W.build_batch(sh, ql, ctx, ph, rng, name="mla_multi_token")
    out, lse = _step(batch).results()
    _compare(batch, out, lse)


GREEN = 4  # FNPU_PLAN_GREEN_CONTEXTS


@pytest.mark.parametrize("share", [0, 20])
def test_green_context_partitions(share):
    """Co-location with the SM split enforced by green contexts (disjoint SM
    partitions for the two phases) gives the results of separate launches;
    the dispatch feedback works on such plans too."""
    import paper_2606_04415_gb300 as fnpu
    sh = W.SHAPES["qwen"]
    rng = np.random.default_rng(77)
    ql = [300, 1, 1, 129, 1] + [1] * 12
    ctx = [300 + 2000, 700, 1500, 129 + 40, 33] + list(rng.integers(20, 3000, size=12))
    ph = [0, 1, 1, 0, 1] + [1] * 12
    batch = W.build_batch(sh, ql, ctx, ph, rng, name="coloc_green")
    st = _step(batch, share=share, flags=GREEN)
    a_out, a_lse = st.results()
    b_out, b_lse = _step(batch, flags=SEPARATE).results()
    _compare(batch, a_out, a_lse)
    assert np.abs(a_out - b_out).max() <= O_TOL and np.abs(a_lse - b_lse).max() <= LSE_TOL
    pre, dec = fnpu.plan_phase_ms(st.plan)
    assert pre > 0 and dec > 0


@pytest.mark.parametrize("flags", [0, 4])
def test_replan_reuses_the_plan_across_steps(flags):
    """fnpu_mixed_attn_replan: one plan re-planned for steps of other shapes
    and decode shares (a larger step grows the workspace, a smaller one
    reuses it; green-context partitions are rebuilt when the share asks for
    another size), each run checked against the oracle."""
    import paper_2606_04415_gb300 as fnpu
    from paper_2606_04415_gb300.step import DeviceStep
    big = W.make_batch("qwen_coloc", seed=2)
    # a small step over a pool of the same descriptor (a re-plan keeps the
    # plan's descriptor: same heads, dims, block size and pool size)
    rng = np.random.default_rng(11)
    small = W.build_batch(W.SHAPES["qwen"], [70, 1, 1, 3], [300, 100, 500, 1000], [0, 1, 1, 1], rng,
                          name="small", num_blocks=big.num_blocks)
    st = DeviceStep(small, opts=fnpu.PlanOpts(0, 0, 0, flags))
    st.run()
    _compare(small, *st.results())
    ws0 = st.plan.info()["workspace_bytes"]
    sbig = DeviceStep(big, opts=fnpu.PlanOpts(0, 20, 0, flags))
    tokens = _sample_tokens(big)
    for share in (20, 12, 20):
        sbig.replan(fnpu.PlanOpts(0, share, 0, flags))
        sbig.run()  # (appending the same new rows again stores the same bits)
        assert fnpu.plan_check(sbig.plan) == fnpu.FNPU_OK
        _compare(big, *sbig.results(), tokens=tokens)
    # the small plan re-planned for the big step (the workspace grows), then back
    b = big
    fnpu.mixed_attn_replan(st.plan, b.query_len, b.context_len, b.phase, b.block_table,
                           opts=fnpu.PlanOpts(0, 16, 0, flags))
    assert st.plan.info()["workspace_bytes"] > ws0
    out = torch.empty_like(sbig.out)
    lse = torch.empty_like(sbig.lse)
    fnpu.mixed_attn_run(st.plan, sbig.q, sbig.k_cache, sbig.v_cache, out, lse)
    assert fnpu.plan_check(st.plan) == fnpu.FNPU_OK
    torch.cuda.synchronize()
    _compare(big, out.float().cpu().numpy(), lse.cpu().numpy(), tokens=tokens)
    grown = st.plan.info()["workspace_bytes"]
    st.replan(fnpu.PlanOpts(0, 0, 0, flags))
    assert st.plan.info()["workspace_bytes"] == grown  # kept, not shrunk
    st.attend()
    assert fnpu.plan_check(st.plan) == fnpu.FNPU_OK
    _compare(small, *st.results())


def test_replan_rejects_bad_metadata_and_keeps_the_plan():
    import paper_2606_04415_gb300 as fnpu
    batch = W.make_batch("tiny", seed=12)
    st = _step(batch)
    bad_ctx = batch.context_len.copy()
    bad_ctx[0] = batch.query_len[0] - 1  # ctx < q
    with pytest.raises(fnpu.FnpuError) as e:
        fnpu.mixed_attn_replan(st.plan, batch.query_len, bad_ctx, batch.phase, batch.block_table)
    assert e.value.code == fnpu.FNPU_EINVAL
    st.attend()
    assert fnpu.plan_check(st.plan) == fnpu.FNPU_OK
    _compare(batch, *st.results())


def test_planner_decode_share_is_reported():
    """A co-located plan reports the decode share it uses: the one it was given
    (to the rounding of SMs), or the planner's own choice, inside the
    controller's range; a plan with one phase has none."""
    import paper_2606_04415_gb300 as fnpu
    from paper_2606_04415_gb300.step import DeviceStep
    st = DeviceStep(W.make_batch("qwen_coloc", seed=0), opts=fnpu.PlanOpts(0, 20, 0, 0))
    assert abs(fnpu.plan_decode_share(st.plan) - 20) <= 1
    st.replan(fnpu.PlanOpts(0, 0, 0, 0))
    assert 1 <= fnpu.plan_decode_share(st.plan) <= 50
    st.run()
    out, lse = st.results()
    _compare(st.batch, out, lse, tokens=_sample_tokens(st.batch, per_seq_rows=4))
    one = DeviceStep(W.make_batch("qwen_prefill", seed=0))
    with pytest.raises(fnpu.FnpuError) as e:
        fnpu.plan_decode_share(one.plan)
    assert e.value.code == fnpu.FNPU_EUNSUPPORTED


@pytest.mark.parametrize("what", ["q", "cache"])
def test_prefill_waits_for_the_kernel_before_it(what):
    """The tcgen05 prefill grid is a programmatic dependent launch of the kernel
    before it on the stream. Here that kernel is not the library's append but a
    copy that writes the queries (or the whole cache) the step then reads,
    replacing NaN: every output must still match the oracle, so the prefill's
    loaders waited for the copy to finish."""
    batch = _coloc_small_batch()
    import paper_2606_04415_gb300 as fnpu
    from paper_2606_04415_gb300.step import DeviceStep
    st = DeviceStep(batch)
    st.append()
    torch.cuda.synchronize()
    dst = st.q if what == "q" else st.k_cache
    good = dst.clone()
    dst.fill_(float("nan"))
    torch.cuda.synchronize()
    dst.copy_(good)  # the kernel just before the attention on the same stream
    st.attend()
    out, lse = st.results()
    assert fnpu.plan_check(st.plan) == fnpu.FNPU_OK
    _compare(batch, out, lse)


def _coloc_small_batch():
    sh = W.SHAPES["qwen"]
    rng = np.random.default_rng(21)
    ql = [400, 1, 1, 129, 1] + [1] * 12
    ctx = [400 + 1700, 700, 1500, 129 + 40, 33] + list(rng.integers(20, 3000, size=12))
    ph = [0, 1, 1, 0, 1] + [1] * 12
    return W.build_batch(sh, ql, ctx, ph, rng, name="coloc_pdl")


def test_prefill_chunk_on_a_very_long_prefix():
    """A Qwen-shape chunk of 256 tokens on a 40000-token prefix (316 key tiles
    per item), beside a few decodes: long tile loops, key splits across CTAs
    and their merge at scale; sampled rows against the oracle."""
    sh = W.SHAPES["qwen"]
    rng = np.random.default_rng(404)
    ql = [256, 1, 1, 1]
    ctx = [40000 + 256, 3000, 17, 40001]
    ph = [0, 1, 1, 1]
    batch = W.build_batch(sh, ql, ctx, ph, rng, name="long_prefix")
    st = _step(batch)
    out, lse = st.results()
    qs = batch.query_start
    toks = np.asarray(sorted({int(qs[0]) + r for r in (0, 1, 35, 36, 127, 200, 255)} | {int(qs[s]) for s in (1, 2, 3)}),
                      np.int64)
    _compare(batch, out, lse, tokens=toks)


@pytest.mark.parametrize("seed", [1, 3, 7])
def test_qwen_coloc_other_seeds_sampled_rows(seed):
    """The co-located Qwen workload at other prefix draws (shorter and longer
    prefixes, other decode shares chosen by the planner): sampled rows."""
    batch = W.make_batch("qwen_coloc", seed=seed)
    st = _step(batch)
    out, lse = st.results()
    _compare(batch, out, lse, tokens=_sample_tokens(batch, per_seq_rows=6, seed=seed))
