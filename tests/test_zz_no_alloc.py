"""The decode entry point that allocates nothing (fnpu_decode_attn_noalloc).

It exists for callers that may not call cudaMalloc (code confined to memory
another framework reserved, or a process whose device memory is fixed at
start): it keeps its split scratch in a fixed array inside the library. These
tests call it through the C ABI, twice in a row where it matters, and check
the results against the fp64 oracle and against the planned path
(fnpu_mixed_attn_plan + fnpu_mixed_attn_run) on the same decode batch, within
the parity tolerances used by the other GPU tests. One test feeds it a context
longer than the bound it was given and a block id outside the pool, laid out
so that even an unchecked read would stay inside allocated memory, and checks
that the kernel skips them and raises the device error flag.

The file is collected last and also passes on its own in a fresh process.
"""
import numpy as np
import pytest

import oracle
import workloads as W

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

O_TOL = 2e-2
LSE_TOL = 1e-3


def _need_gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def _oracle_after_append(batch):
    ref_o, ref_l, _, _ = oracle.run_step(batch)
    return ref_o, ref_l


@pytest.mark.parametrize("split_keys", [0, 256])
def test_noalloc_decode_matches_oracle_and_planned_path_twice(split_keys):
    _need_gpu()
    import paper_2606_04415_gb300 as fnpu
    from paper_2606_04415_gb300.step import DeviceStep

    batch = W.make_batch("qwen_decode", seed=3)
    st = DeviceStep(batch)
    st.run()  # append + planned attention
    plan_o, plan_l = st.results()
    ref_o, ref_l = _oracle_after_append(batch)

    ctx = torch.from_numpy(batch.context_len).cuda()
    bt = torch.from_numpy(batch.block_table).cuda()
    T, Hq, D = st.out.shape
    for call in range(2):
        out = torch.full((T, Hq, D), float("nan"), dtype=torch.bfloat16, device="cuda")
        lse = torch.full((T, Hq), float("nan"), dtype=torch.float32, device="cuda")
        fnpu.decode_attn_noalloc(st.desc, ctx, bt, int(batch.context_len.max()), st.q, st.k_cache,
                                 st.v_cache, out, lse, split_keys=split_keys)
        torch.cuda.synchronize()
        o = out.float().cpu().numpy()
        l = lse.cpu().numpy()
        assert np.isfinite(o).all() and np.isfinite(l).all(), f"call {call}"
        assert np.abs(o - ref_o).max() <= O_TOL, f"call {call}: oracle"
        assert np.abs(l - ref_l).max() <= LSE_TOL, f"call {call}: oracle"
        assert np.abs(o - plan_o).max() <= O_TOL, f"call {call}: planned path"
        assert np.abs(l - plan_l).max() <= LSE_TOL, f"call {call}: planned path"
    assert fnpu.check() == fnpu.FNPU_OK


def test_noalloc_decode_d64_partial_group_single_and_multi_split():
    """head_dim 64 with 3 query heads per kv head (the 8 MMA columns only
    partly filled); contexts from 1 key up to and past one split, so that
    single-split sequences (written directly, no counters) and split ones
    (merged by the last split) both occur, checked against the oracle and the
    planned path on two calls in a row."""
    _need_gpu()
    import paper_2606_04415_gb300 as fnpu
    from paper_2606_04415_gb300.step import DeviceStep

    shape = W.Shape(6, 2, 64, 64, 16, False)
    ctx = np.array([1, 2, 15, 16, 17, 63, 64, 65, 127, 128, 129, 200, 255, 256, 257, 300], np.int32)
    rng = np.random.default_rng(41)
    batch = W.build_batch(shape, np.ones_like(ctx), ctx, np.ones(len(ctx), np.uint8), rng, name="noalloc_d64")
    st = DeviceStep(batch)
    st.run()
    plan_o, plan_l = st.results()
    ref_o, ref_l = _oracle_after_append(batch)

    dctx = torch.from_numpy(batch.context_len).cuda()
    bt = torch.from_numpy(batch.block_table).cuda()
    T, Hq, D = st.out.shape
    for call in range(2):
        out = torch.full((T, Hq, D), float("nan"), dtype=torch.bfloat16, device="cuda")
        lse = torch.full((T, Hq), float("nan"), dtype=torch.float32, device="cuda")
        fnpu.decode_attn_noalloc(st.desc, dctx, bt, int(ctx.max()), st.q, st.k_cache, st.v_cache, out, lse,
                                 split_keys=128)
        torch.cuda.synchronize()
        o = out.float().cpu().numpy()
        l = lse.cpu().numpy()
        assert np.isfinite(o).all() and np.isfinite(l).all(), f"call {call}"
        assert np.abs(o - ref_o).max() <= O_TOL, f"call {call}: oracle"
        assert np.abs(l - ref_l).max() <= LSE_TOL, f"call {call}: oracle"
        assert np.abs(o - plan_o).max() <= O_TOL, f"call {call}: planned path"
        assert np.abs(l - plan_l).max() <= LSE_TOL, f"call {call}: planned path"
    assert fnpu.check() == fnpu.FNPU_OK


def test_noalloc_rejects_requests_beyond_its_scratch():
    _need_gpu()
    import paper_2606_04415_gb300 as fnpu
    desc = fnpu.make_desc(28, 4, 128, 128, 16, 1 << 20)
    n = 4096
    ctx = torch.full((n,), 16384, dtype=torch.int32, device="cuda")
    bt = torch.zeros((n, 1024), dtype=torch.int32, device="cuda")
    dummy = torch.zeros(16, dtype=torch.bfloat16, device="cuda")
    with pytest.raises(fnpu.FnpuError) as e:
        fnpu.decode_attn_noalloc(desc, ctx, bt, 16384, dummy, dummy, dummy, dummy, dummy.float(),
                                 split_keys=64)
    assert e.value.code == fnpu.FNPU_EINVAL


def test_noalloc_skips_and_flags_out_of_range_context_and_block():
    """Sequence 1's context exceeds the max_context_len the call was given and
    sequence 2's block table names a block past desc.num_blocks. The buffers are
    laid out so that neither would leave allocated memory even unchecked: the
    block table is wide enough for the longer context, and the pools hold 8
    blocks more than the descriptor declares. The kernel must skip both (no
    write to sequence 1's rows), raise the flag, and leave the other sequences
    right."""
    _need_gpu()
    import paper_2606_04415_gb300 as fnpu

    shape = W.Shape(6, 2, 64, 64, 16, False)
    ctx = np.array([40, 100, 70, 33], np.int32)
    rng = np.random.default_rng(7)
    batch = W.build_batch(shape, np.ones_like(ctx), ctx, np.ones(len(ctx), np.uint8), rng, name="noalloc_guard",
                          extra_bt_cols=8)
    # reference on the appended cache, before the bad inputs are made
    ref_o, ref_l = _oracle_after_append(batch)
    kc = oracle.kv_append(batch.k_cache, batch.k_new, batch.slot_mapping)
    vc = oracle.kv_append(batch.v_cache, batch.v_new, batch.slot_mapping)
    nb = batch.num_blocks
    pad = np.zeros((8,) + kc.shape[1:], np.uint16)  # 8 allocated blocks past the declared pool
    k_pool = torch.from_numpy(np.concatenate([kc, pad]).view(np.int16)).cuda().view(torch.bfloat16)
    v_pool = torch.from_numpy(np.concatenate([vc, pad]).view(np.int16)).cuda().view(torch.bfloat16)
    q = torch.from_numpy(batch.q.view(np.int16)).cuda().view(torch.bfloat16)
    desc = fnpu.make_desc(6, 2, 64, 64, 16, nb)

    max_ctx = 80           # sequence 1 (100 keys) is beyond it
    bt = batch.block_table.copy()
    assert bt.shape[1] * 16 >= 100  # its row still covers 100 keys
    bt[2, 1] = nb + 3      # sequence 2: a block id past the declared pool, inside the allocation
    dctx = torch.from_numpy(ctx).cuda()
    dbt = torch.from_numpy(bt).cuda()
    T, Hq = len(ctx), 6
    out = torch.full((T, Hq, 64), float("nan"), dtype=torch.bfloat16, device="cuda")
    lse = torch.full((T, Hq), float("nan"), dtype=torch.float32, device="cuda")
    fnpu.decode_attn_noalloc(desc, dctx, dbt, max_ctx, q, k_pool, v_pool, out, lse, split_keys=64)
    assert fnpu.check() == fnpu.FNPU_EDEVICE_RANGE
    assert fnpu.check() == fnpu.FNPU_OK  # read and cleared
    o = out.float().cpu().numpy()
    l = lse.cpu().numpy()
    assert np.isnan(o[1]).all() and np.isnan(l[1]).all()  # skipped: left as it was
    for s in (0, 3):
        assert np.abs(o[s] - ref_o[s]).max() <= O_TOL
        assert np.abs(l[s] - ref_l[s]).max() <= LSE_TOL
