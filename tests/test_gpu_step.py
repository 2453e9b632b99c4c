"""fnpu_mixed_step: the append and the attention of a step in one call.

By default the call is fnpu_kv_append then fnpu_mixed_attn_run (the other GPU
tests run their steps through it). With FNPU_PLAN_FUSED_APPEND, where the
plan's prefill runs on the tcgen05 kernel over a bf16 cache, that kernel's
CTAs write the prefill-path rows themselves (a cooperative grid that waits for
all its CTAs before reading the cache) and a small kernel writes the decode
rows ahead of the decode kernel. Either way the pools and the outputs must be
those of the two calls bit for bit, and those match the oracle.
"""
import numpy as np
import pytest

import oracle
import workloads as W

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

O_TOL = 2e-2
LSE_TOL = 1e-3
SEPARATE, NO_TC, GREEN, FUSED = 1, 2, 4, 8


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2606_04415_gb300 as fnpu
    fnpu.load()


def _two_ways(batch, share=0, flags=0, kv_fp8=False, pool_init=None, fused=True):
    """(step through fnpu_mixed_step, with the fused append when `fused`;
    step through the two calls), each on fresh pools."""
    import paper_2606_04415_gb300 as fnpu
    from paper_2606_04415_gb300.step import DeviceStep
    one = DeviceStep(batch, opts=fnpu.PlanOpts(0, share, 0, flags | (FUSED if fused else 0)), kv_fp8=kv_fp8,
                     pool_init=pool_init)
    one.run()
    two = DeviceStep(batch, opts=fnpu.PlanOpts(0, share, 0, flags), kv_fp8=kv_fp8, pool_init=pool_init)
    two.append()
    two.attend()
    for st in (one, two):
        assert fnpu.plan_check(st.plan) == fnpu.FNPU_OK
    assert fnpu.check() == fnpu.FNPU_OK
    return one, two


def _same(one, two):
    o1, l1 = one.results()
    o2, l2 = two.results()
    assert np.array_equal(o1, o2) and np.array_equal(l1, l2), "outputs differ from the two calls"
    for a, b in zip(one.cache_bits(), two.cache_bits()):
        assert np.array_equal(a, b), "pools differ from the two calls"
    return o1, l1


def _coloc_small():
    rng = np.random.default_rng(31)
    ql = [300, 1, 1, 129, 1, 5, 1] + [1] * 10
    ctx = [300 + 1500, 700, 1500, 129, 33, 5 + 900, 2] + list(rng.integers(20, 3000, size=10))
    ph = [0, 1, 1, 0, 1, 1, 1] + [1] * 10
    return W.build_batch(W.SHAPES["qwen"], ql, ctx, ph, rng, name="step_coloc")


@pytest.mark.parametrize("share", [0, 3, 30])
def test_step_matches_two_calls_colocated(share):
    """Co-located Qwen-shape step (chunks on prefixes, a chunk without one,
    multi-token and one-token decodes) at three decode shares."""
    batch = _coloc_small()
    one, two = _two_ways(batch, share=share)
    assert one.plan.info()["launches_per_run"] >= 2
    out, lse = _same(one, two)
    ref_o, ref_l, _, _ = oracle.run_step(batch)
    assert np.abs(out - ref_o).max() <= O_TOL and np.abs(lse - ref_l).max() <= LSE_TOL


@pytest.mark.parametrize("wl", ["qwen_coloc", "qwen_prefill"])
def test_step_matches_two_calls_full_size(wl):
    """The bench workloads at full size: the co-located step and the
    prefill-only step (no decode rows: the prefill grid appends every row)."""
    one, two = _two_ways(W.make_batch(wl, seed=2))
    _same(one, two)


@pytest.mark.parametrize("flags", [SEPARATE, NO_TC, GREEN])
def test_step_other_launch_modes(flags):
    """Separate launches (the fused prefill after the decode rows' append and
    the decode), the mma.sync prefill and green contexts (both of which keep
    the two calls inside fnpu_mixed_step)."""
    import paper_2606_04415_gb300 as fnpu
    batch = _coloc_small()
    try:
        one, two = _two_ways(batch, share=20, flags=flags)
    except fnpu.FnpuError as e:
        if flags == GREEN and e.code == fnpu.FNPU_EUNSUPPORTED:
            pytest.skip("green contexts unavailable")
        raise
    _same(one, two)


@pytest.mark.parametrize("bs,dim", [(32, 128), (64, 64), (16, 64)])
def test_step_other_shapes(bs, dim):
    """Two kv heads, other block sizes and head widths (the mma.sync decode
    kernel beside the tcgen05 prefill, one phase after the other); padding
    slots (-1) among the new rows are skipped."""
    sh = W.Shape(8, 2, dim, dim, bs, False)
    rng = np.random.default_rng(bs + dim)
    ql, ctx, ph = [1, 63, 130, 1, 7], [37, 63, 131 + 200, 1, 7 + 40], [1, 0, 0, 1, 1]
    batch = W.build_batch(sh, ql, ctx, ph, rng, name="step_shapes")
    one, two = _two_ways(batch)
    _same(one, two)


def test_step_fp8_cache_keeps_two_calls():
    """Over the FP8 cache the step is the quantising append, then the run."""
    import paper_2606_04415_gb300 as fnpu
    batch = _coloc_small()
    init = W.stale_pool_bytes(batch.num_blocks * fnpu.FP8_BLOCK_BYTES, 5)
    one, two = _two_ways(batch, kv_fp8=True, pool_init=init)
    _same(one, two)


def test_step_default_is_the_two_calls():
    """Without the flag the step is the append, then the run."""
    one, two = _two_ways(_coloc_small(), fused=False)
    _same(one, two)


def test_step_flags_a_slot_past_the_pool():
    """A prefill row whose slot lies past the pool: nothing is written for it,
    the library-wide flag reports FNPU_EDEVICE_RANGE (as for fnpu_kv_append),
    and the plan itself stays clean."""
    import paper_2606_04415_gb300 as fnpu
    from paper_2606_04415_gb300.step import DeviceStep
    batch = _coloc_small()
    st = DeviceStep(batch, opts=fnpu.PlanOpts(0, 0, 0, FUSED))
    pool = int(batch.num_blocks * batch.shape.block_size)
    bad = st.slot_mapping.clone()
    bad[3] = pool + 5  # a row of the first (prefill) sequence
    before = [x.copy() for x in st.cache_bits()]
    fnpu.mixed_step(st.plan, st.k_new, st.v_new, bad, st.q, st.k_cache, st.v_cache, st.out, st.lse)
    assert fnpu.plan_check(st.plan) == fnpu.FNPU_OK
    assert fnpu.check() == fnpu.FNPU_EDEVICE_RANGE
    assert fnpu.check() == fnpu.FNPU_OK  # read and cleared
    after = st.cache_bits()
    sm = batch.slot_mapping
    keep = np.ones(pool, bool)
    keep[sm[sm >= 0]] = False  # the slots of the other rows were written
    for a, b in zip(before, after):
        a = a.reshape(pool, -1)
        b = b.reshape(pool, -1)
        assert np.array_equal(a[keep], b[keep]), "a slot outside the step's rows was written"


def test_step_runs_repeatedly():
    """The append count returns to zero after every run: ten steps in a row,
    then the same outputs."""
    import paper_2606_04415_gb300 as fnpu
    from paper_2606_04415_gb300.step import DeviceStep
    batch = _coloc_small()
    st = DeviceStep(batch, opts=fnpu.PlanOpts(0, 0, 0, FUSED))
    st.run()
    o1, l1 = st.results()
    for _ in range(10):
        st.run()
    o2, l2 = st.results()
    assert fnpu.plan_check(st.plan) == fnpu.FNPU_OK
    assert np.array_equal(o1, o2) and np.array_equal(l1, l2)
