"""Randomised mixed steps against the fp64 oracle, every query row (GQA and
absorbed latent attention).

Each case draws a head shape (GQA groups 1 to 8, head widths 64 and 128,
block sizes 16 to 64), a mix of sequences (one-token decodes, multi-token
decodes, prefill chunks with and without a cached prefix, chunks of one row)
and plan options (decode share, key-split length, separate launches, the
mma.sync prefill), runs the append and the attention through the C ABI and
compares O and LSE with the oracle on all rows, then checks that a second
run of the same plan gives the same bits. The draws are seeded, so a failing
case is reproducible from its id.
"""
import numpy as np
import pytest

import oracle
import workloads as W

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

O_TOL = 2e-2
LSE_TOL = 1e-3

# (query heads, kv heads, head width, block size)
SHAPES = [(4, 2, 64, 16), (28, 4, 128, 16), (8, 2, 128, 32), (16, 2, 64, 64),
          (12, 4, 128, 16), (8, 8, 64, 16), (7, 1, 128, 16), (32, 4, 128, 16)]
SEPARATE, NO_TC = 1, 2


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2606_04415_gb300 as fnpu
    fnpu.load()


def _draw(case):
    rng = np.random.default_rng(1000 + case)
    hq, hkv, d, bs = SHAPES[case % len(SHAPES)]
    shape = W.Shape(hq, hkv, d, d, bs, False)
    S = int(rng.integers(2, 13))
    ql, ctx, ph = [], [], []
    for _ in range(S):
        kind = rng.choice(["decode", "decode", "multi", "chunk", "chunk_prefix", "one_row"])
        if kind == "decode":
            c = int(rng.integers(1, 3000))
            ql.append(1), ctx.append(c), ph.append(1)
        elif kind == "multi":
            q = int(rng.integers(2, 8))
            ql.append(q), ctx.append(q + int(rng.integers(0, 2000))), ph.append(1)
        elif kind == "chunk":
            q = int(rng.integers(2, 300))
            ql.append(q), ctx.append(q), ph.append(0)
        elif kind == "chunk_prefix":
            q = int(rng.integers(2, 300))
            ql.append(q), ctx.append(q + int(rng.integers(1, 2500))), ph.append(0)
        else:
            ql.append(1), ctx.append(int(rng.integers(1, 1500))), ph.append(0)
    batch = W.build_batch(shape, ql, ctx, ph, rng, name=f"random_mix_{case}")
    share = int(rng.choice([0, 0, 3, 20, 45]))
    split = int(rng.choice([0, 0, 64, 256]))
    flags = int(rng.choice([0, 0, 0, SEPARATE, NO_TC]))
    return batch, share, split, flags


@pytest.mark.parametrize("case", range(24))
def test_random_mixed_step_all_rows(case):
    import paper_2606_04415_gb300 as fnpu
    from paper_2606_04415_gb300.step import DeviceStep
    batch, share, split, flags = _draw(case)
    st = DeviceStep(batch, opts=fnpu.PlanOpts(split, share, 0, flags))
    st.run()
    out, lse = st.results()
    assert fnpu.plan_check(st.plan) == fnpu.FNPU_OK and fnpu.check() == fnpu.FNPU_OK
    ref_o, ref_l, _, _ = oracle.run_step(batch)
    assert np.isfinite(out).all() and np.isfinite(lse).all()
    eo, el = np.abs(out - ref_o).max(), np.abs(lse - ref_l).max()
    assert eo <= O_TOL, f"case {case} (share {share}, split {split}, flags {flags}): max |dO| = {eo}"
    assert el <= LSE_TOL, f"case {case} (share {share}, split {split}, flags {flags}): max |dLSE| = {el}"
    st.attend()  # the cache already holds the step's rows; same plan, same bits
    out2, lse2 = st.results()
    assert np.array_equal(out, out2) and np.array_equal(lse, lse2)


def _draw_mla(case):
    rng = np.random.default_rng(7000 + case)
    bs = int(rng.choice([16, 32, 64]))
    shape = W.Shape(128, 1, 576, 512, bs, True)
    S = int(rng.integers(2, 7))
    ql, ctx, ph = [], [], []
    for _ in range(S):
        kind = rng.choice(["decode", "decode", "multi", "chunk", "chunk_prefix"])
        if kind == "decode":
            ql.append(1), ctx.append(int(rng.integers(1, 4000))), ph.append(1)
        elif kind == "multi":
            q = int(rng.integers(2, 5))
            ql.append(q), ctx.append(q + int(rng.integers(0, 1500))), ph.append(1)
        elif kind == "chunk":
            q = int(rng.integers(1, 64))
            ql.append(q), ctx.append(q), ph.append(0)
        else:
            q = int(rng.integers(2, 64))
            ql.append(q), ctx.append(q + int(rng.integers(1, 700))), ph.append(0)
    batch = W.build_batch(shape, ql, ctx, ph, rng, name=f"random_mla_{case}")
    return batch, int(rng.choice([0, 0, NO_TC]))


@pytest.mark.parametrize("case", range(10))
def test_random_latent_step_all_rows(case):
    """Absorbed MLA (128 heads on one 576-wide latent row, V its first 512
    columns) on random mixes: latent blocks of 16 to 64 slots, decodes long
    enough to be cut into merged pieces, multi-token decodes and chunks; the
    latent append bit-exact, every row against the oracle, and a second run
    identical."""
    import paper_2606_04415_gb300 as fnpu
    from paper_2606_04415_gb300.step import DeviceStep
    batch, flags = _draw_mla(case)
    st = DeviceStep(batch, opts=fnpu.PlanOpts(0, 0, 0, flags))
    st.run()
    out, lse = st.results()
    assert fnpu.plan_check(st.plan) == fnpu.FNPU_OK and fnpu.check() == fnpu.FNPU_OK
    kc, _ = st.cache_bits()
    assert np.array_equal(kc, oracle.kv_append(batch.k_cache, batch.k_new, batch.slot_mapping))
    ref_o, ref_l, _, _ = oracle.run_step(batch)
    assert np.isfinite(out).all() and np.isfinite(lse).all()
    eo, el = np.abs(out - ref_o).max(), np.abs(lse - ref_l).max()
    assert eo <= O_TOL, f"case {case} (flags {flags}): max |dO| = {eo}"
    assert el <= LSE_TOL, f"case {case} (flags {flags}): max |dLSE| = {el}"
    st.attend()
    out2, lse2 = st.results()
    assert np.array_equal(out, out2) and np.array_equal(lse, lse2)
