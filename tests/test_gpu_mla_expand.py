"""MLA prefill without absorption on the GPU: latent rows expanded into
per-head keys and values (fnpu_mla_expand), then multi-head attention (d_qk
192, d_v 128) over them through the plan / run (the tcgen05 prefill kernel,
or the mma.sync one under FNPU_PLAN_NO_TCGEN05), against the fp64 reference
(oracle.mla_expand + the C oracle).

Expanded rows: the rotary part is a copy (bit-exact); the products are fp32
sums rounded to bf16 against the reference's exactly rounded fp64 sums, so an
element may differ by one bf16 unit where the fp32 sum lands on the other side
of a rounding boundary (about 1% of them, asserted below).

Attention kernel alone (random 192-wide keys and 128-wide values from the
seeded generator): |O - O_ref| <= 2e-2, |LSE - LSE_ref| <= 1e-3 as for every
attention path.

End to end (expansion then attention) the reference attends over its own
expanded rows K_r, V_r and the GPU over K_g, V_g, so the kernel tolerances
hold against attention over K_g, V_g, and the distance between the two
attentions is bounded from the measured differences, per (token, head), with
no fixed constant:
  * score j moves by |<q, K_g,j - K_r,j>| * scale <= ds_j =
    scale * sum_d |q_d| |K_g - K_r|_jd;
  * the log-sum-exp is 1-Lipschitz in the max norm of the scores, so
    |LSE_g - LSE_r| <= 1e-3 + max_j ds_j over the visible keys;
  * with D = max_j ds_j every softmax weight moves by a factor within
    [e^-2D, e^2D], so sum_j |w_g,j - w_r,j| <= e^2D - 1, and per column
    |O_g - O_r| <= 2e-2 + max_j |V_g - V_r|_j + (e^2D - 1) max_j |V_r|_j.
"""
import numpy as np
import pytest

import oracle
import workloads as W
from oracle import mla_expand as X

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


def _expansion_bounds(batch, bt, q_bits, gk, gv, kb, vb, toks):
    """Per checked (token, head): the bound on |LSE_g - LSE_r| and, per column,
    on |O_g - O_r| that the expansion differences allow (module docstring).
    Expanded rows of sequence s are bt[s, 0] * 16 + position."""
    H = gk.shape[1]
    qs = batch.query_start
    seq_of = np.searchsorted(qs, toks, side="right") - 1
    pos = (batch.context_len[seq_of] - batch.query_len[seq_of] + (toks - qs[seq_of])).astype(np.int64)
    first = bt[seq_of, 0].astype(np.int64) * 16
    scale = 1.0 / np.sqrt(192.0)
    qabs = np.abs(X.bf16_bits_to_f64(q_bits[toks]))          # [t, H, 192]
    dk = np.abs(X.bf16_bits_to_f64(gk) - X.bf16_bits_to_f64(kb))  # [n, H, 192]
    dv = np.abs(X.bf16_bits_to_f64(gv) - X.bf16_bits_to_f64(vb))  # [n, H, 128]
    va = np.abs(X.bf16_bits_to_f64(vb))
    n = dk.shape[0]
    rows = np.arange(n)
    vis = (rows[None, :] >= first[:, None]) & (rows[None, :] <= (first + pos)[:, None])
    dmax = np.empty((len(toks), H))
    for h in range(H):
        ds = scale * (qabs[:, h, :] @ dk[:, h, :].T)          # [t, n]
        dmax[:, h] = np.where(vis, ds, 0.0).max(axis=1)
    # maxima over the visible rows j <= pos: running maxima along each sequence
    dv_vis = np.empty((len(toks), H, 128))
    va_vis = np.empty((len(toks), H, 128))
    for s in np.unique(seq_of):
        r0, c = int(bt[s, 0]) * 16, int(batch.context_len[s])
        cdv = np.maximum.accumulate(dv[r0:r0 + c], axis=0)
        cva = np.maximum.accumulate(va[r0:r0 + c], axis=0)
        sel = seq_of == s
        dv_vis[sel] = cdv[pos[sel]]
        va_vis[sel] = cva[pos[sel]]
    lse_bound = LSE_TOL + dmax
    o_bound = O_TOL + dv_vis + np.expm1(2.0 * dmax)[:, :, None] * va_vis
    return lse_bound, o_bound


def _run(q_lens, ctxs, heads=128, seed=0, bs=64, tokens=None, flags=0):
    import paper_2606_04415_gb300 as fnpu
    from paper_2606_04415_gb300.step import ExpandedMlaPrefill
    rng = np.random.default_rng(seed)
    sh = W.Shape(heads, 1, 576, 512, bs, True)
    batch = W.build_batch(sh, q_lens, ctxs, [0] * len(q_lens), rng, name="mla_expand")
    ins = W.mla_expand_inputs(batch, seed)
    slots, bt, nb = W.expanded_layout(batch)
    st = ExpandedMlaPrefill(batch, ins["w_uk"], ins["w_uv"], ins["q"], slots, bt, nb,
                            opts=fnpu.PlanOpts(0, 0, 0, flags))
    st.run()
    assert fnpu.plan_check(st.plan) == fnpu.FNPU_OK and fnpu.check() == fnpu.FNPU_OK
    out, lse = st.results()
    gk, gv = st.expanded_bits()
    lat = oracle.kv_append(batch.k_cache, batch.k_new, batch.slot_mapping)
    kb, vb = X.expand(lat, slots, ins["w_uk"], ins["w_uv"])
    # rotary part copied; products within one bf16 unit plus the fp32
    # accumulation error (512 terms: at most 2^-15 of the sum of |terms|,
    # doubled), and nearly all bit-exact
    assert np.array_equal(gk[:, :, 128:], kb[:, :, 128:])
    c_abs = np.abs(X.latent_rows(lat, slots)[:, :512])
    for g, r, w in ((gk[:, :, :128], kb[:, :, :128], ins["w_uk"]), (gv, vb, ins["w_uv"])):
        gf, rf = X.bf16_bits_to_f64(g), X.bf16_bits_to_f64(r)
        s_abs = np.einsum("nk,hkd->nhd", c_abs, np.abs(X.bf16_bits_to_f64(w)))
        bound = np.abs(rf) * 2.0 ** -7 + s_abs * 2.0 ** -14
        assert np.all(np.abs(gf - rf) <= bound), float(np.max(np.abs(gf - rf) - bound))
        assert np.mean(g == r) > 0.99
    ref_o, ref_l = oracle.attention(batch.query_len, batch.context_len, bt, ins["q"], kb, vb, num_q_heads=heads,
                                    num_kv_heads=heads, head_dim_qk=192, head_dim_v=128, block_size=16,
                                    tokens=tokens)
    toks = np.arange(batch.num_tokens, dtype=np.int64) if tokens is None else np.asarray(tokens, np.int64)
    out, lse = out[toks], lse[toks]
    assert np.isfinite(out).all() and np.isfinite(lse).all()
    lse_bound, o_bound = _expansion_bounds(batch, bt, ins["q"], gk, gv, kb, vb, toks)
    dl, do = np.abs(lse - ref_l), np.abs(out - ref_o)
    assert np.all(dl <= lse_bound), f"max |dLSE| - bound = {float(np.max(dl - lse_bound))}"
    assert np.all(do <= o_bound), f"max |dO| - bound = {float(np.max(do - o_bound))}"
    return st


@pytest.mark.parametrize("flags", [0, 2])
@pytest.mark.parametrize("seed", [0, 1])
def test_attention_kernel_on_192_128_heads(seed, flags):
    """The prefill kernels for 192-wide keys and 128-wide values, one kv head
    per query head (the expanded MLA shape): the tcgen05 kernel (flags 0) and
    the mma.sync one (FNPU_PLAN_NO_TCGEN05), on random bf16 caches: ragged
    chunks on prefixes (rows and keys off every tile boundary, a 600-row
    chunk of three 256-row items, the last one ragged), all rows, the
    attention tolerances."""
    from paper_2606_04415_gb300.step import DeviceStep
    import paper_2606_04415_gb300 as fnpu
    rng = np.random.default_rng(60 + seed)
    sh = W.Shape(16, 16, 192, 128, 16, False)
    batch = W.build_batch(sh, [1, 17, 64, 130, 600], [1, 40, 364, 700, 1000], [0, 0, 0, 0, 0], rng,
                          name="mha192")
    st = DeviceStep(batch, opts=fnpu.PlanOpts(0, 0, 0, flags))
    st.run()
    assert fnpu.plan_check(st.plan) == fnpu.FNPU_OK
    out, lse = st.results()
    ref_o, ref_l, _, _ = oracle.run_step(batch)
    assert np.isfinite(out).all()
    assert np.abs(out - ref_o).max() <= O_TOL and np.abs(lse - ref_l).max() <= LSE_TOL


@pytest.mark.parametrize("flags", [0, 2])
@pytest.mark.parametrize("heads", [128, 16])
def test_ragged_chunks_on_prefixes(heads, flags):
    """Chunks of 1, 17, 64 and 200 rows on prefixes of 0, 23, 300 and 824
    (rows and keys off every tile boundary), latent blocks of 64; the tcgen05
    and the mma.sync attention."""
    _run([1, 17, 64, 200], [1, 40, 364, 1024], heads=heads, seed=1, flags=flags)


def test_latent_blocks_of_16():
    _run([33, 128], [33, 500], heads=128, seed=2, bs=16)


def test_full_size_prefill_chunk_sampled_rows():
    """The 1024-token DeepSeek-R1 prefill chunk of the MLA co-located workload
    (no prefix, 128 heads): all of it expanded and attended on the GPU, the
    reference on rows at tile boundaries and at random."""
    rng = np.random.default_rng(5)
    rows = sorted({0, 1, 63, 64, 127, 128, 511, 512, 1023} | set(rng.integers(0, 1024, 12).tolist()))
    _run([1024], [1024], heads=128, seed=3, tokens=np.asarray(rows, np.int64))


def test_out_of_range_slot_gives_zero_row_and_flag():
    import paper_2606_04415_gb300 as fnpu
    st = _run([8], [8], heads=16, seed=4)
    bad = torch.tensor([st.latent_desc.num_blocks * st.latent_desc.block_size + 5, -1], dtype=torch.int64,
                       device="cuda")
    k = torch.full((2, 16, 192), 1.0, dtype=torch.bfloat16, device="cuda")
    v = torch.full((2, 16, 128), 1.0, dtype=torch.bfloat16, device="cuda")
    ws = torch.empty((2, 512), dtype=torch.bfloat16, device="cuda")
    fnpu.mla_expand(st.latent_desc, st.latent, bad, st.w_uk, st.w_uv, ws, k, v)
    assert fnpu.check() == fnpu.FNPU_EDEVICE_RANGE
    assert not k.float().abs().sum().item() and not v.float().abs().sum().item()


@pytest.mark.parametrize("case", range(4))
def test_random_chunks_on_prefixes(case):
    """Random chunk lengths (1 to 160 rows), prefixes (0 to 500), latent block
    sizes and head counts, on the tcgen05 and the mma.sync attention; every
    row within the derived bounds."""
    rng = np.random.default_rng(900 + case)
    S = int(rng.integers(1, 4))
    q = [int(rng.integers(1, 161)) for _ in range(S)]
    ctx = [x + int(rng.integers(0, 501)) for x in q]
    _run(q, ctx, heads=int(rng.choice([16, 128])), seed=20 + case, bs=int(rng.choice([16, 32, 64])),
         flags=int(rng.choice([0, 2])))
