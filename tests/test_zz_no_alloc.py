"""The decode entry point that allocates nothing (fnpu_decode_attn_noalloc).

It exists for callers that may not call cudaMalloc (code confined to memory
another framework reserved, or a process whose device memory is fixed at
start): it keeps its split scratch in a fixed array inside the library. This
test calls it through the C ABI twice in a row and checks both results
against the planned path (fnpu_mixed_attn_plan + fnpu_mixed_attn_run) on the
same decode batch, within the parity tolerances used by the other GPU tests.
It lives in its own file, collected last, and also passes on its own in a
fresh process.
"""
import numpy as np
import pytest

import workloads as W

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

O_TOL = 2e-2
LSE_TOL = 1e-3


@pytest.mark.parametrize("split_keys", [0, 256])
def test_noalloc_decode_matches_planned_path_twice(split_keys):
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2606_04415_gb300 as fnpu
    from paper_2606_04415_gb300.step import DeviceStep

    batch = W.make_batch("qwen_decode", seed=3)
    st = DeviceStep(batch)
    st.run()  # append + planned attention
    ref_o, ref_l = st.results()

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
        assert np.abs(o - ref_o).max() <= O_TOL, f"call {call}"
        assert np.abs(l - ref_l).max() <= LSE_TOL, f"call {call}"


def test_noalloc_rejects_requests_beyond_its_scratch():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
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
