"""Host-side checks of the C ABI that need no GPU: the library builds, loads
and exports every entry point declared in include/fnpu.h, and argument
validation rejects bad metadata before any CUDA call is made."""
import ctypes
import os
import re

import numpy as np
import pytest

import paper_2606_04415_gb300 as fnpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared_symbols():
    names = set()
    for fn in os.listdir(os.path.join(ROOT, "include")):
        if fn.endswith(".h"):
            src = open(os.path.join(ROOT, "include", fn)).read()
            src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
            names |= set(re.findall(r"\b(fnpu_[a-z_0-9]+)\s*\(", src))
    return names


def test_library_exports_every_declared_symbol():
    lib = fnpu.load()
    declared = _declared_symbols()
    assert declared, "no declarations found"
    assert declared == set(fnpu.EXPORTED)
    for name in declared:
        assert hasattr(lib, name), name


def test_status_strings_and_version():
    assert fnpu.status_str(fnpu.FNPU_OK) == "ok"
    assert "invalid" in fnpu.status_str(fnpu.FNPU_EINVAL)
    assert fnpu.status_str(12345) == "unknown status"
    assert fnpu.version() >= 100


def _plan_rc(desc, ql, cl, ph, bt, opts=None):
    lib = fnpu.load()
    ql = np.ascontiguousarray(ql, np.int32)
    cl = np.ascontiguousarray(cl, np.int32)
    ph = np.ascontiguousarray(ph, np.uint8)
    bt = np.ascontiguousarray(bt, np.int32)
    out = ctypes.c_void_p()
    return lib.fnpu_mixed_attn_plan_ex(ctypes.byref(desc), len(ql), ql.ctypes.data, cl.ctypes.data,
                                       ph.ctypes.data, bt.ctypes.data, bt.shape[1],
                                       None if opts is None else ctypes.byref(opts), None,
                                       ctypes.byref(out))


QWEN = dict(num_q_heads=28, num_kv_heads=4, head_dim_qk=128, head_dim_v=128, block_size=16,
            num_blocks=100)


@pytest.mark.parametrize("case", [
    "ctx_lt_q", "q_zero", "phase_2", "block_oob", "block_neg", "stride_short",
])
def test_plan_rejects_bad_metadata(case):
    desc = fnpu.make_desc(**QWEN)
    ql, cl, ph = [4, 1], [10, 40], [0, 1]
    bt = np.zeros((2, 4), np.int32)
    if case == "ctx_lt_q":
        cl = [3, 40]
    elif case == "q_zero":
        ql = [0, 1]
    elif case == "phase_2":
        ph = [0, 2]
    elif case == "block_oob":
        bt[1, 2] = 100
    elif case == "block_neg":
        bt[0, 0] = -1
    elif case == "stride_short":
        bt = np.zeros((2, 2), np.int32)
    assert _plan_rc(desc, ql, cl, ph, bt) == fnpu.FNPU_EINVAL


def test_plan_accepts_multi_token_decode():
    """A decode of several tokens (speculative verification) is valid
    metadata: without a GPU the plan then fails on the device, not on the
    arguments."""
    desc = fnpu.make_desc(**QWEN)
    bt = np.zeros((2, 4), np.int32)
    assert _plan_rc(desc, [4, 3], [10, 40], [0, 1], bt) != fnpu.FNPU_EINVAL


def test_plan_rejects_bad_shape_and_options():
    bt = np.zeros((1, 4), np.int32)
    bad = fnpu.make_desc(**dict(QWEN, num_q_heads=30))  # not a multiple of Hkv
    assert _plan_rc(bad, [1], [5], [1], bt) == fnpu.FNPU_EINVAL
    bad = fnpu.make_desc(**dict(QWEN, block_size=0))
    assert _plan_rc(bad, [1], [5], [1], bt) == fnpu.FNPU_EINVAL
    opts = fnpu.PlanOpts(-5, 0, 0, 0)
    assert _plan_rc(fnpu.make_desc(**QWEN), [1], [5], [1], bt, opts) == fnpu.FNPU_EINVAL
    opts = fnpu.PlanOpts(0, 101, 0, 0)
    assert _plan_rc(fnpu.make_desc(**QWEN), [1], [5], [1], bt, opts) == fnpu.FNPU_EINVAL


def test_plan_reports_unsupported_head_dims():
    bt = np.zeros((1, 4), np.int32)
    desc = fnpu.make_desc(**dict(QWEN, head_dim_qk=96, head_dim_v=96))
    assert _plan_rc(desc, [1], [5], [1], bt) == fnpu.FNPU_EUNSUPPORTED
    # latent layout: 576 / 512 with a multiple of 64 query heads only
    lat = fnpu.make_desc(100, 1, 576, 512, 64, 8, latent=True)
    assert _plan_rc(lat, [1], [5], [1], bt) == fnpu.FNPU_EUNSUPPORTED
    lat = fnpu.make_desc(128, 1, 320, 256, 64, 8, latent=True)
    assert _plan_rc(lat, [1], [5], [1], bt) == fnpu.FNPU_EUNSUPPORTED


def test_append_and_run_reject_null_pointers():
    lib = fnpu.load()
    desc = fnpu.make_desc(**QWEN)
    rc = lib.fnpu_kv_append(ctypes.byref(desc), None, None, None, 4, None, None, None)
    assert rc == fnpu.FNPU_EINVAL
    rc = lib.fnpu_kv_append(ctypes.byref(desc), 16, 32, 64, -1, 128, 256, None)
    assert rc == fnpu.FNPU_EINVAL
    rc = lib.fnpu_kv_append(ctypes.byref(desc), 17, 32, 64, 4, 128, 256, None)  # misaligned
    assert rc == fnpu.FNPU_EINVAL
    assert lib.fnpu_mixed_attn_run(None, None, None, None, None, None, None) == fnpu.FNPU_EINVAL
    assert lib.fnpu_plan_check(None, None) == fnpu.FNPU_EINVAL
    assert lib.fnpu_mixed_attn_replan(None, 0, None, None, None, None, 1, None, None) == fnpu.FNPU_EINVAL
    share = ctypes.c_int32(-1)
    assert lib.fnpu_plan_decode_share(None, ctypes.byref(share)) == fnpu.FNPU_EINVAL and share.value == -1
    assert lib.fnpu_mixed_step(None, 16, 32, 64, 128, 256, 512, 1024, 2048, None) == fnpu.FNPU_EINVAL
    lib.fnpu_plan_destroy(None)  # ignored


def test_fp8_cache_validation():
    """The FP8 cache: kv_fp8 outside {0, 1} is invalid; other shapes and latent
    caches are unsupported; all decided on the host before any CUDA call.
    Plans with prefill work are valid (without a GPU they fail later)."""
    lib = fnpu.load()
    bt = np.zeros((2, 4), np.int32)
    bad = fnpu.make_desc(**QWEN)
    bad.kv_fp8 = 2
    assert _plan_rc(bad, [1], [5], [1], bt[:1]) == fnpu.FNPU_EINVAL
    assert lib.fnpu_kv_append(ctypes.byref(bad), 16, 32, 64, 4, 128, 256, None) == fnpu.FNPU_EINVAL
    fp8 = fnpu.make_desc(**QWEN, kv_fp8=True)
    assert _plan_rc(fp8, [8, 1], [8, 20], [0, 1], bt) not in (fnpu.FNPU_EUNSUPPORTED, fnpu.FNPU_EINVAL)
    assert _plan_rc(fp8, [3], [20], [1], bt[:1]) not in (fnpu.FNPU_EUNSUPPORTED, fnpu.FNPU_EINVAL)
    for other in (dict(head_dim_qk=64, head_dim_v=64), dict(num_kv_heads=2, num_q_heads=14),
                  dict(block_size=32), dict(num_q_heads=36)):
        d = fnpu.make_desc(**dict(QWEN, **other), kv_fp8=True)
        assert _plan_rc(d, [1], [5], [1], bt[:1]) == fnpu.FNPU_EUNSUPPORTED, other
        assert lib.fnpu_kv_append(ctypes.byref(d), 16, 32, 64, 4, 128, 256, None) == fnpu.FNPU_EUNSUPPORTED
    lat = fnpu.make_desc(128, 1, 576, 512, 64, 8, latent=True, kv_fp8=True)
    assert _plan_rc(lat, [1], [5], [1], bt[:1]) == fnpu.FNPU_EUNSUPPORTED
    # the allocation-free decode entry point takes bf16 caches only
    rc = lib.fnpu_decode_attn_noalloc(ctypes.byref(fp8), 1, 16, 32, 4, 5, 0, 48, 64, 80, 96, 112, None)
    assert rc == fnpu.FNPU_EUNSUPPORTED
    assert fnpu.FP8_BLOCK_BYTES == 8448


def test_mla_expand_validation_and_expanded_shape():
    """fnpu_mla_expand rejects non-latent descriptors, other widths, bad
    pointers; the expanded shape (192 / 128, Hkv = Hq) plans prefill only."""
    lib = fnpu.load()
    lat = fnpu.make_desc(128, 1, 576, 512, 64, 8, latent=True)
    ok_ptrs = (16, 32, 4, 48, 64, 80, 96, 112)
    assert lib.fnpu_mla_expand(ctypes.byref(lat), *ok_ptrs[:2], 0, *ok_ptrs[3:], None) == fnpu.FNPU_OK  # n = 0
    assert lib.fnpu_mla_expand(ctypes.byref(lat), 16, 32, -1, 48, 64, 80, 96, 112, None) == fnpu.FNPU_EINVAL
    assert lib.fnpu_mla_expand(ctypes.byref(lat), 16, 33, 4, 48, 64, 80, 96, 112, None) == fnpu.FNPU_EINVAL
    assert lib.fnpu_mla_expand(ctypes.byref(lat), 16, 32, 4, 48, 64, 81, 96, 112, None) == fnpu.FNPU_EINVAL
    assert lib.fnpu_mla_expand(ctypes.byref(lat), None, 32, 4, 48, 64, 80, 96, 112, None) == fnpu.FNPU_EINVAL
    plain = fnpu.make_desc(**QWEN)
    assert lib.fnpu_mla_expand(ctypes.byref(plain), 16, 32, 4, 48, 64, 80, 96, 112, None) == fnpu.FNPU_EINVAL
    other = fnpu.make_desc(128, 1, 320, 256, 64, 8, latent=True)
    assert lib.fnpu_mla_expand(ctypes.byref(other), 16, 32, 4, 48, 64, 80, 96, 112, None) == fnpu.FNPU_EUNSUPPORTED
    exp = fnpu.make_desc(128, 128, 192, 128, 16, 100)
    bt = np.zeros((1, 4), np.int32)
    assert _plan_rc(exp, [1], [5], [1], bt) == fnpu.FNPU_EUNSUPPORTED   # no decode kernel for it
    assert _plan_rc(exp, [3], [5], [0], bt) != fnpu.FNPU_EUNSUPPORTED   # prefill: valid (fails later without a GPU)
