"""Plant one plausible mistake at a time in a copy of the numpy references
(the FP8 cache and the MLA expansion, on the CPU) and check that their pins
catch every one. The copy of the `oracle` package goes to a temporary
directory that the child pytest run imports first; the committed references
are never modified."""
import os
import shutil
import subprocess
import sys

import pytest

import oracle

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

MUTANTS = {
    # FP8 cache (oracle/fp8.py), pinned by tests/test_oracle_fp8.py
    "fp8_kpos_k_c_swapped": ("fp8.py", "return 32 * c + 4 * k + r", "return 16 * c + 4 * k + r"),
    "fp8_vpos_transposed": ("fp8.py", "    return 4 * c + r\n", "    return 4 * r + c\n"),
    "fp8_scale_447": ("fp8.py", "amax / np.float32(E4M3_MAX)", "amax / np.float32(447.0)"),
    "fp8_ties_away_from_zero": ("fp8.py", "m = np.rint(np.ldexp(a, 3 - E))", "m = np.floor(np.ldexp(a, 3 - E) + 0.5)"),
    "fp8_no_saturation": ("fp8.py", "a = np.minimum(np.abs(x), np.float32(E4M3_MAX))", "a = np.abs(x)"),
    "fp8_subnormals_as_normals": ("fp8.py", "    E[a < 2.0 ** -6] = -6", "    E[a < 0] = -6"),
    "fp8_zero_row_scale_zero": ("fp8.py", "amax / np.float32(E4M3_MAX), np.float32(1.0))", "amax / np.float32(E4M3_MAX), np.float32(0.0))"),
    "fp8_v_scaled_by_k_scale": ("fp8.py", "vals = e4m3_decode(v_codes[blk, idx % BS]) * v_scales[blk, idx % BS]",
                                "vals = e4m3_decode(v_codes[blk, idx % BS]) * k_scales[blk, idx % BS]"),
    "fp8_append_skips_slot0": ("fp8.py", "        if s < 0:\n            continue", "        if s <= 0:\n            continue"),
    "fp8_causal_off_by_one": ("fp8.py", "x = keys[:pos + 1, kvh, :] @ qf[t, h] * sc", "x = keys[:pos, kvh, :] @ qf[t, h] * sc"),
    # MLA expansion (oracle/mla_expand.py), pinned by tests/test_oracle_mla_expand.py
    "mla_rope_from_c": ("mla_expand.py", "k[:, h, DN:] = r", "k[:, h, DN:] = c[:, :R]"),
    "mla_value_weights_for_keys": ("mla_expand.py", "k[:, h, :DN] = c @ wk[h]", "k[:, h, :DN] = c @ wv[h]"),
    "mla_head_weights_shifted": ("mla_expand.py", "v[:, h, :] = c @ wv[h]", "v[:, h, :] = c @ wv[(h + 1) % H]"),
    "mla_double_rounding": ("mla_expand.py", "    x = np.asarray(x, np.float64)\n    m, e = np.frexp(x)",
                            "    x = np.asarray(x, np.float64).astype(np.float32).astype(np.float64)\n    m, e = np.frexp(x)"),
    "mla_negative_slot_not_zero": ("mla_expand.py", "    rows[s < 0] = 0.0\n", ""),
}

PINS = {"fp8.py": "test_oracle_fp8.py", "mla_expand.py": "test_oracle_mla_expand.py"}


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_pins_catch_mutant(name, tmp_path):
    fname, a, b = MUTANTS[name]
    src_dir = os.path.join(ROOT, "oracle")
    dst_dir = tmp_path / "oracle"
    shutil.copytree(src_dir, dst_dir, ignore=shutil.ignore_patterns("_build", "__pycache__"))
    path = dst_dir / fname
    src = path.read_text()
    assert a in src, f"mutation site for {name} not found"
    path.write_text(src.replace(a, b, 1))
    # the copy uses the committed C oracle's library (the mutants are in the numpy parts)
    env = dict(os.environ, FNPU_ORACLE_LIB=oracle.build(),
               PYTHONPATH=os.pathsep.join([str(tmp_path), ROOT, os.environ.get("PYTHONPATH", "")]))
    r = subprocess.run([sys.executable, "-m", "pytest", "-x", "-q", "-p", "no:cacheprovider",
                        os.path.join(ROOT, "tests", PINS[fname])],
                       cwd=str(tmp_path), env=env, capture_output=True, text=True, timeout=600)
    assert "passed" in r.stdout or "failed" in r.stdout, r.stdout[-2000:] + r.stderr[-2000:]
    assert r.returncode != 0, f"mutant {name} survived the pins:\n{r.stdout[-2000:]}"
