"""Plant one plausible mistake at a time in a copy of the oracle (on the CPU)
and check that the pins in test_oracle.py catch every one of them.

Each mutant is compiled into a temporary directory and loaded by a child
pytest run through FNPU_ORACLE_LIB; the committed oracle is never modified.
"""
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "oracle", "fnpu_oracle.c")

MUTANTS = {
    "mask_excludes_self": ("for (int32_t j = 0; j <= pos; ++j) {", "for (int32_t j = 0; j < pos; ++j) {"),
    "position_off_by_one": ("- a->query_len[s] + i;", "- a->query_len[s] + i - 1;"),
    "gqa_interleaved_map": ("const int32_t kvh = h / (a->hq / a->hkv);", "const int32_t kvh = h % a->hkv;"),
    "block_offset_swapped": ("int64_t slot = blk * a->bs + j % a->bs;",
                             "int64_t slot = blk * a->bs + (j / a->bs) % a->bs;"),
    "scale_dropped": ("score[j] = a->scale * dot;", "score[j] = dot;"),
    "lse_log2": ("*lse = m + log(l);", "*lse = m + log2(l);"),
    "lse_without_max": ("*lse = m + log(l);", "*lse = log(l);"),
    "default_scale_uses_dv": ("scale > 0 ? scale : 1.0 / sqrt((double)dqk)",
                              "scale > 0 ? scale : 1.0 / sqrt((double)dv)"),
    "latent_v_from_tail": ("if (a->latent) return a->k_cache + slot * a->dqk; /* V",
                           "if (a->latent) return a->k_cache + slot * a->dqk + (a->dqk - a->dv); /* V"),
    "exp_sign_flipped": ("double e = exp(score[j] - m);", "double e = exp(m - score[j]);"),
    "append_skips_slot0": ("if (s < 0) continue;", "if (s <= 0) continue;"),
}


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_pins_catch_mutant(name, tmp_path):
    a, b = MUTANTS[name]
    src = open(SRC).read()
    assert a in src, f"mutation site for {name} not found"
    mutated = tmp_path / "mut.c"
    mutated.write_text(src.replace(a, b, 1))
    lib = tmp_path / "libmut.so"
    subprocess.check_call(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fopenmp",
                           str(mutated), "-o", str(lib), "-lm"])
    env = dict(os.environ, FNPU_ORACLE_LIB=str(lib))
    r = subprocess.run([sys.executable, "-m", "pytest", "-x", "-q", "-p", "no:cacheprovider",
                        os.path.join(ROOT, "tests", "test_oracle.py")],
                       cwd=ROOT, env=env, capture_output=True, text=True, timeout=600)
    assert r.returncode != 0, f"mutant {name} survived the oracle pins:\n{r.stdout[-2000:]}"
