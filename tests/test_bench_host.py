"""The bench's CPU legs on small batches (no GPU): the reference timings of
the default path, the FP8 cache and the expanded MLA prefill return a
positive throughput and say what they sampled; the reference arm prints one
line with the contract's keys."""
import json

import numpy as np

import bench
import workloads as W


def _check(r):
    assert r["value"] > 0 and r["kind"] == "oracle" and r["cores"] >= 1 and r["sample"]
    assert r["step_seconds_extrapolated"] > 0


def test_cpu_baseline_default_path():
    _check(bench.cpu_baseline(W.make_batch("tiny", 0), target_seconds=0.3))


def test_cpu_baseline_fp8_mixed_batch():
    rng = np.random.default_rng(0)
    b = W.build_batch(W.Shape(28, 4, 128, 128, 16, False), [20, 1, 1], [60, 300, 45], [0, 1, 1], rng,
                      name="fp8_small", seed=0)
    _check(bench.cpu_baseline_fp8(b, target_seconds=0.5))


def test_cpu_baseline_expanded_mla():
    rng = np.random.default_rng(1)
    b = W.build_batch(W.Shape(4, 1, 576, 512, 64, True), [16, 5], [16, 70], [0, 0], rng, name="mla_small", seed=1)
    ins = W.mla_expand_inputs(b, seed=1)
    slots, bt, _ = W.expanded_layout(b)
    _check(bench.cpu_baseline_mla_expand(b, ins, slots, bt, target_seconds=0.3))


def test_reference_arm_line(capsys):
    assert bench.main(["--impl", "reference", "--workload", "tiny", "--steps", "1", "--warmup", "3",
                       "--ref-seconds", "0.2"]) == 0
    line = json.loads(capsys.readouterr().out.strip().splitlines()[-1])
    for key in ("impl", "metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step",
                "higher_is_better", "config", "cpu_baseline", "e2e"):
        assert key in line
    assert line["impl"] == "reference" and line["value"] > 0
