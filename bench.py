"""Benchmark of one mixed prefill/decode paged-attention step on GB300.

A step is the whole hot path over one synthetic batch: KV append of the
step's new tokens, then attention of every query (prefill chunk + decodes)
through the C ABI. Default workload: the Qwen2.5-7B-shaped co-located step
(one 2048-token prefill chunk on a cached prefix ~ U[0, 8192] plus 128
decodes with log-normal contexts, 28/4 heads, d 128, block size 16).

Prints one JSON line (rank 0): query tokens/s for the whole job, the roofline
fraction of the dominant kernel, the end-to-end figure through host buffers,
the oracle's CPU time on the host cores, and clocks seen during the timed
region.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME]
  python bench.py --impl reference ...   # the fp64 oracle on the host cores
  python bench.py --workload qwen_decode --kv-fp8   # decode over the FP8 (e4m3) cache
  python bench.py --workload mla_prefill --mla-expand   # MLA prefill without absorption

Under torchrun each rank runs an independent replica (seed + rank): the path
has no exchange step, so there is no collective on the data path.
"""
from __future__ import annotations

import argparse
import json
import math
import os
import ctypes
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import workloads as W  # noqa: E402

METRIC = "mixed PD attention query tokens/s at 1 GB300; % of max(FLOP,HBM) roofline"
UNIT = "query tokens/s"
L2_FLUSH_BYTES = 512 << 20  # > 129 MB L2

# DRAM bytes (read + write) of one attention call, from ncu captures of the
# current kernels (dram__bytes_read.sum + dram__bytes_write.sum; for the
# co-located step the sum over its prefill and decode launches); the
# summaries with the commands are under profiles/. Set to None for a
# workload whose kernels change until they are captured again.
NCU_TRAFFIC = {
    # co-located workloads: the prefill kernel (the dominant one), captured alone
    "qwen_coloc": 33.6e6,        # prefill_tc 33.3 MB read + 0.32 MB write
    "qwen_decode": 308.9e6,      # decode_tma 308.15 MB read + 0.7 MB write
    "qwen_decode_fp8": 159.6e6,  # decode_fp8 159.16 MB read + 0.4 MB write
    "mla_prefill_expand": 200.9e6,  # prefill_tc<192, 128> 186.8 MB read + 14.0 MB write
}


def _flush_l2(wbuf, rbuf):
    """Evict L2 between timed steps: write a buffer larger than L2, then read
    another one so that L2 is left holding clean lines (otherwise the timed
    kernel would pay for writing back ~126 MB of dirty flush data). A short
    device-side sleep follows, so that the host has queued the timed step's
    launches before the device reaches them: the device-timed region then
    measures kernel execution, not host enqueue latency (that is what the
    end-to-end figure covers)."""
    import torch
    wbuf.zero_()
    rbuf.sum()
    torch.cuda._sleep(200_000)


def _peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return {"hbm_gbs": float(d["hbm_gbs"]), "bf16_tflops": float(d["bf16_tflops"]),
                "bf16_tflops_sustained": float(d.get("bf16_tflops_sustained", d["bf16_tflops"])),
                "source": "measured"}
    except (OSError, KeyError, ValueError):
        return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0,
                "source": "fallback"}


def _dist():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def max_over_ranks(value, ws, device):
    """The largest of each rank's value: a job's step time is its slowest
    replica's. Every rank gets the same result."""
    if ws <= 1:
        return value
    import torch
    import torch.distributed as dist
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(ws, tokens_per_rank, ms):
    """Whole-job query tokens/s: every replica processes its own batch of
    tokens_per_rank tokens in the job's step time (weak scaling)."""
    return ws * tokens_per_rank / (ms * 1e-3)


class ClockSampler:
    """nvidia-smi clocks/throttle reasons sampled every 200 ms while active."""

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.path = None

    def __enter__(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.index}", f"--query-gpu={q}", "--format=csv,noheader,nounits",
                 "-lms", "200"], stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None
        time.sleep(0.3)
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
        if self.proc is None or not self.path:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        rows = []
        with open(self.path) as f:
            for line in f:
                parts = [x.strip() for x in line.split(",")]
                if len(parts) >= 9:
                    rows.append(parts)
        os.unlink(self.path)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i].lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": reasons,
                "samples": len(rows)}


def _sample_rows(batch, target_pairs: int):
    """Evenly spaced query rows whose visible pairs sum to about target_pairs."""
    T = batch.num_tokens
    seq_of = np.repeat(np.arange(batch.num_seqs), batch.query_len)
    idx = np.arange(T) - batch.query_start[seq_of]
    pos = batch.context_len[seq_of] - batch.query_len[seq_of] + idx
    row_pairs = (pos + 1).astype(np.int64)
    total = int(row_pairs.sum())
    frac = min(1.0, max(target_pairs, 1) / total)
    n = max(1, int(round(T * frac)))
    rows = np.unique(np.linspace(0, T - 1, n).round().astype(np.int64))
    return rows, int(row_pairs[rows].sum()), total


def cpu_baseline(batch, target_seconds: float = 15.0, reps: int = 1):
    """Time the fp64 oracle on a bounded, evenly spaced sample of the step's
    query rows on all host cores; extrapolate to the whole step by visible
    (query, key) pairs."""
    import oracle
    threads = oracle.max_threads()
    sh = batch.shape
    t0 = time.perf_counter()
    kc = oracle.kv_append(batch.k_cache, batch.k_new, batch.slot_mapping)
    vc = None if sh.latent else oracle.kv_append(batch.v_cache, batch.v_new, batch.slot_mapping)
    t_append = time.perf_counter() - t0
    kw = dict(num_q_heads=sh.num_q_heads, num_kv_heads=sh.num_kv_heads, head_dim_qk=sh.head_dim_qk,
              head_dim_v=sh.head_dim_v, block_size=sh.block_size, latent=sh.latent)
    # calibrate the oracle's pair rate: grow a sample until it takes >= 0.2 s
    target = max(1, W.pairs(batch) // 4096)
    while True:
        rows, sp, total = _sample_rows(batch, target_pairs=target)
        t0 = time.perf_counter()
        oracle.attention(batch.query_len, batch.context_len, batch.block_table, batch.q, kc, vc,
                         tokens=rows, **kw)
        dt = time.perf_counter() - t0
        if dt >= 0.2 or sp >= total:
            break
        target *= 4
    rate = sp / max(dt, 1e-6)
    rows, sp, total = _sample_rows(batch, target_pairs=int(rate * target_seconds))
    times = []
    for _ in range(reps):
        t0 = time.perf_counter()
        oracle.attention(batch.query_len, batch.context_len, batch.block_table, batch.q, kc, vc,
                         tokens=rows, **kw)
        times.append(time.perf_counter() - t0)
    t_sample = statistics.median(times)
    t_step = t_append + t_sample * total / sp
    return {"value": batch.num_tokens / t_step, "unit": UNIT, "cores": threads, "kind": "oracle",
            "sample": (f"{len(rows)} of {batch.num_tokens} query rows (every ~{batch.num_tokens // max(len(rows), 1)}th, "
                       f"{sp / total:.4f} of the visible pairs), fp64 C oracle with OpenMP; "
                       f"step time extrapolated by pairs plus the full KV append"),
            "sample_seconds": t_sample, "step_seconds_extrapolated": t_step}


def cpu_baseline_fp8(batch, target_seconds: float = 15.0):
    """Time the fp64 FP8 reference: the step's append (all new rows, on the
    whole pool) and the attention of an evenly spaced sample of the query rows,
    extrapolated to the step by visible pairs. The sampled rows' sequences get
    their prefix rows into the reference pools first, untimed."""
    from oracle import fp8 as F8
    sh = batch.shape
    init = W.stale_pool_bytes(batch.num_blocks * F8.block_bytes(sh.num_kv_heads), batch.seed)
    starts = batch.query_start
    seq_q = np.repeat(np.arange(batch.num_seqs), batch.query_len)
    pos = batch.context_len[seq_q] - batch.query_len[seq_q] + (np.arange(batch.num_tokens) - starts[seq_q])
    row_pairs = (pos + 1).astype(np.int64)

    def pick(n):
        return np.unique(np.linspace(0, batch.num_tokens - 1, min(n, batch.num_tokens)).round().astype(np.int64))

    def pools_for(rows):  # the reference pools with the prefix rows of the rows' sequences
        seqs = np.unique(seq_q[rows])
        k, v, sl = W.prefix_rows(batch)
        pre = (batch.context_len - batch.query_len).astype(np.int64)
        p0 = np.concatenate([[0], np.cumsum(pre)])
        pi = np.concatenate([np.arange(p0[s], p0[s + 1]) for s in seqs])
        return F8.kv_append(init[0], init[1], k[pi], v[pi], sl[pi], sh.num_kv_heads)

    # calibrate on 4 rows, then take about a third of the budget of rows
    rows = pick(4)
    kp, vp = pools_for(rows)  # (the step's own rows are not in yet: the time does not depend on values)
    t0 = time.perf_counter()
    F8.attention(batch.query_len, batch.context_len, batch.block_table, batch.q, kp, vp,
                 num_q_heads=sh.num_q_heads, num_kv_heads=sh.num_kv_heads, tokens=rows)
    per_pair = (time.perf_counter() - t0) / float(row_pairs[rows].sum())
    n = int(target_seconds / 3 / max(per_pair * float(row_pairs.mean()), 1e-9))
    rows = pick(max(4, n))
    kp, vp = pools_for(rows)
    t0 = time.perf_counter()
    kp, vp = F8.kv_append(kp, vp, batch.k_new, batch.v_new, batch.slot_mapping, sh.num_kv_heads)
    t_append = time.perf_counter() - t0
    t0 = time.perf_counter()
    F8.attention(batch.query_len, batch.context_len, batch.block_table, batch.q, kp, vp,
                 num_q_heads=sh.num_q_heads, num_kv_heads=sh.num_kv_heads, tokens=rows)
    t_sample = time.perf_counter() - t0
    frac = float(row_pairs[rows].sum()) / float(row_pairs.sum())
    t_step = t_append + t_sample / frac
    return {"value": batch.num_tokens / t_step, "unit": UNIT, "cores": 1, "kind": "oracle",
            "sample": (f"attention of {len(rows)} of {batch.num_tokens} query rows (evenly spaced, {frac:.4f} of "
                       f"the visible pairs), fp64 numpy FP8 reference; step time = full append + sample / pair "
                       f"fraction"),
            "sample_seconds": t_sample, "step_seconds_extrapolated": t_step}


def run_reference(args):
    ws, rank, _ = _dist()
    if rank != 0:
        return 0
    batch = W.make_batch(args.workload, seed=args.seed)
    if args.kv_fp8:
        _fp8_workload_ok(batch)
    if args.mla_expand:
        ins = W.mla_expand_inputs(batch, seed=args.seed)
        slots, bt, _ = W.expanded_layout(batch)
    per = []
    # a bounded run: short warm-up samples, and timed samples that share about
    # 150 s (at most --ref-seconds each)
    timed_s = min(args.ref_seconds, max(1.0, 150.0 / max(args.steps, 1)))
    for i in range(args.warmup + args.steps):
        tgt = 0.5 if i < args.warmup else timed_s
        if args.mla_expand:
            r = cpu_baseline_mla_expand(batch, ins, slots, bt, target_seconds=tgt)
        else:
            r = (cpu_baseline_fp8 if args.kv_fp8 else cpu_baseline)(batch, target_seconds=tgt)
        if i >= args.warmup:
            per.append(r)
    step_s = statistics.median(x["step_seconds_extrapolated"] for x in per)
    value = batch.num_tokens / step_s
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": step_s * 1e3,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": {"workload": args.workload, "seed": args.seed,
                                            "kv_cache": "fp8_e4m3" if args.kv_fp8 else "bf16",
                                            "path": "mla_expand" if args.mla_expand else "default"},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": per[0]["cores"], "kind": "oracle",
                             "sample": per[0]["sample"]},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
            "gpu_launches": 0}
    print(json.dumps(line), flush=True)
    return 0


def cpu_baseline_mla_expand(batch, ins, slots, bt, target_seconds: float = 15.0):
    """Time the fp64 reference of the expanded MLA prefill: the latent append,
    the expansion of every row (numpy), and the C oracle's attention on an
    evenly spaced sample of the query rows, extrapolated by visible pairs."""
    import oracle
    from oracle import mla_expand as X
    sh = batch.shape
    t0 = time.perf_counter()
    lat = oracle.kv_append(batch.k_cache, batch.k_new, batch.slot_mapping)
    kb, vb = X.expand(lat, slots, ins["w_uk"], ins["w_uv"])
    t_expand = time.perf_counter() - t0
    kw = dict(num_q_heads=sh.num_q_heads, num_kv_heads=sh.num_q_heads, head_dim_qk=192, head_dim_v=128,
              block_size=16)
    target = max(1, W.pairs(batch) // 4096)
    while True:
        rows, sp, total = _sample_rows(batch, target_pairs=target)
        t0 = time.perf_counter()
        oracle.attention(batch.query_len, batch.context_len, bt, ins["q"], kb, vb, tokens=rows, **kw)
        dt = time.perf_counter() - t0
        if dt >= 0.2 or sp >= total:
            break
        target *= 4
    rate = sp / max(dt, 1e-6)
    rows, sp, total = _sample_rows(batch, target_pairs=int(rate * max(target_seconds - t_expand, 1.0)))
    t0 = time.perf_counter()
    oracle.attention(batch.query_len, batch.context_len, bt, ins["q"], kb, vb, tokens=rows, **kw)
    t_sample = time.perf_counter() - t0
    t_step = t_expand + t_sample * total / sp
    return {"value": batch.num_tokens / t_step, "unit": UNIT, "cores": oracle.max_threads(), "kind": "oracle",
            "sample": (f"append + expansion of all {len(slots)} rows (numpy fp64), attention of {len(rows)} of "
                       f"{batch.num_tokens} query rows ({sp / total:.4f} of the pairs, fp64 C oracle with OpenMP), "
                       f"extrapolated by pairs"),
            "sample_seconds": t_sample, "step_seconds_extrapolated": t_step}


def run_fnpu_mla_expand(args):
    """MLA prefill without absorption (latent append + expansion + MHA)."""
    import torch
    import paper_2606_04415_gb300 as fnpu
    from paper_2606_04415_gb300.step import ExpandedMlaPrefill

    ws, rank, local = _dist()
    if ws > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    fnpu.load()
    peaks = _peaks()
    batch = W.make_batch(args.workload, seed=args.seed + rank)
    if not batch.shape.latent or np.any(batch.phase != 0):
        raise SystemExit("--mla-expand needs a latent prefill workload (mla_prefill)")
    ins = W.mla_expand_inputs(batch, seed=args.seed + rank)
    slots, bt, nb = W.expanded_layout(batch)
    st = ExpandedMlaPrefill(batch, ins["w_uk"], ins["w_uv"], ins["q"], slots, bt, nb, device=str(dev))
    stream = torch.cuda.current_stream(dev)
    flush = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device=dev)
    flush_r = torch.zeros(L2_FLUSH_BYTES // 8, dtype=torch.float32, device=dev)
    for _ in range(args.warmup):
        _flush_l2(flush, flush_r)
        st.run()
    torch.cuda.synchronize(dev)
    if fnpu.plan_check(st.plan) != fnpu.FNPU_OK or fnpu.check() != fnpu.FNPU_OK:
        raise RuntimeError("device error flag raised during warm-up")
    K = args.steps
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(K)]
    if ws > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize(dev)
    # events only around the whole step (the attention grid is a dependent
    # launch of the expansion; an event between them delays it)
    with ClockSampler(local) as clocks:
        for i in range(K):
            _flush_l2(flush, flush_r)
            ev[i][0].record(stream)
            st.append()
            st.expand()
            st.attend()
            ev[i][1].record(stream)
        torch.cuda.synchronize(dev)
        if ws > 1:
            torch.distributed.barrier()
    clk = clocks.summary()
    step_ms = max_over_ranks(sum(ev[i][0].elapsed_time(ev[i][1]) for i in range(K)) / K, ws, dev)
    # the split of a step into its three calls, from a separate loop of K steps
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(K)]
    for i in range(K):
        _flush_l2(flush, flush_r)
        evs[i][0].record(stream)
        st.append()
        evs[i][1].record(stream)
        st.expand()
        evs[i][2].record(stream)
        st.attend()
        evs[i][3].record(stream)
    torch.cuda.synchronize(dev)
    seg = [[evs[i][j].elapsed_time(evs[i][j + 1]) for i in range(K)] for j in range(3)]
    t_app, t_exp, t_att = (sum(x) / K for x in seg)

    bf = torch.bfloat16
    h_q = torch.from_numpy(ins["q"]).view(bf).pin_memory()
    h_k = torch.from_numpy(batch.k_new).view(bf).pin_memory()
    h_s = torch.from_numpy(batch.slot_mapping).pin_memory()
    h_o = torch.empty(st.out.shape, dtype=bf).pin_memory()
    h_l = torch.empty(st.lse.shape, dtype=torch.float32).pin_memory()
    h2d = sum(x.numel() * x.element_size() for x in (h_q, h_k, h_s))
    d2h = h_o.numel() * h_o.element_size() + h_l.numel() * h_l.element_size()
    e2e_ms = []
    for i in range(args.warmup + K):
        _flush_l2(flush, flush_r)
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record(stream)
        st.q.copy_(h_q, non_blocking=True)
        st.k_new.copy_(h_k, non_blocking=True)
        st.slot_mapping.copy_(h_s, non_blocking=True)
        st.run()
        h_o.copy_(st.out, non_blocking=True)
        h_l.copy_(st.lse, non_blocking=True)
        b.record(stream)
        b.synchronize()
        if i >= args.warmup:
            e2e_ms.append(a.elapsed_time(b))
    e2e = max_over_ranks(sum(e2e_ms) / len(e2e_ms), ws, dev)

    H = batch.shape.num_q_heads
    n = len(slots)
    F_gemm = 2.0 * n * 512 * 128 * H * 2
    F_attn = 2.0 * H * W.pairs(batch) * (192 + 128)
    roof = {"bound": "tensor", "achieved": F_attn / (t_att * 1e-3) / 1e12, "peak": peaks["bf16_tflops"],
            "unit": "TFLOP/s", "kernel": "prefill_tc_kernel<192, 128> (the attention call)"}
    roof["frac"] = roof["achieved"] / roof["peak"]
    roof["traffic"] = args.traffic if args.traffic is not None else NCU_TRAFFIC.get(args.workload + "_expand")
    roof["peak_source"] = peaks["source"] + " burst"
    T = batch.num_tokens
    line = {
        "metric": METRIC, "value": job_throughput(ws, T, step_ms), "unit": UNIT, "n_gpus": ws, "steps": K,
        "warmup": args.warmup, "ms_per_step": step_ms, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": args.workload, "seed": args.seed, "query_tokens": T, "path": "mla_expand",
                   "expanded_rows": n, "heads": H, "flops_expand": F_gemm, "flops_attention": F_attn,
                   "l2": "flushed between timed steps (512 MB write, then 256 MB read)", "plan": st.plan.info()},
        "roofline": roof,
        "roofline_step_frac": {"burst": (F_gemm + F_attn) / (peaks["bf16_tflops"] * 1e12) / (step_ms * 1e-3),
                               "denominator": "(F_expand + F_attention) / bf16 peak of measured"},
        "kernel_ms": {"append": t_app, "expand": t_exp, "attention": t_att},
        "e2e": {"value": job_throughput(ws, T, e2e), "unit": UNIT, "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h, "ms_per_step": e2e},
        "gpu_launches": K * (3 + st.plan.info()["launches_per_run"]),  # append, gather, GEMM, attention
        "clocks": clk,
    }
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline_mla_expand(batch, ins, slots, bt, target_seconds=args.ref_seconds)
    elif rank == 0:
        line["cpu_baseline"] = None
    if rank == 0:
        print(json.dumps(line), flush=True)
    if ws > 1:
        torch.distributed.barrier()
        torch.distributed.destroy_process_group()
    return 0


def _replan_c_ms(st, batch, opts, stream_handle, n=20):
    """Host times (ms) of n re-plans of the batch through the C ABI
    (fnpu_mixed_attn_replan), with the arguments marshalled once."""
    import paper_2606_04415_gb300 as fnpu
    lib = fnpu.load()
    ql = np.ascontiguousarray(batch.query_len, np.int32)
    cl = np.ascontiguousarray(batch.context_len, np.int32)
    ph = np.ascontiguousarray(batch.phase, np.uint8)
    bt = np.ascontiguousarray(batch.block_table, np.int32)
    args = (st.plan.handle, int(ql.shape[0]), ql.ctypes.data, cl.ctypes.data, ph.ctypes.data, bt.ctypes.data,
            int(bt.shape[1]), ctypes.byref(opts), stream_handle)
    out = []
    for _ in range(n):
        t0 = time.perf_counter()
        rc = lib.fnpu_mixed_attn_replan(*args)
        out.append((time.perf_counter() - t0) * 1e3)
        if rc != fnpu.FNPU_OK:
            raise RuntimeError(f"re-plan failed: {fnpu.status_str(rc)}")
    return out


def pipelined_e2e(st, host_in, host_out, steps, warmup, replan_opts=None):
    """End-to-end steps overlapped as a serving loop runs them: step n's inputs
    go up (pinned host -> device, on a copy stream) and step n - 1's outputs
    come down while step n - 1 computes; two device buffer sets alternate, with
    events ordering each set's reuse. With replan_opts, every step is also
    re-planned from its host metadata (fnpu_mixed_attn_replan) while the device
    works on the step before. Returns (ms per step of device time from the
    first copy up to the last copy down, over `steps` steps after `warmup`;
    ms per step the host took to issue them). No L2
    flush here: a step reads far more than L2 holds."""
    import torch
    comp = torch.cuda.current_stream()
    up = torch.cuda.Stream()
    down = torch.cuda.Stream()
    names = ("q", "k_new", "v_new", "slot_mapping")
    bufs = [{n: getattr(st, n) for n in names},
            {n: None if getattr(st, n) is None else torch.empty_like(getattr(st, n)) for n in names}]
    outs = [(st.out, st.lse), (torch.empty_like(st.out), torch.empty_like(st.lse))]
    hout = [host_out, tuple(torch.empty_like(x).pin_memory() for x in host_out)]
    ready = [torch.cuda.Event() for _ in range(2)]
    done = [torch.cuda.Event() for _ in range(2)]
    drained = [torch.cuda.Event() for _ in range(2)]
    total = warmup + steps
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    orig = {n: getattr(st, n) for n in names}
    orig_out = (st.out, st.lse)
    try:
        for i in range(total):
            b = i & 1
            if i == warmup:
                torch.cuda.synchronize()
                t0.record(up)
                h0 = time.perf_counter()
            with torch.cuda.stream(up):
                if i >= 2:
                    up.wait_event(done[b])  # the set's previous step has read its inputs
                for n in names:
                    if host_in[n] is not None:
                        bufs[b][n].copy_(host_in[n], non_blocking=True)
                    # (the copies read pinned host memory that no step writes)
                ready[b].record(up)
            if replan_opts is not None:
                st.replan(replan_opts, stream=comp)
            comp.wait_event(ready[b])
            if i >= 2:
                comp.wait_event(drained[b])  # its previous outputs are down
            for n in names:
                setattr(st, n, bufs[b][n])
            st.out, st.lse = outs[b]
            st.run(stream=comp)
            done[b].record(comp)
            with torch.cuda.stream(down):
                down.wait_event(done[b])
                hout[b][0].copy_(outs[b][0], non_blocking=True)
                hout[b][1].copy_(outs[b][1], non_blocking=True)
                drained[b].record(down)
        t1.record(down)
        host_ms = (time.perf_counter() - h0) * 1e3 / steps  # enqueueing only (no sync inside the loop)
        torch.cuda.synchronize()
    finally:
        for n in names:
            setattr(st, n, orig[n])
        st.out, st.lse = orig_out
    return t0.elapsed_time(t1) / steps, host_ms


def _fp8_workload_ok(batch):
    sh = batch.shape
    if sh.latent or sh.num_kv_heads != 4 or sh.head_dim_qk != 128 or sh.block_size != 16:
        raise SystemExit("--kv-fp8 needs the Qwen shape (4 kv heads, d 128, 16-slot blocks)")


def run_fnpu(args):
    import torch
    import torch.distributed as dist

    import paper_2606_04415_gb300 as fnpu
    from paper_2606_04415_gb300.step import DeviceStep

    ws, rank, local = _dist()
    if ws > 1:
        dist.init_process_group("nccl" if torch.cuda.is_available() else "gloo")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    fnpu.load()
    peaks = _peaks()

    batch = W.make_batch(args.workload, seed=args.seed + rank)
    work = W.algorithmic_work(batch, kv_fp8=args.kv_fp8)
    opts = fnpu.PlanOpts(args.split, args.decode_share, 0, args.flags)
    if args.kv_fp8:
        _fp8_workload_ok(batch)
        init = W.stale_pool_bytes(batch.num_blocks * fnpu.FP8_BLOCK_BYTES, batch.seed)
        st = DeviceStep(batch, opts=opts, device=str(dev), kv_fp8=True, pool_init=init)
    else:
        st = DeviceStep(batch, opts=opts, device=str(dev))
    # the plan (host: validation, work lists, one async upload), timed apart
    # from the step: median host time of re-plans of the batch into one plan
    # (the steady state of a serving loop, which plans every step), and of
    # new plans (which also allocate the workspace, staging, streams, events)
    torch.cuda.synchronize(dev)
    planner_ms, first_ms = [], []
    extra = None
    for _ in range(5):
        t0 = time.perf_counter()
        extra = fnpu.mixed_attn_plan(st.desc, batch.query_len, batch.context_len, batch.phase, batch.block_table,
                                     opts=opts)
        first_ms.append((time.perf_counter() - t0) * 1e3)
        extra.destroy()
    stream = torch.cuda.current_stream(dev)
    planner_ms = _replan_c_ms(st, batch, opts, stream.cuda_stream)
    torch.cuda.synchronize(dev)
    info = st.plan.info()
    flush = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device=dev)
    flush_r = torch.zeros(L2_FLUSH_BYTES // 8, dtype=torch.float32, device=dev)

    # warm-up; with --dispatch feedback each warm-up step also feeds its phase
    # times to the decode-share controller and the next step is planned with
    # the share it returns (Sec. 3.4 dispatch ratio)
    # (the controller starts from the share the planner chose)
    share = args.decode_share
    if share <= 0:
        try:
            share = fnpu.plan_decode_share(st.plan)
        except fnpu.FnpuError:  # one phase only: no share
            share = 24
    trace = []
    for w in range(args.warmup):
        if args.dispatch == "feedback":
            _flush_l2(flush, flush_r)
        st.run()
        if args.dispatch == "feedback" and w > 0:  # the first run is cold (module load, first touch)
            try:
                pre_ms, dec_ms = fnpu.plan_phase_ms(st.plan)
            except fnpu.FnpuError:  # one phase only: nothing to balance
                break
            nxt = fnpu.dispatch_next_share(share, pre_ms, dec_ms)
            trace.append([share, round(pre_ms * 1e3, 1), round(dec_ms * 1e3, 1)])
            if nxt != share:
                share = nxt
                st.replan(fnpu.PlanOpts(args.split, share, 0, args.flags))
                info = st.plan.info()
    torch.cuda.synchronize(dev)
    if fnpu.plan_check(st.plan) != fnpu.FNPU_OK or fnpu.check() != fnpu.FNPU_OK:
        raise RuntimeError("device error flag raised during warm-up")
    # re-plans at the decode share the dispatch settled on: what a serving loop
    # pays every step once its controller has converged
    share_opts = fnpu.PlanOpts(args.split, share if args.dispatch == "feedback" else args.decode_share, 0,
                               args.flags)
    # (plan_ms: the C-ABI call alone, as a native serving loop calls it;
    # plan_py_ms: through the Python binding)
    plan_ms = _replan_c_ms(st, batch, share_opts, stream.cuda_stream)
    plan_py_ms = []
    for _ in range(20):
        t0 = time.perf_counter()
        st.replan(share_opts)
        plan_py_ms.append((time.perf_counter() - t0) * 1e3)
    torch.cuda.synchronize(dev)

    K = args.steps
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(K)]
    if ws > 1:
        dist.barrier()
    torch.cuda.synchronize(dev)
    # the timed steps: fnpu_mixed_step (the append, then the attention), events
    # only around the whole step (an event between the append and the
    # attention sits between the append and the prefill grid that is its
    # dependent launch, and costs the step about 2 us)
    with ClockSampler(local) as clocks:
        for i in range(K):
            _flush_l2(flush, flush_r)  # evict L2 between timed steps (outside the events)
            ev[i][0].record(stream)
            st.run()
            ev[i][1].record(stream)
        torch.cuda.synchronize(dev)
        if ws > 1:
            dist.barrier()
    clk = clocks.summary()
    t_step = [ev[i][0].elapsed_time(ev[i][1]) for i in range(K)]
    step_ms = max_over_ranks(sum(t_step) / K, ws, dev)
    # the append / attention split of a step, from a separate loop of K steps
    # with an event between the two calls
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(K)]
    for i in range(K):
        _flush_l2(flush, flush_r)
        evs[i][0].record(stream)
        st.append()
        evs[i][1].record(stream)
        st.attend()
        evs[i][2].record(stream)
    torch.cuda.synchronize(dev)
    t_append = [evs[i][0].elapsed_time(evs[i][1]) for i in range(K)]
    t_attn = [evs[i][1].elapsed_time(evs[i][2]) for i in range(K)]
    attn_ms = sum(t_attn) / K

    # for a co-located plan, in a separate loop of K steps, the phase times of
    # the attention call (fork to the end of the prefill kernel on its stream,
    # and to the end of the decode kernel and merge on theirs)
    phase = []
    if info["launches_per_run"] >= 2 and not batch.shape.latent:
        for i in range(K):
            _flush_l2(flush, flush_r)
            st.run()
            try:
                phase.append(fnpu.plan_phase_ms(st.plan))
            except fnpu.FnpuError:  # not co-located
                break
    torch.cuda.synchronize(dev)
    if fnpu.plan_check(st.plan) != fnpu.FNPU_OK or fnpu.check() != fnpu.FNPU_OK:
        raise RuntimeError("device error flag raised in the timed steps")

    # end to end through host buffers: H2D of the step's inputs, append + attention,
    # D2H of the outputs, all inside the timed region
    bf = torch.bfloat16
    h_q = torch.from_numpy(batch.q).view(bf).pin_memory()
    h_k = torch.from_numpy(batch.k_new).view(bf).pin_memory()
    h_v = None if batch.v_new is None else torch.from_numpy(batch.v_new).view(bf).pin_memory()
    h_s = torch.from_numpy(batch.slot_mapping).pin_memory()
    h_o = torch.empty(st.out.shape, dtype=bf).pin_memory()
    h_l = torch.empty(st.lse.shape, dtype=torch.float32).pin_memory()
    h2d = sum(x.numel() * x.element_size() for x in (h_q, h_k, h_v, h_s) if x is not None)
    d2h = h_o.numel() * h_o.element_size() + h_l.numel() * h_l.element_size()
    # (a second pass re-plans the step from its host metadata every step, as a
    # serving loop whose metadata changes does: the device is idle when the
    # timed region starts, so the plan's host time, the enqueueing and the
    # metadata upload all lie inside it)
    e2e_by_mode = {}
    for mode in ("plan_once", "replan_every_step"):
        e2e_ms = []
        for i in range(args.warmup + K):
            _flush_l2(flush, flush_r)
            a = torch.cuda.Event(enable_timing=True)
            b = torch.cuda.Event(enable_timing=True)
            if mode == "replan_every_step":
                torch.cuda.synchronize(dev)
            a.record(stream)
            if mode == "replan_every_step":
                st.replan(share_opts)
            st.q.copy_(h_q, non_blocking=True)
            st.k_new.copy_(h_k, non_blocking=True)
            if h_v is not None:
                st.v_new.copy_(h_v, non_blocking=True)
            st.slot_mapping.copy_(h_s, non_blocking=True)
            st.run()
            h_o.copy_(st.out, non_blocking=True)
            h_l.copy_(st.lse, non_blocking=True)
            b.record(stream)
            b.synchronize()
            if i >= args.warmup:
                e2e_ms.append(a.elapsed_time(b))
        e2e_by_mode[mode] = max_over_ranks(sum(e2e_ms) / len(e2e_ms), ws, dev)
    e2e = e2e_by_mode["plan_once"]
    e2e_replan = e2e_by_mode["replan_every_step"]
    host_in = {"q": h_q, "k_new": h_k, "v_new": h_v, "slot_mapping": h_s}
    e2e_pipe, host_pipe = pipelined_e2e(st, host_in, (h_o, h_l), K, args.warmup)
    e2e_pipe = max_over_ranks(e2e_pipe, ws, dev)
    e2e_pipe_replan, host_pipe_replan = pipelined_e2e(st, host_in, (h_o, h_l), K, args.warmup,
                                                      replan_opts=share_opts)
    e2e_pipe_replan = max_over_ranks(e2e_pipe_replan, ws, dev)

    # roofline of the dominant kernel: for a co-located step the prefill
    # kernel (its tile FLOPs over the prefill phase of the step, from the fork
    # to the end of the prefill stream), else the attention call (FLOPs and
    # bytes per run over its duration)
    F = work["flops"]
    B_attn = work["bytes"] - work["append_bytes"] - 8 * batch.num_tokens
    t_s = attn_ms * 1e-3
    tf_time = F / (peaks["bf16_tflops"] * 1e12)
    hb_time = B_attn / (peaks["hbm_gbs"] * 1e9)
    if phase:
        pre_ms = sum(x[0] for x in phase) / len(phase)
        F_pre = W.prefill_path_flops(batch)
        roof = {"bound": "tensor", "achieved": F_pre / (pre_ms * 1e-3) / 1e12, "peak": peaks["bf16_tflops"],
                "unit": "TFLOP/s", "kernel": "prefill_tc_kernel (fork to the end of the prefill stream)",
                "flops": F_pre, "ms": pre_ms}
    elif tf_time >= hb_time:
        roof = {"bound": "tensor", "achieved": F / t_s / 1e12, "peak": peaks["bf16_tflops"],
                "unit": "TFLOP/s", "kernel": "the attention call"}
    else:
        roof = {"bound": "hbm", "achieved": B_attn / t_s / 1e9, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                "kernel": "the attention call"}
    roof["frac"] = roof["achieved"] / roof["peak"]
    roof["traffic"] = args.traffic if args.traffic is not None else \
        NCU_TRAFFIC.get(args.workload + ("_fp8" if args.kv_fp8 else ""))
    roof["peak_source"] = peaks["source"] + " burst"
    step_roof = max(F / (peaks["bf16_tflops"] * 1e12), work["bytes"] / (peaks["hbm_gbs"] * 1e9))
    step_roof_sus = max(F / (peaks["bf16_tflops_sustained"] * 1e12), work["bytes"] / (peaks["hbm_gbs"] * 1e9))

    T = batch.num_tokens
    line = {
        "metric": METRIC, "value": job_throughput(ws, T, step_ms), "unit": UNIT, "n_gpus": ws,
        "steps": K, "warmup": args.warmup, "ms_per_step": step_ms, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "fp8-e4m3 KV, f16 products" if args.kv_fp8 else "bf16",
        "data": "synthetic",
        "config": {"workload": args.workload, "seed": args.seed, "query_tokens": T,
                   "num_seqs": batch.num_seqs, "prefill_ctx": int(batch.context_len[0]),
                   "flops": F, "bytes": work["bytes"], "l2": "flushed between timed steps (512 MB write, then 256 MB read)",
                   "plan": info, "plan_host_ms": round(statistics.median(plan_ms), 4),
                   "plan_host_ms_python": round(statistics.median(plan_py_ms), 4),
                   "plan_host_ms_planner_share": round(statistics.median(planner_ms), 4),
                   "plan_host_ms_new_plan": round(statistics.median(first_ms), 3),
                   "dispatch": args.dispatch, "kv_cache": "fp8_e4m3" if args.kv_fp8 else "bf16"},
        "roofline": roof,
        "roofline_step_frac": {"burst": step_roof / (step_ms * 1e-3),
                               "sustained": step_roof_sus / (step_ms * 1e-3),
                               "denominator": "max(F/bf16 peak, B/HBM peak) of measured"},
        "kernel_ms": {"append": sum(t_append) / K, "attention": attn_ms,
                      "step_median": statistics.median(t_step), "step_min": min(t_step),
                      "step_max": max(t_step),
                      "prefill_phase": (sum(x[0] for x in phase) / len(phase)) if phase else None,
                      "decode_phase": (sum(x[1] for x in phase) / len(phase)) if phase else None},
        # end to end as a serving loop runs it: every step's inputs up from pinned
        # host memory and its outputs down, on copy streams that overlap the
        # step before; the same with the copies and the step one after the
        # other below ("serial")
        "e2e": {"value": job_throughput(ws, T, e2e_pipe), "unit": UNIT, "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h, "ms_per_step": e2e_pipe,
                "how": "pipelined: step n's copies up and step n-1's copies down overlap step n-1's compute "
                       "(copy streams, two buffer sets), timed from the first copy up to the last copy down "
                       "over the K steps; no L2 flush, a step reads > L2",
                "host_ms_per_step": host_pipe,
                "replan_every_step": {"value": job_throughput(ws, T, e2e_pipe_replan),
                                      "ms_per_step": e2e_pipe_replan, "host_ms_per_step": host_pipe_replan},
                "serial": {"value": job_throughput(ws, T, e2e), "ms_per_step": e2e,
                           "how": "each step's copies up, step, copies down, one after the other; "
                                  "L2 flushed between steps",
                           "replan_every_step": {"value": job_throughput(ws, T, e2e_replan),
                                                 "ms_per_step": e2e_replan}}},
        "gpu_launches": K * (1 + info["launches_per_run"]),  # the append and the run's launches
        "clocks": clk,
    }
    if args.dispatch == "feedback":
        line["config"]["decode_share_pct"] = share
        line["config"]["dispatch_trace"] = trace  # [share %, prefill us, decode us] per warm-up step
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = (cpu_baseline_fp8 if args.kv_fp8 else cpu_baseline)(batch, target_seconds=args.ref_seconds)
    elif rank == 0:
        line["cpu_baseline"] = None
    if rank == 0:
        print(json.dumps(line), flush=True)
    if ws > 1:
        dist.barrier()
        dist.destroy_process_group()
    return 0


def main(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="fnpu", choices=["fnpu", "reference"])
    ap.add_argument("--workload", default="qwen_coloc", choices=list(W.CONFIG_NAMES))
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--split", type=int, default=0, help="decode split keys (0 = planner)")
    ap.add_argument("--decode-share", type=int, default=0)
    ap.add_argument("--dispatch", default="feedback", choices=["planner", "feedback"],
                    help="decode share of a co-located step: the phase-time feedback loop run over "
                         "the warm-up steps (default), or the planner's model alone")
    ap.add_argument("--flags", type=int, default=0)
    ap.add_argument("--ref-seconds", type=float, default=15.0)
    ap.add_argument("--traffic", type=float, default=None,
                    help="ncu dram bytes per attention launch, if measured for this kernel")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--mla-expand", action="store_true",
                    help="MLA prefill without absorption: latent rows expanded into per-head K/V, then MHA "
                         "(latent prefill workloads: mla_prefill)")
    ap.add_argument("--kv-fp8", action="store_true",
                    help="FP8 (e4m3) KV cache (Qwen-shaped workloads)")
    args = ap.parse_args(argv)
    args.warmup = max(args.warmup, 3)  # at least three untimed warm-up steps
    if args.impl == "reference":
        return run_reference(args)
    if args.mla_expand:
        return run_fnpu_mla_expand(args)
    return run_fnpu(args)


if __name__ == "__main__":
    sys.exit(main())
