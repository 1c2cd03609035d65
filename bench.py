"""Decode-step throughput of the budgeted KV-eviction hot path on GB300.

One step = dc_decode_step + dc_evict over every layer and sequence of the
workload: Mistral-7B KV shape (32 layers, 32 query / 8 KV heads, head_dim 128),
batch 8, 32K-token prompt compressed to a 25% budget (8192 tokens per row), one
token appended and one evicted per row per step. Inputs are synthetic and
seeded; the prompt compression (first decode step) happens before warm-up.

Prints one JSON line (rank 0). ``--impl reference`` times the fp64 CPU oracle
on the host cores instead (a bounded sample of the same workload).
"""

from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "decode steps/s and HBM GB/s (% of 8 TB/s) at Mistral-7B shape, 25% budget"
UNIT = "decode steps/s"
NOMINAL_HBM_GBS = 8000.0


def measured_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return json.load(f), "measured"
    except Exception:
        return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0}, "fallback"


_OVERRIDES = {}


def workload():
    """The benchmark workload (Mistral-7B KV shape, 32 layers, batch 8, 32K
    context, 25% budget); --layers / --batch shrink it for profiling."""
    from paper_2608_08878_gb300 import synth
    wl = synth.MISTRAL_FULL
    if _OVERRIDES:
        wl = wl.with_(**_OVERRIDES)
        wl = wl.with_(name=f"{wl.name} [profiling case: {wl.layers} layers, batch {wl.batch}, "
                           f"{wl.q_heads}q/{wl.kv_heads}kv heads, context {wl.prompt_len}, budget {wl.budget}]")
    return wl


def row_bytes_per_step(n: int, d: int, alpha_mode: int = 0) -> int:
    """Algorithmic HBM bytes of one row's decode step over n tokens (after the
    append): K and V read once (4d bytes per token), position read (4), window
    sums S and Z read and written (32), cumulative alpha read and written in
    alpha_mode 1 (8)."""
    return n * (4 * d + 36 + (8 if alpha_mode else 0))


def step_bytes(wl, n: int, moved_per_row: float = 1.0) -> float:
    """Whole-step algorithmic bytes: every row's pass over its n tokens, the
    append (new key and value, 4d bytes, plus 20 bytes of position and window
    state written) and the compaction moves (each moved token's K/V and 20
    bytes of state read and written; one per row in the steady state)."""
    d = wl.head_dim
    per_row = row_bytes_per_step(n, d, wl.alpha_mode) + (4 * d + 20) + moved_per_row * 2 * (4 * d + 20)
    return wl.rows * per_row


def step_bytes_global(wl, n: int, moved_per_seq: float = 1.0) -> float:
    """Whole-step algorithmic bytes of the global token mode: every row's K, V
    and positions read once (4d + 4 bytes per token-row); per sequence and
    token, the window sums read and written (32), the ring's previous and
    departing query terms read and this query's written (24), cumulative alpha
    in alpha_mode 1 (8); the append; each sequence's moves, on every row. The
    rows' partial sums are the implementation's exchange, not counted."""
    d = wl.head_dim
    per_seq_tok = 32 + 24 + (8 if wl.alpha_mode else 0)
    return (wl.rows * n * (4 * d + 4) + wl.batch * n * per_seq_tok + wl.rows * (4 * d + 20)
            + moved_per_seq * wl.rows * 2 * (4 * d + 20))


# The fused kernel's source: the kernel template and every header it includes.
FUSED_KERNEL_SOURCES = ["dc_fused_kernel.cuh", "dc_common.cuh", "dc_fused.h", "dc_kernels.h", "dc_select.cuh",
                        "dc_sm100.cuh"]


def fused_kernel_source_sha() -> str:
    """sha256 of the fused kernel's source files, concatenated in the order above."""
    import hashlib
    h = hashlib.sha256()
    for f in FUSED_KERNEL_SOURCES:
        with open(os.path.join(ROOT, "paper_2608_08878_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()


def fused_traffic_per_token_row():
    """DRAM bytes per token-row of the fused kernel from the committed one-pass
    ncu capture of the benchmark workload at full size, or None if the kernel
    source changed since it was captured."""
    import re
    prof = os.path.join(ROOT, "profiles", "fused_kernel_mistral7b_32L_b8_ctx32k_dram_traffic.md")
    try:
        text = open(prof).read()
        t = float(re.search(r"traffic_bytes_per_token_row:\s*([0-9.]+)", text).group(1))
        sha = re.search(r"kernel_source_sha256_prefix:\s*([0-9a-f]+)", text).group(1)
        return t if fused_kernel_source_sha()[:len(sha)] == sha else None
    except Exception:
        return None


class ClockSampler:
    """nvidia-smi clock/throttle samples while the timed region runs."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    PERIOD_MS = 20

    def __init__(self, index: str):
        self.index = index
        self.proc = None
        self.lines = []
        self.ready = threading.Event()

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", self.index, f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", str(self.PERIOD_MS)],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
            # the timed region starts once nvidia-smi is sampling (its start-up
            # takes longer than a short timed region)
            self.ready.wait(timeout=5.0)
            self.lines.clear()
        except Exception:
            self.proc = None
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())
            self.ready.set()

    def __exit__(self, *a):
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()
            self.thread.join(timeout=2)

    def summary(self):
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                mx = float(parts[2])
            except ValueError:
                continue
            for nm, val in zip(names, parts[5:9]):
                if val.lower().startswith("active"):
                    reasons.add(nm)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": mx,
                "reasons": sorted(reasons), "samples": len(sm), "period_ms": self.PERIOD_MS}


def gpu_index_for_smi(local_rank: int) -> str:
    vis = os.environ.get("CUDA_VISIBLE_DEVICES")
    if vis:
        ids = [x.strip() for x in vis.split(",") if x.strip()]
        if local_rank < len(ids):
            return ids[local_rank]
    return str(local_rank)


# ---------------------------------------------------------------------------
# CPU oracle leg (cpu_baseline and --impl reference)
# ---------------------------------------------------------------------------

def oracle_sample(wl, seconds: float = 12.0, threads: int | None = None, warm_steps: int | None = None):
    """Times the fp64 oracle on a bounded sample: `threads` rows of the steady
    state (n = budget + 1 after the append), each run for several decode steps
    with a full entropy window, rows in parallel on host threads. Returns
    decode steps/s of the whole workload extrapolated from the sample."""
    import numpy as np
    import oracle
    from paper_2608_08878_gb300 import synth
    oracle.build()
    cores = os.cpu_count() or 1
    threads = threads or max(1, min(16, cores))
    warm_steps = wl.window if warm_steps is None else warm_steps
    blob = synth.policy_weights(wl.policy_seed, wl.mlp_hidden)
    sample_rows = [int(r) for r in np.linspace(0, wl.rows - 1, threads).astype(int)]
    rows = {}

    def setup(r):
        layer, b, g = wl.row_coords(r)
        o = oracle.OracleRow(wl.head_dim, wl.group, wl.window, wl.alpha_mode, wl.budget + 2)
        k, v = synth.prompt_row(wl, layer, b, g, 0, wl.budget)
        o.append(k, v)
        for s in range(warm_steps):
            qb, kb, vb = synth.step_row(wl, s, layer, b, g)
            o.step(qb, kb, vb, blob, wl.mlp_hidden, wl.layernorm)
            o.evict(wl.budget)
        rows[r] = o

    ts = [threading.Thread(target=setup, args=(r,)) for r in sample_rows]
    [t.start() for t in ts]
    [t.join() for t in ts]
    # timed: each thread steps its row until the time budget is used
    counts = {r: 0 for r in sample_rows}
    deadline = [0.0]

    def run(r):
        layer, b, g = wl.row_coords(r)
        o = rows[r]
        s = warm_steps
        while time.perf_counter() < deadline[0] or counts[r] == 0:
            qb, kb, vb = synth.step_row(wl, s, layer, b, g)
            o.step(qb, kb, vb, blob, wl.mlp_hidden, wl.layernorm)
            o.evict(wl.budget)
            counts[r] += 1
            s += 1

    t0 = time.perf_counter()
    deadline[0] = t0 + seconds
    ts = [threading.Thread(target=run, args=(r,)) for r in sample_rows]
    [t.start() for t in ts]
    [t.join() for t in ts]
    el = time.perf_counter() - t0
    row_steps = sum(counts.values())
    steps_per_s = row_steps / wl.rows / el
    # the same on one host thread: one sampled row for a third of the time
    r1 = sample_rows[0]
    counts = {r1: 0}
    t1 = time.perf_counter()
    deadline[0] = t1 + seconds / 3
    run(r1)
    el1 = time.perf_counter() - t1
    return {"value": steps_per_s, "unit": UNIT, "cores": len(sample_rows), "host_cores": cores,
            "kind": "oracle", "extrapolated": True, "row_steps_run": row_steps, "seconds": el,
            "sample": (f"{len(sample_rows)} rows (of {wl.rows}) at the steady state n={wl.budget + 1}, "
                       f"full w={wl.window} window, {row_steps} row-steps in {el:.1f}s on "
                       f"{len(sample_rows)} host threads (of {cores} host cores); whole decode steps/s "
                       f"extrapolated as row-steps / rows / s (rows are independent)"),
            "single_thread": {"value": counts[r1] / wl.rows / el1, "unit": UNIT, "cores": 1,
                              "host_cores": cores, "extrapolated": True, "row_steps_run": counts[r1],
                              "sample": f"row {r1}, {counts[r1]} row-steps in {el1:.1f}s on one host thread"}}


# ---------------------------------------------------------------------------
# GPU leg
# ---------------------------------------------------------------------------

def bench_config(wl, args, world: int) -> dict:
    """The workload description both arms print (the same dict for the same
    flags): shape, budget rule, selection mode and scorer."""
    n_steady = wl.budget + 1
    bytes_step = step_bytes_global(wl, n_steady) if args.global_tokens else step_bytes(wl, n_steady)
    return {"workload": wl.name, "layers": wl.layers, "batch": wl.batch, "q_heads": wl.q_heads,
            "kv_heads": wl.kv_heads, "head_dim": wl.head_dim, "context": wl.prompt_len,
            "budget": wl.budget, "window": wl.window, "policy": f"5-{wl.mlp_hidden}-LN-ReLU-1",
            "parallelism": f"replicas x{world}",
            "selection": "per sequence (global token mode)" if args.global_tokens else
            "per (layer, KV head) row" + (", head-level hybrid budgets" if args.hybrid else ""),
            "scorer": ["policy MLP", "H2O (cumulative attention)", "StreamingLLM (sinks + recent)"][args.scorer],
            "budget_rule": (f"dynamic: max(floor({args.budget_ratio} x tokens seen), 32)"
                            if args.budget_ratio > 0 else "fixed"),
            "timed_state": (f"after the prompt compression and {wl.window} + warm-up decode steps: "
                            f"a full w = {wl.window} entropy window, every step subtracts a departing query"),
            "l2": f"inputs larger than L2: {bytes_step / 1e9:.2f} GB streamed per step vs 129 MB L2",
            "steady_tokens_per_row": n_steady}


def job_throughput(el_ms: float, steps: int, dist=None, device="cpu"):
    """(max elapsed ms over ranks, whole-job decode steps/s): every rank runs
    `steps` steps of its own replica and the job ends with the slowest rank."""
    world = 1
    if dist is not None:
        import torch
        world = dist.get_world_size()
        t = torch.tensor([el_ms], dtype=torch.float64, device=device)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        el_ms = float(t.item())
    return el_ms, world * steps / (el_ms / 1e3)


def roofline_of(prof, wl, n_steady, engine, global_tokens=False):
    """(dominant phase, per-launch ms, algorithmic bytes per launch, launches)
    from the library's per-launch CUDA events: the fused kernel's bytes are
    the whole step's but the append (K/V, positions, window sums, one move
    per row); the split engine's kernels count their own reads and writes."""
    dom = max((ph for ph in prof if prof[ph][1] > 0), key=lambda ph: prof[ph][0])
    dom_ms, dom_n = prof[dom]
    d = wl.head_dim
    if dom == "attend" and engine.startswith("fused") and global_tokens:
        alg = wl.rows * n_steady * (4 * d + 4)  # the rows' pass: K/V and positions
    elif dom == "attend" and engine.startswith("fused"):
        alg = wl.rows * (row_bytes_per_step(n_steady, d, wl.alpha_mode) + 2 * (4 * d + 20))
    elif dom == "attend":
        alg = wl.rows * n_steady * (2 * d + 36)  # K read + positions + window sums R/W
    elif dom == "score":
        alg = wl.rows * n_steady * (2 * d + 20)  # V read + positions + window sums read
    else:
        alg = wl.rows * row_bytes_per_step(n_steady, d, wl.alpha_mode)
    return dom, dom_ms / dom_n, alg, dom_n


def timed_steps(cache, inputs, s0, K, out, stream, index):
    """K dc_step calls from inputs[s0], CUDA events on the launching stream,
    clocks sampled meanwhile: (ms per step, clocks summary)."""
    import torch
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    with ClockSampler(index) as clk:
        ev0.record(stream)
        for s in range(s0, s0 + K):
            cache.step(*inputs[s], out=out)
        ev1.record(stream)
        torch.cuda.synchronize()
    cache.sync()  # device-side status of every timed step (raises on error)
    return ev0.elapsed_time(ev1) / K, clk.summary()


def timed_then_profiled(cache, inputs, s0, K, out, stream, index):
    """For steps of tens of microseconds, where the library's per-launch
    events would add to the step time: K steps timed with launch counting
    only, then the same K inputs again with per-launch events (for the
    roofline). Returns (ms per step, clocks, per-launch profile)."""
    cache.profile(False)  # counts launches, records no events
    ms, clocks = timed_steps(cache, inputs, s0, K, out, stream, index)
    cache.profile(True)
    for s in range(s0, s0 + K):
        cache.step(*inputs[s], out=out)
    prof = cache.profile_read()
    cache.profile(False)
    return ms, clocks, prof


def warm_modules(wl, args):
    """Runs the prompt compression's kernels once on a small cache of the
    workload's head shape (one layer, one sequence, a prompt past the on-chip
    logit capacity), so that the timed first step does not include the lazy
    loading of their modules."""
    import torch
    from paper_2608_08878_gb300 import dc, synth_device
    small = wl.with_(layers=1, batch=1, prompt_len=12000, budget=3000)
    c = dc.DistillCache(1, wl.kv_heads, wl.head_dim, small.prompt_len + 8, small.budget, batch=1,
                        q_heads=wl.q_heads, window=wl.window, mlp_hidden=wl.mlp_hidden, layernorm=wl.layernorm,
                        engine=args.engine)
    k, v = synth_device.prompt(small, 0, small.prompt_len)
    c.append(k, v)
    q, kn, vn = synth_device.step_inputs(small, 0)
    c.decode_step(q, kn, vn)
    c.evict()
    c.step(*synth_device.step_inputs(small, 1))
    c.sync()
    c.close()
    torch.cuda.synchronize()


def run_gpu(args):
    import torch
    from paper_2608_08878_gb300 import build, dc, synth, synth_device
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local_rank)
    dist = None
    if world > 1:
        import torch.distributed as tdist
        tdist.init_process_group("nccl", device_id=torch.device("cuda", local_rank))
        dist = tdist
    if local_rank == 0:
        build.build()
    if dist:
        dist.barrier()
    wl0 = workload()
    wl = wl0.with_(seed=wl0.seed + 1000 * rank)
    K, W = args.steps, args.warmup
    # untimed decode steps after the prompt compression, so that the entropy
    # window is full: every timed step adds the previous query's window terms
    # and subtracts a departing query's
    F = wl.window
    stream = torch.cuda.current_stream()
    cache = make_cache(wl, args)
    if args.scorer == 1:  # H2O ranks by cumulative attention (alpha_mode 1 state)
        wl = wl.with_(alpha_mode=1)
    chunk = 4096
    # all step inputs resident in HBM before timing
    inputs = [synth_device.step_inputs(wl, s) for s in range(1 + F + W + K)]
    out = torch.empty((wl.layers, wl.batch, wl.q_heads, wl.head_dim), dtype=torch.float32, device="cuda")
    # step 0: prompt compression (32769 -> 8192 tokens per row), timed apart,
    # after the kernels it runs are loaded (CUDA loads a module at the first
    # launch of one of its kernels, inside the launch call)
    warm_modules(wl, args)
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    cache.profile(True)
    ev0.record(stream)
    cache.step(*inputs[0], out=out)
    ev1.record(stream)
    torch.cuda.synchronize()
    first_ms = ev0.elapsed_time(ev1)
    first_prof = cache.profile_read()
    cache.profile(False)
    # the prompt compression (first step): per-phase kernel time, and the
    # slot moves of its many-eviction compaction (a slot below the budget
    # holds a position at or above it only if a survivor moved there)
    first = {"ms": first_ms, "phases_ms": {k: v[0] for k, v in first_prof.items() if v[1]}}
    if not (args.hybrid or args.budget_ratio > 0 or args.global_tokens):
        pos = cache.buffer(dc.BUF_POS)[:, :wl.budget]
        moved = int((pos >= wl.budget).sum().item())
        del pos
        mv_bytes = moved * 2 * (4 * wl.head_dim + 20)
        first["moved_slots"] = moved
        first["move_bytes"] = mv_bytes
        if "evict" in first["phases_ms"]:
            first["evict_move_gbs"] = mv_bytes / (first["phases_ms"]["evict"] / 1e3) / 1e9
        torch.cuda.empty_cache()

    for s in range(1, 1 + F + W):
        cache.step(*inputs[s], out=out)
    n_steady = cache.length()[0] + 1
    if args.hybrid or args.budget_ratio > 0:  # mean row length after the next append
        n_steady = float(cache.row_lengths().mean()) + 1
    engine = cache.engine()
    # steps taken so far >= w: the next (first timed) step has a departing query
    window_full = cache.length()[1] - wl.prompt_len >= wl.window
    cache.profile(True)
    torch.cuda.synchronize()
    if dist:
        dist.barrier()
    ms_per_step, clocks = timed_steps(cache, inputs, 1 + F + W, K, out, stream, gpu_index_for_smi(local_rank))
    prof = cache.profile_read()
    cache.profile(False)
    el_ms, value = job_throughput(ms_per_step * K, K, dist, device="cuda")
    ms_per_step = el_ms / K
    bytes_step = step_bytes_global(wl, n_steady) if args.global_tokens else step_bytes(wl, n_steady)
    gbs = bytes_step / (ms_per_step / 1e3) / 1e9
    peaks, peak_src = measured_peaks()

    # dominant kernel: roofline from the live per-launch events
    dom, per_launch_ms, alg, _ = roofline_of(prof, wl, n_steady, engine, args.global_tokens)
    achieved = alg / (per_launch_ms / 1e3) / 1e9
    traffic = None
    if dom == "attend" and engine.startswith("fused") and not (args.global_tokens or args.hybrid or args.scorer):
        tpr = fused_traffic_per_token_row()
        if tpr is not None:
            traffic = wl.rows * n_steady * tpr  # the full-size capture's bytes per token-row
    gpu_launches = int(sum(v[1] for v in prof.values()))
    # full-cache comparator on the same inputs (the uncompressed prompt)
    full = None
    if not args.no_full and rank == 0:
        del cache
        torch.cuda.empty_cache()
        fc = dc.DistillCache(wl.layers, wl.kv_heads, wl.head_dim, wl.prompt_len + 1, wl.budget,
                             batch=wl.batch, q_heads=wl.q_heads, window=wl.window, engine=args.engine)
        for t0 in range(0, wl.prompt_len, chunk):
            k, v = synth_device.prompt(wl, t0, min(chunk, wl.prompt_len - t0))
            fc.append(k, v)
            del k, v
        for s in range(W):
            fc.full_decode(inputs[s][0], out=out)
        kf = min(K, 32)
        torch.cuda.synchronize()
        ev0.record(stream)
        for s in range(kf):
            fc.full_decode(inputs[1 + F + W + s][0], out=out)
        ev1.record(stream)
        torch.cuda.synchronize()
        fms = ev0.elapsed_time(ev1) / kf
        fbytes = wl.rows * wl.prompt_len * 4 * wl.head_dim
        full = {"ms_per_step": fms, "steps_per_s": 1e3 / fms, "n_tokens_per_row": wl.prompt_len,
                "gbs": fbytes / (fms / 1e3) / 1e9, "speedup_of_eviction_step": fms / ms_per_step}
        del fc
        torch.cuda.empty_cache()
        cache = None

    # end to end through the public API with host buffers (every rank its own
    # replica)
    e2e = None
    if not args.no_e2e:
        e2e = run_e2e(wl, args, inputs, F)
    del inputs
    torch.cuda.empty_cache()

    # the other workloads, each in the bench's launch configuration (rank 0 of
    # a one-GPU run)
    extra = {}
    if not args.no_extra and rank == 0 and world == 1 and not _OVERRIDES:
        extra = run_extra_workloads(args, peaks, stream, gpu_index_for_smi(local_rank))

    res = None
    if rank == 0:
        cfg = bench_config(wl0, args, world)
        cfg["steady_tokens_per_row"] = n_steady
        res = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": K, "warmup": W,
            "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "bf16", "data": "synthetic",
            "config": cfg,
            "engine": engine,
            "window_full": bool(window_full),
            "untimed_steps_before_warmup": 1 + F,
            "hbm": {"algorithmic_bytes_per_step": bytes_step, "gbs": gbs,
                    "frac_of_8tbs": gbs / NOMINAL_HBM_GBS,
                    "frac_of_measured": gbs / peaks["hbm_gbs"], "peak_source": peak_src},
            "first_step_ms": first_ms,
            "first_step": first,
            "roofline": {"bound": "hbm", "kernel": dom, "achieved": achieved, "peak": peaks["hbm_gbs"],
                         "unit": "GB/s", "frac": achieved / peaks["hbm_gbs"], "traffic": traffic,
                         "peak_source": f"{peak_src} copy bandwidth",
                         "per_launch_ms": per_launch_ms, "algorithmic_bytes_per_launch": alg},
            "phases_ms_per_step": {k: v[0] / K for k, v in prof.items() if v[1]},
            "gpu_launches": gpu_launches,
            "clocks": clocks,
            "full_cache": full,
            "e2e": e2e,
        }
        res.update(extra)
    if dist:
        dist.barrier()
        dist.destroy_process_group()
    return res


def make_cache(wl, args):
    """The cache of the timed run, with the mode the flags select, holding the
    workload's prompt."""
    from paper_2608_08878_gb300 import dc, synth_device
    cap = wl.capacity
    if args.hybrid:  # full-cache rows grow by one token per step
        cap = wl.prompt_len + 2 + args.warmup + args.steps
    cache = dc.DistillCache(wl.layers, wl.kv_heads, wl.head_dim, cap, wl.budget,
                            batch=wl.batch, q_heads=wl.q_heads, window=wl.window,
                            mlp_hidden=wl.mlp_hidden, layernorm=wl.layernorm, engine=args.engine,
                            seed=wl.policy_seed, global_tokens=args.global_tokens, scorer=args.scorer,
                            budget_ratio=args.budget_ratio)
    if args.hybrid:
        # head-level hybrid (Sec. 5): every fifth row (20% of the heads) keeps its
        # full cache, the others share the rest of a 25% overall budget
        cache.set_row_budgets(dc.head_level_hybrid_budgets(wl.rows, wl.prompt_len,
                                                           range(0, wl.rows, 5), 0.25))
    chunk = 4096
    for t0 in range(0, wl.prompt_len, chunk):
        k, v = synth_device.prompt(wl, t0, min(chunk, wl.prompt_len - t0))
        cache.append(k, v)
        del k, v
    return cache


def run_e2e(wl, args, inputs, F):
    """The same steps through the host-buffer API: every step copies its pinned
    host inputs in and the attention output out (dc_step_host_async, in the
    handle's stream order; one synchronisation at the end of the timed region,
    which therefore holds every copy). The same untimed steps come first."""
    import torch
    cache = make_cache(wl, args)
    host = [tuple(x.cpu().pin_memory() for x in inp) for inp in inputs]
    out = torch.empty((wl.layers, wl.batch, wl.q_heads, wl.head_dim), dtype=torch.float32).pin_memory()
    W, K = args.warmup, args.steps
    for s in range(0, 1 + F + W):
        cache.step_host(*host[s], out)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    for s in range(1 + F + W, 1 + F + W + K):
        cache.step_host_async(*host[s], out)
    cache.sync()
    el = time.perf_counter() - t0
    h2d = sum(x.numel() * x.element_size() for x in host[0])
    d2h = out.numel() * out.element_size()
    cache.close()
    return {"value": K / el, "unit": UNIT, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
            "ms_per_step": el / K * 1e3}


def run_reference(args):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return None
    wl = workload()
    cb = oracle_sample(wl, seconds=args.cpu_seconds)
    world = int(os.environ.get("WORLD_SIZE", "1"))
    return {"impl": "reference", "metric": METRIC, "value": cb["value"], "unit": UNIT,
            "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": 1e3 / cb["value"], "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "extrapolated": True,
            "timing_note": (f"not {args.steps} whole steps: {cb['row_steps_run']} row-steps of {wl.rows}-row "
                            f"decode steps in {cb['seconds']:.1f}s on {cb['cores']} host threads, "
                            f"extrapolated to whole steps (rows are independent)"),
            "config": bench_config(wl, args, world),
            "cpu_baseline": cb,
            "e2e": {"value": cb["value"], "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}


# ---------------------------------------------------------------------------
# Throughput sweep (batch x context x budget ratio), one JSON line per point
# ---------------------------------------------------------------------------

SWEEP_BATCH = (1, 4, 16, 64)
SWEEP_CONTEXT = (4096, 16384, 32768)
SWEEP_RATIO = (0.10, 0.25, 0.50)


def sweep_point_run(b, c, r, K, W, engine_flag, peaks, stream, index, with_full=True):
    """One sweep point: the steady cache (B prompt tokens, then steps that
    append one token and evict one, the state after prompt compression), W
    warm-up and K timed dc_step calls, roofline of the dominant kernel from
    the library's per-launch events, and (with_full) full-cache attention over
    context + 1 tokens, timed on as many layers as fit in 48 GB and scaled to
    32 layers (its time is linear in the rows)."""
    import torch
    from paper_2608_08878_gb300 import dc, synth, synth_device
    wl = synth.sweep_point(b, c, r)
    B, d = wl.budget, wl.head_dim
    cache = dc.DistillCache(wl.layers, wl.kv_heads, d, B + 1, B, batch=b, q_heads=wl.q_heads,
                            window=wl.window, mlp_hidden=wl.mlp_hidden, layernorm=wl.layernorm,
                            seed=wl.policy_seed, engine=engine_flag)
    chunk = max(1, min(B, (1 << 31) // (wl.rows * d * 2)))
    for t0 in range(0, B, chunk):
        k, v = synth_device.prompt(wl, t0, min(chunk, B - t0))
        cache.append(k, v)
        del k, v
    inputs = [synth_device.step_inputs(wl, s) for s in range(W + K)]
    out = torch.empty((wl.layers, b, wl.q_heads, d), dtype=torch.float32, device="cuda")
    for s in range(W):
        cache.step(*inputs[s], out=out)
    engine = cache.engine()
    ms, clocks, prof = timed_then_profiled(cache, inputs, W, K, out, stream, index)
    dom, per_launch_ms, alg, _ = roofline_of(prof, wl, B + 1, engine)
    achieved = alg / (per_launch_ms / 1e3) / 1e9
    bytes_step = step_bytes(wl, B + 1)
    del cache, inputs, out
    torch.cuda.empty_cache()
    gbs = bytes_step / (ms / 1e3) / 1e9
    res = {"sweep_point": f"{b}x{c}x{int(round(r * 100))}", "workload": wl.name, "batch": b, "context": c,
           "ratio": r, "budget": B, "rows": wl.rows, "engine": engine, "steps": K, "warmup": W,
           "ms_per_step": ms, "steps_per_s": 1e3 / ms, "gbs": gbs,
           "frac_of_8tbs": gbs / NOMINAL_HBM_GBS, "frac_of_measured": gbs / peaks["hbm_gbs"],
           "roofline": {"bound": "hbm", "kernel": dom, "achieved": achieved, "peak": peaks["hbm_gbs"],
                        "unit": "GB/s", "frac": achieved / peaks["hbm_gbs"], "per_launch_ms": per_launch_ms,
                        "algorithmic_bytes_per_launch": alg},
           "footprint_steady_gb": wl.rows * (B + 1) * (4 * d + 20) / 1e9,
           "footprint_prompt_gb": wl.rows * (c + 1) * (4 * d + 20) / 1e9,
           "clocks": clocks, "data": "synthetic"}
    if not with_full:
        return res
    per_layer = b * wl.kv_heads * (c + 1) * (4 * d + 20)
    lf = max(1, min(wl.layers, int(48e9 // per_layer)))
    wf = wl.with_(layers=lf)
    full = dc.DistillCache(lf, wl.kv_heads, d, c + 1, c, batch=b, q_heads=wl.q_heads)
    chunk = max(1, min(c + 1, (1 << 31) // (wf.rows * d * 2)))
    for t0 in range(0, c + 1, chunk):
        k, v = synth_device.prompt(wf, t0, min(chunk, c + 1 - t0))
        full.append(k, v)
        del k, v
    qf = synth_device.step_inputs(wf, 0)[0]
    for _ in range(2):
        full.full_decode(qf)
    torch.cuda.synchronize()
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    reps = 5
    ev0.record(stream)
    for _ in range(reps):
        full.full_decode(qf)
    ev1.record(stream)
    torch.cuda.synchronize()
    full_ms = ev0.elapsed_time(ev1) / reps * wl.layers / lf
    del full, qf
    torch.cuda.empty_cache()
    res.update({"full_cache_ms_per_step": full_ms, "full_cache_layers_timed": lf,
                "speedup_vs_full": full_ms / ms})
    return res


def workload_run(wl, steps_total, W, engine_flag, peaks, stream, index):
    """A workload as its configuration states it: the prompt, then
    `steps_total` decode steps (dc_step) of which the first is the prompt
    compression (timed apart), the next W warm-up and the rest timed; roofline
    of the dominant kernel from the library's per-launch events."""
    import torch
    from paper_2608_08878_gb300 import dc, synth_device
    cache = dc.DistillCache(wl.layers, wl.kv_heads, wl.head_dim, wl.capacity, wl.budget, batch=wl.batch,
                            q_heads=wl.q_heads, window=wl.window, mlp_hidden=wl.mlp_hidden,
                            layernorm=wl.layernorm, seed=wl.policy_seed, engine=engine_flag)
    chunk = max(1, min(wl.prompt_len, (1 << 31) // (wl.rows * wl.head_dim * 2)))
    for t0 in range(0, wl.prompt_len, chunk):
        k, v = synth_device.prompt(wl, t0, min(chunk, wl.prompt_len - t0))
        cache.append(k, v)
        del k, v
    inputs = [synth_device.step_inputs(wl, s) for s in range(steps_total)]
    out = torch.empty((wl.layers, wl.batch, wl.q_heads, wl.head_dim), dtype=torch.float32, device="cuda")
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    ev0.record(stream)
    cache.step(*inputs[0], out=out)
    ev1.record(stream)
    torch.cuda.synchronize()
    first_ms = ev0.elapsed_time(ev1)
    for s in range(1, 1 + W):
        cache.step(*inputs[s], out=out)
    engine = cache.engine()
    K = steps_total - 1 - W
    ms, clocks, prof = timed_then_profiled(cache, inputs, 1 + W, K, out, stream, index)
    n = wl.budget + 1
    dom, per_launch_ms, alg, _ = roofline_of(prof, wl, n, engine)
    achieved = alg / (per_launch_ms / 1e3) / 1e9
    bytes_step = step_bytes(wl, n)
    del cache, inputs, out
    torch.cuda.empty_cache()
    gbs = bytes_step / (ms / 1e3) / 1e9
    return {"workload": wl.name, "rows": wl.rows, "tokens_per_row": n, "engine": engine,
            "decode_steps": steps_total, "first_step_ms": first_ms, "warmup": W, "steps": K,
            "ms_per_step": ms, "us_per_step": ms * 1e3, "steps_per_s": 1e3 / ms,
            "hbm": {"algorithmic_bytes_per_step": bytes_step, "gbs": gbs,
                    "frac_of_measured": gbs / peaks["hbm_gbs"]},
            "roofline": {"bound": "hbm", "kernel": dom, "achieved": achieved, "peak": peaks["hbm_gbs"],
                         "unit": "GB/s", "frac": achieved / peaks["hbm_gbs"], "per_launch_ms": per_launch_ms,
                         "algorithmic_bytes_per_launch": alg},
            "clocks": clocks, "data": "synthetic"}


SWEEP_WORST = ((1, 4096, 0.10), (4, 4096, 0.10), (64, 4096, 0.10), (1, 32768, 0.50))


def run_extra_workloads(args, peaks, stream, index):
    """The other configurations next to the headline, each timed the same
    way: the Mistral-7B single layer (8 rows of 2049 tokens, 128 decode
    steps, latency-bound), the aggressive 10% workload (32 layers, batch 16,
    hot sets reshuffled every 16 steps, 64 decode steps) and the sweep's
    slowest points (short rows at 10%, one 32K row set at 50%)."""
    from paper_2608_08878_gb300 import synth
    W = args.warmup
    out = {"config2": workload_run(synth.MISTRAL_1L, synth.MISTRAL_1L.steps, W, args.engine, peaks, stream, index)}
    out["config2"]["note"] = ("9 MB of algorithmic traffic per step: bound by launch and per-row latency, "
                              "not HBM; the roofline fraction is reported for completeness")
    out["config4"] = workload_run(synth.AGGRESSIVE, synth.AGGRESSIVE.steps, W, args.engine, peaks, stream, index)
    out["sweep_worst"] = [sweep_point_run(b, c, r, 32, W, args.engine, peaks, stream, index, with_full=False)
                          for b, c, r in SWEEP_WORST]
    return out


def run_sweep(args):
    """Steady-state decode steps/s per point of the sweep (batch x context x
    budget ratio), one JSON line each, next to full-cache attention on the
    same shapes."""
    import torch
    from paper_2608_08878_gb300 import build
    torch.cuda.set_device(0)
    build.build()
    peaks, _ = measured_peaks()
    stream = torch.cuda.current_stream()
    pts = [(b, c, r) for b in SWEEP_BATCH for c in SWEEP_CONTEXT for r in SWEEP_RATIO]
    if args.sweep_points:
        keep = set(args.sweep_points.split(","))
        pts = [p for p in pts if f"{p[0]}x{p[1]}x{int(round(p[2] * 100))}" in keep]
    for b, c, r in pts:
        print(json.dumps(sweep_point_run(b, c, r, args.steps, args.warmup, args.engine, peaks, stream,
                                         gpu_index_for_smi(0))), flush=True)


def run_train(args):
    """Training-side kernels (App. C) at the paper's training scale (L = 4096
    tokens, B = 1024): the exact Plackett-Luce log-partition and Gumbel-top-B
    with log-probabilities, for 64 sequences; one JSON line."""
    import torch
    from paper_2608_08878_gb300 import build, dc
    torch.cuda.set_device(0)
    build.build()
    rows, L, B, tau = 64, 4096, 1024, 1.0
    g = torch.Generator(device="cuda").manual_seed(5)
    s = torch.randn((rows, L), device="cuda", generator=g) * 3.0
    u = torch.rand((rows, L), device="cuda", generator=g).clamp_(1e-12, 1.0 - 1e-7)
    gum = -torch.log(-torch.log(u))
    stream = torch.cuda.current_stream()
    out = {}
    for name, fn in (("log_partition", lambda: dc.pl_log_partition(s, B, tau)),
                     ("gumbel_top_b_with_logp", lambda: dc.gumbel_top_b(s, gum, B, tau))):
        for _ in range(3):
            fn()
        torch.cuda.synchronize()
        ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        reps = 10
        ev0.record(stream)
        for _ in range(reps):
            fn()
        ev1.record(stream)
        torch.cuda.synchronize()
        ms = ev0.elapsed_time(ev1) / reps
        out[name] = {"ms_per_call": ms, "dp_cells_per_s": rows * L * B / (ms / 1e3)}
    print(json.dumps({"training_kernels": out, "rows": rows, "L": L, "B": B, "tau": tau,
                      "data": "synthetic"}), flush=True)


def main():
    ap = argparse.ArgumentParser(description=__doc__.splitlines()[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--engine", type=int, default=0, help="0 auto, 1 split, 2 fused")
    ap.add_argument("--cpu-seconds", type=float, default=12.0)
    ap.add_argument("--no-cpu", action="store_true")
    ap.add_argument("--no-full", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-extra", action="store_true",
                    help="skip the other workloads (single layer, aggressive 10%%, the sweep's slowest points)")
    ap.add_argument("--layers", type=int, default=None, help="profiling: fewer layers than the workload's 32")
    ap.add_argument("--batch", type=int, default=None, help="profiling: another batch than the workload's 8")
    ap.add_argument("--context", type=int, default=None, help="profiling: another prompt length than 32768")
    ap.add_argument("--budget", type=int, default=None, help="profiling: another budget than 8192")
    ap.add_argument("--q-heads", type=int, default=None, help="profiling: query heads per layer (32)")
    ap.add_argument("--kv-heads", type=int, default=None, help="profiling: KV heads per layer (8)")
    ap.add_argument("--sweep", action="store_true",
                    help="throughput sweep (batch x context x ratio): one JSON line per point")
    ap.add_argument("--sweep-points", default=None, help="e.g. 1x4096x10,64x32768x50 (default: all 36)")
    ap.add_argument("--train", action="store_true", help="time the training-side kernels (App. C)")
    ap.add_argument("--hybrid", action="store_true",
                    help="head-level hybrid: 20%% of the rows keep the full cache, the rest share a 25%% budget")
    ap.add_argument("--scorer", type=int, choices=[0, 1, 2], default=0,
                    help="0 policy MLP, 1 H2O, 2 StreamingLLM (the heuristic scorers on the same path)")
    ap.add_argument("--budget-ratio", type=float, default=0.0,
                    help="> 0: dynamic budget B_t = max(floor(r x tokens seen), 32) instead of the fixed 8192")
    ap.add_argument("--global-tokens", action="store_true",
                    help="the global token mode (features over all heads and layers, one selection per sequence)")
    args = ap.parse_args()
    if args.layers:
        _OVERRIDES["layers"] = args.layers
    if args.batch:
        _OVERRIDES["batch"] = args.batch
    if args.context:
        _OVERRIDES["prompt_len"] = args.context
    if args.budget:
        _OVERRIDES["budget"] = args.budget
    if args.q_heads:
        _OVERRIDES["q_heads"] = args.q_heads
    if args.kv_heads:
        _OVERRIDES["kv_heads"] = args.kv_heads
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    if args.sweep:
        run_sweep(args)
        return
    if args.train:
        run_train(args)
        return
    if args.impl == "reference":
        res = run_reference(args)
        if res:
            print(json.dumps(res), flush=True)
        return
    # the oracle's host threads start before any GPU work
    cpu = None
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    if not args.no_cpu and rank == 0 and world == 1:
        cpu = oracle_sample(workload(), seconds=args.cpu_seconds)
    res = run_gpu(args)
    if res is not None:
        res["cpu_baseline"] = cpu
        print(json.dumps(res), flush=True)


if __name__ == "__main__":
    main()
