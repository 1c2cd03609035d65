"""Multi-rank host logic of the benchmark on CPU (gloo, world size 2): the
job time is the slowest rank's, the rate counts every rank's replica, and the
reference arm runs on rank 0 only."""

import os
import socket

import pytest
import torch.multiprocessing as mp


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, world, port, q):
    import torch.distributed as dist
    import bench
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    el, rate = bench.job_throughput(100.0 + 50.0 * rank, 10, dist, device="cpu")
    ref = bench.run_reference(type("A", (), {"steps": 1, "warmup": 3, "cpu_seconds": 0.01})()) if rank else "skip"
    q.put((rank, el, rate, ref))
    dist.barrier()
    dist.destroy_process_group()


def test_job_throughput_takes_slowest_rank_and_counts_all_replicas():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    out = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, el, rate, ref in out:
        assert el == pytest.approx(150.0)
        assert rate == pytest.approx(2 * 10 / 0.150)
        if rank == 1:
            assert ref is None  # the reference arm does no work off rank 0


def test_single_rank_throughput():
    import bench
    el, rate = bench.job_throughput(200.0, 40)
    assert el == 200.0 and rate == pytest.approx(200.0)


def test_algorithmic_bytes_are_the_documented_per_unit_figures():
    """The roofline's numerator: 548 B per token-row of a steady step (K and V
    read, 4d = 512 B at d = 128; position read, 4 B; window sums read and
    written, 32 B; cumulative alpha read and written, 8 B more, in alpha_mode 1),
    plus per row the append (4d + 20 B) and one compaction move (2 x (4d + 20) B).
    At the benchmark shape (2048 rows of 8193 tokens) that is 9.198 GB a step."""
    import bench
    from paper_2608_08878_gb300 import synth
    assert bench.row_bytes_per_step(1, 128) == 548
    assert bench.row_bytes_per_step(1, 128, alpha_mode=1) == 556
    assert bench.row_bytes_per_step(1, 64) == 292
    wl = synth.MISTRAL_FULL
    assert (wl.rows, wl.head_dim, wl.alpha_mode) == (2048, 128, 0)
    assert bench.step_bytes(wl, 8193) == 2048 * (8193 * 548 + 532 + 2 * 532)
    assert round(bench.step_bytes(wl, 8193) / 1e9, 3) == 9.198
    assert bench.step_bytes(wl, 8193, moved_per_row=0) == 2048 * (8193 * 548 + 532)


def test_reference_arm_line_on_rank_zero(monkeypatch):
    """The reference arm's line (the fp64 oracle on the host's cores, a bounded
    sample extrapolated to whole steps): the GPU arm's metric, unit, direction
    and config dict; the sample described in cpu_baseline; an e2e entry with
    no host-device copies."""
    import json
    import types
    import bench
    monkeypatch.delenv("RANK", raising=False)
    monkeypatch.delenv("WORLD_SIZE", raising=False)
    args = types.SimpleNamespace(steps=2, warmup=3, cpu_seconds=0.3, global_tokens=False, hybrid=False, scorer=0,
                                 budget_ratio=0.0)
    line = bench.run_reference(args)
    json.dumps(line)
    assert line["impl"] == "reference"
    assert (line["metric"], line["unit"], line["higher_is_better"]) == (bench.METRIC, bench.UNIT, True)
    assert line["config"] == bench.bench_config(bench.workload(), args, 1)
    assert line["n_gpus"] == 1 and (line["steps"], line["warmup"]) == (2, 3)
    cb = line["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["host_cores"] >= cb["cores"] and cb["sample"]
    assert cb["value"] == line["value"] > 0 and cb["row_steps_run"] >= 1
    assert line["extrapolated"] is True and line["ms_per_step"] == pytest.approx(1e3 / line["value"])
    assert line["e2e"] == {"value": line["value"], "unit": bench.UNIT, "h2d_bytes_per_step": 0,
                           "d2h_bytes_per_step": 0}
