"""The N > 1 host path of bench.py on CPU: N independent replicas, one per
process, each timing its own steps; the job's time is the maximum over the
ranks (an all-reduce), its value the units of all ranks over that time, and
under the reference arm only rank 0 runs and prints.  Two gloo processes on
127.0.0.1, no GPU."""
import os
import socket
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    import torch.distributed as dist
    import bench
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    dist.barrier()
    local = [10.0 + 5.0 * rank, 30.0 - 10.0 * rank, 7.0]  # per-rank step totals (ms)
    times = bench.max_over_ranks(local, world)
    rate = bench.job_rate(1000.0, 4, world, times[0])
    out.put((rank, times, rate))
    dist.barrier()
    dist.destroy_process_group()


def test_max_over_ranks_and_job_rate_gloo():
    world = 2
    ctx = mp.get_context("spawn")
    out = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, world, port, out)) for r in range(world)]
    for p in procs:
        p.start()
    got = [out.get(timeout=120) for _ in range(world)]
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    for rank, times, rate in got:
        assert times == [15.0, 30.0, 7.0], rank          # every rank sees the maxima
        assert rate == pytest.approx(1000.0 * 4 * 2 / 0.015)


def test_single_process_is_identity():
    import bench
    assert bench.max_over_ranks([1.5, 2.5], 1) == [1.5, 2.5]
    assert bench.job_rate(10, 2, 1, 4.0) == pytest.approx(5000.0)


def test_reference_arm_runs_on_rank_0_only(capsys):
    import bench

    class Args:
        workload = "tiny"
        steps = 1
        warmup = 0
    bench.run_reference(Args(), rank=1, world=2)     # other ranks exit without work
    assert capsys.readouterr().out == ""


def test_reference_arm_line_on_rank_0(capsys):
    """The reference arm's JSON line (the oracle timed on the host cores) on the
    tiny configuration: the contract's keys, impl, and an e2e equal to the value."""
    import json
    import bench

    class Args:
        workload = "tiny"
        steps = 1
        warmup = 0
    bench.run_reference(Args(), rank=0, world=1)
    line = json.loads(capsys.readouterr().out.strip().splitlines()[-1])
    for k in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better", "scaling",
              "vs_baseline", "dtype", "data", "config", "cpu_baseline", "e2e"):
        assert k in line, k
    assert line["impl"] == "reference" and line["value"] > 0
    assert line["e2e"]["value"] == line["value"] and line["e2e"]["h2d_bytes_per_step"] == 0
    assert line["cpu_baseline"]["kind"] == "oracle"
