"""The multi-process path of bench.py on the CPU (gloo, world size 2).

The step partitions by batch element with no exchange, so under torchrun
every rank verifies its own replica of the workload and the only
collectives are the timing ones: a barrier on both sides of the timed
region and an all-reduce MAX of the elapsed time.  These tests run those
collectives over gloo in two spawned processes and check that every rank
ends with the slowest rank's time and the whole-job throughput built from
it; and that the reference arm runs on rank 0 alone.
"""
import json
import os
import socket

import pytest

import bench


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out_dir):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        dist.barrier()
        ms = bench.max_over_ranks(1.5 + 2.0 * rank, dist, "cpu")   # rank 1 is the slow one
        value = bench.aggregate_rows_per_s(world, 512, ms / 100)
        dist.barrier()
        with open(os.path.join(out_dir, f"rank{rank}.json"), "w") as f:
            json.dump({"ms": ms, "value": value}, f)
    finally:
        dist.destroy_process_group()


def test_two_ranks_take_the_slowest_time(tmp_path):
    import torch.multiprocessing as mp
    world = 2
    mp.start_processes(_worker, args=(world, _free_port(), str(tmp_path)), nprocs=world,
                       join=True, start_method="spawn")
    got = [json.load(open(tmp_path / f"rank{r}.json")) for r in range(world)]
    assert [g["ms"] for g in got] == [3.5, 3.5]
    # 2 replicas x 512 rows per step, 0.035 ms per step
    assert got[0]["value"] == pytest.approx(2 * 512 / 0.035e-3)
    assert got[0]["value"] == got[1]["value"]


def test_single_process_needs_no_group():
    assert bench.max_over_ranks(2.25) == 2.25
    assert bench.aggregate_rows_per_s(1, 512, 0.14) == pytest.approx(512 / 0.14e-3)


def test_reference_arm_runs_on_rank_zero_only(capsys):
    class Args:
        mode, steps, warmup = "stochastic", 1, 0

    from paper_2608_26004_gb300 import synth
    bench.run_reference(Args, synth.CONFIGS[bench.WORKLOAD_CFG], rank=1, world=2)
    assert capsys.readouterr().out == ""
