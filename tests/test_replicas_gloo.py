"""Host logic of the benchmark's replica mode on CPU (two gloo ranks).

The decode step shards by sequence with no exchange, so N GPUs run N
independent replicas: each rank times its own steps, the slowest rank's time
sets the job's, and the job's rate is the steps of all ranks over that time.
The reference arm runs on rank 0 only; the other ranks exit without work.
"""

import multiprocessing as mp
import socket

import pytest

import bench


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, elapsed, out):
    import torch.distributed as dist
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=world)
    try:
        el = bench.max_over_ranks(elapsed[rank], world, "cpu")
        dist.barrier()
        out.put((rank, el, bench.job_rate(world, 64, el)))
    finally:
        dist.destroy_process_group()


@pytest.mark.timeout(120)
def test_slowest_rank_sets_the_job_time():
    ctx = mp.get_context("spawn")
    out = ctx.Queue()
    elapsed = [0.25, 0.5]
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, 2, port, elapsed, out)) for r in range(2)]
    for p in procs:
        p.start()
    got = sorted(out.get(timeout=90) for _ in procs)
    for p in procs:
        p.join(timeout=30)
        assert p.exitcode == 0
    assert [g[1] for g in got] == [0.5, 0.5]
    # 2 replicas x 64 steps in 0.5 s
    assert [g[2] for g in got] == [256.0, 256.0]


def test_one_rank_is_its_own_job():
    assert bench.max_over_ranks(0.3, 1, "cpu") == 0.3
    assert bench.job_rate(1, 10, 0.5) == 20.0


def test_reference_arm_runs_on_rank_zero_only():
    args = bench.parse_args(["--impl", "reference", "--gpus", "2", "--steps", "1", "--warmup", "0"])
    assert bench.run_reference(args, 1, 2) == 0  # returns at once: no oracle work on rank 1
