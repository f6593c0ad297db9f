"""The multi-GPU path of bench.py is replicas (every rank runs its own copy of
the workload, no data-path collective).  What is host logic is checked here
with two gloo ranks on the CPU: the max-over-ranks timing, the whole-job rate
built from it, and that the reference arm runs on rank 0 only."""
import os
import socket
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    times = [12.5, 40.0]  # this rank's timed region (ms): rank 1 is the slowest
    m = bench.max_over_ranks(times[rank])
    rate = bench.whole_job_rate(world, 1000, 10, m)
    dist.barrier()
    dist.destroy_process_group()
    out.put((rank, m, rate))


def test_two_gloo_ranks_take_the_slowest_rank():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    got = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, m, rate in got:
        assert m == 40.0  # every rank sees the max
        assert rate == pytest.approx(2 * 1000 * 10 / 0.040)  # all ranks' units / slowest time


def test_single_process_is_identity():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.max_over_ranks(3.25) == 3.25
    assert bench.whole_job_rate(1, 4096, 2, 1.0) == pytest.approx(4096 * 2 / 1e-3)


def test_reference_arm_runs_on_rank_zero_only(monkeypatch, capsys):
    """Under torchrun the oracle arm prints from rank 0; other ranks exit at once."""
    sys.path.insert(0, ROOT)
    import bench
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("WORLD_SIZE", "2")

    class Args:
        workload, steps, warmup = "gla_bf16_4k", 1, 3
    bench.run_reference(Args())  # would take minutes if rank 1 did any work
    assert capsys.readouterr().out == ""
