"""The N > 1 path of bench.py on CPU: two ranks over gloo (127.0.0.1).

Every (batch, head) unit is independent, so N GPUs run N replicas of the
workload with no data-path collective; the only exchange is the timing: the
job's step time is the maximum over ranks, and the job's throughput counts the
units of every rank over that time.  Rank 0 alone reports, and the reference
arm runs on rank 0 only (the other ranks exit without work)."""
import multiprocessing as mp
import os
import socket
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank: int, world: int, port: int, q) -> None:
    try:
        os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), LOCAL_RANK=str(rank),
                          WORLD_SIZE=str(world))
        sys.path.insert(0, ROOT)
        import torch.distributed as tdist
        import argparse
        import bench
        from synth.workloads import WORKLOADS
        tdist.init_process_group("gloo", rank=rank, world_size=world)
        mine = 1.5 + 2.0 * rank  # this rank's step time (ms)
        step_ms = bench.max_over_ranks(mine, "cpu", world)
        rate = bench.job_throughput(1000, world, step_ms)
        args = argparse.Namespace(steps=1, warmup=0, cpu_seconds=1.0, ch_rms_target=0.0)
        ref = bench.run_reference(args, WORKLOADS["tiny_f32"])
        tdist.barrier()
        tdist.destroy_process_group()
        q.put((rank, bench.dist_env(), step_ms, rate, None if ref is None else (ref["impl"], ref["n_gpus"])))
    except Exception as e:  # reported to the parent
        q.put((rank, "error", repr(e), None, None))


def test_two_ranks_over_gloo():
    world = 2
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    out = sorted(q.get(timeout=240) for _ in range(world))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, env, step_ms, rate, ref in out:
        assert env != "error", step_ms
        assert env == (rank, rank, world)
        assert step_ms == pytest.approx(3.5)                    # the slowest rank's time
        assert rate == pytest.approx(1000 * world / 3.5e-3)     # units of all ranks over that time
        if rank == 0:
            assert ref == ("reference", world)                  # rank 0 runs the reference arm
        else:
            assert ref is None                                  # the others exit without work
