"""The multi-rank logic of bench.py on CPU: two ranks over gloo (127.0.0.1).

bench.py under torchrun runs one replica of the step per rank (weak scaling, no
collective on the data path) and reports the whole-job aggregate over the slowest
rank's step time; the reference arm runs on rank 0 only.  The GPU parts need a GPU;
what is checked here is the rank arithmetic and the process-group plumbing.
"""
import os
import socket

import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist  # noqa: E402
import torch.multiprocessing as mp  # noqa: E402


def _free_port() -> int:
    with socket.socket(socket.AF_INET, socket.SOCK_STREAM) as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out_q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    step_ms = 2.0 + rank  # the last rank is the slowest
    ms = bench.max_over_ranks(step_ms, dist, "cpu")
    value = bench.job_tflops(world, ms)

    class Args:  # the reference arm: ranks other than 0 return at once, doing no work
        steps, warmup, ref_rows = 1, 3, 1
    ref_rc = bench.run_reference(Args) if rank != 0 else 0
    dist.barrier()
    out_q.put((rank, ms, value, ref_rc, bench.dist_env()))
    dist.destroy_process_group()


def test_two_ranks_report_the_slowest_step_and_the_job_total():
    world = 2
    ctx = mp.get_context("spawn")
    q = ctx.SimpleQueue()
    mp.start_processes(_worker, args=(world, _free_port(), q), nprocs=world, join=True, start_method="spawn")
    got = sorted(q.get() for _ in range(world))
    import bench
    for rank, ms, value, ref_rc, env in got:
        assert ms == pytest.approx(3.0), "max over ranks"
        assert value == pytest.approx(world * bench.STEP_FLOPS / 3.0e-3 / 1e12), "whole-job aggregate"
        assert ref_rc == 0
        assert env == (rank, rank, world)


def test_single_process_has_no_group():
    import bench
    assert bench.max_over_ranks(1.5, None, "cpu") == 1.5
    assert bench.job_tflops(1, 1.0) == pytest.approx(bench.STEP_FLOPS / 1e-3 / 1e12)
