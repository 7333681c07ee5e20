"""The multi-GPU path of bench.py is replicas only: every rank runs its own
generation and the ranks meet only to agree on the job's step time (the
slowest rank) and the whole-job throughput.  Checked here with two gloo
processes on the CPU."""
import os
import socket

import pytest
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    import torch.distributed as dist
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    ms = 10.0 + 5.0 * rank                      # rank 1 is the slower replica
    job_ms = bench.slowest_rank_ms(ms, world, None)
    q.put((rank, job_ms, bench.job_tokens_per_s(32760, world, job_ms)))
    dist.barrier()
    dist.destroy_process_group()


def test_two_replicas_report_the_slowest_rank_and_the_job_total():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    res = sorted(q.get(timeout=10) for _ in range(2))
    for rank, job_ms, tps in res:
        assert job_ms == 15.0                   # both ranks agree on the slowest
        assert tps == pytest.approx(2 * 32760 / 0.015)


def test_single_rank_is_unchanged():
    import bench
    assert bench.slowest_rank_ms(7.5, 1) == 7.5
    assert bench.job_tokens_per_s(1000, 1, 10.0) == pytest.approx(1e5)
