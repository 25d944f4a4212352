"""The multi-GPU path of the benchmark is replicas only (the path shards by
(sequence, kv head) with no exchange): each rank runs the whole workload and
the job's time is the slowest rank's.  Checked here with two gloo ranks on
the CPU: the reduction takes every value's maximum over the ranks and the
whole-job throughput counts the bytes of all ranks."""
import os
import socket

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, out):
    import sys

    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    import bench
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        # rank r took (1 + r) s for the draft phase and (3 - r) s for the step
        draft_s, step_s = bench.max_over_ranks([1.0 + rank, 3.0 - rank], world, "cpu")
        dist.barrier()
        out[rank] = (draft_s, step_s, bench.whole_job_gbs(world, 4e9, 10, draft_s))
    finally:
        dist.destroy_process_group()


def test_two_replicas_take_the_slowest_rank():
    world = 2
    port = _free_port()
    ctx = mp.get_context("spawn")
    with ctx.Manager() as m:
        out = m.dict()
        procs = [ctx.Process(target=_rank, args=(r, world, port, out)) for r in range(world)]
        for p in procs:
            p.start()
        for p in procs:
            p.join(120)
            assert p.exitcode == 0
        res = dict(out)
    for r in range(world):
        draft_s, step_s, gbs = res[r]
        assert draft_s == 2.0 and step_s == 3.0          # max over ranks, per value
        assert gbs == pytest.approx(2 * 4e9 * 10 / 2.0 / 1e9)  # both ranks' bytes / slowest time


def test_one_rank_keeps_its_own_values():
    import sys
    sys.path.insert(0, ROOT)
    import bench
    assert bench.max_over_ranks([1.5, 2.5], 1, "cpu") == [1.5, 2.5]
    assert bench.whole_job_gbs(1, 1e9, 3, 1.5) == pytest.approx(2.0)
