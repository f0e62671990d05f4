"""Host logic of `bench.py --gpus N` (N independent replicas, weak scaling) on CPU ranks: two
`gloo` processes stand in for two GPUs. The forward itself has no exchange step, so the only
cross-rank operations are the barrier around the timed region and the max over the ranks'
timed seconds; the whole-job throughput divides every rank's tokens by that maximum."""
import os
import socket

import pytest

import bench


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, secs, out):
    import torch.distributed as dist
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        dist.barrier()
        m = bench.max_over_ranks(secs[rank], dist, world, device="cpu")
        out[rank] = (m, bench.job_throughput(32, 10, world, m))
        dist.barrier()
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_agree_on_the_slowest_time_and_job_throughput():
    import torch.multiprocessing as mp
    world, secs = 2, [1.5, 2.5]
    with mp.Manager() as mgr:
        out = mgr.dict()
        mp.spawn(_rank_main, args=(world, _free_port(), secs, out), nprocs=world, join=True)
        res = dict(out)
    assert sorted(res) == [0, 1]
    for rank in range(world):
        m, v = res[rank]
        assert m == pytest.approx(2.5)
        # 32 tokens per step, 10 steps, on each of the 2 replicas, over the slowest 2.5 s
        assert v == pytest.approx(32 * 10 * 2 / 2.5)


def test_single_process_needs_no_collective():
    assert bench.max_over_ranks(1.25, None, 1) == 1.25
    assert bench.job_throughput(32, 4, 1, 2.0) == pytest.approx(64.0)


def test_reference_arm_runs_on_rank_zero_only():
    # a non-zero rank returns at once, without touching the oracle or the inputs
    class Args:
        steps, warmup, seed, ref_budget = 1, 1, 0, 1.0

    assert bench.run_reference(Args(), None, rank=1) is None
