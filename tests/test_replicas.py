"""Multi-rank host logic of the replicas-only layout, on CPU with gloo (world size 2)."""

import os
import socket

import pytest
import torch.multiprocessing as mp

from paper_2608_02134_gb300 import replicas


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, times, out):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        ms = replicas.max_over_ranks(times[rank])
        imgs = replicas.shard_images(32, rank, world)
        dist.barrier()
        out[rank] = (ms, replicas.job_rate(world, len(imgs), ms), imgs)
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_agree_on_the_slowest_step_and_split_the_batch():
    world, port = 2, _free_port()
    times = [1.25, 2.5]
    with mp.Manager() as m:
        out = m.dict()
        mp.spawn(_worker, args=(world, port, times, out), nprocs=world, join=True)
        res = dict(out)
    assert res[0][0] == res[1][0] == 2.5                      # every rank sees the max
    assert res[0][1] == res[1][1] == pytest.approx(2 * 16 * 1000.0 / 2.5)
    assert sorted(res[0][2] + res[1][2]) == list(range(32))   # each image exactly once


def test_single_process_defaults():
    assert replicas.max_over_ranks(3.0) == 3.0
    assert replicas.rank_info({}) == (0, 1, 0)
    assert replicas.job_rate(4, 1, 0.5) == 8000.0
    for B, W in [(1, 2), (5, 3), (32, 8), (7, 7)]:
        parts = [replicas.shard_images(B, r, W) for r in range(W)]
        assert sorted(sum(parts, [])) == list(range(B))
        assert max(map(len, parts)) - min(map(len, parts)) <= 1
    with pytest.raises(ValueError):
        replicas.shard_images(4, 2, 2)
    with pytest.raises(ValueError):
        replicas.job_rate(1, 1, 0.0)
