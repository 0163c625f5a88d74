"""Multi-rank host logic of the data-parallel path, run as two gloo ranks on CPU."""
import os
import socket

import pytest
import torch.distributed as dist
import torch.multiprocessing as mp

from paper_2601_02819_gb300.sharding import max_over_ranks, rank_seed, shard_sequences


@pytest.mark.parametrize("batch,world", [(1, 1), (8, 2), (7, 2), (3, 4), (2, 8)])
def test_shards_cover_every_sequence_once(batch, world):
    shards = [shard_sequences(batch, world, r) for r in range(world)]
    flat = [s for sh in shards for s in sh]
    assert sorted(flat) == list(range(batch))
    sizes = [len(sh) for sh in shards]
    assert max(sizes) - min(sizes) <= 1


def test_seeds_depend_on_the_sequence_not_the_rank_count():
    assert rank_seed(10, 3) == rank_seed(10, 3)
    assert len({rank_seed(10, s) for s in range(100)}) == 100


def _worker(rank, world, port, q):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        mine = shard_sequences(6, world, rank)
        elapsed = 10.0 + rank  # a per-rank time; the job's time is the slowest rank's
        dist.barrier()
        q.put((rank, mine, max_over_ranks(elapsed)))
    finally:
        dist.destroy_process_group()


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def test_two_gloo_ranks_shard_and_reduce_the_time():
    world = 2
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    out = sorted(q.get(timeout=120) for _ in range(world))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert [o[1] for o in out] == [[0, 1, 2], [3, 4, 5]]
    assert all(o[2] == 11.0 for o in out)
