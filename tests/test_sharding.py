"""Multi-rank bench logic on the CPU: two gloo ranks split the sequences and combine their
timings the way the bench does on GPUs (max of device times, sum of committed bytes)."""
import os
import socket

import pytest
import torch.multiprocessing as mp

import bench


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, batch, out):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        seqs = bench.rank_sequences(rank, world, batch)
        ms = 10.0 + 5.0 * rank                  # rank 1 is the slow one
        committed = 100 * (rank + 1)
        e2e = 1000.0 * (rank + 1)
        got = bench.combine_over_ranks(dist, "cpu", ms, committed, e2e)
        gathered = [None] * world
        dist.all_gather_object(gathered, seqs)
        out[rank] = (got, gathered)
    finally:
        dist.destroy_process_group()


def test_rank_sequences_partition_the_batch():
    world, batch = 4, 3
    ids = [i for r in range(world) for i in bench.rank_sequences(r, world, batch)]
    assert ids == list(range(world * batch))
    with pytest.raises(ValueError):
        bench.rank_sequences(4, 4, 3)


def test_single_rank_passes_through():
    assert bench.combine_over_ranks(None, "cpu", 3.5, 7, 9.0) == (3.5, 7, 9.0)


def test_two_gloo_ranks_combine_like_the_bench():
    world, batch = 2, 5
    ctx = mp.get_context("spawn")
    with ctx.Manager() as m:
        out = m.dict()
        port = _free_port()
        procs = [ctx.Process(target=_rank, args=(r, world, port, batch, out)) for r in range(world)]
        for p in procs:
            p.start()
        for p in procs:
            p.join(120)
        assert all(p.exitcode == 0 for p in procs), [p.exitcode for p in procs]
        res = dict(out)
    for r in range(world):
        (ms, committed, e2e), gathered = res[r]
        assert ms == 15.0                    # slowest rank
        assert committed == 300              # bytes of all ranks
        assert e2e == 3000.0
        flat = sorted(i for g in gathered for i in g)
        assert flat == list(range(world * batch))   # disjoint, covering
