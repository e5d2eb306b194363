"""Multi-rank host logic of the weak-scaling bench, on CPU with the gloo backend
(world size 2): disjoint layer shards and the max-time / sum-units reduction."""

import os
import socket

import pytest
import torch.multiprocessing as mp

from paper_2609_11687_gb300 import shard


def test_schedule_single_and_disjoint():
    assert shard.layer_schedule(0, 1, 5) == [0, 1, 2, 3, 4]
    a = shard.layer_schedule(0, 2, 16)
    b = shard.layer_schedule(1, 2, 16)
    assert set(a).isdisjoint(b) and sorted(a + b) == list(range(32))
    with pytest.raises(ValueError):
        shard.layer_schedule(2, 2, 1)


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    import torch.distributed as dist
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        layers = shard.layer_schedule(rank, world, 4)
        elapsed = [10.0, 25.0][rank]                       # the slower rank sets the time
        t, units = shard.aggregate(elapsed, 100.0 * len(layers))
        out[rank] = (t, units, layers)
        dist.barrier()
    finally:
        dist.destroy_process_group()


def test_gloo_two_ranks_aggregate():
    ctx = mp.get_context("spawn")
    mgr = ctx.Manager()
    out = mgr.dict()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, out)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    for r in range(2):
        t, units, layers = out[r]
        assert t == 25.0 and units == 800.0
    assert set(out[0][2]).isdisjoint(out[1][2])


def test_aggregate_without_process_group():
    assert shard.aggregate(3.0, 7.0) == (3.0, 7.0)
