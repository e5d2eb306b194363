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


def _compute_worker(rank, world, port, out):
    """Each rank decomposes its shard of a small synthetic stack with the oracle (the
    stand-in for its GPU on this CPU test), then the ranks gather their codes and
    centres; only rank 0's gathered result is returned."""
    import numpy as np
    import torch
    import torch.distributed as dist
    from oracle import kashin_oracle as ko
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        n_layers, n, m = 4, 32, 6
        mine = {}
        for L in shard.layer_schedule(rank, world, n_layers // world, n_layers):
            x = np.random.default_rng(100 + L).standard_t(4, size=(n, m)) * 0.015
            d = ko.decompose(x, ko.sign_mask(L, n), 3)
            cu = ko.centres(d.coeffs[0], d.coeffs[1])
            mine[L] = (ko.pack_codes(ko.codes(d.u, cu)), cu)
        t, units = shard.aggregate(1.0 + rank, float(len(mine) * n * m))
        gathered = [None] * world
        dist.all_gather_object(gathered, mine)
        if rank == 0:
            allres = {}
            for part in gathered:
                assert set(part).isdisjoint(allres)
                allres.update(part)
            out["res"] = {L: (c.tolist(), e.tolist()) for L, (c, e) in allres.items()}
            out["agg"] = (t, units)
        dist.barrier()
    finally:
        dist.destroy_process_group()


def test_gloo_two_ranks_sharded_decomposition_equals_one_rank():
    """World size 2: the layers split with no exchange, every layer is decomposed by
    exactly one rank, and the gathered codes and centres equal a one-process run."""
    import numpy as np
    from oracle import kashin_oracle as ko
    ctx = mp.get_context("spawn")
    mgr = ctx.Manager()
    out = mgr.dict()
    port = _free_port()
    procs = [ctx.Process(target=_compute_worker, args=(r, 2, port, out)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=180)
        assert p.exitcode == 0
    res = out["res"]
    assert sorted(res) == [0, 1, 2, 3]
    assert out["agg"] == (2.0, 4 * 32 * 6.0)
    for L in range(4):
        x = np.random.default_rng(100 + L).standard_t(4, size=(32, 6)) * 0.015
        d = ko.decompose(x, ko.sign_mask(L, 32), 3)
        cu = ko.centres(d.coeffs[0], d.coeffs[1])
        assert np.array_equal(np.array(res[L][0], dtype=np.uint32), ko.pack_codes(ko.codes(d.u, cu)))
        assert np.array_equal(np.array(res[L][1]), cu)
