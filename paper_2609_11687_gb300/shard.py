"""Weak-scaling shards for multi-GPU runs: every matrix (and every vector) is
decomposed independently and each matrix's sign set comes from its own seed, so
ranks split the work with no data exchange.  The only collectives are the
timing barrier and the reductions below."""

from __future__ import annotations

from typing import List, Tuple


def layer_schedule(rank: int, world: int, steps: int, n_layers: int = 32) -> List[int]:
    """Layers a rank decomposes, one per step: rank, rank + world, ... (mod n_layers).
    For world <= n_layers the ranks' first ceil(n_layers / world) steps are disjoint."""
    if not (0 <= rank < world):
        raise ValueError("rank out of range")
    return [(rank + world * i) % n_layers for i in range(steps)]


def aggregate(elapsed_ms: float, units: float, group=None) -> Tuple[float, float]:
    """(max elapsed over ranks, total units over ranks).  Whole-job throughput is
    total units / max elapsed; without an initialised process group this is the
    single-rank identity."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()):
        return float(elapsed_ms), float(units)
    dev = torch.device("cuda", torch.cuda.current_device()) if dist.get_backend(group) == "nccl" else "cpu"
    t = torch.tensor([float(elapsed_ms)], dtype=torch.float64, device=dev)
    u = torch.tensor([float(units)], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX, group=group)
    dist.all_reduce(u, op=dist.ReduceOp.SUM, group=group)
    return float(t.item()), float(u.item())
