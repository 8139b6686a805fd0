"""Row sharding of a layer across ranks (one GPU per rank).

The objective separates over output rows (Sec. 3.3, "each column can be
refined independently"), so N ranks refine disjoint contiguous row ranges of
a layer with no communication on the data path.  These helpers give each
rank its range and, for callers that want the whole layer on every rank,
gather the refined scales and codes at the end (one all-gather per tensor).
"""
from __future__ import annotations


def row_range(dout: int, rank: int, world: int):
    """Contiguous [start, stop) of the rows owned by `rank` (balanced split)."""
    if world < 1 or not 0 <= rank < world:
        raise ValueError("bad rank/world")
    base, extra = divmod(dout, world)
    start = rank * base + min(rank, extra)
    return start, start + base + (1 if rank < extra else 0)


def gather_rows(local, dout: int, group=None):
    """All-gather row shards (torch tensors, leading dim = rows) into [dout, ...]."""
    import torch
    import torch.distributed as dist
    world = dist.get_world_size(group)
    sizes = [row_range(dout, r, world) for r in range(world)]
    maxn = max(b - a for a, b in sizes)
    pad = torch.zeros((maxn,) + tuple(local.shape[1:]), dtype=local.dtype, device=local.device)
    pad[: local.shape[0]] = local
    outs = [torch.empty_like(pad) for _ in range(world)]
    dist.all_gather(outs, pad, group=group)
    return torch.cat([o[: b - a] for o, (a, b) in zip(outs, sizes)], dim=0)


def token_range(n: int, rank: int, world: int):
    """Contiguous [start, stop) of the calibration tokens a rank accumulates.

    The Hessian H = X^T X + nu^2 I (Eq. strict_target) is a sum over tokens, so
    the tokens shard across ranks with one exchange: each rank forms the
    partial product of its tokens (``jarq_accumulate_hessian``) and the
    partials are summed on every rank (``allreduce_hessian``)."""
    return row_range(n, rank, world)


def allreduce_hessian(H_local, group=None):
    """Sum the ranks' partial Hessians in place (one all-reduce); returns H."""
    import torch.distributed as dist
    dist.all_reduce(H_local, op=dist.ReduceOp.SUM, group=group)
    return H_local
