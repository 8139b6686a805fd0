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
