"""Query sharding over processes (one process per GPU).

A query's result depends only on the query and the index (the per-query
state of Algorithm 1 and the order-independence of Sec. 4.3), so with the
index replicated on every GPU the queries split into contiguous shards and no
collective touches the data path.  The one exchange is the host-side
concatenation of the shards' [nq][k] results and probe counts, done here over
any ``torch.distributed`` process group (gloo on the host; the tensors are
moved to the host first).
"""
from __future__ import annotations

import torch


def query_shard(nq: int, world: int, rank: int) -> tuple[int, int]:
    """Half-open row range [lo, hi) of the queries that ``rank`` searches:
    contiguous, sizes differing by at most one, earlier ranks larger."""
    if world < 1 or not 0 <= rank < world:
        raise ValueError(f"rank {rank} outside a world of {world}")
    base, extra = divmod(int(nq), world)
    lo = rank * base + min(rank, extra)
    return lo, lo + base + (1 if rank < extra else 0)


def _world(group):
    import torch.distributed as dist
    if not dist.is_available() or not dist.is_initialized():
        return 1, 0
    return dist.get_world_size(group), dist.get_rank(group)


def barrier(group=None) -> None:
    """Barrier over the group (no-op without an initialised process group)."""
    import torch.distributed as dist
    if _world(group)[0] > 1:
        dist.barrier(group=group)


def max_over_ranks(x: float, group=None, device="cpu") -> float:
    """The largest of every rank's x (the whole job's time is its slowest rank's)."""
    import torch.distributed as dist
    if _world(group)[0] == 1:
        return float(x)
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX, group=group)
    return float(t.item())


def sum_over_ranks(x: float, group=None, device="cpu") -> float:
    import torch.distributed as dist
    if _world(group)[0] == 1:
        return float(x)
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.SUM, group=group)
    return float(t.item())


def gather_results(ids, scores, count, probes, nq: int, group=None):
    """Concatenate every rank's shard of (ids [m][k], scores [m][k], count [m],
    probes [m]) in rank order into the full [nq] arrays, on every rank.

    Each rank passes the results of its ``query_shard(nq, world, rank)`` rows
    (torch tensors on any device, or numpy arrays).  Shards are padded to the
    largest shard for the all-gather and trimmed afterwards.  Returns host
    torch tensors (ids int64, scores float32, count int32, probes int32).
    """
    import torch.distributed as dist
    parts = [torch.as_tensor(x).detach().cpu() for x in (ids, scores, count, probes)]
    world, rank = _world(group)
    lo, hi = query_shard(nq, world, rank)
    if parts[0].shape[0] != hi - lo:
        raise ValueError(f"rank {rank} holds {parts[0].shape[0]} rows, its shard is {hi - lo}")
    if world == 1:
        return tuple(parts)
    k = parts[0].shape[1]
    m = query_shard(nq, world, 0)[1]              # the largest shard
    # one int64 buffer per rank: ids | scores (bit pattern) | count | probes
    buf = torch.zeros((m, 2 * k + 2), dtype=torch.int64)
    n = hi - lo
    buf[:n, :k] = parts[0].to(torch.int64)
    buf[:n, k:2 * k] = parts[1].to(torch.float32).contiguous().view(torch.int32).to(torch.int64)
    buf[:n, 2 * k] = parts[2].to(torch.int64)
    buf[:n, 2 * k + 1] = parts[3].to(torch.int64)
    got = [torch.empty_like(buf) for _ in range(world)]
    dist.all_gather(got, buf, group=group)
    rows = []
    for r in range(world):
        a, b = query_shard(nq, world, r)
        rows.append(got[r][:b - a])
    full = torch.cat(rows, 0)
    out_ids = full[:, :k].contiguous()
    out_scores = full[:, k:2 * k].to(torch.int32).view(torch.float32).contiguous()
    return out_ids, out_scores, full[:, 2 * k].to(torch.int32), full[:, 2 * k + 1].to(torch.int32)
