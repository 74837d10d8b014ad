"""Multi-GPU exhaustive search by index ranges: the split and the one exchange step.

The joint space [0, |Lambda|) (Eq. 1) is cut into one contiguous range per rank;
each rank searches its range on its own GPU (mf_search_range) and keeps its top-k
and feasible count.  The exchange is an all-gather of the k (score, index) pairs
and the counts, merged on every rank by the total order of the search (score
descending, index ascending), so the result does not depend on the number of
ranks.  This module holds only that host logic; it does not load the CUDA library.
"""
from __future__ import annotations

import numpy as np

EMPTY = (1 << 64) - 1


def shard_range(total: int, rank: int, world: int) -> tuple[int, int]:
    """Contiguous [lo, hi) of rank `rank` among `world`; sizes differ by at most one."""
    if world < 1 or not 0 <= rank < world:
        raise ValueError("need 0 <= rank < world")
    base, extra = divmod(int(total), world)
    lo = rank * base + min(rank, extra)
    return lo, lo + base + (1 if rank < extra else 0)


def merge_results(parts: list[dict], k: int) -> dict:
    """Merge per-range results (topk_idx uint64 [k], topk_score float32 [k], count).

    Empty slots (index 2**64 - 1, score -inf) sort last.  Ranges are disjoint, so no
    index appears twice."""
    idx = np.concatenate([np.asarray(p["topk_idx"], dtype=np.uint64) for p in parts])
    sc = np.concatenate([np.asarray(p["topk_score"], dtype=np.float32) for p in parts])
    live = idx != np.uint64(EMPTY)
    idx, sc = idx[live], sc[live]
    order = np.lexsort((idx, -sc.astype(np.float64)))[:k]
    out_i = np.full(k, EMPTY, dtype=np.uint64)
    out_s = np.full(k, -np.inf, dtype=np.float32)
    out_i[:order.size] = idx[order]
    out_s[:order.size] = sc[order]
    count = int(sum(int(p["count"]) for p in parts))
    return dict(best_idx=int(out_i[0]), best_score=float(out_s[0]), count=count,
                topk_idx=out_i, topk_score=out_s)


def gather_merge(local: dict, k: int, group=None, device=None) -> dict:
    """All-gather every rank's result over torch.distributed and merge it.

    `device` is where the exchange tensors live: a CUDA device for NCCL, None (CPU)
    for gloo.  Indices travel as int64 bit patterns."""
    import torch
    import torch.distributed as dist

    world = dist.get_world_size(group)
    ti = torch.from_numpy(np.asarray(local["topk_idx"], dtype=np.uint64).view(np.int64).copy())
    ts = torch.from_numpy(np.asarray(local["topk_score"], dtype=np.float32).copy())
    tc = torch.tensor([int(local["count"])], dtype=torch.int64)
    if device is not None:
        ti, ts, tc = ti.to(device), ts.to(device), tc.to(device)
    gi = [torch.empty_like(ti) for _ in range(world)]
    gs = [torch.empty_like(ts) for _ in range(world)]
    gc = [torch.empty_like(tc) for _ in range(world)]
    dist.all_gather(gi, ti, group=group)
    dist.all_gather(gs, ts, group=group)
    dist.all_gather(gc, tc, group=group)
    parts = [dict(topk_idx=a.cpu().numpy().view(np.uint64), topk_score=b.cpu().numpy(), count=int(c.item()))
             for a, b, c in zip(gi, gs, gc)]
    return merge_results(parts, k)


def search_sharded(ctx, k: int, group=None, chunk: int = 0, device=None) -> dict:
    """Exhaustive search of ctx's whole space, this rank's range on this rank's GPU."""
    import torch.distributed as dist

    lo, hi = shard_range(ctx.space_size, dist.get_rank(group), dist.get_world_size(group))
    local = ctx.search(k, lo=lo, hi=hi, chunk=chunk)
    return gather_merge(local, k, group=group, device=device)
