"""Host-side sharding of a candidate set across ranks (one GPU per rank).

Candidates are independent, so N ranks price disjoint index ranges with no
exchange on the data path; the only exchange is the final merge of the
per-rank top-k lists (k entries each), done on the host over a gloo group.
The merge uses the same strict order as the kernels: higher throughput
nM / T first (exact integer cross-multiplication), then the smaller global
index, so the merged list equals the top-k of the union.
"""

from __future__ import annotations

import functools

import numpy as np


def shard_range(n: int, rank: int, world: int) -> tuple[int, int]:
    """Contiguous candidate range [lo, hi) of ``rank``."""
    return n * rank // world, n * (rank + 1) // world


def _cmp(a, b):
    l, r = int(a[2]) * int(b[1]), int(b[2]) * int(a[1])
    if l != r:
        return -1 if l > r else 1
    return -1 if a[0] < b[0] else (1 if a[0] > b[0] else 0)


def merge_topk(lists, k: int) -> dict:
    """Merge top-k dicts (idx, T, nM) into the top-k of their union."""
    items = [(int(i), int(t), int(m)) for d in lists for i, t, m in zip(d["idx"], d["T"], d["nM"])]
    items.sort(key=functools.cmp_to_key(_cmp))
    items = items[:k]
    return {"k": k, "count": len(items), "idx": np.array([e[0] for e in items], np.int64),
            "T": np.array([e[1] for e in items], np.int64), "nM": np.array([e[2] for e in items], np.uint32)}


def init(world: int):
    """Process group for the host-side exchange (None for one rank)."""
    if world <= 1:
        return None
    import torch.distributed as dist
    if not dist.is_initialized():
        dist.init_process_group("gloo")
    return dist.group.WORLD


def barrier(group):
    if group is not None:
        import torch.distributed as dist
        dist.barrier(group)


def max_over_ranks(group, value: float) -> float:
    if group is None:
        return value
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(value)], dtype=torch.float64)
    dist.all_reduce(t, op=dist.ReduceOp.MAX, group=group)
    return float(t.item())


def merge_topk_across_ranks(group, local: dict, k: int) -> dict:
    if group is None:
        return merge_topk([local], k)
    import torch.distributed as dist
    out = [None] * dist.get_world_size(group)
    dist.all_gather_object(out, {key: np.asarray(local[key]).tolist() for key in ("idx", "T", "nM")},
                           group=group)
    return merge_topk(out, k)
