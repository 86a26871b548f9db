"""Data-parallel sharding of the loss head across ranks (host logic).

The loss head is row-independent except inside one trajectory (the advantage
scan), so a batch shards by whole trajectories with no exchange on the data
path. The only cross-rank quantity is the denominator of the token mean (the
number of action tokens of the whole batch): each rank passes the all-reduced
count as ``n_norm`` to the policy-loss and value-loss calls, after which the
per-rank losses and weight gradients simply add up (the trainer's usual
gradient all-reduce).
"""
from __future__ import annotations

from typing import List, Tuple

import numpy as np


def shard_trajectories(cu_seqlens, world: int) -> List[Tuple[int, int]]:
    """Split trajectories into `world` contiguous ranges with balanced token
    counts. Returns [(b_begin, b_end)] per rank; every trajectory appears in
    exactly one range (a range may be empty)."""
    cu = np.asarray(cu_seqlens, np.int64)
    B = len(cu) - 1
    total = int(cu[-1]) if B > 0 else 0
    bounds = [0]
    for r in range(1, world):
        target = total * r / world
        # first trajectory boundary at or after the target token count
        b = int(np.searchsorted(cu, target, side="left"))
        b = min(max(b, bounds[-1]), B)
        bounds.append(b)
    bounds.append(B)
    return [(bounds[r], bounds[r + 1]) for r in range(world)]


def local_batch(wl_arrays: dict, cu_seqlens, shard: Tuple[int, int]):
    """Slice per-token arrays (keys ending in '_tok') and per-trajectory arrays
    (keys ending in '_traj') to one shard; returns (arrays, local cu_seqlens)."""
    cu = np.asarray(cu_seqlens, np.int64)
    b0, b1 = shard
    t0, t1 = int(cu[b0]), int(cu[b1])
    out = {}
    for k, a in wl_arrays.items():
        if k.endswith("_tok"):
            out[k] = a[t0:t1]
        elif k.endswith("_traj"):
            out[k] = a[b0:b1]
        else:
            out[k] = a
    return out, (cu[b0:b1 + 1] - t0).astype(np.int32)


def global_action_count(local_count: int, group=None) -> int:
    """All-reduce (sum) of the local action-token count: the n_norm every rank
    passes to sao_policy_loss_fwd / _bwd."""
    import torch
    import torch.distributed as dist
    t = torch.tensor([int(local_count)], dtype=torch.int64)
    if dist.is_available() and dist.is_initialized():
        if dist.get_backend(group) == "nccl":
            t = t.cuda()
        dist.all_reduce(t, op=dist.ReduceOp.SUM, group=group)
    return int(t.item())
