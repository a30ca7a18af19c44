"""Host-side layout helpers for the sharded step (gnmr_step_partials +
gnmr_finish): with ZeRO-style sharding, a flat gradient buffer of N elements
is split into contiguous per-rank shards, and every unit's elements inside a
rank's shard form that rank's local layout.  Pure index arithmetic."""
from __future__ import annotations

import numpy as np


def even_shards(total_elems: int, world: int, align: int = 1):
    """Contiguous shards [start, start + elems) covering [0, total_elems),
    one per rank, sizes equal up to `align`-element rounding."""
    if world < 1 or total_elems < 0 or align < 1:
        raise ValueError("world >= 1, total_elems >= 0 and align >= 1 required")
    per = -(-total_elems // world)
    per = -(-per // align) * align
    out = []
    for r in range(world):
        s = min(r * per, total_elems)
        e = min(s + per, total_elems)
        out.append((s, e - s))
    return out


def shard_layout(offsets, lengths, shard_start: int, shard_elems: int):
    """Local (offsets, lengths) of every unit inside the shard
    [shard_start, shard_start + shard_elems), relative to the shard's first
    element.  A unit with no element in the shard gets offset 0, length 0."""
    off = np.asarray(offsets, dtype=np.int64)
    ln = np.asarray(lengths, dtype=np.int64)
    lo = np.maximum(off, shard_start)
    hi = np.minimum(off + ln, shard_start + shard_elems)
    local_len = np.maximum(hi - lo, 0)
    local_off = np.where(local_len > 0, lo - shard_start, 0)
    return local_off.astype(np.int64), local_len.astype(np.int64)


def sharded_step(mon, local_arena, *, group=None, sumsq=None, mask=None, stats=None):
    """One step of the sharded path for a rank whose gradient shard is
    `local_arena` (a handle created with the rank's `shard_layout`):
    this rank's per-unit sums of squares (gnmr_step_partials), their sum over
    the ranks of `group` (torch.distributed all-reduce, U fp64 values), then
    Algorithms 1-2 on the summed sums (gnmr_finish).  Every rank passes the
    same sums to the same deterministic controller, so every rank gets the
    same mask.  All three run on torch's current stream, which the
    all-reduce orders against.  Returns the mask tensor."""
    import torch.distributed as dist
    sums = mon.step_partials(local_arena, sumsq=sumsq)
    dist.all_reduce(sums, op=dist.ReduceOp.SUM, group=group)
    return mon.finish(sums, mask=mask, stats=stats)
