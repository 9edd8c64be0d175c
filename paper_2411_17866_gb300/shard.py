"""Parameter shards of one model over G processes: host-side logic of the multi-GPU path.

Every step of Algorithm 1 (arXiv 2411.17866, Sec. 3) is elementwise in the
parameters: the local steps update each element of each worker's copy on its
own, and the global step's only cross-worker operation, the all-reduce
average, combines the n copies of one element.  Cutting the model's
parameters into G contiguous ranges therefore gives G independent problems
(each holds all n worker copies of its range) with no communication on the
data path.  Rank r runs the library on its range, a dsm_layout whose
``first_element`` places it in the whole model, so the synthetic gradients,
the initial model and the randomized signs are those of the whole model, and
the G shards together compute exactly what one process computes on it.

This module holds no arithmetic of the method: it cuts a tensor list into
pieces and sums the per-tensor statistics of the pieces back per tensor.
"""
from __future__ import annotations

import dataclasses
from typing import List, Sequence, Tuple

STAT_SUMS = ("delta_sq", "drift")
STAT_COUNTS = ("zero_sign", "flips", "unanimous", "clamped")


@dataclasses.dataclass(frozen=True)
class Piece:
    """The part of one tensor of the whole model that lies in a shard."""
    name: str
    numel: int
    kind: int
    grad_scale: float
    wd: int
    tensor: int          # index of the tensor in the whole model's list
    offset: int          # first element of the piece within that tensor


@dataclasses.dataclass(frozen=True)
class Shard:
    rank: int
    world: int
    first_element: int   # of the shard in the whole model (a multiple of `align`)
    count: int           # elements of the shard
    pieces: Tuple[Piece, ...]

    @property
    def tensors(self) -> Tuple[Piece, ...]:
        """The shard's layout (pieces have numel, grad_scale, kind and wd, as tensors do)."""
        return self.pieces


def shard_bounds(d: int, world: int, align: int = 64) -> List[Tuple[int, int]]:
    """Contiguous element ranges [start, end) of G = world shards of a d-element model: boundaries at
    multiples of `align` (the library needs multiples of 4; 64 keeps every shard's buffers 256-byte aligned),
    as equal as that allows; the last shard ends at d."""
    if world < 1 or align < 4 or align % 4:
        raise ValueError("world must be >= 1 and align a positive multiple of 4")
    cuts = [min(d, (r * d // world) // align * align) for r in range(world)] + [d]
    return [(cuts[r], cuts[r + 1]) for r in range(world)]


def shard_layout(tensors: Sequence, world: int, rank: int, align: int = 64) -> Shard:
    """Shard `rank` of `world` of the model whose tensor list is `tensors` (objects with numel, kind,
    grad_scale and, optionally, wd and name)."""
    d = sum(int(t.numel) for t in tensors)
    a, b = shard_bounds(d, world, align)[rank]
    pieces = []
    start = 0
    for i, t in enumerate(tensors):
        end = start + int(t.numel)
        lo, hi = max(a, start), min(b, end)
        if hi > lo:
            pieces.append(Piece(getattr(t, "name", f"t{i}"), hi - lo, int(t.kind), float(t.grad_scale),
                                int(getattr(t, "wd", 1)), i, lo - start))
        start = end
    return Shard(rank, world, a, b - a, tuple(pieces))


def repeated_model(tensors: Sequence, copies: int) -> list:
    """The tensor list of a model made of `copies` copies of `tensors` (the weak-scaling model: G shards
    of one copy each)."""
    return [t for _ in range(copies) for t in tensors]


def stats_by_tensor(shard: Shard, piece_stats: Sequence[dict], num_tensors: int) -> List[dict]:
    """The statistics of a shard's pieces placed at their tensors of the whole model (zeros elsewhere)."""
    out = [dict({k: 0.0 for k in STAT_SUMS}, **{k: 0 for k in STAT_COUNTS}) for _ in range(num_tensors)]
    for p, st in zip(shard.pieces, piece_stats):
        o = out[p.tensor]
        for k in STAT_SUMS:
            o[k] += float(st[k])
        for k in STAT_COUNTS:
            o[k] += int(st[k])
    return out


def reduce_stats(per_rank: Sequence[Sequence[dict]]) -> List[dict]:
    """Sum per-tensor statistics over shards (each a list over the whole model's tensors)."""
    num = len(per_rank[0])
    out = [dict({k: 0.0 for k in STAT_SUMS}, **{k: 0 for k in STAT_COUNTS}) for _ in range(num)]
    for stats in per_rank:
        for o, st in zip(out, stats):
            for k in STAT_SUMS:
                o[k] += float(st[k])
            for k in STAT_COUNTS:
                o[k] += int(st[k])
    return out


def all_reduce_stats(stats: Sequence[dict]):
    """Sum per-tensor statistics over the ranks of the default torch.distributed group (host tensors:
    float64 sums, int64 counts), in place of a gather; returns the reduced list."""
    import torch
    import torch.distributed as dist
    sums = torch.tensor([[float(s[k]) for k in STAT_SUMS] for s in stats], dtype=torch.float64)
    counts = torch.tensor([[int(s[k]) for k in STAT_COUNTS] for s in stats], dtype=torch.int64)
    dist.all_reduce(sums)
    dist.all_reduce(counts)
    return [dict({k: float(sums[T, j]) for j, k in enumerate(STAT_SUMS)},
                 **{k: int(counts[T, j]) for j, k in enumerate(STAT_COUNTS)}) for T in range(len(stats))]
