"""Partitioning one parameter set over ranks (ZeRO-1 style).

The delayed step is elementwise, so it splits along the flat concatenation
of the tensors: rank r owns one contiguous range and keeps the optimizer
state of that range only. The one quantity that crosses ranks is the
squared gradient norm for global clipping (App. E.1): each rank adds its
share with ``grad_sqnorm``, ``dpo.allreduce_sqnorm`` sums the shares, and
every rank's step clips from the total (``set_clip_source``). The
reduce-scatter of gradients before the step and the all-gather of weights
after it belong to the training framework around this library.
"""
from __future__ import annotations

from typing import List, Optional, Sequence, Tuple

from .dpo import ALIGN_ELEMS, DelayedAdamW, Layout

Piece = Tuple[int, int, int]   # (tensor index, start, stop) within that tensor


def bounds(total: int, world: int, rank: int, align: int = ALIGN_ELEMS) -> Tuple[int, int]:
    """[lo, hi) of rank's range of ``total`` flat elements: near-equal
    shares, every inner boundary a multiple of ``align`` (so each shard's
    pieces start on a vector boundary of their tensors' flat layout)."""
    if world < 1 or not 0 <= rank < world:
        raise ValueError(f"rank {rank} outside a world of {world}")
    if total < 0:
        raise ValueError("negative element count")
    cut = lambda r: total if r == world else min(total, (total * r // world) // align * align)
    return cut(rank), cut(rank + 1)


def partition(numels: Sequence[int], world: int, rank: int,
              align: int = ALIGN_ELEMS) -> List[Piece]:
    """The pieces of rank's range, one per tensor it overlaps, in tensor
    order. Over all ranks the pieces tile every tensor exactly once."""
    lo, hi = bounds(sum(int(n) for n in numels), world, rank, align)
    pieces, off = [], 0
    for i, n in enumerate(numels):
        n = int(n)
        a, b = max(lo, off), min(hi, off + n)
        if a < b:
            pieces.append((i, a - off, b - off))
        off += n
    return pieces


def shard_optimizer(numels: Sequence[int], world: int, rank: int, *,
                    wd_on: Optional[Sequence[bool]] = None,
                    sync: Optional[Sequence[bool]] = None, x0=None,
                    **kwargs) -> Tuple[DelayedAdamW, List[Piece]]:
    """A DelayedAdamW over rank's pieces. Each piece keeps the weight-decay
    and synchronous flags of the tensor it comes from. ``x0`` seeds the
    shard's master copy: the full flat fp32 weights (a torch tensor on any
    device), or a function ``x0(start, out)`` that writes the weights of flat
    elements [start, start + out.numel()) into the fp32 device tensor ``out``
    (so no rank holds the whole set). Pass ``max_grad_norm`` in ``kwargs``
    and a clip source to clip globally."""
    pieces = partition(numels, world, rank)
    lay = Layout.of([b - a for _, a, b in pieces])
    buf = None
    if x0 is not None:
        import torch
        starts = [0]
        for n in numels:
            starts.append(starts[-1] + int(n))
        dev = kwargs.get("device") if callable(x0) else x0.device
        buf = torch.zeros(lay.total, dtype=torch.float32, device=dev)
        for j, (i, a, b) in enumerate(pieces):
            out = buf[lay.offsets[j]:lay.offsets[j] + b - a]
            if callable(x0):
                x0(starts[i] + a, out)
            else:
                out.copy_(x0[starts[i] + a:starts[i] + b])
    opt = DelayedAdamW(
        lay.numels,
        wd_on=[wd_on[i] for i, _, _ in pieces] if wd_on is not None else None,
        sync=[sync[i] for i, _, _ in pieces] if sync is not None else None,
        x0=buf, **kwargs)
    return opt, pieces
