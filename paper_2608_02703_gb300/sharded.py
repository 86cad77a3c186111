"""Vocabulary-parallel evaluation of the packed head: one process per GPU,
each holding a contiguous block of vocabulary rows.

The forward is row-separable (paper, Section 3.2, Eq. 7): logit y[m][n]
involves only row n of the V-indexed stored components (residual codes and
group scales, the core's left factor, the correction's left factor and row
scales) plus the d-side factors, which every rank keeps whole.  So

  - logits need no exchange: each rank writes its own block of columns;
  - cross entropy needs one exchange of three floats per token: every rank
    computes (max, sum of exp, target logit or -inf) over its rows
    (archead_forward_lse_partial), the ranks all-gather them, and one
    deterministic combine in shard order gives ce = max + log(sum) - y_t
    (archead_lse_combine);
  - greedy output exchanges (largest logit, its row) per token and keeps the
    largest, the lowest global row on ties (archead_argmax_combine).

This module only marshals arguments and makes the exchange (an all-gather
over a torch.distributed process group: NCCL on GPUs, gloo works as well);
every step of the forward and both combines run in the library's kernels.
"""

from __future__ import annotations

import dataclasses
from typing import Dict, Optional, Tuple

import numpy as np

from . import archead

# Canonical arrays indexed by vocabulary row, per packed format.
_ROW_ARRAYS = {
    "int8": ("res_codes", "res_scales", "core_u", "corr_a", "corr_a_scale"),
    "sc4": ("res_codes", "res_scale_codes", "res_row_scale", "core_u5", "corr_a", "corr_a_scale"),
}
# Arrays every shard holds whole (indexed by d or by rank column).
_SHARED_ARRAYS = ("core_u_scale", "core_v", "core_v_scale", "corr_b", "corr_b_scale")


def shard_rows(V: int, world: int, rank: int, align: int = 128) -> Tuple[int, int]:
    """(first global row, number of rows) of `rank`'s block: contiguous blocks
    of whole 128-row tiles, as even as the tiles allow; every rank gets at
    least one row while V >= world."""
    if world < 1 or not 0 <= rank < world:
        raise ValueError("rank must lie in [0, world)")
    if V < world:
        raise ValueError("fewer vocabulary rows than ranks")
    tiles = -(-V // align)
    if tiles >= world:
        t0 = tiles * rank // world
        t1 = tiles * (rank + 1) // world
        r0, r1 = t0 * align, min(V, t1 * align)
    else:  # fewer tiles than ranks: plain row blocks
        r0, r1 = V * rank // world, V * (rank + 1) // world
    return r0, r1 - r0


def shard_head(head: Dict[str, np.ndarray], shape, row0: int, rows: int):
    """The packed head of global rows [row0, row0 + rows): the V-indexed
    arrays sliced, the d-side arrays shared, and its shape (V = rows)."""
    fmt = getattr(shape, "fmt", "int8")
    if row0 < 0 or rows < 1 or row0 + rows > shape.V:
        raise ValueError("row block outside the head")
    out = {}
    for k in _ROW_ARRAYS[fmt]:
        out[k] = np.ascontiguousarray(head[k][row0:row0 + rows])
    for k in _SHARED_ARRAYS:
        out[k] = head[k]
    return out, dataclasses.replace(shape, V=rows)


def exchange(t, group=None):
    """All-gather of one tensor from every rank of `group`, stacked in rank
    order: [world, *t.shape].  The only data exchange of the sharded head."""
    import torch
    import torch.distributed as dist

    world = dist.get_world_size(group)
    parts = [torch.empty_like(t) for _ in range(world)]
    dist.all_gather(parts, t.contiguous(), group=group)
    return torch.stack(parts)


class ShardedHead:
    """This rank's block of a packed head, on the current CUDA device."""

    def __init__(self, head: Dict[str, np.ndarray], shape, group=None, rank: Optional[int] = None,
                 world: Optional[int] = None):
        import torch.distributed as dist

        if rank is None or world is None:
            rank, world = dist.get_rank(group), dist.get_world_size(group)
        self.group, self.rank, self.world = group, rank, world
        self.full_shape = shape
        self.row0, self.rows = shard_rows(shape.V, world, rank)
        sub, self.shape = shard_head(head, shape, self.row0, self.rows)
        self.pack = archead.archead_pack_create(sub, self.shape)

    def close(self) -> None:
        self.pack.close()

    def logits(self, x, M: int, out, out_dtype: int = archead.OUT_BF16, path: int = archead.PATH_AUTO) -> None:
        """Logits of this rank's rows, out [M][rows] (global columns row0 ...)."""
        archead.archead_forward_path(self.pack, x, M, out, out_dtype, path)

    def cross_entropy(self, x, M: int, targets, ce, path: int = archead.PATH_AUTO) -> None:
        """Per-token CE over the whole vocabulary (targets: global rows), the
        same on every rank."""
        import torch

        parts = torch.empty((M, 3), dtype=torch.float32, device=x.device)
        archead.archead_forward_lse_partial(self.pack, x, M, targets, self.row0, parts, path)
        gathered = exchange(parts, self.group)
        archead.archead_lse_combine(gathered, self.world, M, ce)

    def greedy(self, x, M: int, index, value=None, path: int = archead.PATH_AUTO) -> None:
        """Greedy next token (global row) per row of x, the same on every rank."""
        import torch

        dev = x.device
        idx = torch.empty(M, dtype=torch.int32, device=dev)
        val = torch.empty(M, dtype=torch.float32, device=dev)
        archead.archead_forward_argmax_path(self.pack, x, M, idx, val, path)
        vals, idxs = exchange(val, self.group), exchange(idx, self.group)
        row0s = exchange(torch.tensor([self.row0], dtype=torch.int32, device=dev), self.group)
        archead.archead_argmax_combine(vals, idxs, row0s, self.world, M, index, value)
