"""Data-parallel token sharding of the LoRA linear (host logic only).

The layer shards by tokens.  Every rank keeps the frozen W and the adapter
A, B, and runs the library on its own contiguous slice of the tokens: the
forward (y, su) and the input gradient dx are row-local, so they need
nothing from other ranks.  dA = s (dy B)^T x and dB = s dy^T (x A^T) are
sums over tokens, so the gradient of the whole batch is the sum of the
ranks' gradients; that sum is the one exchange of a data-parallel step.

The exchange is a host hook the caller supplies: a callable that sums one
contiguous fp32 tensor across ranks in place (torch.distributed.all_reduce
by default).  The library itself never runs a collective.  This module is
argument marshalling around that hook: it computes slices and packs the
gradients into one buffer so that a step makes one call of the hook.
"""
from __future__ import annotations

from typing import Callable, Sequence, Tuple

ROW_ALIGN = 8  # token counts the library accepts are multiples of 8


def token_slice(T: int, rank: int, world: int, align: int = ROW_ALIGN) -> Tuple[int, int]:
    """Contiguous token range [t0, t1) of `rank` among `world` ranks.

    Boundaries fall on multiples of `align` (T must be one); the slices
    cover [0, T) without overlap and differ in length by at most `align`.
    A rank may get an empty slice when T / align < world."""
    if T % align or T < 0:
        raise ValueError(f"T={T} is not a non-negative multiple of {align}")
    if not 0 <= rank < world:
        raise ValueError(f"rank {rank} outside world of {world}")
    blocks = T // align
    base, extra = divmod(blocks, world)
    b0 = rank * base + min(rank, extra)
    b1 = b0 + base + (1 if rank < extra else 0)
    return b0 * align, b1 * align


def sum_adapter_grads(grads: Sequence, all_reduce: Callable | None = None) -> None:
    """Sums fp32 gradient tensors (dA and dB of every projection) across
    ranks in place, through one call of `all_reduce` on a packed buffer.

    `all_reduce(buf)` must replace the 1-D fp32 tensor `buf` by its sum over
    ranks; the default is torch.distributed.all_reduce (SUM) on the default
    process group.  Every rank passes tensors of the same shapes in the same
    order."""
    import torch

    if all_reduce is None:
        import torch.distributed as dist

        def all_reduce(buf):
            dist.all_reduce(buf, op=dist.ReduceOp.SUM)

    grads = list(grads)
    if not grads:
        return
    for g in grads:
        if g.dtype != torch.float32:
            raise TypeError("adapter gradients are fp32")
    buf = torch.cat([g.reshape(-1) for g in grads])
    all_reduce(buf)
    off = 0
    for g in grads:
        n = g.numel()
        g.copy_(buf[off:off + n].view_as(g))
        off += n
