"""Multi-process host logic: one process per GPU, launched by torchrun.

L_JAB evaluations are independent units (candidates, blocks, batches), so ranks need no exchange on
the data path. The one real exchange is when one evaluation's sequences are sharded across ranks:
L and the scale gradient are sums over sequences (Eq. 3 is a sum over the batch before the mean), so
the full-batch values are the size-weighted sum of the shard values, combined with one all-reduce of
the gradient (D x d/G floats) and the loss.
"""
from __future__ import annotations

import os
from typing import Tuple

import torch


def dist_env() -> Tuple[int, int, int]:
    """(world_size, rank, local_rank) from the torchrun environment (1, 0, 0 when absent)."""
    return (int(os.environ.get("WORLD_SIZE", "1")), int(os.environ.get("RANK", "0")),
            int(os.environ.get("LOCAL_RANK", "0")))


def max_over_ranks(x: float, device=None) -> float:
    """Maximum of a host float over all ranks (the timed region ends when the slowest rank does)."""
    import torch.distributed as dist
    if not dist.is_available() or not dist.is_initialized() or dist.get_world_size() == 1:
        return float(x)
    t = torch.tensor([float(x)], dtype=torch.float64, device=device or "cpu")
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def shard_sequences(batch: int, world: int, rank: int) -> Tuple[int, int]:
    """Contiguous sequence range [start, stop) of `rank` when `batch` sequences are split over
    `world` ranks as evenly as possible (the first batch % world ranks get one more)."""
    if world < 1 or not 0 <= rank < world:
        raise ValueError("bad world/rank")
    base, extra = divmod(batch, world)
    start = rank * base + min(rank, extra)
    return start, start + base + (1 if rank < extra else 0)


def combine_shards(loss: torch.Tensor, grad: torch.Tensor, n_local: int, n_total: int):
    """Full-batch L_JAB and scale gradient from per-shard values computed on n_local of n_total
    sequences: each shard's mean-normalised values are weighted by n_local / n_total and summed over
    ranks with one all-reduce of a single fp64 buffer holding the loss and the gradient (1 + D d/G
    values), written back in place into `loss` and `grad`."""
    import torch.distributed as dist
    w = float(n_local) / float(n_total)
    if dist.is_available() and dist.is_initialized() and dist.get_world_size() > 1:
        buf = torch.cat([loss.reshape(-1).double(), grad.reshape(-1).double()]).mul_(w)
        dist.all_reduce(buf)
        loss.copy_(buf[:loss.numel()].view_as(loss))
        grad.copy_(buf[loss.numel():].view_as(grad))
    else:
        loss.mul_(w)
        grad.mul_(w)
    return loss, grad


def fisher_score_from_shards(grad_w: torch.Tensor, n_local: int, n_total: int) -> float:
    """Fisher-coupling score of one evaluation whose sequences are sharded over the ranks: the weight
    gradient dL/dw_hat (jab_loss_backward_weights' grad_w of this rank's shard) is additive over
    sequences like the scale gradient, but its squared norm is not, so the shards' gradients are
    combined first (one all-reduce of D x d floats, in place) and the norm is taken of the sum."""
    import torch.distributed as dist
    grad_w.mul_(float(n_local) / float(n_total))
    if dist.is_available() and dist.is_initialized() and dist.get_world_size() > 1:
        dist.all_reduce(grad_w)
    return float((grad_w.double() ** 2).sum())

