"""Data-parallel plumbing of the DendSN layer step.

Neurons are independent, so a batch splits across ranks with no exchange in the
forward; the only exchange is the sum of the parameter gradients (2K + 2Kb floats
per channel, plus one for dL/dbeta when the somatic decay is learnable) after the
backward. These helpers hold that host-side logic; the arithmetic stays in the CUDA
library.
"""
from __future__ import annotations

from typing import Dict, Tuple

import torch
import torch.distributed as dist


def shard_range(n: int, world: int, rank: int) -> Tuple[int, int]:
    """Contiguous [start, stop) share of n items for `rank` of `world` (sizes differ by <= 1)."""
    if world < 1 or not 0 <= rank < world:
        raise ValueError(f"bad rank {rank} of world {world}")
    base, extra = divmod(n, world)
    start = rank * base + min(rank, extra)
    return start, start + base + (1 if rank < extra else 0)


def _sizes(C: int, K: int, Kb: int, with_beta: bool):
    return [C * K, C * K, C * Kb, C * Kb] + ([C] if with_beta else [])


def param_grad_buffer(C: int, K: int, Kb: int, device=None, with_beta: bool = False
                      ) -> Tuple[torch.Tensor, Dict[str, torch.Tensor]]:
    """One flat float32 buffer holding the parameter gradients, and views into it.

    galpha, gxi [C, K], gzeta, gkappa [C, Kb], and with_beta also gbeta [C] (the
    per-channel dL/dbeta of a learnable somatic decay). A single buffer lets one
    all-reduce sum all of them.
    """
    flat = torch.zeros(sum(_sizes(C, K, Kb, with_beta)), dtype=torch.float32, device=device)
    return flat, split_param_grads(flat, C, K, Kb, with_beta, as_dict=True)


def split_param_grads(flat: torch.Tensor, C: int, K: int, Kb: int, with_beta: bool = False,
                      as_dict: bool = False):
    """Views of one flat parameter-gradient row: (galpha, gxi, gzeta, gkappa[, gbeta]), or a
    dict with those keys."""
    parts = torch.split(flat, _sizes(C, K, Kb, with_beta))
    views = [parts[0].view(C, K), parts[1].view(C, K), parts[2].view(C, Kb),
             parts[3].view(C, Kb)] + ([parts[4]] if with_beta else [])
    if as_dict:
        return dict(zip(("galpha", "gxi", "gzeta", "gkappa", "gbeta"), views))
    return tuple(views)


def sum_param_grads(flat: torch.Tensor, group=None) -> torch.Tensor:
    """Sums the parameter-gradient buffer over the ranks of `group` in place."""
    if dist.is_available() and dist.is_initialized() and dist.get_world_size(group) > 1:
        dist.all_reduce(flat, op=dist.ReduceOp.SUM, group=group)
    return flat
