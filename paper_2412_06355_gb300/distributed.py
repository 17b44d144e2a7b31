"""Data-parallel plumbing of the DendSN layer step.

Neurons are independent, so a batch splits across ranks with no exchange in the
forward; the only exchange is the sum of the parameter gradients (2K + 2Kb floats
per channel) after the backward. These helpers hold that host-side logic; the
arithmetic stays in the CUDA library.
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


def param_grad_buffer(C: int, K: int, Kb: int, device=None) -> Tuple[torch.Tensor, Dict[str, torch.Tensor]]:
    """One flat float32 buffer holding the four parameter gradients, and views into it.

    A single buffer lets one all-reduce sum all four.
    """
    flat = torch.zeros(2 * C * K + 2 * C * Kb, dtype=torch.float32, device=device)
    ga, gxi, gz, gk = torch.split(flat, [C * K, C * K, C * Kb, C * Kb])
    return flat, {"galpha": ga.view(C, K), "gxi": gxi.view(C, K), "gzeta": gz.view(C, Kb),
                  "gkappa": gk.view(C, Kb)}


def split_param_grads(flat: torch.Tensor, C: int, K: int, Kb: int):
    """(galpha, gxi, gzeta, gkappa) views of one flat parameter-gradient row."""
    ga, gxi, gz, gk = torch.split(flat, [C * K, C * K, C * Kb, C * Kb])
    return ga.view(C, K), gxi.view(C, K), gz.view(C, Kb), gk.view(C, Kb)


def sum_param_grads(flat: torch.Tensor, group=None) -> torch.Tensor:
    """Sums the parameter-gradient buffer over the ranks of `group` in place."""
    if dist.is_available() and dist.is_initialized() and dist.get_world_size(group) > 1:
        dist.all_reduce(flat, op=dist.ReduceOp.SUM, group=group)
    return flat
