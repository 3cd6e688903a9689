"""Fixed-order FP16 gradient all-reduce for data-parallel training (host code).

The paper trains on 8 to 128 GPUs (Sec. 5.1), each with its own batch and its
own BatchNorm statistics; before every SGD step the GPUs' gradients are
averaged, and in the pure-FP16 method that average is FP16 arithmetic too
(Sec. 5.2).  A ring all-reduce adds the ranks' values in an order that
depends on the ring position of each chunk, so its FP16 result differs from
rank to rank and run to run.  Here the order is fixed: every element is the
pairwise tree over the ranks in rank order, then one scaling by rn(1/world)
(pf16_allreduce_combine), and every rank ends with the same bits.

Transport (torch.distributed; NCCL on GPUs, gloo on CPU ranks), for a flat
gradient of n values padded to world * chunk:
  1. all_to_all: rank r receives chunk r of every rank's gradient, in rank
     order -- the reduce-scatter's traffic, without its arithmetic;
  2. combine: rank r reduces its `world` planes with the fixed tree;
  3. all_gather: every rank receives every combined chunk.
Each rank sends and receives (world - 1) / world of the gradient twice, the
bytes of a bandwidth-optimal all-reduce.

The combining step is `pf16.allreduce_combine` on device tensors.  A caller
may pass another `combine` with the same contract (planes [world][chunk] ->
chunk); the CPU-rank tests pass the oracle's.
"""
from __future__ import annotations

import numpy as np
import torch
import torch.distributed as dist

from . import pf16


def inv_world_bits(world: int) -> int:
    """rn(1/world) as binary16 bits (exact for a power of two)."""
    return int(np.array([1.0 / world], np.float64).astype(np.float16).view(np.uint16)[0])


def chunk_size(n: int, world: int) -> int:
    """Elements of each rank's chunk: n / world rounded up to a multiple of 8
    (16-byte rows for the combining kernel)."""
    per = -(-n // world)
    return -(-per // 8) * 8


def _device_combine(planes: torch.Tensor, world: int, chunk: int, scale: int) -> torch.Tensor:
    out = torch.empty(chunk, dtype=torch.int16, device=planes.device)
    pf16.allreduce_combine(planes, world, chunk, chunk, scale, out)
    return out


def allreduce_mean_(grad: torch.Tensor, group=None, combine=None) -> torch.Tensor:
    """Average the binary16 gradient `grad` (a flat int16 tensor of bit
    patterns) over the ranks of `group`, in place, with the fixed FP16 order.
    Returns grad.  Every rank must call it with a gradient of the same size."""
    world = dist.get_world_size(group)
    if world == 1:
        return grad
    n = grad.numel()
    chunk = chunk_size(n, world)
    send = torch.zeros(world * chunk, dtype=torch.int16, device=grad.device)
    send[:n].copy_(grad.view(-1))
    recv = torch.empty_like(send)
    # the transport moves bit patterns; float16 is a dtype every backend carries
    dist.all_to_all_single(recv.view(torch.float16), send.view(torch.float16), group=group)
    comb = combine if combine is not None else _device_combine
    mine = comb(recv, world, chunk, inv_world_bits(world))
    gathered = torch.empty(world * chunk, dtype=torch.int16, device=grad.device)
    dist.all_gather_into_tensor(gathered.view(torch.float16), mine.view(torch.float16), group=group)
    grad.view(-1).copy_(gathered[:n])
    return grad
