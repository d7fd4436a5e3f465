"""Data-parallel training over ranks (one process per GPU).

The scan is independent across the batch, so ranks split B and need no
exchange during the forward or the reverse pass.  The one exchange is the
sum of the gradients that reduce over the batch: dW of the dense layers and
the learnable beta / threshold / alpha gradients of the scans.  The loss is
normalised by the global batch in the loss kernel (``batch_total``), so the
per-rank results are partial sums of the global ones and a plain SUM
all-reduce (NCCL on GPUs, gloo on CPU) completes them; no rescaling step.

Only host logic lives here: how the batch is split and which buffers are
summed.
"""
from __future__ import annotations

from typing import Iterable, Optional, Tuple

import torch
import torch.distributed as dist


def shard_range(B: int, world: int, rank: int) -> Tuple[int, int]:
    """Contiguous samples [b0, b1) of rank `rank`: the first B % world ranks
    take one sample more than the others."""
    if world < 1 or not 0 <= rank < world or B < 0:
        raise ValueError("shard_range: need world >= 1, 0 <= rank < world, B >= 0")
    q, r = divmod(B, world)
    b0 = rank * q + min(rank, r)
    return b0, b0 + q + (1 if rank < r else 0)


def allreduce_sum_(tensors: Iterable[torch.Tensor], group: Optional[dist.ProcessGroup] = None):
    """Sum each tensor over the ranks, in place (no-op without a process
    group or with one rank)."""
    if not dist.is_available() or not dist.is_initialized() or dist.get_world_size(group) == 1:
        return
    for t in tensors:
        if t is not None:
            dist.all_reduce(t, op=dist.ReduceOp.SUM, group=group)


def grad_buffers(net):
    """The buffers a replica's gradients and loss live in: dW of every layer
    (one flat buffer), the learnable betas' gradients if the net has them
    (the convolutional SNN), and the loss."""
    return [net.dW_flat, getattr(net, "dbeta_flat", None), net.loss]


class DataParallelDenseSNN:
    """A network replica (DenseSNN or ConvSNN) per rank training on its
    shard of each global batch: forward and BPTT on the shard (loss
    normalised by the global batch), SUM all-reduce of the gradients (one
    flat buffer per kind), then the same AdamW update on every rank, so the
    replicas stay identical."""

    def __init__(self, net, global_batch: int, group: Optional[dist.ProcessGroup] = None):
        self.net = net
        self.global_batch = global_batch
        self.group = group
        net.batch_total = global_batch

    def train_step(self, X_shard, labels_shard, stream=None):
        net = self.net
        net.forward(X_shard, labels_shard, stream)
        net.backward(X_shard, stream)
        allreduce_sum_(grad_buffers(net), self.group)
        net.update(stream)
        return net.loss


DataParallelConvSNN = DataParallelDenseSNN
