"""Data-parallel training of NOBLE layers: token sharding and the gradient all-reduce.

The paper trains its decoders on 8 GPUs with data parallelism (Section 4.1.1).
Each rank holds a full copy of the layer's parameters and a contiguous share of
the step's tokens.  The forward pass needs no exchange.  Every parameter
gradient of the layer (dW, dbias, dW_down, dW_up, dM, domega, dphi) is a sum
over tokens, so the gradient of the whole batch is the sum of the ranks'
gradients: one all-reduce (sum) per layer, of the flat bucket that
``noble_linear_grad_bucket`` lays out and ``noble_linear_bwd`` writes into.
dx stays on its rank (it is per token).

The collective is torch.distributed's (NCCL between GPUs, gloo on the host).
Each bucket's all-reduce is started as soon as that layer's backward has been
enqueued, with ``async_op``: NCCL runs it on its own stream after the work
already queued on the caller's stream, so it overlaps the backward of the
next layer; ``wait`` orders the caller's stream after every pending
reduction.  No kernel of this library reads a peer's memory.
"""
from __future__ import annotations


def token_shard(T: int, rank: int, world: int) -> tuple[int, int]:
    """[start, stop) of rank's contiguous share of T tokens; the first
    T % world ranks take one token more."""
    if world < 1 or not 0 <= rank < world or T < 0:
        raise ValueError("bad shard request")
    base, extra = divmod(T, world)
    start = rank * base + min(rank, extra)
    return start, start + base + (1 if rank < extra else 0)


class GradAllReduce:
    """Sum-all-reduce of gradient buckets across the ranks of ``group``.

    ``launch(bucket)`` starts the reduction of one flat fp32 bucket (a torch
    tensor, on the device for NCCL or on the host for gloo) and returns at
    once; ``wait()`` completes every pending reduction (for NCCL: makes the
    current stream wait for them).  The result is the plain sum over ranks;
    dividing by the world size, if the loss is a mean over the global batch,
    is left to the caller.
    """

    def __init__(self, group=None):
        self.group = group
        self._pending = []

    def launch(self, bucket):
        import torch.distributed as dist
        self._pending.append(dist.all_reduce(bucket, op=dist.ReduceOp.SUM, group=self.group, async_op=True))

    def wait(self):
        pending, self._pending = self._pending, []
        for work in pending:
            work.wait()

    @property
    def pending(self) -> int:
        return len(self._pending)
