"""Data-parallel block training across replicas: the one exchange step.

Every replica holds the same weights (same seeds, same updates) and runs the
block step of Sec. 3.3 on its own shard of the batch.  Nothing crosses
replicas during the forward or the local backward; the single exchange sits
between the backward and IntegerSGD (Algorithm 1): the int64 weight
gradients dW and dW_lr are summed over the replicas, and every replica then
applies IntegerSGD to that sum.

* Integer addition is associative, so the summed gradient equals the one a
  single replica would compute on the whole batch, bit for bit and modulo
  2^64 like the single-replica sum, in any reduction order.
* The floor of Algorithm 1 comes after the sum: floor(sum dW / gamma) differs
  from sum floor(dW / gamma) in general, so replicas must not update first
  and average weights afterwards.
* Status bits (OVERFLOW, bad label) are OR-ed over replicas: a value that
  overflows on one shard overflows on the whole batch.  The SSE is summed and
  the loss recomputed as floor(SSE / 2).

The reductions go through torch.distributed (NCCL for CUDA tensors, gloo for
CPU tensors).  Dropout masks index samples within a replica's shard, so a
data-parallel run with dropout is not bit-identical to a single replica on the
whole batch; without dropout it is.
"""
import torch
import torch.distributed as dist

from . import binding as nb

STATUS_BITS = (nb.STATUS_BIT_OVERFLOW, nb.STATUS_BIT_BAD_LABEL, nb.STATUS_BIT_TIMEOUT)


def _world(group):
    return dist.get_world_size(group) if dist.is_available() and dist.is_initialized() else 1


def allreduce_grads(grads, group=None):
    """Sums int64 weight-gradient tensors over all replicas, in place.  The
    result is exact (integer addition, wrapping modulo 2^64 as the
    single-replica sum does).  No-op for one replica."""
    if _world(group) == 1:
        return grads
    for g in grads:
        if g.dtype != torch.int64:
            raise TypeError("weight gradients are int64")
        dist.all_reduce(g, op=dist.ReduceOp.SUM, group=group)
    return grads


def combine_status(bits, group=None, device="cpu"):
    """OR of the replicas' status words (each bit's maximum)."""
    bits = int(bits)
    if _world(group) == 1:
        return bits
    t = torch.tensor([1 if bits & b else 0 for b in STATUS_BITS], dtype=torch.int64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX, group=group)
    return sum(b for b, v in zip(STATUS_BITS, t.tolist()) if v)


def _wrap64(v):
    v &= (1 << 64) - 1
    return v - (1 << 64) if v >= 1 << 63 else v


def combine_loss(sse, group=None, device="cpu"):
    """(summed SSE, floor(SSE / 2)) over the replicas, SSE modulo 2^64."""
    t = torch.tensor([_wrap64(int(sse))], dtype=torch.int64, device=device)
    if _world(group) > 1:
        dist.all_reduce(t, op=dist.ReduceOp.SUM, group=group)
    total = _wrap64(int(t.item()))
    return total, total // 2


def shard(n, rank, world):
    """[start, stop) of this replica's contiguous share of n samples."""
    base, extra = divmod(int(n), int(world))
    start = rank * base + min(rank, extra)
    return start, start + base + (1 if rank < extra else 0)


class DataParallelNet:
    """A chain of block handles on this replica's GPU trained data-parallel:
    forward and backward of every block on the local shard, the exact int64
    gradient exchange, then IntegerSGD from the summed gradients.  Every
    replica must be built with the same layers and seeds."""

    def __init__(self, blocks, group=None):
        self.blocks = list(blocks)
        self.group = group

    def grads(self):
        out = []
        for g in self.blocks:
            for i in range(len(g.layers)):
                out.append(g.grad_device(nb.NITRO_T_DW, i))
            out.append(g.grad_device(nb.NITRO_T_DWLR, 0))
        return out

    def step(self, x, labels, losses, stream=None):
        """One step on this replica's shard: x int8 [b, in], labels int32 [b],
        losses int64 [blocks] (the local losses).  Collectives run on the
        current stream after the backward passes."""
        acts = [x]
        for g in self.blocks:
            out = (torch.empty((x.shape[0], g.out_features), dtype=torch.int8, device=x.device)
                   if g.layers else None)
            g.forward(acts[-1], out, stream=stream)
            acts.append(out if out is not None else acts[-1])
        for i, g in enumerate(self.blocks):
            g.backward(acts[i], labels, losses[i:i + 1], stream=stream)
        allreduce_grads(self.grads(), self.group)
        for g in self.blocks:
            g.sgd(stream=stream)
