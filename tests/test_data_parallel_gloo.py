"""Data-parallel exchange step on CPU ranks (gloo, world size 2).

Two replicas each train the same network on half of every batch, sum their
int64 weight gradients with the library's exchange step and apply IntegerSGD
to the sum (Algorithm 1, floor after the sum).  Their weights must equal,
bit for bit, those of one replica trained on the whole batch.  The arithmetic
on both sides is the oracle's; what is under test is the exchange: the
reduction, the shard split, the status OR and the loss from the summed SSE.
"""
import os
import socket
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

NETS = {
    # conv block with pool and a second conv, then the output block
    "conv": dict(shape=(8, 8, 3), blocks=[
        {"layers": [(0, 3, 8, 8, 8, 1), (0, 8, 8, 4, 4, 0)], "in_features": 8 * 8 * 3},
        {"layers": [], "in_features": 4 * 4 * 8}]),
    # two linear blocks and the output block, with weight decay and trunc rounding
    "mlp": dict(shape=(24,), hyper=dict(eta_inv_fw=25000, eta_inv_lr=3000, sgd_round=1), blocks=[
        {"layers": [(1, 24, 16, 1, 1, 0)], "in_features": 24},
        {"layers": [(1, 16, 12, 1, 1, 0)], "in_features": 16},
        {"layers": [], "in_features": 12}]),
}
BATCH, STEPS = 10, 4


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _blocks(net):
    import oracle as O
    spec = NETS[net]
    return [O.OracleBlock([O.LayerDesc(*l) for l in b["layers"]], in_features=b["in_features"],
                          seed=40 + i, **spec.get("hyper", {}))
            for i, b in enumerate(spec["blocks"])]


def _data(net, step):
    from paper_2407_11698_gb300 import synth
    x = synth.images(17, step, BATCH, NETS[net]["shape"]).reshape(BATCH, -1).astype(np.int64)
    y = synth.labels(17, step, BATCH).astype(np.int64)
    return x, y


def _replica_step(blocks, x, y, exchange, group=None):
    """Forward and backward on (x, y), then (if exchange) the gradient sum,
    status OR and loss over the replicas, then IntegerSGD."""
    import torch
    from paper_2407_11698_gb300 import data_parallel as dp
    acts = [x]
    for b in blocks:
        acts.append(b.forward(acts[-1]))
    for i, b in enumerate(blocks):
        b.backward(acts[i], y)
    losses = []
    for b in blocks:
        if exchange:
            grads = [torch.from_numpy(np.ascontiguousarray(g, dtype=np.int64)) for g in b.dW]
            grads.append(torch.from_numpy(np.ascontiguousarray(b.dWlr, dtype=np.int64)))
            dp.allreduce_grads(grads, group)
            for i in range(len(b.dW)):
                b.dW[i] = grads[i].numpy().reshape(b.dW[i].shape)
            b.dWlr = grads[-1].numpy().reshape(b.dWlr.shape)
            b.status = dp.combine_status(b.status, group)
            losses.append(dp.combine_loss(b.sse, group)[1])
        else:
            losses.append(b.loss)
    for b in blocks:
        b.sgd()
    return losses


def _rank_main(rank, world, port, net, q):
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    from paper_2407_11698_gb300 import data_parallel as dp
    dist.init_process_group("gloo", init_method="tcp://127.0.0.1:%d" % port, rank=rank,
                            world_size=world)
    try:
        blocks = _blocks(net)
        lo, hi = dp.shard(BATCH, rank, world)
        losses = []
        for s in range(STEPS):
            x, y = _data(net, s)
            losses.append(_replica_step(blocks, x[lo:hi], y[lo:hi], True))
        q.put((rank, losses, [[w.copy() for w in b.W] + [b.Wlr.copy()] for b in blocks],
               [b.status for b in blocks]))
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("net", sorted(NETS))
def test_two_replicas_on_half_batches_match_one_replica_on_the_whole_batch(net):
    import torch.multiprocessing as mp
    sys.path.insert(0, ROOT)
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, net, q)) for r in range(2)]
    for p in procs:
        p.start()
    got = sorted((q.get(timeout=300) for _ in procs), key=lambda t: t[0])
    for p in procs:
        p.join(60)
        assert p.exitcode == 0
    # one replica, whole batch
    ref = _blocks(net)
    ref_losses = []
    for s in range(STEPS):
        x, y = _data(net, s)
        ref_losses.append(_replica_step(ref, x, y, False))
    ref_w = [[w for w in b.W] + [b.Wlr] for b in ref]
    for rank, losses, weights, status in got:
        assert losses == ref_losses, "rank %d losses" % rank
        assert status == [b.status for b in ref]
        for bw, rw in zip(weights, ref_w):
            for w, r in zip(bw, rw):
                assert np.array_equal(w, r), "rank %d weights differ" % rank
    # the exchange is what makes them equal: a replica that updates from its
    # own half-batch gradient ends elsewhere
    alone = _blocks(net)
    for s in range(STEPS):
        x, y = _data(net, s)
        _replica_step(alone, x[:BATCH // 2], y[:BATCH // 2], False)
    assert any(not np.array_equal(w, r) for b, rb in zip(alone, ref)
               for w, r in zip(b.W + [b.Wlr], rb.W + [rb.Wlr]))


def test_floor_comes_after_the_sum():
    # Algorithm 1 on the summed gradient differs from summing per-replica updates
    import oracle as O
    w = np.array([100, -7, 0, 5], dtype=np.int64)
    g0 = np.array([300, -300, 511, 1], dtype=np.int64)
    g1 = np.array([300, -300, 1, 511], dtype=np.int64)
    once = O.integersgd(w, g0 + g1, 512, 0)
    twice = w - (w - O.integersgd(w, g0, 512, 0)) - (w - O.integersgd(w, g1, 512, 0))
    assert not np.array_equal(once, twice)
    assert once.tolist() == [99, -5, -1, 4]


def test_shard_split_and_single_replica_helpers():
    sys.path.insert(0, ROOT)
    import torch
    from paper_2407_11698_gb300 import data_parallel as dp
    assert [dp.shard(10, r, 3) for r in range(3)] == [(0, 4), (4, 7), (7, 10)]
    assert [dp.shard(4, r, 2) for r in range(2)] == [(0, 2), (2, 4)]
    assert dp.shard(2, 2, 3) == (2, 2)
    # one replica: no process group needed, nothing changes
    g = torch.tensor([5, -3], dtype=torch.int64)
    assert dp.allreduce_grads([g])[0].tolist() == [5, -3]
    assert dp.combine_status(3) == 3
    assert dp.combine_loss(7) == (7, 3)
    assert dp.combine_loss(-7) == (-7, -4)
    assert dp.combine_loss(2**64 - 2) == (-2, -1)     # SSE kept modulo 2^64
