"""The data-parallel exchange point on the GPU library (one replica, GPU).

The gradient views that the exchange step reduces are the block's own int64
gradients: after the backward they equal the tensors the block reports, and
what is written into them is what IntegerSGD applies.  With one replica the
data-parallel step is the plain block step, bit-exact with the oracle.
"""
import numpy as np
import pytest

import oracle as O
from paper_2407_11698_gb300 import binding as nb
from paper_2407_11698_gb300 import data_parallel as dp
from paper_2407_11698_gb300 import synth

from netpair import NetPair

pytestmark = pytest.mark.gpu

C, L = nb.NITRO_CONV3X3, nb.NITRO_LINEAR
BLOCKS = [{"layers": [(C, 4, 64, 16, 16, 1), (C, 64, 64, 8, 8, 0)], "in_features": 16 * 16 * 4},
          {"layers": [(L, 8 * 8 * 64, 32, 1, 1, 0)], "in_features": 8 * 8 * 64},
          {"layers": [], "in_features": 32}]


@pytest.fixture(scope="module")
def torch():
    t = pytest.importorskip("torch")
    if not t.cuda.is_available():
        pytest.skip("no CUDA device")
    nb.lib()
    return t


def test_gradient_views_are_what_integersgd_applies(torch):
    B = 6
    pair = NetPair(BLOCKS, B, seed=21)
    try:
        x = synth.images(4, 0, B, (16, 16, 4))
        y = synth.labels(4, 0, B)
        xs = torch.from_numpy(x).cuda().reshape(B, -1)
        ys = torch.from_numpy(y.astype(np.int32)).cuda()
        acts = [xs]
        for g in pair.gb:
            out = torch.empty((B, g.out_features), dtype=torch.int8, device="cuda") if g.layers else None
            g.forward(acts[-1], out)
            acts.append(out if out is not None else acts[-1])
        for i, g in enumerate(pair.gb):
            g.backward(acts[i], ys, None)
        oacts = [x.astype(np.int64)]
        for o in pair.ob:
            oacts.append(o.forward(oacts[-1]))
        for i, o in enumerate(pair.ob):
            o.backward(oacts[i], y.astype(np.int64))
        for g, o in zip(pair.gb, pair.ob):
            for i in range(len(g.layers)):
                v = g.grad_device(nb.NITRO_T_DW, i)
                torch.cuda.synchronize()
                assert np.array_equal(v.cpu().numpy(), g.get(nb.NITRO_T_DW, i, check=False))
                assert np.array_equal(v.cpu().numpy(), np.asarray(o.dW[i]).reshape(-1))
                # an exchange step writes the summed gradient here: stand in
                # for a second replica with the same gradient
                v.mul_(2)
                o.dW[i] = o.dW[i] * 2
            v = g.grad_device(nb.NITRO_T_DWLR, 0)
            v.mul_(2)
            o.dWlr = o.dWlr * 2
        torch.cuda.synchronize()
        for g, o in zip(pair.gb, pair.ob):
            g.sgd()
            o.sgd()
        pair.compare("after the doubled update")
    finally:
        pair.close()


def test_one_replica_data_parallel_step_is_the_block_step(torch):
    B = 5
    pair = NetPair(BLOCKS, B, seed=33)
    try:
        net = dp.DataParallelNet(pair.gb)
        for s in range(3):
            x = synth.images(6, s, B, (16, 16, 4))
            y = synth.labels(6, s, B)
            losses = torch.zeros(len(pair.gb), dtype=torch.int64, device="cuda")
            net.step(torch.from_numpy(x).cuda().reshape(B, -1),
                     torch.from_numpy(y.astype(np.int32)).cuda(), losses)
            torch.cuda.synchronize()
            ol = O.train_step(pair.ob, x.astype(np.int64), y.astype(np.int64))
            assert losses.cpu().tolist() == ol
            pair.compare("step %d" % s)
    finally:
        pair.close()


def test_gradient_view_rejects_other_tensors(torch):
    blk = nb.Block([(L, 16, 8, 1, 1, 0)], 16, seed=1, max_batch=2)
    try:
        for which, layer in ((nb.NITRO_T_W, 0), (nb.NITRO_T_DW, 1), (nb.NITRO_T_DWLR, 1),
                             (nb.NITRO_T_ACT, 0)):
            with pytest.raises(nb.NitroError):
                blk.grad_device(which, layer)
        assert blk.grad_device(nb.NITRO_T_DW, 0).numel() == 16 * 8
        assert blk.grad_device(nb.NITRO_T_DWLR, 0).numel() == 10 * 8
    finally:
        blk.close()
