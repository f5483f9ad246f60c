"""Bit-exact parity of learning-layer pooling and linear-block dropout with the
CPU oracle, through the C-ABI (GPU).

Learning-layer pooling: the block output is max-pooled to at most d_lr
features before the learning layer (Sec. 3.3 z^mp; App. B d^lr = 4096).
Dropout: the outputs of linear forward layers are dropped at rate
dropout_p16 / 2^16 (App. B p_l), with masks from the block's SplitMix64
stream indexed by the device-side step counter.  Every exposed tensor,
including the pooled learning input, its window positions and the step
counter, must equal the oracle's after every step.
"""
import numpy as np
import pytest

from paper_2407_11698_gb300 import binding as nb
from paper_2407_11698_gb300 import synth
from paper_2407_11698_gb300 import workloads as WL

from netpair import NetPair, run_workload

pytestmark = pytest.mark.gpu

C, L = nb.NITRO_CONV3X3, nb.NITRO_LINEAR


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    nb.lib()


def _b(layers, in_features):
    return {"layers": layers, "in_features": in_features}


def _run(blocks, batch, steps, input_shape, **hyper):
    pair = NetPair(blocks, batch, **hyper)
    try:
        for s in range(steps):
            x = synth.images(9, s, batch, input_shape)
            y = synth.labels(9, s, batch, hyper.get("num_classes", 10))
            gl, ol = pair.step(x, y)
            assert gl == ol, "step %d losses gpu %s oracle %s" % (s, gl, ol)
            pair.compare("step %d" % s)
        return pair
    finally:
        pair.close()


# ------------------------------------------------------- learning-layer pooling
def test_vgg_blocks_pool_learning_input_to_4096():
    # App. B's d^lr = 4096 on the VGG-style network: block 1 (64 x 16 x 16)
    # pools 2 x 2, block 2 (128 x 8 x 8) 2 x 1, block 3 (256 x 4 x 4) none
    run_workload(WL.WORKLOADS["vgg_64_128_256_b128"], steps=3, batch=16, d_lr=4096)


def test_cnn_blocks_pool_with_ragged_windows():
    # d_lr = 1000: block 1 (32 x 14 x 14) takes 4 x 2 windows and drops two
    # rows; block 2 (64 x 7 x 7) 2 x 2 and drops a row and a column
    run_workload(WL.WORKLOADS["cnn_32_64_b64"], steps=4, batch=24, d_lr=1000)


def test_last_layer_without_pool_and_ragged_map():
    # a conv output that is not 2x2-pooled feeds the learning pool directly;
    # 10 x 10 maps leave partial windows
    blocks = [_b([(C, 3, 8, 10, 10, 0)], 10 * 10 * 3), _b([], 10 * 10 * 8)]
    _run(blocks, 5, steps=3, input_shape=(10, 10, 3), d_lr=100)
    blocks = [_b([(C, 3, 16, 8, 8, 0)], 8 * 8 * 3), _b([], 8 * 8 * 16)]
    _run(blocks, 4, steps=2, input_shape=(8, 8, 3), d_lr=64)
    # six channels: the one-channel-per-thread routing kernel
    blocks = [_b([(C, 3, 6, 8, 8, 1)], 8 * 8 * 3), _b([], 4 * 4 * 6)]
    _run(blocks, 5, steps=2, input_shape=(8, 8, 3), d_lr=20)


def test_pooled_tensor_core_layers_and_many_classes():
    # 32-channel layers on the tensor-core path, G = 20 (the unfused
    # learning-weight gradient), a learning pool of 4 x 4 windows
    blocks = [_b([(C, 3, 32, 16, 16, 0), (C, 32, 32, 16, 16, 1)], 16 * 16 * 3),
              _b([], 8 * 8 * 32)]
    _run(blocks, 8, steps=3, input_shape=(16, 16, 3), d_lr=128, num_classes=20)


def test_learning_pool_with_thirteen_classes():
    # G = 13: the routing kernel's batched loads for up to 16 classes (G = 10
    # and G = 20 take the other two forms above)
    blocks = [_b([(C, 3, 16, 16, 16, 1)], 16 * 16 * 3), _b([], 8 * 8 * 16)]
    _run(blocks, 6, steps=3, input_shape=(16, 16, 3), d_lr=256, num_classes=13)


def test_pooled_block_exposes_window_geometry():
    blk = nb.Block([(C, 4, 16, 16, 16, 1)], 16 * 16 * 4, seed=3, max_batch=2, d_lr=256)
    plain = nb.Block([(C, 4, 16, 16, 16, 1)], 16 * 16 * 4, seed=3, max_batch=2)
    try:
        # 16 x 8 x 8 = 1024 -> 2 x 1 -> 2 x 2: 16 x 4 x 4 = 256 learning inputs
        assert blk.get(nb.NITRO_T_WLR, 0).size == 10 * 256
        # a block without learning-layer pooling has no pooled input to read
        with pytest.raises(nb.NitroError):
            plain.get(nb.NITRO_T_LR_IN)
    finally:
        blk.close()
        plain.close()


# ------------------------------------------------------- dropout
def test_mlp_dropout_fifteen_percent():
    # p_l = 0.15 (App. B, VGG8B on CIFAR-10) on every linear block of the MLP
    run_workload(WL.WORKLOADS["mlp_784_100_50_10_b64"], steps=12, check_every=3,
                 dropout_p16=9830)


def test_dropout_all_and_none():
    blocks = [_b([(L, 40, 24, 1, 1, 0), (L, 24, 16, 1, 1, 0)], 40), _b([], 16)]
    _run(blocks, 7, steps=2, input_shape=(40,), dropout_p16=65536)
    _run(blocks, 7, steps=2, input_shape=(40,), dropout_p16=1)


def test_dropout_rate_change_and_step_counter_resume():
    blocks = [_b([(L, 30, 20, 1, 1, 0)], 30), _b([], 20)]
    a = NetPair(blocks, 6, seed=21, dropout_p16=20000)
    b = NetPair(blocks, 6, seed=21, dropout_p16=20000)
    try:
        for s in range(3):
            x, y = synth.images(8, s, 6, (30,)), synth.labels(8, s, 6)
            gl, ol = a.step(x, y)
            assert gl == ol
        a.compare("before resume")
        # b resumes from a's state: weights and the step counter of the masks
        for ga, gb_, oa, ob in zip(a.gb, b.gb, a.ob, b.ob):
            for i in range(len(oa.layers)):
                gb_.set(nb.NITRO_T_W, i, ga.get(nb.NITRO_T_W, i))
                ob.W[i] = oa.W[i].copy()
            gb_.set(nb.NITRO_T_WLR, 0, ga.get(nb.NITRO_T_WLR, 0))
            ob.Wlr = oa.Wlr.copy()
            gb_.set(nb.NITRO_T_STEP, 0, ga.get(nb.NITRO_T_STEP, 0))
            ob.t = oa.t
        for s in range(3, 5):
            x, y = synth.images(8, s, 6, (30,)), synth.labels(8, s, 6)
            la, _ = a.step(x, y)
            lb, ol = b.step(x, y)
            assert la == lb == ol
        b.compare("after resume")
        # a rate change between steps (e.g. 0 for inference) takes effect at
        # the next forward on both sides
        for g, o in zip(b.gb, b.ob):
            g.set_dropout(0)
            o.dropout_p16 = 0
        x, y = synth.images(8, 5, 6, (30,)), synth.labels(8, 5, 6)
        gl, ol = b.step(x, y)
        assert gl == ol
        b.compare("rate 0")
        assert not np.any(b.gb[0].get(nb.NITRO_T_REGION, 0) == 4)
        with pytest.raises(nb.NitroError):
            b.gb[0].set_dropout(65537)
    finally:
        a.close()
        b.close()


def test_dropout_masks_advance_across_cuda_graph_replays():
    # the step counter lives on the device: replays of one captured step draw
    # a fresh mask each time, like the oracle's successive steps
    torch = pytest.importorskip("torch")
    blocks = [_b([(L, 48, 32, 1, 1, 0)], 48), _b([], 32)]
    B = 8
    pair = NetPair(blocks, B, seed=13, dropout_p16=16384)
    try:
        x = synth.images(6, 0, B, (48,))
        y = synth.labels(6, 0, B)
        xs = torch.from_numpy(x).cuda().reshape(B, -1)
        ys = torch.from_numpy(y.astype(np.int32)).cuda()
        a1 = torch.empty((B, 32), dtype=torch.int8, device="cuda")
        losses = [torch.zeros(1, dtype=torch.int64, device="cuda") for _ in pair.gb]

        def step():
            pair.gb[0].forward(xs, a1)
            pair.gb[1].forward(a1, None)
            pair.gb[0].backward(xs, ys, losses[0])
            pair.gb[1].backward(a1, ys, losses[1])
            for g in pair.gb:
                g.sgd()

        step()                                   # eager step 0
        torch.cuda.synchronize()
        assert [int(l.item()) for l in losses] == pair.step_oracle(x, y)
        side = torch.cuda.Stream()
        side.wait_stream(torch.cuda.current_stream())
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.stream(side):
            with torch.cuda.graph(graph, stream=side):
                step()
        torch.cuda.current_stream().wait_stream(side)
        # capture queued nothing: the device state is still after step 0
        for s in range(1, 4):
            graph.replay()
            torch.cuda.synchronize()
            assert [int(l.item()) for l in losses] == pair.step_oracle(x, y), s
            pair.compare("replay %d" % s)
    finally:
        pair.close()


# ------------------------------------------------------- paper-scale networks
@pytest.mark.parametrize("name,batch,steps", [
    ("vgg8b_cifar10_b64", 4, 2), ("vgg11b_cifar10_b64", 2, 2),
    ("mlp3_mnist_b64", 16, 3), ("mlp4_cifar10_b64", 8, 2)])
def test_paper_scale_networks(name, batch, steps):
    # Table 1's VGG8B / VGG11B / MLP3 / MLP4 with App. B's hyper-parameters
    # (d^lr = 4096, weight decay, dropout on the linear blocks)
    run_workload(WL.WORKLOADS[name], steps=steps, batch=batch)
