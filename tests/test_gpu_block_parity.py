"""Bit-exact parity of the GPU library with the CPU oracle, through the C-ABI.

Every exposed tensor (weights, weight gradients, activations, ReLU region and
pool argmax codes, deltas, loss gradient, SSE, loss, status bits) must be equal
after every training step.
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


# ---------------------------------------------------------------- workloads
def test_conv1_b16_three_steps():
    run_workload(WL.WORKLOADS["conv1_b16"], steps=3)


def test_mlp_784_100_50_10_b64_100_steps():
    run_workload(WL.WORKLOADS["mlp_784_100_50_10_b64"], steps=100, check_every=10)


def test_cnn_32_64_b64_100_steps():
    run_workload(WL.WORKLOADS["cnn_32_64_b64"], steps=100, check_every=25)


def test_vgg_64_128_256_b128_50_steps():
    # Full-size VGG-style network for all 50 steps of the workload: the first
    # step drives the first conv of each block to multi-limb weights (|W| ~
    # 1e6) and deltas (~7e5); around step 4 deltas leave int32 (OVERFLOW on
    # both sides, identical wrap), so later steps run with four-limb operands.
    run_workload(WL.WORKLOADS["vgg_64_128_256_b128"], steps=50, check_every=5)


def test_blocks_on_their_own_streams():
    # blocks share no gradients (Sec. 3.3): with a stream per block, block i's
    # backward and update overlap the forward of the blocks after it; the
    # results stay bit-identical to the oracle, through the first steps of limb
    # growth and into the int32 overflow regime of the VGG-style network
    run_workload(WL.WORKLOADS["cnn_32_64_b64"], steps=20, check_every=5, concurrent=True)
    run_workload(WL.WORKLOADS["vgg_64_128_256_b128"], steps=8, check_every=2, concurrent=True)


# ---------------------------------------------------------------- edge cases
def _run(blocks, batch, steps=2, input_shape=None, **hyper):
    pair = NetPair(blocks, batch, **hyper)
    try:
        for s in range(steps):
            x = synth.images(3, s, batch, input_shape or (blocks[0]["in_features"],))
            y = synth.labels(3, s, batch, hyper.get("num_classes", 10))
            gl, ol = pair.step(x, y)
            assert gl == ol
            pair.compare("step %d" % s)
    finally:
        pair.close()


def _b(layers, in_features):
    return {"layers": layers, "in_features": in_features}


def test_ragged_conv_shapes_odd_pool():
    # 7x5 input, odd pool (drops the last row), Cin/Cout not multiples of anything
    blocks = [_b([(C, 5, 7, 7, 5, 1), (C, 7, 3, 3, 2, 0)], 7 * 5 * 5), _b([], 3 * 2 * 3)]
    _run(blocks, 3, steps=3, input_shape=(7, 5, 5))


def test_conv_then_linear_in_one_block():
    blocks = [_b([(C, 3, 8, 6, 6, 1), (L, 3 * 3 * 8, 12, 1, 1, 0)], 6 * 6 * 3), _b([], 12)]
    _run(blocks, 5, steps=3, input_shape=(6, 6, 3))


def test_linear_layers_on_tensor_cores():
    # input widths that are multiples of 8 run the forward on the tcgen05 GEMM:
    # three row tiles (batch 257), a ragged column tile, a K split (3000-wide
    # input against few output tiles), weight decay and dropout on top
    blocks = [_b([(L, 136, 200, 1, 1, 0), (L, 200, 72, 1, 1, 0)], 136), _b([], 72)]
    _run(blocks, 257, steps=3, eta_inv_fw=25000, eta_inv_lr=3000, dropout_p16=6554)
    blocks = [_b([(L, 3000, 40, 1, 1, 0)], 3000), _b([], 40)]
    _run(blocks, 20, steps=3)


def test_batch_of_one_and_max_batch():
    blocks = [_b([(L, 20, 9, 1, 1, 0)], 20)]
    _run(blocks, 1, steps=2)
    _run(blocks, 257, steps=2)


def test_trunc_rounding_with_weight_decay_and_other_alpha():
    blocks = [_b([(C, 2, 6, 8, 8, 1)], 8 * 8 * 2), _b([], 4 * 4 * 6)]
    for alpha in (4, 100):
        _run(blocks, 6, steps=3, input_shape=(8, 8, 2), alpha_inv=alpha, sgd_round=nb.NITRO_ROUND_TRUNC,
             eta_inv_fw=25000, eta_inv_lr=3000)
    _run(blocks, 6, steps=3, input_shape=(8, 8, 2), eta_inv_fw=25000, eta_inv_lr=3000)


def test_gamma_plateau_schedule_changes_updates_like_oracle():
    """App. B schedule: gamma_inv x3 on a plateau, pushed through
    nitro_block_set_hyper between steps; the oracle blocks take the same
    values.  Weight decay switched on at the same time."""
    from paper_2407_11698_gb300.schedule import GammaPlateau
    blocks = [_b([(C, 2, 8, 8, 8, 1)], 8 * 8 * 2), _b([], 4 * 4 * 8)]
    pair = NetPair(blocks, 6, seed=77)
    sched = GammaPlateau(512, patience=1)
    try:
        for s in range(6):
            x = synth.images(5, s, 6, (8, 8, 2))
            y = synth.labels(5, s, 6)
            gl, ol = pair.step(x, y)
            assert gl == ol
            pair.compare("step %d" % s)
            if sched.step(0.5):                # a flat metric: every call past the first raises
                sched.apply(pair.gb, eta_inv_fw=25000, eta_inv_lr=3000)
                for o in pair.ob:
                    o.gamma_inv_lr = sched.gamma_inv
                    o.eta_inv_fw, o.eta_inv_lr = 25000, 3000
        assert sched.gamma_inv == 512 * 3 ** 5
        with pytest.raises(nb.NitroError):
            pair.gb[0].set_hyper(0)
    finally:
        pair.close()


def test_other_class_counts():
    blocks = [_b([(L, 16, 8, 1, 1, 0)], 16), _b([], 8)]
    _run(blocks, 9, steps=3, num_classes=3)
    _run(blocks, 9, steps=2, num_classes=16)     # widest fused learning-layer backward
    _run(blocks, 9, steps=2, num_classes=40)


def test_empty_batch():
    torch = pytest.importorskip("torch")
    blk = nb.Block([(C, 1, 4, 4, 4, 1)], 16, seed=1, max_batch=4)
    w0 = blk.get(nb.NITRO_T_W, 0)
    x = torch.empty((0, 16), dtype=torch.int8, device="cuda")
    y = torch.empty((0,), dtype=torch.int32, device="cuda")
    loss = torch.full((1,), 5, dtype=torch.int64, device="cuda")
    blk.forward(x, None)
    blk.backward(x, y, loss)
    blk.sgd()
    assert int(loss.item()) == 0
    assert np.array_equal(blk.get(nb.NITRO_T_W, 0), w0)
    assert not np.any(blk.get(nb.NITRO_T_DW, 0))
    assert blk.status() == nb.NITRO_OK
    blk.close()


def test_batch_above_max_is_rejected():
    torch = pytest.importorskip("torch")
    blk = nb.Block([(L, 8, 4, 1, 1, 0)], 8, seed=1, max_batch=2)
    x = torch.zeros((3, 8), dtype=torch.int8, device="cuda")
    assert nb.nitro_block_forward(blk.h, nb._ptr(x), 3, None) == nb.NITRO_ERR_ARG
    # backward must follow a forward of the same batch
    assert nb.nitro_block_backward(blk.h, nb._ptr(x), nb._ptr(x), 1, None) == nb.NITRO_ERR_ARG
    blk.close()


def test_bad_label_sets_status_like_oracle():
    torch = pytest.importorskip("torch")
    blocks = [_b([(L, 8, 4, 1, 1, 0)], 8)]
    pair = NetPair(blocks, 3)
    try:
        x = synth.images(1, 0, 3, (8,))
        y = np.array([1, 10, -1], dtype=np.int32)
        pair.step(x, y)
        pair.compare()
        assert pair.gb[0].status() == nb.NITRO_ERR_ARG
        assert pair.gb[0].status(clear=True) == nb.NITRO_ERR_ARG
        assert pair.gb[0].status() == nb.NITRO_OK
    finally:
        pair.close()


def test_overflow_is_flagged_like_oracle():
    # learning weights of 2^29 make delta_fw leave int32; a forward weight at
    # the int32 edge leaves it on update.  Both sides flag and wrap alike.
    blocks = [_b([(L, 8, 4, 1, 1, 0)], 8)]
    pair = NetPair(blocks, 3)
    try:
        wlr = np.full((10, 4), 2**29, dtype=np.int64)
        pair.ob[0].Wlr = wlr.copy()
        pair.gb[0].set(nb.NITRO_T_WLR, 0, wlr)
        x = synth.images(2, 0, 3, (8,))
        y = synth.labels(2, 0, 3)
        pair.step(x, y)
        pair.compare()
        assert pair.gb[0].status() == nb.NITRO_ERR_OVERFLOW
    finally:
        pair.close()


def test_checkpoint_resume_is_bit_exact():
    blocks = [_b([(C, 1, 8, 8, 8, 1)], 64), _b([], 4 * 4 * 8)]
    a = NetPair(blocks, 4, seed=5)
    b = NetPair(blocks, 4, seed=99)
    try:
        for s in range(2):
            a.step(synth.images(4, s, 4, (8, 8, 1)), synth.labels(4, s, 4))
        # copy every weight tensor of a into b (GPU and oracle sides)
        for ga, gb_, oa, ob in zip(a.gb, b.gb, a.ob, b.ob):
            for i in range(len(oa.layers)):
                gb_.set(nb.NITRO_T_W, i, ga.get(nb.NITRO_T_W, i))
                ob.W[i] = oa.W[i].copy()
            gb_.set(nb.NITRO_T_WLR, 0, ga.get(nb.NITRO_T_WLR, 0))
            ob.Wlr = oa.Wlr.copy()
            gb_.set(nb.NITRO_T_STEP, 0, ga.get(nb.NITRO_T_STEP, 0))
            ob.t = oa.t
        for s in range(2, 4):
            x, y = synth.images(4, s, 4, (8, 8, 1)), synth.labels(4, s, 4)
            la, _ = a.step(x, y)
            lb, _ = b.step(x, y)
            assert la == lb
        for ga, gb_ in zip(a.gb, b.gb):
            assert np.array_equal(ga.get(nb.NITRO_T_WLR, 0), gb_.get(nb.NITRO_T_WLR, 0))
        b.compare()
    finally:
        a.close()
        b.close()
