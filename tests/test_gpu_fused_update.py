"""Backward and IntegerSGD in one call (GPU): nitro_block_backward_update.

The tensor-core weight-gradient kernels apply Algorithm 1 to each output tile
once its sum is final (after the last K split arrives, or straight from the
accumulators without a split).  Every exposed tensor must stay bit-identical
to the oracle's step: weights, weight gradients, deltas, codes, loss and
status, through the growth of the weights to several limbs and into the int32
overflow regime, with decay and both rounding modes.
"""
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


def test_vgg_style_network_fused_update_into_overflow_regime():
    # batch 128: the weight gradients run with K splits (per-slot tickets);
    # deltas leave int32 around step 4
    run_workload(WL.WORKLOADS["vgg_64_128_256_b128"], steps=12, check_every=3, fused_update=True)


def test_vgg_style_network_fused_update_on_block_streams():
    run_workload(WL.WORKLOADS["vgg_64_128_256_b128"], steps=6, check_every=2, fused_update=True,
                 concurrent=True)


def test_cnn_with_narrow_first_layer_fused_update():
    # the 1-channel first conv updates through IntegerSGD, the 32 -> 64 conv in
    # its weight-gradient kernel
    run_workload(WL.WORKLOADS["cnn_32_64_b64"], steps=20, check_every=5, fused_update=True)


def _run(blocks, batch, steps, shape, **hyper):
    pair = NetPair(blocks, batch, fused_update=True, **hyper)
    try:
        for s in range(steps):
            x = synth.images(23, s, batch, shape)
            y = synth.labels(23, s, batch)
            gl, ol = pair.step(x, y)
            assert gl == ol
            pair.compare("step %d" % s)
    finally:
        pair.close()


@pytest.mark.parametrize("sgd_round", [nb.NITRO_ROUND_FLOOR, nb.NITRO_ROUND_TRUNC])
def test_fused_update_with_decay_and_rounding(sgd_round):
    blocks = [{"layers": [(C, 8, 64, 16, 16, 1), (C, 64, 40, 8, 8, 0)], "in_features": 16 * 16 * 8},
              {"layers": [], "in_features": 8 * 8 * 40}]
    _run(blocks, 6, 4, (16, 16, 8), eta_inv_fw=25000, eta_inv_lr=3000, sgd_round=sgd_round)


def test_fused_update_without_k_split_and_ragged_channels():
    # batch 2 on 8x8 maps: one K split per tile, the update from the
    # accumulators; 40 output channels leave part of the last column tile empty
    blocks = [{"layers": [(C, 64, 64, 8, 8, 0), (C, 64, 40, 8, 8, 1)], "in_features": 8 * 8 * 64},
              {"layers": [(L, 4 * 4 * 40, 16, 1, 1, 0)], "in_features": 4 * 4 * 40},
              {"layers": [], "in_features": 16}]
    _run(blocks, 2, 4, (8, 8, 64))


def test_fused_and_separate_calls_interleave():
    # tickets return to zero after every launch: alternate the two call forms
    blocks = [{"layers": [(C, 32, 64, 16, 16, 0), (C, 64, 64, 16, 16, 1)], "in_features": 16 * 16 * 32},
              {"layers": [], "in_features": 8 * 8 * 64}]
    pair = NetPair(blocks, 16)
    try:
        for s in range(6):
            pair.fused_update = s % 2 == 0
            x = synth.images(29, s, 16, (16, 16, 32))
            y = synth.labels(29, s, 16)
            gl, ol = pair.step(x, y)
            assert gl == ol
            pair.compare("step %d" % s)
    finally:
        pair.close()
