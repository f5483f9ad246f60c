"""Tensor-core (tcgen05) conv path: bit-exact against the oracle through the
C-ABI on shapes that exercise ragged tiles, batch padding, 1..4 limb operands
and narrow (image-channel) inputs that run as im2col rows.  Every block has two conv layers, so fwd, wgrad and dgrad of the
second layer and the fwd of the first all run on tensor cores when the
channel counts are multiples of 64."""
import numpy as np
import pytest

from paper_2407_11698_gb300 import binding as nb
from paper_2407_11698_gb300 import synth

from netpair import NetPair

pytestmark = pytest.mark.gpu
C = nb.NITRO_CONV3X3


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    nb.lib()


def _two_conv_block(B, h, w, c0, c1, c2, pool, pool_first=False):
    h1, w1 = (h // 2, w // 2) if pool_first else (h, w)
    oh, ow = (h1 // 2, w1 // 2) if pool else (h1, w1)
    return [{"layers": [(C, c0, c1, h, w, int(pool_first)), (C, c1, c2, h1, w1, int(pool))],
             "in_features": h * w * c0},
            {"layers": [], "in_features": oh * ow * c2}]


def _widen(pair, scale):
    """Multiply every forward weight by `scale` on both sides (more limbs)."""
    for g, o in zip(pair.gb, pair.ob):
        for i in range(len(o.layers)):
            w = (o.W[i] * scale).astype(np.int64)
            assert np.abs(w).max() < 2**31
            o.W[i] = w
            g.set(nb.NITRO_T_W, i, w.astype(np.int32))


@pytest.mark.parametrize("B,h,w,c0,c1,c2,pool,scale", [
    (8, 8, 8, 64, 64, 64, True, 1),
    (3, 12, 9, 64, 128, 64, True, 1),          # ragged tiles in x and y, batch pad
    (5, 8, 8, 192, 64, 128, False, 3),         # N = 64 tiles, 2-image pixel tiles
    (8, 16, 16, 64, 128, 128, True, 1000),     # two-limb weights
    (4, 8, 8, 64, 64, 64, True, 70001),        # three-limb weights
    (4, 8, 8, 64, 64, 64, False, 2**22),       # four-limb weights
    (130, 8, 16, 64, 64, 64, True, 1),         # batch over 128 (wgrad batch blocks)
    (13, 4, 4, 64, 64, 128, True, 1),          # 4 x 4 maps: 8-image forward tiles, ragged batch
    (9, 4, 4, 128, 128, 64, False, 70001),     # 4 x 4 maps, three-limb weights, N = 64 tiles
])
def test_two_conv_block_parity(B, h, w, c0, c1, c2, pool, scale):
    _run_two_conv(B, h, w, c0, c1, c2, pool, scale, False)


@pytest.mark.parametrize("B,h,w,c0,c1,c2,pool,scale", [
    (4, 16, 16, 64, 64, 64, False, 1),         # pooled lower layer: dgrad routes to argmax
    (3, 17, 18, 64, 128, 64, True, 300),       # odd pooled lower layer (dropped row)
    (5, 16, 32, 64, 64, 128, False, 70001),    # wide weights through the pooled path
])
def test_two_conv_block_pooled_lower_layer(B, h, w, c0, c1, c2, pool, scale):
    _run_two_conv(B, h, w, c0, c1, c2, pool, scale, True)


@pytest.mark.parametrize("B,h,w,c0,c1,c2,pool,scale", [
    (8, 8, 8, 3, 64, 64, True, 1),             # image channels: im2col rows on tcgen05
    (3, 12, 9, 1, 16, 64, False, 1),           # one input channel, 16 outputs (ragged N tile)
    (5, 16, 16, 7, 128, 64, True, 300),        # 63 of the 64 im2col entries, two-limb weights
    (4, 10, 12, 5, 48, 64, False, 70001),      # 48 outputs, three-limb weights
    (130, 8, 16, 3, 64, 64, True, 2**22),      # batch over 128, four-limb weights
])
def test_narrow_input_first_layer(B, h, w, c0, c1, c2, pool, scale):
    _run_two_conv(B, h, w, c0, c1, c2, pool, scale, False)


def _run_two_conv(B, h, w, c0, c1, c2, pool, scale, pool_first):
    blocks = _two_conv_block(B, h, w, c0, c1, c2, pool, pool_first)
    pair = NetPair(blocks, B, seed=31)
    try:
        if scale != 1:
            _widen(pair, scale)
        for s in range(3):
            x = synth.images(13, s, B, (h, w, c0))
            y = synth.labels(13, s, B)
            gl, ol = pair.step(x, y)
            assert gl == ol, (s, gl, ol)
            pair.compare("step %d" % s)
    finally:
        pair.close()


@pytest.mark.parametrize("c0", [64, 3])
def test_tensor_core_kernels_ran(c0):
    """The tc kernels are the ones launched for a 64-channel layer and for a
    3-channel (image) layer."""
    torch = pytest.importorskip("torch")
    import ctypes
    L = nb.lib()
    blocks = _two_conv_block(8, 8, 8, c0, 64, 64, True)
    pair = NetPair(blocks, 8, seed=2)
    try:
        L.nitro_profile_reset()
        L.nitro_profile_enable(1)
        pair.step_gpu(synth.images(1, 0, 8, (8, 8, c0)), synth.labels(1, 0, 8))
        L.nitro_profile_enable(0)
        names = {}
        for k in range(L.nitro_profile_kernel_count()):
            n, ms, ops, by = ctypes.c_uint64(), ctypes.c_double(), ctypes.c_double(), ctypes.c_double()
            L.nitro_profile_read(k, ctypes.byref(n), ctypes.byref(ms), ctypes.byref(ops), ctypes.byref(by))
            names[L.nitro_profile_kernel_name(k).decode()] = n.value
        L.nitro_profile_reset()
        assert names["tc_conv_fwd"] == 2 and names["tc_conv_wgrad"] == 2 and names["tc_conv_dgrad"] == 1
        assert names["simt_conv_fwd"] == 0 and names["simt_conv_wgrad"] == 0
    finally:
        pair.close()


def test_linear_tensor_core_weights_from_a_checkpoint():
    """Weights written through set_tensor reach the tensor-core linear forward
    (input width a multiple of 8): the layer's limb planes are rebuilt from the
    new int32 weights, here widened to three limbs on both sides."""
    blocks = [{"layers": [(nb.NITRO_LINEAR, 136, 64, 1, 1, 0)], "in_features": 136},
              {"layers": [], "in_features": 64}]
    pair = NetPair(blocks, 12, seed=8)
    try:
        x, y = synth.images(21, 0, 12, (136,)), synth.labels(21, 0, 12)
        gl, ol = pair.step(x, y)
        assert gl == ol
        _widen(pair, 70001)      # max |W| 21 after one step -> 1.47e6: three limbs
        for s in range(1, 3):
            x, y = synth.images(21, s, 12, (136,)), synth.labels(21, s, 12)
            gl, ol = pair.step(x, y)
            assert gl == ol, (s, gl, ol)
            pair.compare("step %d" % s)
    finally:
        pair.close()
