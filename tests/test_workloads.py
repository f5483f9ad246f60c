"""The synthetic workloads have the shapes they stand for (CPU).

Each of the five workloads is checked against its stated structure: input
shape, batch, steps, the layers of every block and the chain of flattened
sizes between blocks (through the oracle's own layer arithmetic), with G = 10
classes and, for the networks, an output block at the end.
"""
import numpy as np

import oracle as O
from paper_2407_11698_gb300 import workloads as WL


def _chain(wl, output_block=True):
    blocks = [O.OracleBlock([O.LayerDesc(*l) for l in b["layers"]], in_features=b["in_features"],
                            seed=i, **wl.get("hyper", {}))
              for i, b in enumerate(wl["blocks"])]
    in_f = int(np.prod(wl["input_shape"]))
    for blk in blocks:
        assert blk.in_features == in_f
        if blk.layers:
            in_f = blk.layers[-1].out_features
    assert all(blk.G == 10 for blk in blocks)
    assert (blocks[-1].layers == []) == output_block
    return blocks


def _convs(wl):
    return [(l[1], l[2], l[3], bool(l[5])) for b in wl["blocks"] for l in b["layers"]]


def test_single_conv_block():
    wl = WL.WORKLOADS["conv1_b16"]
    assert wl["batch"] == 16 and wl["steps"] == 3 and wl["input_shape"] == (28, 28, 1)
    assert _convs(wl) == [(1, 32, 28, True)]
    blocks = _chain(wl, output_block=False)  # one block: its learning layer classifies
    assert len(blocks) == 1 and blocks[0].d == 14 * 14 * 32


def test_mlp_784_100_50_10():
    wl = WL.WORKLOADS["mlp_784_100_50_10_b64"]
    assert wl["batch"] == 64 and wl["steps"] == 100
    widths = [b["layers"][0][1:3] for b in wl["blocks"] if b["layers"]]
    assert widths == [(784, 100), (100, 50)]
    assert _chain(wl)[-1].in_features == 50


def test_cnn_32_64():
    wl = WL.WORKLOADS["cnn_32_64_b64"]
    assert wl["batch"] == 64 and wl["steps"] == 100 and wl["input_shape"] == (28, 28, 1)
    assert _convs(wl) == [(1, 32, 28, True), (32, 64, 14, True)]
    assert _chain(wl)[-1].in_features == 7 * 7 * 64


def test_vgg_64_128_256():
    wl = WL.WORKLOADS["vgg_64_128_256_b128"]
    assert wl["batch"] == 128 and wl["steps"] == 50 and wl["input_shape"] == (32, 32, 3)
    assert _convs(wl) == [(3, 64, 32, False), (64, 64, 32, True), (64, 128, 16, False),
                          (128, 128, 16, True), (128, 256, 8, False), (256, 256, 8, True)]
    assert [len(b["layers"]) for b in wl["blocks"]] == [2, 2, 2, 0]
    blocks = _chain(wl)
    assert [b.d for b in blocks] == [16384, 8192, 4096, 4096]


def test_kernel_sweep_shapes():
    assert sorted(set(hw for _, hw, _ in WL.SWEEP_CONV)) == [8, 16, 32]
    assert sorted(set(c for _, _, c in WL.SWEEP_CONV)) == [64, 128, 256, 512]
    assert all(b == 256 for b, _, _ in WL.SWEEP_CONV)
    assert WL.SWEEP_GEMM == [1024, 4096, 8192]
