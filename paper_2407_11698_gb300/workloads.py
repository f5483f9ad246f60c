"""The five synthetic workloads, as lists of blocks.

A layer is ``(kind, cin, cout, h, w, pool)`` with kind 0 = 3x3 conv (stride 1,
pad 1) and 1 = linear; ``h``/``w`` are the layer's input size (1 for linear).
A block is ``{"layers": [...], "in_features": n}``; a block with no layers is
the network's output block.  Shapes follow Table 1 of the paper (MLP widths,
VGG-style 3x3 conv stacks with 2x2 max-pool) at the sizes of the datasets of
Sec. 4 (28x28x1, 32x32x3, G = 10).
"""

CONV, LINEAR = 0, 1


def _conv(cin, cout, hw, pool):
    return (CONV, cin, cout, hw, hw, bool(pool))


def _lin(cin, cout):
    return (LINEAR, cin, cout, 1, 1, False)


def _blk(layers, in_features):
    return {"layers": list(layers), "in_features": int(in_features)}


WORKLOADS = {
    # 1 conv local-loss block 1->32 @ 28x28 with max-pool, batch 16, 3 steps
    "conv1_b16": dict(
        input_shape=(28, 28, 1), batch=16, steps=3,
        blocks=[_blk([_conv(1, 32, 28, True)], 784)]),
    # MLP 784-100-50-10: two linear local-loss blocks and an output block
    "mlp_784_100_50_10_b64": dict(
        input_shape=(28, 28, 1), batch=64, steps=100,
        blocks=[_blk([_lin(784, 100)], 784), _blk([_lin(100, 50)], 100), _blk([], 50)]),
    # CNN: conv 1->32 @28 pool, conv 32->64 @14 pool, output block 3136->10
    "cnn_32_64_b64": dict(
        input_shape=(28, 28, 1), batch=64, steps=100,
        blocks=[_blk([_conv(1, 32, 28, True)], 784),
                _blk([_conv(32, 64, 14, True)], 14 * 14 * 32),
                _blk([], 7 * 7 * 64)]),
    # VGG-style: 3 blocks of two 3x3 convs (64, 128, 256) + pool, output block
    "vgg_64_128_256_b128": dict(
        input_shape=(32, 32, 3), batch=128, steps=50,
        blocks=[_blk([_conv(3, 64, 32, False), _conv(64, 64, 32, True)], 32 * 32 * 3),
                _blk([_conv(64, 128, 16, False), _conv(128, 128, 16, True)], 16 * 16 * 64),
                _blk([_conv(128, 256, 8, False), _conv(256, 256, 8, True)], 8 * 8 * 128),
                _blk([], 4 * 4 * 256)]),
}


def _vgg_b(spec, hw, cin):
    # one local-loss block per layer: (cout, pool) convs, then linear widths
    blocks = []
    for cout, pool in spec:
        blocks.append(_blk([_conv(cin, cout, hw, pool)], hw * hw * cin))
        cin, hw = cout, hw // 2 if pool else hw
    return blocks, hw * hw * cin


def _paper_vgg(spec):
    blocks, flat = _vgg_b(spec, 32, 3)
    blocks.append(_blk([_lin(flat, 1024)], flat))
    blocks.append(_blk([], 1024))
    return blocks


def _paper_mlp(widths):
    blocks = [_blk([_lin(a, b)], a) for a, b in zip(widths[:-1], widths[1:])]
    blocks.append(_blk([], widths[-1]))
    return blocks


# Paper-scale networks of Table 1 with the CIFAR-10 / MNIST hyper-parameters
# of App. B (gamma_inv = 512; Table 6's decay rates taken as eta_inv; d^lr;
# the linear blocks' dropout p_l in units of 2^-16).  Every IntConv2D (with the
# MaxPool2D after it) and every hidden IntLinear is a local-loss block.  Batch
# 64 as in App. B.  Used for timing; parity runs them at smaller batches.
PAPER_WORKLOADS = {
    # VGG8B, CIFAR-10: d^lr 4096, lambda 25000 / 3000, p_l = 0.15
    "vgg8b_cifar10_b64": dict(
        input_shape=(32, 32, 3), batch=64, steps=10,
        hyper=dict(d_lr=4096, eta_inv_fw=25000, eta_inv_lr=3000, dropout_p16=9830),
        blocks=_paper_vgg([(128, False), (256, True), (256, False), (512, True), (512, True),
                           (512, True)])),
    # VGG11B, CIFAR-10: d^lr 4096, lambda 28000 / 4500, p_l = 0
    "vgg11b_cifar10_b64": dict(
        input_shape=(32, 32, 3), batch=64, steps=10,
        hyper=dict(d_lr=4096, eta_inv_fw=28000, eta_inv_lr=4500),
        blocks=_paper_vgg([(128, False), (128, False), (128, False), (256, True), (256, False),
                           (512, True), (512, False), (512, True), (512, True)])),
    # MLP3, MNIST: 784-1024-1024-1024-10, lambda 28000 / 5000
    "mlp3_mnist_b64": dict(
        input_shape=(28, 28, 1), batch=64, steps=10,
        hyper=dict(eta_inv_fw=28000, eta_inv_lr=5000),
        blocks=_paper_mlp([784, 1024, 1024, 1024])),
    # MLP4, CIFAR-10: 1024-3000-3000-3000-10 (Table 1 gives a 1024-wide input:
    # one 32 x 32 channel), lambda 19000 / 7500, p_l = 0.10
    "mlp4_cifar10_b64": dict(
        input_shape=(32, 32, 1), batch=64, steps=10,
        hyper=dict(eta_inv_fw=19000, eta_inv_lr=7500, dropout_p16=6554),
        blocks=_paper_mlp([1024, 3000, 3000, 3000])),
}
WORKLOADS.update(PAPER_WORKLOADS)

# Kernel sweep: conv fwd / dgrad / wgrad at batch 256 and int GEMM sizes.
SWEEP_CONV = [(256, hw, c) for hw in (32, 16, 8) for c in (64, 128, 256, 512)]
SWEEP_GEMM = [1024, 4096, 8192]
