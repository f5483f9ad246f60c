"""Pins of the oracle's learning-layer pooling and dropout (no GPU needed).

Learning-layer pooling (Sec. 3.3: a block's output is downsampled to z^mp
before its learning layers; App. B: d^lr input features) is tied to
hand-worked windows (tests/golden/lr_pool_window.txt), to numpy's reshape-max
and first-occurrence argmax, to the separately pinned 2x2 max-pool, and to the
adjoint identity of max-pool backward.  Dropout (App. B, p_l) is tied to its
closed cases (p = 0 keeps all, p = 1 drops all), to the binomial law of the
dropped fraction, to the independence of masks across steps and layers, and at
block level to the all-zero learning input, whose loss the paper's formulas
give in closed form.
"""
import numpy as np
import pytest

import oracle as O
from oracle import nitro as N
from paper_2407_11698_gb300 import synth

RNG = np.random.default_rng(2407)


# ------------------------------------------------------- window rule
def test_lr_pool_window_golden(golden):
    for C, H, W, d_lr, kh, kw, d in golden("lr_pool_window.txt"):
        assert N.lr_pool_window(C, H, W, d_lr) == (kh, kw), (C, H, W, d_lr)
        assert C * (H // kh) * (W // kw) == d


def test_lr_pool_window_properties():
    # the window is a power of two on each side that fits the map; it reaches
    # d <= d_lr unless the map is exhausted (neither side can double)
    for C in (1, 3, 32, 128, 512):
        for H in (1, 2, 3, 7, 8, 14, 16, 32):
            for d_lr in (1, 10, 100, 1000, 4096):
                kh, kw = N.lr_pool_window(C, H, H, d_lr)
                assert kh & (kh - 1) == 0 and kw & (kw - 1) == 0
                assert kh <= H and kw <= H
                # on a square map the height leads the width by at most one doubling
                assert kw <= kh <= 2 * kw
                d = C * (H // kh) * (H // kw)
                if d > d_lr:
                    assert 2 * kh > H and 2 * kw > H
                if d_lr >= C * H * H:
                    assert (kh, kw) == (1, 1)


# ------------------------------------------------------- pooling forward / backward
def _numpy_winpool(a, kh, kw):
    B, H, W, C = a.shape
    Ho, Wo = H // kh, W // kw
    v = a[:, :Ho * kh, :Wo * kw, :].reshape(B, Ho, kh, Wo, kw, C)
    v = v.transpose(0, 1, 3, 5, 2, 4).reshape(B, Ho, Wo, C, kh * kw)
    return v.max(axis=-1), v.argmax(axis=-1)   # argmax: first occurrence


@pytest.mark.parametrize("kh,kw", [(1, 1), (2, 1), (2, 2), (4, 2), (8, 4), (3, 5)])
def test_winpool_matches_numpy_reshape_max(kh, kw):
    for H, W in ((16, 16), (17, 11), (9, 23)):
        if H < kh or W < kw:
            continue
        # a narrow value range forces many ties: the first maximum must win
        a = RNG.integers(-3, 3, size=(2, H, W, 5))
        out, am = O.nitro.winpool_fwd(a, kh, kw)
        want, want_am = _numpy_winpool(a, kh, kw)
        assert np.array_equal(out, want)
        assert np.array_equal(am, want_am)


def test_winpool_2x2_equals_maxpool():
    a = RNG.integers(-128, 128, size=(3, 10, 14, 6))
    out, am = O.nitro.winpool_fwd(a, 2, 2)
    out2, am2 = O.maxpool_fwd(a)
    assert np.array_equal(out, out2) and np.array_equal(am, am2)
    g = RNG.integers(-1000, 1000, size=out.shape)
    assert np.array_equal(O.nitro.winpool_bwd(g, am, 10, 14, 2, 2),
                          O.maxpool_bwd(g, am2, 10, 14))


@pytest.mark.parametrize("kh,kw", [(2, 1), (4, 4), (8, 4)])
def test_winpool_backward_adjoint_and_routing(kh, kw):
    H, W = 2 * kh + 1, 3 * kw + 1          # ragged: the floor drops a row and a column
    a = RNG.integers(-128, 128, size=(2, H, W, 3))
    out, am = O.nitro.winpool_fwd(a, kh, kw)
    g = RNG.integers(-10**6, 10**6, size=out.shape)
    gi = O.nitro.winpool_bwd(g, am, H, W, kh, kw)
    # <pool(a), g> = <a, bwd(g)>: the gradient lands where the maximum was read
    assert int((out * g).sum()) == int((a * gi).sum())
    # one nonzero per window at most, none outside the pooled area
    assert np.count_nonzero(gi) <= np.count_nonzero(g)
    assert not gi[:, (H // kh) * kh:, :, :].any() and not gi[:, :, (W // kw) * kw:, :].any()
    assert gi.sum() == g.sum()


# ------------------------------------------------------- dropout mask
def test_dropout_closed_cases():
    assert not N.dropout_mask(5000, 9, 0, 0, 0).any()
    assert N.dropout_mask(5000, 9, 3, 2, 65536).all()


@pytest.mark.parametrize("p16", [6554, 9830, 32768])
def test_dropout_fraction_is_binomial(p16):
    n = 200000
    k = int(N.dropout_mask(n, 20240716, 5, 1, p16).sum())
    p = p16 / 65536.0
    assert abs(k - n * p) < 5 * np.sqrt(n * p * (1 - p))


def test_dropout_masks_independent_across_steps_and_layers():
    n, p16 = 100000, 32768
    m = [N.dropout_mask(n, 77, t, l, p16) for t, l in ((0, 0), (1, 0), (0, 1), (2, 3))]
    for i in range(len(m)):
        for j in range(i + 1, len(m)):
            # agreement of two independent fair masks: n/2 +- 5 sigma
            agree = int((m[i] == m[j]).sum())
            assert abs(agree - n / 2) < 5 * np.sqrt(n / 4)
    # the step counter is taken modulo 2^28
    assert np.array_equal(N.dropout_mask(1000, 77, 2**28 + 1, 0, p16), m[1][:1000])


def test_dropout_matches_splitmix64_stream():
    # element e of layer l at step t reads output 2^63 + t 2^35 + l 2^31 + e
    # of the block's SplitMix64 stream (itself pinned to its published vector)
    for t, l, e in ((0, 0, 0), (3, 1, 17), (2**27, 14, 2**31 - 1)):
        u = O.splitmix64_at(99, 2**63 + t * 2**35 + l * 2**31 + e)
        for p16 in (0, 1, 9830, 65535, 65536):
            assert N.dropout_drop(99, t, l, e, p16) == int((u >> 48) < p16)


# ------------------------------------------------------- block level
def _mlp_block(**kw):
    return O.OracleBlock([O.LayerDesc(O.LINEAR, 48, 20)], seed=4, **kw)


def test_block_dropout_zero_is_plain_block():
    x = RNG.integers(-128, 128, size=(6, 48))
    y = RNG.integers(0, 10, size=6)
    a, b = _mlp_block(), _mlp_block(dropout_p16=0)
    for _ in range(3):
        assert O.train_step([a], x, y) == O.train_step([b], x, y)
    assert np.array_equal(a.W[0], b.W[0]) and np.array_equal(a.Wlr, b.Wlr)


def test_block_dropout_all_drops_everything():
    # every output dropped: the learning layer sees zeros, so y_hat = 0 and the
    # RSS loss is (32^2 / 2) per sample = 512 B; no gradient reaches the layer
    B = 5
    x = RNG.integers(-128, 128, size=(B, 48))
    y = RNG.integers(0, 10, size=B)
    blk = _mlp_block(dropout_p16=65536)
    w0 = blk.W[0].copy()
    assert O.train_step([blk], x, y) == [512 * B]
    assert not blk.act[0].any()
    assert (blk.region[0] == 4).all()
    assert not blk.delta[0].any() and not blk.dW[0].any()
    assert np.array_equal(blk.W[0], w0)


def test_block_dropout_mask_follows_step_counter():
    x = RNG.integers(-128, 128, size=(4, 48))
    y = RNG.integers(0, 10, size=4)
    blk = _mlp_block(dropout_p16=16384)
    for t in range(3):
        O.train_step([blk], x, y)
        drop = N.dropout_mask(4 * 20, 4, t, 0, 16384).reshape(4, 20)
        assert blk.t == t + 1
        assert ((blk.region[0] == 4) == (drop == 1)).all()
        assert not blk.act[0][drop == 1].any()
        assert not blk.delta[0][drop == 1].any()


def _conv_block(d_lr, pool=True, hw=8, cout=8):
    return O.OracleBlock([O.LayerDesc(O.CONV, 3, cout, hw, hw, pool)], seed=6, d_lr=d_lr)


def test_block_lr_pool_large_d_is_identity():
    x = synth.images(1, 0, 4, (8, 8, 3)).reshape(4, -1)
    y = synth.labels(1, 0, 4)
    a, b = _conv_block(0), _conv_block(10**6)
    assert a.d == b.d == 4 * 4 * 8
    for _ in range(2):
        assert O.train_step([a], x, y) == O.train_step([b], x, y)
    assert np.array_equal(a.dW[0], b.dW[0]) and np.array_equal(a.Wlr, b.Wlr)


@pytest.mark.parametrize("pool,hw,d_lr", [(True, 8, 32), (False, 8, 100), (True, 10, 20)])
def test_block_lr_pool_brute_force(pool, hw, d_lr):
    # the learning part of the step recomputed with numpy alone on a tiny block:
    # z^mp by reshape-max, the scaled learning layer, grad_L, dW_lr, and
    # delta_fw scattered back to the first maximum of each window
    B, C = 3, 8
    blk = _conv_block(d_lr, pool=pool, hw=hw, cout=C)
    x = synth.images(2, 0, B, (hw, hw, 3)).reshape(B, -1)
    y = synth.labels(2, 0, B)
    Wlr0 = blk.Wlr.copy()
    blk.forward(x)
    loss = blk.backward(x, y)
    oh = hw // 2 if pool else hw
    kh, kw = blk.lr_win
    assert (kh, kw) != (1, 1)
    a = blk.out.reshape(B, oh, oh, C)
    zmp, am = _numpy_winpool(a, kh, kw)
    zf = zmp.reshape(B, -1)
    assert blk.d == zf.shape[1] and np.array_equal(blk.lr_in, zf)
    z = zf @ Wlr0.T
    yhat = z // (256 * blk.d)
    t = np.zeros_like(yhat)
    t[np.arange(B), y] = 32
    gl = yhat - t
    assert np.array_equal(blk.grad_l, gl)
    assert loss == int((gl * gl).sum()) // 2
    assert np.array_equal(blk.dWlr, gl.T @ zf)
    # delta_fw at the pooled features, then routed to the window maxima
    dfw = (gl @ Wlr0).reshape(zmp.shape)
    g_out = np.zeros_like(a)
    Ho, Wo = zmp.shape[1], zmp.shape[2]
    for b in range(B):
        for i in range(Ho):
            for j in range(Wo):
                for c in range(C):
                    k = am[b, i, j, c]
                    g_out[b, i * kh + k // kw, j * kw + k % kw, c] = dfw[b, i, j, c]
    # then the layer's own pool and NITRO-ReLU backward, pinned elsewhere
    g = g_out
    if pool:
        g = O.maxpool_bwd(g, blk.argmax[0], hw, hw)
    assert np.array_equal(blk.delta[0], O.nitro.relu_bwd_vec(g, blk.region[0], 10))


def test_block_lr_pool_rejects_wide_windows():
    with pytest.raises(ValueError):
        O.OracleBlock([O.LayerDesc(O.CONV, 1, 1, 64, 64, False)], d_lr=1)


# ------------------------------------------------------- paper-scale networks
def test_paper_workloads_chain_and_pool_to_d_lr():
    from paper_2407_11698_gb300 import workloads as WL
    for name, wl in WL.PAPER_WORKLOADS.items():
        hyper = wl.get("hyper", {})
        blocks = [O.OracleBlock([O.LayerDesc(*l) for l in b["layers"]],
                                in_features=b["in_features"], seed=i, **hyper)
                  for i, b in enumerate(wl["blocks"])]
        in_f = int(np.prod(wl["input_shape"]))
        for blk in blocks:
            assert blk.in_features == in_f, name
            if blk.layers:
                in_f = blk.layers[-1].out_features
                if hyper.get("d_lr"):
                    assert blk.d <= hyper["d_lr"], name
        assert blocks[-1].layers == [] and blocks[-1].G == 10
    # VGG8B's learning layers all see 4096 features except the 2 x 2 x 512
    # block and the linear block (2048 and 1024 outputs)
    ds = [O.OracleBlock([O.LayerDesc(*l) for l in b["layers"]], in_features=b["in_features"],
                        **WL.PAPER_WORKLOADS["vgg8b_cifar10_b64"]["hyper"]).d
          for b in WL.PAPER_WORKLOADS["vgg8b_cifar10_b64"]["blocks"][:-1]]
    assert ds == [4096, 4096, 4096, 4096, 4096, 2048, 1024]
