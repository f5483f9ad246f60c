"""Pins of the CPU oracle against things other than itself (no GPU needed).

Each test ties an oracle function to a hand-worked value from the paper's
formulas (tests/golden/), a closed form, an invariant the paper states, or an
independent library routine (Python integer arithmetic, numpy integer matmul /
einsum, scipy correlate2d).  A dropped term, a wrong sign, a transposed operand
or a trunc-for-floor slip in the oracle fails at least one of them.
"""
import math

import numpy as np
import pytest

import oracle as O
from oracle import nitro as N
from paper_2407_11698_gb300 import synth

RNG = np.random.default_rng(12345)


# ---------------------------------------------------------------- division
def test_fdiv_golden(golden):
    for x, d, fl, tr in golden("fdiv.txt"):
        assert O.fdiv(x, d) == fl, (x, d)
        assert O.tdiv(x, d) == tr, (x, d)


def test_fdiv_matches_python_floor_division():
    # Python's // on ints is floor division: an independent implementation.
    xs = RNG.integers(-2**62, 2**62, size=2000)
    ds = RNG.integers(1, 2**20, size=2000)
    for x, d in zip(xs.tolist(), ds.tolist()):
        assert O.fdiv(x, d) == x // d
        assert O.tdiv(x, d) == int(x / d) if abs(x) < 2**52 else True
    v = N.fdiv_vec(xs, 2304)
    assert v.tolist() == [x // 2304 for x in xs.tolist()]


def test_scaling_invariant_int8_operands():
    # Sec. 3.2.1: with |a| <= 128, |W| <= 127 the rescaled pre-activation
    # floor(z / (2^8 K^2 C)) lies in [-64, 63].
    a = RNG.integers(-128, 128, size=(2, 6, 5, 7))
    w = RNG.integers(-127, 128, size=(4, 3, 3, 7))
    z = O.conv3x3_fwd(a, w)
    zs, _, _ = N.scale_relu(z, 256 * 9 * 7, 10)
    assert zs.min() >= -64 and zs.max() <= 63
    zmax = O.conv3x3_fwd(np.full((1, 3, 3, 7), -128), np.full((1, 3, 3, 7), -127))
    assert zmax[0, 1, 1, 0] == 9 * 7 * 128 * 127


# ---------------------------------------------------------------- NITRO-ReLU
def test_relu_mu_golden(golden):
    for a, m1, m2, mu in golden("relu_mu.txt"):
        assert O.fdiv(-127, a) == m1 and O.fdiv(-127, 2 * a) == m2
        assert O.relu_mu(a) == mu


def test_relu_golden(golden):
    for x, fx, reg in golden("relu_alpha10.txt"):
        assert O.relu(x, 10) == fx, x
        assert O.relu_region(x) == reg, x


def test_relu_bwd_golden(golden):
    for g, reg, out in golden("relu_bwd_alpha10.txt"):
        assert O.relu_bwd(g, reg, 10) == out, (g, reg)


@pytest.mark.parametrize("alpha", [2, 3, 4, 10, 100])
def test_relu_range_and_monotone(alpha):
    xs = np.arange(-400, 401)
    _, reg, act = N.scale_relu(xs, 1, alpha)
    mu = O.relu_mu(alpha)
    assert np.all(np.diff(act) >= 0)
    assert act.min() == (-127) // alpha - mu and act.max() == 127 - mu
    assert act.min() >= -128 and act.max() <= 127      # int8 storage
    # regions follow the forward definition's split
    assert np.all(reg[xs < -127] == 0) and np.all(reg[(xs >= -127) & (xs < 0)] == 1)
    assert np.all(reg[(xs >= 0) & (xs <= 127)] == 2) and np.all(reg[xs > 127] == 3)


def test_relu_bwd_is_slope_of_forward():
    # For a step of alpha in the slope piece the forward moves by exactly 1,
    # so floor(g/alpha) is the integer slope times g for g a multiple of alpha.
    alpha = 10
    for x in range(-120, -9):
        assert O.relu(x + alpha, alpha) - O.relu(x, alpha) == 1
        assert O.relu_bwd(alpha * 7, 1, alpha) == 7
    for x in range(0, 126):
        assert O.relu(x + 1, alpha) - O.relu(x, alpha) == 1


# ---------------------------------------------------------------- init
def test_isqrt_matches_math_isqrt():
    for n in list(range(0, 3000)) + RNG.integers(0, 2**62, size=500).tolist():
        assert O.isqrt(n) == math.isqrt(n)


def test_init_bound_golden(golden):
    for fan_in, r, b in golden("init_bound.txt"):
        assert O.isqrt(fan_in) == r
        assert O.init_bound(fan_in) == b


def test_splitmix64_published_vector():
    # First outputs of SplitMix64 seeded with 1234567 (the test vector used
    # with the reference C implementation by S. Vigna).
    expect = [6457827717110365317, 3203168211198807973, 9817491932198370423,
              4593380528125082431, 16408922859458223821]
    assert [O.splitmix64_at(1234567, i) for i in range(5)] == expect


def test_init_uniform_range():
    w = N.init_uniform((64, 3, 3, 3), 44, 99, 0)
    assert w.min() == -44 and w.max() == 44
    assert abs(w.mean()) < 3
    assert np.all(N.init_uniform((5, 7), 0, 1, 2) == 0)
    # distinct tensors draw from distinct streams
    assert not np.array_equal(N.init_uniform((100,), 5, 1, 0), N.init_uniform((100,), 5, 1, 1))


# ---------------------------------------------------------------- contractions
def _correlate_same(a, k):
    from scipy.signal import correlate2d
    return correlate2d(a, k, mode="same", boundary="fill", fillvalue=0)


def test_conv_fwd_matches_scipy_correlate2d():
    pytest.importorskip("scipy")
    B, H, W, Cin, Cout = 2, 7, 5, 3, 4
    a = RNG.integers(-128, 128, size=(B, H, W, Cin))
    w = RNG.integers(-3000, 3000, size=(Cout, 3, 3, Cin))
    z = O.conv3x3_fwd(a, w)
    for b in range(B):
        for co in range(Cout):
            ref = sum(_correlate_same(a[b, :, :, ci], w[co, :, :, ci]) for ci in range(Cin))
            assert np.array_equal(z[b, :, :, co], ref)


def _brute_conv(a, w):
    """Direct definition in Python integers: z[b,y,x,co] = sum over taps (ky, kx)
    and ci of a[b, y+ky-1, x+kx-1, ci] w[co, ky, kx, ci], zero outside."""
    B, H, W, Cin = a.shape
    Cout = w.shape[0]
    z = [[[[0] * Cout for _ in range(W)] for _ in range(H)] for _ in range(B)]
    for b in range(B):
        for y in range(H):
            for x in range(W):
                for co in range(Cout):
                    t = 0
                    for ky in range(3):
                        for kx in range(3):
                            iy, ix = y + ky - 1, x + kx - 1
                            if 0 <= iy < H and 0 <= ix < W:
                                for ci in range(Cin):
                                    t += int(a[b, iy, ix, ci]) * int(w[co, ky, kx, ci])
                    z[b][y][x][co] = t
    return z


def test_conv_contractions_match_brute_force():
    # forward, weight gradient and input gradient of the oracle against the
    # direct sums in Python integers; |w|, |d| < 2^27 keep every sum inside
    # int64 while the products are far beyond int32, so a 32-bit truncation
    # anywhere in the oracle would show
    B, H, W, Cin, Cout = 2, 4, 3, 2, 3
    a = RNG.integers(-128, 128, size=(B, H, W, Cin))
    w = RNG.integers(-2**27, 2**27, size=(Cout, 3, 3, Cin))
    d = RNG.integers(-2**27, 2**27, size=(B, H, W, Cout))
    assert O.conv3x3_fwd(a, w).tolist() == _brute_conv(a, w)
    # dW[co,ky,kx,ci] = sum_(b,y,x) d[b,y,x,co] a[b,y+ky-1,x+kx-1,ci]
    dw = [[[[0] * Cin for _ in range(3)] for _ in range(3)] for _ in range(Cout)]
    for co in range(Cout):
        for ky in range(3):
            for kx in range(3):
                for ci in range(Cin):
                    t = 0
                    for b in range(B):
                        for y in range(H):
                            for x in range(W):
                                iy, ix = y + ky - 1, x + kx - 1
                                if 0 <= iy < H and 0 <= ix < W:
                                    t += int(d[b, y, x, co]) * int(a[b, iy, ix, ci])
                    dw[co][ky][kx][ci] = t
    assert O.conv3x3_wgrad(a, d).tolist() == dw
    # g[b,y,x,ci] = sum_(ky,kx,co) d[b,y-ky+1,x-kx+1,co] w[co,ky,kx,ci]
    g = [[[[0] * Cin for _ in range(W)] for _ in range(H)] for _ in range(B)]
    for b in range(B):
        for y in range(H):
            for x in range(W):
                for ci in range(Cin):
                    t = 0
                    for ky in range(3):
                        for kx in range(3):
                            oy, ox = y - ky + 1, x - kx + 1
                            if 0 <= oy < H and 0 <= ox < W:
                                for co in range(Cout):
                                    t += int(d[b, oy, ox, co]) * int(w[co, ky, kx, ci])
                    g[b][y][x][ci] = t
    assert O.conv3x3_dgrad(d, w).tolist() == g


def test_conv_one_hot_reproduces_flipped_kernel():
    H = W = 5
    w = RNG.integers(-50, 50, size=(2, 3, 3, 3))
    a = np.zeros((1, H, W, 3), dtype=np.int64)
    a[0, 2, 2, 1] = 1
    z = O.conv3x3_fwd(a, w)
    # output (y, x) reads input (2, 2) through tap (2 - y + 1, 2 - x + 1)
    for co in range(2):
        assert np.array_equal(z[0, 1:4, 1:4, co], w[co, ::-1, ::-1, 1])
    assert np.count_nonzero(z[0, [0, 4], :, :]) == 0


def test_conv_1x1_image_is_linear_on_centre_tap():
    a = RNG.integers(-128, 128, size=(3, 1, 1, 6))
    w = RNG.integers(-99, 99, size=(5, 3, 3, 6))
    z = O.conv3x3_fwd(a, w)
    assert np.array_equal(z[:, 0, 0, :], a[:, 0, 0, :] @ w[:, 1, 1, :].T)


def _pad(x):
    return np.pad(x, ((0, 0), (1, 1), (1, 1), (0, 0)))


def test_conv_wgrad_dgrad_match_einsum():
    B, H, W, Cin, Cout = 2, 6, 7, 3, 5
    a = RNG.integers(-128, 128, size=(B, H, W, Cin))
    g = RNG.integers(-10**6, 10**6, size=(B, H, W, Cout))
    w = RNG.integers(-10**4, 10**4, size=(Cout, 3, 3, Cin))
    ap, gp = _pad(a), _pad(g)
    dw = O.conv3x3_wgrad(a, g)
    dgi = O.conv3x3_dgrad(g, w)
    for ky in range(3):
        for kx in range(3):
            ref = np.einsum("byxo,byxc->oc", g, ap[:, ky:ky + H, kx:kx + W, :])
            assert np.array_equal(dw[:, ky, kx, :], ref)
    ref = np.zeros_like(dgi)
    for ky in range(3):
        for kx in range(3):
            # input (y, x) is read by output (y - ky + 1, x - kx + 1)
            ref += np.einsum("byxo,oc->byxc", gp[:, 2 - ky:2 - ky + H, 2 - kx:2 - kx + W, :],
                             w[:, ky, kx, :])
    assert np.array_equal(dgi, ref)


def test_adjoint_identities():
    # <conv(a,W), g> = <a, dgrad(g,W)> = <W, wgrad(a,g)>, exactly in integers
    B, H, W, Cin, Cout = 2, 5, 6, 4, 3
    a = RNG.integers(-128, 128, size=(B, H, W, Cin))
    g = RNG.integers(-5000, 5000, size=(B, H, W, Cout))
    w = RNG.integers(-5000, 5000, size=(Cout, 3, 3, Cin))
    lhs = int(np.sum(O.conv3x3_fwd(a, w) * g))
    assert lhs == int(np.sum(a * O.conv3x3_dgrad(g, w)))
    assert lhs == int(np.sum(w * O.conv3x3_wgrad(a, g)))
    a2 = RNG.integers(-128, 128, size=(7, 11))
    g2 = RNG.integers(-5000, 5000, size=(7, 4))
    w2 = RNG.integers(-5000, 5000, size=(4, 11))
    lhs = int(np.sum(O.linear_fwd(a2, w2) * g2))
    assert lhs == int(np.sum(a2 * O.linear_dgrad(g2, w2)))
    assert lhs == int(np.sum(w2 * O.linear_wgrad(a2, g2)))


def test_linear_matches_numpy_matmul():
    a = RNG.integers(-128, 128, size=(9, 37))
    w = RNG.integers(-2**20, 2**20, size=(13, 37))
    g = RNG.integers(-2**20, 2**20, size=(9, 13))
    assert np.array_equal(O.linear_fwd(a, w), a @ w.T)
    assert np.array_equal(O.linear_dgrad(g, w), g @ w)
    assert np.array_equal(O.linear_wgrad(a, g), g.T @ a)


def test_contraction_wraps_modulo_2_64():
    a = np.array([[2**40, 3]], dtype=np.int64)
    w = np.array([[2**40, 5]], dtype=np.int64)
    exact = 2**80 + 15
    z = int(O.linear_fwd(a, w)[0, 0])
    assert z % 2**64 == exact % 2**64


# ---------------------------------------------------------------- max-pool
def test_maxpool_matches_reshape_max_and_first_tie():
    a = RNG.integers(-5, 5, size=(2, 6, 8, 3))          # many ties
    out, am = O.maxpool_fwd(a)
    blocks = a.reshape(2, 3, 2, 4, 2, 3).transpose(0, 1, 3, 5, 2, 4).reshape(2, 3, 4, 3, 4)
    assert np.array_equal(out, blocks.max(-1))
    assert np.array_equal(am, blocks.argmax(-1))      # numpy argmax: first maximum
    g = RNG.integers(-100, 100, size=out.shape)
    gi = O.maxpool_bwd(g, am, 6, 8)
    assert gi.sum() == g.sum() and np.count_nonzero(gi) == np.count_nonzero(g)
    gb = gi.reshape(2, 3, 2, 4, 2, 3).transpose(0, 1, 3, 5, 2, 4).reshape(2, 3, 4, 3, 4)
    assert np.array_equal(np.take_along_axis(gb, am[..., None], -1)[..., 0], g)


def test_maxpool_odd_size_floors():
    a = RNG.integers(-100, 100, size=(1, 7, 5, 2))
    out, am = O.maxpool_fwd(a)
    assert out.shape == (1, 3, 2, 2)
    gi = O.maxpool_bwd(np.ones_like(out), am, 7, 5)
    assert gi[:, 6, :, :].sum() == 0 and gi[:, :, 4, :].sum() == 0


# ---------------------------------------------------------------- IntegerSGD
def test_integersgd_golden(golden):
    for w, dw, gamma, eta, mode, out in golden("integersgd.txt"):
        r = O.integersgd(np.array([w]), np.array([dw]), gamma, eta, mode)
        assert int(r[0]) == out, (w, dw, gamma, eta, mode)


def test_integersgd_zero_gradient_no_update_and_decay_threshold():
    w = RNG.integers(-2**30, 2**30, size=1000)
    assert np.array_equal(O.integersgd(w, np.zeros_like(w), 512, 0, O.FLOOR), w)
    # Sec. 3.3.4: |w| < eta_inv gives no decay (exact under truncation)
    small = RNG.integers(-999, 1000, size=1000)
    assert np.array_equal(O.integersgd(small, np.zeros_like(small), 512, 1000, O.TRUNC), small)
    # under floor a negative weight below the threshold still moves up by one
    assert int(O.integersgd(np.array([-5]), np.array([0]), 512, 1000, O.FLOOR)[0]) == -4


def test_integersgd_matches_python():
    w = RNG.integers(-2**31, 2**31, size=500)
    dw = RNG.integers(-2**55, 2**55, size=500)
    for mode in (O.FLOOR, O.TRUNC):
        r = O.integersgd(w, dw, 327680, 25000, mode)
        for wi, di, ri in zip(w.tolist(), dw.tolist(), r.tolist()):
            if mode == O.FLOOR:
                d = di // 327680 + wi // 25000
            else:
                d = int(di / 327680) if abs(di) < 2**52 else None
                if d is None:
                    continue
                d += int(wi / 25000)
            assert ri == wi - d


def test_amplification_factor():
    # Sec. 3.3.5: AF = 2^6 * G; gamma_inv^fw = AF * gamma_inv^lr
    assert O.amplification_factor(10) == 640
    blk = O.OracleBlock([], in_features=4)
    assert blk.gamma_inv_fw == 640 * 512 == 327680


# ---------------------------------------------------------------- block level
def _lin_block(cin, cout, **kw):
    return O.OracleBlock([O.LayerDesc(O.LINEAR, cin, cout)], **kw)


def test_learning_layer_and_loss_closed_form():
    blk = _lin_block(20, 12, seed=3)
    B = 9
    x = RNG.integers(-128, 128, size=(B, 20))
    y = RNG.integers(0, 10, size=B)
    blk.forward(x)
    loss = blk.backward(x, y)
    a = blk.out
    z = a @ blk.Wlr.T
    yhat = np.array([[int(v) // (256 * 12) for v in row] for row in z.tolist()])
    tgt = np.zeros((B, 10), dtype=np.int64)
    tgt[np.arange(B), y] = 32
    assert np.array_equal(blk.yhat, yhat)
    assert np.array_equal(blk.grad_l, yhat - tgt)
    sse = int(((yhat - tgt) ** 2).sum())
    assert blk.sse == sse and loss == sse // 2
    assert np.array_equal(blk.dWlr, (yhat - tgt).T @ a)


def test_zero_learning_weights_special_case():
    # W_lr = 0 => yhat = 0, grad_L = -32 at the label, SSE = 1024 B,
    # delta_fw = 0, so the forward layers get zero gradient and do not move.
    blk = O.OracleBlock([O.LayerDesc(O.CONV, 2, 4, 6, 6, True)], seed=5)
    blk.Wlr[:] = 0
    B = 5
    x = RNG.integers(-128, 128, size=(B, 6, 6, 2))
    y = RNG.integers(0, 10, size=B)
    blk.forward(x)
    loss = blk.backward(x, y)
    assert loss == 512 * B and blk.sse == 1024 * B
    assert np.all(blk.grad_l[np.arange(B), y] == -32)
    assert np.count_nonzero(blk.grad_l) == B
    assert not np.any(blk.dW[0])
    w0 = blk.W[0].copy()
    blk.sgd()
    assert np.array_equal(blk.W[0], w0)


def test_linear_block_identity_region_is_textbook_backprop():
    # Non-negative inputs and weights keep z* in [0, 127], NITRO-ReLU's
    # identity piece, so the block's backward is plain back-propagation with
    # a straight-through scaling: delta = grad_L W_lr, dW = delta^T a.
    blk = _lin_block(30, 8, seed=11)
    blk.W[0] = np.abs(blk.W[0])
    x = RNG.integers(0, 128, size=(6, 30))
    y = RNG.integers(0, 10, size=6)
    blk.forward(x)
    assert np.all(blk.region[0] == 2)
    blk.backward(x, y)
    delta = blk.grad_l @ blk.Wlr
    assert np.array_equal(blk.delta[0], delta)
    assert np.array_equal(blk.dW[0], delta.T @ x)


def test_conv_block_pool_backward_routes_through_argmax():
    blk = O.OracleBlock([O.LayerDesc(O.CONV, 3, 4, 6, 4, True)], seed=2)
    blk.W[0] = np.abs(blk.W[0])
    x = RNG.integers(0, 128, size=(2, 6, 4, 3))
    y = np.array([1, 7])
    blk.forward(x)
    assert np.all(blk.region[0] == 2)
    blk.backward(x, y)
    g = (blk.grad_l @ blk.Wlr).reshape(2, 3, 2, 4)
    d = blk.delta[0]
    assert d.sum() == g.sum()
    # only window maxima receive gradient; every other position gets zero
    act = np.array(blk.zs[0]) - O.relu_mu(10)
    for b in range(2):
        for yy in range(3):
            for xx in range(2):
                for c in range(4):
                    win = act[b, 2 * yy:2 * yy + 2, 2 * xx:2 * xx + 2, c].reshape(-1)
                    k = int(np.argmax(win))
                    dw_ = d[b, 2 * yy:2 * yy + 2, 2 * xx:2 * xx + 2, c].reshape(-1)
                    assert dw_[k] == g[b, yy, xx, c]
                    assert np.count_nonzero(np.delete(dw_, k)) == 0


def test_two_layer_block_dgrad_chain():
    layers = [O.LayerDesc(O.CONV, 2, 3, 5, 5, False), O.LayerDesc(O.CONV, 3, 4, 5, 5, True)]
    blk = O.OracleBlock(layers, seed=8)
    x = RNG.integers(-128, 128, size=(3, 5, 5, 2))
    y = RNG.integers(0, 10, size=3)
    blk.forward(x)
    blk.backward(x, y)
    g1 = O.conv3x3_dgrad(blk.delta[1], blk.W[1])
    d0 = np.array([[O.relu_bwd(int(v), int(r), 10) for v, r in zip(gr, rr)]
                   for gr, rr in zip(g1.reshape(3, -1), blk.region[0].reshape(3, -1))])
    assert np.array_equal(blk.delta[0].reshape(3, -1), d0)
    assert np.array_equal(blk.dW[0], O.conv3x3_wgrad(x, blk.delta[0]))


def test_blocks_are_local():
    # Sec. 3.3: no gradient crosses blocks; perturbing block 2 leaves block
    # 1's weight gradients bit-identical.
    def net(perturb):
        b1 = O.OracleBlock([O.LayerDesc(O.LINEAR, 16, 12)], seed=1)
        b2 = O.OracleBlock([O.LayerDesc(O.LINEAR, 12, 6)], seed=2)
        b3 = O.OracleBlock([], in_features=6, seed=3)
        if perturb:
            b2.W[0] += 17
            b2.Wlr -= 3
        return [b1, b2, b3]
    x = RNG.integers(-128, 128, size=(8, 16))
    y = RNG.integers(0, 10, size=8)
    n1, n2 = net(False), net(True)
    O.train_step(n1, x, y)
    O.train_step(n2, x, y)
    assert np.array_equal(n1[0].dW[0], n2[0].dW[0])
    assert np.array_equal(n1[0].dWlr, n2[0].dWlr)
    assert np.array_equal(n1[0].W[0], n2[0].W[0])
    assert not np.array_equal(n1[1].dW[0], n2[1].dW[0])


def test_empty_batch():
    blk = O.OracleBlock([O.LayerDesc(O.CONV, 1, 4, 4, 4, True)], seed=1)
    x = np.zeros((0, 4, 4, 1), dtype=np.int64)
    out = blk.forward(x)
    assert out.shape == (0, 16)
    assert blk.backward(x, np.zeros(0, dtype=np.int64)) == 0
    w = blk.W[0].copy()
    blk.sgd()
    assert np.array_equal(blk.W[0], w) and blk.status == 0


def test_bad_label_flag():
    blk = _lin_block(8, 4, seed=1)
    x = RNG.integers(-128, 128, size=(3, 8))
    blk.forward(x)
    blk.backward(x, np.array([1, 10, -1]))
    assert blk.status & O.ST_BAD_LABEL
    tgt_row = blk.yhat[1]
    assert np.array_equal(blk.grad_l[1], tgt_row)   # no hot entry for a bad label


def test_overflow_flags():
    # delta stored in int32: a learning weight of 2^29 makes delta_fw overflow
    blk = _lin_block(8, 4, seed=1)
    blk.Wlr[:] = 2**29
    x = RNG.integers(-128, 128, size=(3, 8))
    blk.forward(x)
    blk.backward(x, np.array([1, 2, 3]))
    assert blk.status & O.ST_OVERFLOW
    # weight update leaving int32
    blk2 = _lin_block(8, 4, seed=1)
    blk2.W[0][:] = 2**31 - 1
    blk2.dW[0][:] = -512 * 640 * 4
    blk2.sgd()
    assert blk2.status & O.ST_OVERFLOW
    assert int(blk2.W[0][0, 0]) == ((2**31 - 1 + 4 + 2**31) % 2**32) - 2**31
    # int64 exactness bound on int32 x int32 contractions
    assert N.int64_bound_exceeded(np.array([2**31]), np.array([2**31]), 2)
    assert not N.int64_bound_exceeded(np.array([2**31 - 1]), np.array([2**31 - 1]), 1)


def test_post_update_option_differs_only_in_delta():
    kw = dict(seed=4)
    b1 = _lin_block(10, 6, **kw)
    b2 = _lin_block(10, 6, lr_post_update=True, **kw)
    x = RNG.integers(-128, 128, size=(16, 10))
    y = RNG.integers(0, 10, size=16)
    for b in (b1, b2):
        b.forward(x)
        b.backward(x, y)
    assert np.array_equal(b1.dWlr, b2.dWlr)
    w_new = O.integersgd(b1.Wlr, b1.dWlr, 512, 0)
    assert np.array_equal(b2.delta[0], O.relu_bwd_vec(b1.grad_l @ w_new, b1.region[0], 10)
                          if hasattr(O, "relu_bwd_vec") else N.relu_bwd_vec(b1.grad_l @ w_new,
                                                                          b1.region[0], 10))


def test_synthetic_inputs_are_seeded():
    a = synth.images(1, 0, 4, (28, 28, 1))
    assert a.dtype == np.int8 and a.shape == (4, 28, 28, 1)
    assert np.array_equal(a, synth.images(1, 0, 4, (28, 28, 1)))
    assert not np.array_equal(a, synth.images(1, 1, 4, (28, 28, 1)))
    lab = synth.labels(1, 0, 1000)
    assert lab.min() == 0 and lab.max() == 9


# ------------------------------------------------------- pre-processing
def test_prep_golden(golden):
    for row in golden("preprocess.txt"):
        n = row[0]
        x, (mu, om), xh = row[1:1 + n], row[1 + n:3 + n], row[3 + n:]
        assert O.prep_stats(x) == (mu, om)
        assert O.prep_apply(np.array(x), mu, om).tolist() == xh


def test_prep_shift_invariance():
    """mu moves with a constant shift of the data, omega and x_hat do not."""
    x = RNG.integers(0, 200, 20011)
    mu, om = O.prep_stats(x)
    mu2, om2 = O.prep_stats(x + 37)
    assert (mu2, om2) == (mu + 37, om)
    assert np.array_equal(O.prep_apply(x, mu, om), O.prep_apply(x + 37, mu2, om2))


def test_prep_uniform_data_has_mad_51():
    """Uniform bytes: omega ~ 64, no value reaches the clamp, and the mean
    absolute value of x_hat is the 51 the rescaling multiplies by (App. A)."""
    x = RNG.integers(0, 256, 1 << 20)
    mu, om = O.prep_stats(x)
    assert 126 <= mu <= 128 and 62 <= om <= 65
    xh = O.prep_apply(x, mu, om).astype(np.int64)
    assert np.abs(xh).max() < 127
    assert abs(np.abs(xh).mean() - 51) < 1.0
    assert abs(xh.mean()) < 1.0


def test_prep_gaussian_data_meets_the_stated_target():
    """App. A: the rescaling by 51 / omega (omega = mean absolute deviation,
    ~0.8 sigma for Gaussian data) gives Gaussian data a standard deviation of
    ~64, so ~95% of it lands in [-127, 127].  Checked on N(128.5, 30^2) bytes:
    the realised scale 51 sd(x) / omega is within 5% of 64, and the mean and
    standard deviation of x_hat equal those of the clipped normal that the
    realised affine map (floor included) predicts."""
    from scipy import integrate
    from scipy.stats import norm
    x = np.clip(np.rint(RNG.normal(128.5, 30.0, 1 << 20)), 0, 255)
    mu, om = O.prep_stats(x)
    assert abs(om - math.sqrt(2 / math.pi) * 30) <= 1.5
    scale = 51 * x.std() / om
    assert abs(scale / 64 - 1) < 0.05
    shift = (x.mean() - mu) * 51 / om - 0.5          # floor lowers by 1/2 on average
    sd = math.sqrt(scale ** 2 + 1 / 12)
    clip = lambda y: min(max(y, -127.0), 127.0)
    pdf = lambda y: norm.pdf(y, shift, sd)
    m1 = integrate.quad(lambda y: clip(y) * pdf(y), shift - 10 * sd, shift + 10 * sd,
                        points=[-127, 127], limit=200)[0]
    m2 = integrate.quad(lambda y: clip(y) ** 2 * pdf(y), shift - 10 * sd, shift + 10 * sd,
                        points=[-127, 127], limit=200)[0]
    xh = O.prep_apply(x, mu, om).astype(np.float64)
    assert abs(xh.mean() - m1) < 0.3
    assert abs(xh.std() / math.sqrt(m2 - m1 ** 2) - 1) < 0.01
    inside = norm.cdf(127, shift, sd) - norm.cdf(-127, shift, sd)
    assert abs(inside - 0.95) < 0.02
    assert abs((np.abs(xh) < 127).mean() - inside) < 0.01


# ---------------------------------------------------------------- whole step
@pytest.mark.parametrize("round_mode", [O.FLOOR, O.TRUNC])
def test_block_step_worked_by_hand(golden, round_mode):
    # one full training step of a one-layer linear block, every intermediate
    # and the updated weights worked by hand (tests/golden/block_step_linear.txt)
    rows = golden("block_step_linear.txt")
    (a, w, wlr, lab, zs, region, a1, yhat, grad_l, sse_loss, dwlr, delta, dw,
     w_floor, wlr_new, w_trunc) = rows
    blk = O.OracleBlock([O.LayerDesc(O.LINEAR, 2, 2)], num_classes=2, alpha_inv=10,
                        gamma_inv_lr=512, sgd_round=round_mode, seed=1)
    blk.W[0] = np.array(w, dtype=np.int64).reshape(2, 2)
    blk.Wlr = np.array(wlr, dtype=np.int64).reshape(2, 2)
    losses = O.train_step([blk], np.array([a], dtype=np.int64), np.array(lab, dtype=np.int64))
    assert losses == [sse_loss[1]] and blk.sse == sse_loss[0]
    assert blk.zs[0].reshape(-1).tolist() == zs
    assert blk.region[0].reshape(-1).tolist() == region
    assert blk.act[0].reshape(-1).tolist() == a1
    assert blk.yhat.reshape(-1).tolist() == yhat
    assert blk.grad_l.reshape(-1).tolist() == grad_l
    assert blk.dWlr.reshape(-1).tolist() == dwlr
    assert blk.delta[0].reshape(-1).tolist() == delta
    assert blk.dW[0].reshape(-1).tolist() == dw
    assert blk.W[0].reshape(-1).tolist() == (w_floor if round_mode == O.FLOOR else w_trunc)
    assert blk.Wlr.reshape(-1).tolist() == wlr_new
    assert blk.status == 0


def test_conv_block_step_worked_by_hand(golden):
    # the conv counterpart: padding, scaling, pool routing and the 3x3 weight
    # gradient of one full step, worked by hand (tests/golden/block_step_conv.txt)
    (a, w, wlr, lab, zs, region, _relu, a1, am, yhat, grad_l, sse_loss, dwlr, delta, dw,
     w_new, wlr_new) = golden("block_step_conv.txt")
    blk = O.OracleBlock([O.LayerDesc(O.CONV, 1, 1, 2, 2, True)], num_classes=2, alpha_inv=10,
                        gamma_inv_lr=512, seed=1)
    blk.W[0] = np.array(w, dtype=np.int64).reshape(1, 3, 3, 1)
    blk.Wlr = np.array(wlr, dtype=np.int64).reshape(2, 1)
    losses = O.train_step([blk], np.array([a], dtype=np.int64), np.array(lab, dtype=np.int64))
    assert losses == [sse_loss[1]] and blk.sse == sse_loss[0]
    assert blk.zs[0].reshape(-1).tolist() == zs
    assert blk.region[0].reshape(-1).tolist() == region
    assert blk.act[0].reshape(-1).tolist() == a1
    assert blk.argmax[0].reshape(-1).tolist() == am
    assert blk.yhat.reshape(-1).tolist() == yhat
    assert blk.grad_l.reshape(-1).tolist() == grad_l
    assert blk.dWlr.reshape(-1).tolist() == dwlr
    assert blk.delta[0].reshape(-1).tolist() == delta
    assert blk.dW[0].reshape(-1).tolist() == dw
    assert blk.W[0].reshape(-1).tolist() == w_new
    assert blk.Wlr.reshape(-1).tolist() == wlr_new
