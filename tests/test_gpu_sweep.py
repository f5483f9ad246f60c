"""Kernel sweep: conv forward / weight gradient / input gradient and the
integer GEMM through the kernel-level C-ABI calls, bit-exact against the
oracle.  Small ragged shapes are compared element by element; the sweep's full
sizes (batch 256, 32x32 / 16x16 / 8x8, 64..512 channels; GEMM up to 8192^3)
are compared on sampled outputs that the oracle computes one by one from
cropped inputs.  Operands span one to four int8 limbs."""
import numpy as np
import pytest

import oracle as O
from paper_2407_11698_gb300 import binding as nb
from paper_2407_11698_gb300 import synth
from paper_2407_11698_gb300 import workloads as WL

pytestmark = pytest.mark.gpu

# value ranges whose max |x| needs exactly 1, 2, 3 and 4 limbs
RANGES = {1: (-127, 127), 2: (-32639, 32639), 3: (-8355711, 8355711), 4: (-2**31, 2**31 - 1)}


@pytest.fixture(scope="module")
def torch():
    t = pytest.importorskip("torch")
    if not t.cuda.is_available():
        pytest.skip("no CUDA device")
    nb.lib()
    return t


def _dev(torch, x, dtype):
    return torch.from_numpy(np.ascontiguousarray(x).astype(dtype)).cuda()


def _wrap64(x):
    return (np.asarray(x, dtype=np.int64))


@pytest.mark.parametrize("B,h,w,cin,cout,lw,ld", [
    (3, 12, 9, 64, 128, 1, 2),
    (2, 8, 8, 192, 64, 3, 1),
    (5, 16, 16, 128, 128, 2, 4),
    (2, 7, 7, 64, 64, 4, 3),       # 7x7: forward / dgrad on CUDA cores, wgrad on tcgen05
    (4, 8, 8, 32, 64, 2, 2),       # 32 input channels (padded to a 64-wide K-block)
    (9, 10, 11, 64, 48, 1, 1),     # 48 output channels: masked columns
    (3, 12, 9, 3, 64, 3, 4),       # 3 input channels: im2col rows (27 of 64 K entries)
    (2, 8, 10, 7, 16, 4, 2),       # 7 input channels (63 entries), 16 output channels
    (2, 9, 8, 1, 128, 2, 3),       # single input channel, N = 128 tiles
])
def test_conv_contractions_full(torch, B, h, w, cin, cout, lw, ld):
    a = synth.images(21, 0, B, (h, w, cin)).astype(np.int64)
    W = synth.int_tensor(22, (cout, 3, 3, cin), *RANGES[lw])
    d = synth.int_tensor(23, (B, h, w, cout), *RANGES[ld])
    conv = nb.Conv3x3(B, h, w, cin, cout)
    try:
        ad, Wd, dd = _dev(torch, a, np.int8), _dev(torch, W, np.int32), _dev(torch, d, np.int32)
        z = torch.empty((B, h, w, cout), dtype=torch.int64, device="cuda")
        conv.contract(nb.NITRO_CONTRACT_FWD, ad, Wd, z)
        assert np.array_equal(z.cpu().numpy(), O.conv3x3_fwd(a, W))
        dw = torch.empty((cout, 3, 3, cin), dtype=torch.int64, device="cuda")
        conv.contract(nb.NITRO_CONTRACT_WGRAD, ad, dd, dw)
        assert np.array_equal(dw.cpu().numpy(), O.conv3x3_wgrad(a, d))
        g = torch.empty((B, h, w, cin), dtype=torch.int64, device="cuda")
        conv.contract(nb.NITRO_CONTRACT_DGRAD, dd, Wd, g)
        assert np.array_equal(g.cpu().numpy(), O.conv3x3_dgrad(d, W))
        assert conv.status() == nb.NITRO_OK
    finally:
        conv.close()


@pytest.mark.parametrize("edge", [127, 128, 32639, 32640, 8355711, 8355712, 2**31 - 1, -2**31])
def test_limb_count_boundaries(torch, edge):
    # operands whose max |x| sits exactly at (or one past) a limb-count boundary
    # of the canonical split; every contraction must stay exact
    B, h, w, c = 2, 8, 8, 64
    a = synth.images(71, 0, B, (h, w, c)).astype(np.int64)
    W = synth.int_tensor(72, (c, 3, 3, c), -100, 100)
    d = synth.int_tensor(73, (B, h, w, c), -100, 100)
    W.flat[5] = edge
    W.flat[-3] = -edge if edge > -2**31 else 2**31 - 1
    d.flat[7] = edge
    conv = nb.Conv3x3(B, h, w, c, c)
    try:
        ad, Wd, dd = _dev(torch, a, np.int8), _dev(torch, W, np.int32), _dev(torch, d, np.int32)
        z = torch.empty((B, h, w, c), dtype=torch.int64, device="cuda")
        conv.contract(nb.NITRO_CONTRACT_FWD, ad, Wd, z)
        assert np.array_equal(z.cpu().numpy(), O.conv3x3_fwd(a, W))
        dw = torch.empty((c, 3, 3, c), dtype=torch.int64, device="cuda")
        conv.contract(nb.NITRO_CONTRACT_WGRAD, ad, dd, dw)
        assert np.array_equal(dw.cpu().numpy(), O.conv3x3_wgrad(a, d))
        g = torch.empty((B, h, w, c), dtype=torch.int64, device="cuda")
        conv.contract(nb.NITRO_CONTRACT_DGRAD, dd, Wd, g)
        # the int64 wrap of an int32 x int32 contraction is the oracle's too
        assert np.array_equal(g.cpu().numpy(), O.conv3x3_dgrad(d, W))
    finally:
        conv.close()


def _patch(x, b, y, xx):
    """3x3 neighbourhood of pixel (y, xx) of image b, zero outside the image."""
    B, H, W, C = x.shape
    p = np.zeros((1, 3, 3, C), dtype=np.int64)
    for dy in range(3):
        for dx in range(3):
            iy, ix = y + dy - 1, xx + dx - 1
            if 0 <= iy < H and 0 <= ix < W:
                p[0, dy, dx] = x[b, iy, ix]
    return p


@pytest.mark.parametrize("B,hw,c", WL.SWEEP_CONV)
def test_conv_sweep_sampled(torch, B, hw, c):
    rng = np.random.default_rng(hw * 1000 + c)
    lw = 1 + (hw + c // 64) % 3              # weights: 1..3 limbs across the sweep
    ld = 4 - (hw + c // 64) % 3              # deltas: 2..4 limbs
    a = synth.images(31, hw, B, (hw, hw, c))
    W = synth.int_tensor(32, (c, 3, 3, c), *RANGES[lw], dtype=np.int32)
    d = synth.int_tensor(33, (B, hw, hw, c), *RANGES[ld], dtype=np.int32)
    conv = nb.Conv3x3(B, hw, hw, c, c)
    try:
        ad, Wd, dd = _dev(torch, a, np.int8), _dev(torch, W, np.int32), _dev(torch, d, np.int32)
        out = torch.empty((B, hw, hw, c), dtype=torch.int64, device="cuda")
        samples = [(int(rng.integers(B)), int(rng.integers(hw)), int(rng.integers(hw)))
                   for _ in range(24)] + [(0, 0, 0), (B - 1, hw - 1, hw - 1)]
        W64 = W.astype(np.int64)
        # forward: z at sampled pixels, all output channels
        conv.contract(nb.NITRO_CONTRACT_FWD, ad, Wd, out)
        z = out.cpu().numpy()
        for b, y, x in samples:
            ref = O.conv3x3_fwd(_patch(a, b, y, x), W64)[0, 1, 1]
            assert np.array_equal(z[b, y, x], ref), ("fwd", b, y, x)
        # input gradient at the same pixels
        conv.contract(nb.NITRO_CONTRACT_DGRAD, dd, Wd, out)
        g = out.cpu().numpy()
        for b, y, x in samples:
            ref = O.conv3x3_dgrad(_patch(d, b, y, x), W64)[0, 1, 1]
            assert np.array_equal(g[b, y, x], ref), ("dgrad", b, y, x)
        # weight gradient: sampled (co, ci) pairs, all nine taps, full batch
        dw = torch.empty((c, 3, 3, c), dtype=torch.int64, device="cuda")
        conv.contract(nb.NITRO_CONTRACT_WGRAD, ad, dd, dw)
        dwh = dw.cpu().numpy()
        for co, ci in [(int(rng.integers(c)), int(rng.integers(c))) for _ in range(4)] + [(c - 1, 0)]:
            ref = O.conv3x3_wgrad(a[..., ci:ci + 1].astype(np.int64), d[..., co:co + 1].astype(np.int64))
            assert np.array_equal(dwh[co, :, :, ci], ref[0, :, :, 0]), ("wgrad", co, ci)
        assert conv.status() == nb.NITRO_OK
    finally:
        conv.close()


@pytest.mark.parametrize("m,n,k,lb", [(1024, 1024, 1024, 1), (1024, 1024, 1024, 3),
                                      (4096, 4096, 4096, 1), (8192, 8192, 8192, 2),
                                      (300, 200, 136, 4), (130, 70, 12, 2),
                                      # few output tiles: K split across CTAs
                                      (64, 3000, 3000, 2), (20, 40, 3000, 3), (64, 1024, 2048, 1)])
def test_int_gemm(torch, m, n, k, lb):
    a = synth.int_tensor(41, (m, k), -128, 127, dtype=np.int8)
    b = synth.int_tensor(42, (n, k), *RANGES[lb], dtype=np.int32)
    gm = nb.IntGemm(m, n, k)
    try:
        c = torch.empty((m, n), dtype=torch.int64, device="cuda")
        gm.run(_dev(torch, a, np.int8), _dev(torch, b, np.int32), c)
        ch = c.cpu().numpy()
        if m * n * k <= 2**30:
            assert np.array_equal(ch, O.linear_fwd(a.astype(np.int64), b.astype(np.int64)))
        else:
            rows = sorted({0, m - 1} | set(np.random.default_rng(m).integers(0, m, 6).tolist()))
            ref = O.linear_fwd(a[rows].astype(np.int64), b.astype(np.int64))
            assert np.array_equal(ch[rows], ref)
        assert gm.status() == nb.NITRO_OK
    finally:
        gm.close()


# every limb at -128 (the canonical split's top limb of an int32 stops at -127)
_ALL_LIMBS_MIN = -128 * (1 + 256 + 65536) - 127 * 2**24


@pytest.mark.parametrize("k", [1024, 576, 3000])
def test_extreme_limb_products_gemm(torch, k):
    # half of the output columns see products of 2^14 in every limb pair, so the
    # exact chunk sums reach 2^24 (1024 products per chunk at k = 1024); the
    # other half stays small: drains with both large and small accumulator
    # values, on either side of the 2^22 range of the add-based conversion
    m, n = 256, 192
    a = np.full((m, k), -128, dtype=np.int8)
    a[1::7] = 127
    b = synth.int_tensor(45, (n, k), -90, 90, dtype=np.int32)
    b[: n // 2] = _ALL_LIMBS_MIN
    b[n // 2: n // 2 + 8] = -128
    gm = nb.IntGemm(m, n, k)
    try:
        c = torch.empty((m, n), dtype=torch.int64, device="cuda")
        gm.run(_dev(torch, a, np.int8), _dev(torch, b, np.int32), c)
        assert np.array_equal(c.cpu().numpy(), O.linear_fwd(a.astype(np.int64), b.astype(np.int64)))
        assert gm.status() == nb.NITRO_OK
    finally:
        gm.close()


def test_extreme_limb_products_conv(torch):
    # the three conv contractions with operands whose limbs all sit at -128 in
    # half of the channels (chunk sums of 576 products of 2^14 = 9.4e6 > 2^22)
    B, h, w, c = 2, 8, 8, 128
    a = np.full((B, h, w, c), -128, dtype=np.int64)
    W = synth.int_tensor(46, (c, 3, 3, c), -90, 90)
    W[: c // 2] = _ALL_LIMBS_MIN
    d = synth.int_tensor(47, (B, h, w, c), -90, 90)
    d[..., : c // 2] = _ALL_LIMBS_MIN
    conv = nb.Conv3x3(B, h, w, c, c)
    try:
        ad, Wd, dd = _dev(torch, a, np.int8), _dev(torch, W, np.int32), _dev(torch, d, np.int32)
        z = torch.empty((B, h, w, c), dtype=torch.int64, device="cuda")
        conv.contract(nb.NITRO_CONTRACT_FWD, ad, Wd, z)
        assert np.array_equal(z.cpu().numpy(), O.conv3x3_fwd(a, W))
        dw = torch.empty((c, 3, 3, c), dtype=torch.int64, device="cuda")
        conv.contract(nb.NITRO_CONTRACT_WGRAD, ad, dd, dw)
        assert np.array_equal(dw.cpu().numpy(), O.conv3x3_wgrad(a, d))
        g = torch.empty((B, h, w, c), dtype=torch.int64, device="cuda")
        conv.contract(nb.NITRO_CONTRACT_DGRAD, dd, Wd, g)
        assert np.array_equal(g.cpu().numpy(), O.conv3x3_dgrad(d, W))
    finally:
        conv.close()
