"""Caller buffers need only the alignment of their element type: the block
step and the kernel-level contractions give the same results for input,
output and operand pointers offset by one element into a larger buffer as for
freshly allocated (256-byte aligned) ones, and the contractions stay equal to
the oracle."""
import numpy as np
import pytest

import oracle as O
from paper_2407_11698_gb300 import binding as nb
from paper_2407_11698_gb300 import synth

pytestmark = pytest.mark.gpu
C = nb.NITRO_CONV3X3


@pytest.fixture(scope="module")
def torch():
    t = pytest.importorskip("torch")
    if not t.cuda.is_available():
        pytest.skip("no CUDA device")
    nb.lib()
    return t


def _at(torch, arr, dtype, shift):
    """Device copy of `arr` starting `shift` elements into a larger buffer."""
    host = torch.from_numpy(np.ascontiguousarray(arr).astype(dtype).reshape(-1))
    buf = torch.zeros(host.numel() + 32, dtype=host.dtype, device="cuda")
    view = buf[shift:shift + host.numel()]
    view.copy_(host.cuda())
    return view.view(*arr.shape)


def _empty_at(torch, shape, dtype, shift):
    n = int(np.prod(shape))
    buf = torch.zeros(n + 32, dtype=dtype, device="cuda")
    return buf[shift:shift + n].view(*shape)


@pytest.mark.parametrize("layers,in_shape", [
    ([(C, 64, 64, 8, 8, 1)], (8, 8, 64)),      # tcgen05 forward, vector input pack
    ([(C, 3, 64, 8, 8, 0)], (8, 8, 3)),        # im2col rows
    ([(C, 3, 16, 6, 6, 1)], (6, 6, 3)),        # CUDA-core narrow-input forward
])
def test_block_step_with_offset_buffers(torch, layers, in_shape):
    B = 5
    feat = int(np.prod(in_shape))
    x = synth.images(7, 0, B, (feat,))
    y = synth.labels(7, 0, B)
    results = []
    for shift in (0, 1, 3):
        blk = nb.Block(layers, feat, seed=4, max_batch=B)
        try:
            xd = _at(torch, x, np.int8, shift)
            yd = _at(torch, y, np.int32, 1 if shift else 0)
            out = _empty_at(torch, (B, blk.out_features), torch.int8, shift)
            loss = _empty_at(torch, (1,), torch.int64, 1 if shift else 0)
            blk.forward(xd, out)
            blk.backward(xd, yd, loss)
            blk.sgd()
            torch.cuda.synchronize()
            act = blk.get(nb.NITRO_T_ACT, 0, check=False)
            assert np.array_equal(out.cpu().numpy().reshape(-1), act)
            results.append((act, blk.get(nb.NITRO_T_W, 0, check=False),
                            blk.get(nb.NITRO_T_DELTA, 0, check=False), int(loss.item())))
        finally:
            blk.close()
    for r in results[1:]:
        assert all(np.array_equal(a, b) for a, b in zip(results[0][:3], r[:3]))
        assert r[3] == results[0][3]


@pytest.mark.parametrize("B,h,w,cin,cout", [(2, 8, 8, 64, 64), (2, 9, 8, 3, 64)])
def test_contractions_with_offset_operands(torch, B, h, w, cin, cout):
    a = synth.images(51, 0, B, (h, w, cin)).astype(np.int64)
    W = synth.int_tensor(52, (cout, 3, 3, cin), -2**20, 2**20)
    d = synth.int_tensor(53, (B, h, w, cout), -2**30, 2**30)
    conv = nb.Conv3x3(B, h, w, cin, cout)
    try:
        ad = _at(torch, a, np.int8, 1)
        Wd = _at(torch, W, np.int32, 1)
        dd = _at(torch, d, np.int32, 1)
        z = _empty_at(torch, (B, h, w, cout), torch.int64, 1)
        conv.contract(nb.NITRO_CONTRACT_FWD, ad, Wd, z)
        assert np.array_equal(z.cpu().numpy(), O.conv3x3_fwd(a, W))
        dw = _empty_at(torch, (cout, 3, 3, cin), torch.int64, 1)
        conv.contract(nb.NITRO_CONTRACT_WGRAD, ad, dd, dw)
        assert np.array_equal(dw.cpu().numpy(), O.conv3x3_wgrad(a, d))
        g = _empty_at(torch, (B, h, w, cin), torch.int64, 1)
        conv.contract(nb.NITRO_CONTRACT_DGRAD, dd, Wd, g)
        assert np.array_equal(g.cpu().numpy(), O.conv3x3_dgrad(d, W))
        assert conv.status() == nb.NITRO_OK
    finally:
        conv.close()


def test_gemm_with_offset_operands(torch):
    m, n, k = 130, 72, 64
    a = synth.int_tensor(61, (m, k), -128, 127, dtype=np.int8)
    b = synth.int_tensor(62, (n, k), -2**31, 2**31 - 1, dtype=np.int32)
    gm = nb.IntGemm(m, n, k)
    try:
        c = _empty_at(torch, (m, n), torch.int64, 1)
        gm.run(_at(torch, a, np.int8, 3), _at(torch, b, np.int32, 1), c)
        assert np.array_equal(c.cpu().numpy(), O.linear_fwd(a.astype(np.int64), b.astype(np.int64)))
        assert gm.status() == nb.NITRO_OK
    finally:
        gm.close()
