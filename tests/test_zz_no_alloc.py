"""The allocation-free conv forward against the block forward and the oracle (GPU).

nitro_conv3x3_forward_noalloc serves callers that cannot allocate device
memory while running; it keeps its int64 scratch in a fixed array inside the
library.  This file is named to be collected last, so a run that stops at
the first failure has run every other test before it.
"""
import numpy as np
import pytest

import oracle as O
from paper_2407_11698_gb300 import binding as nb
from paper_2407_11698_gb300 import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def torch():
    t = pytest.importorskip("torch")
    if not t.cuda.is_available():
        pytest.skip("no CUDA device")
    nb.lib()
    return t


def _block_forward(torch, blk, x):
    out = torch.empty((x.shape[0], blk.out_features), dtype=torch.int8, device="cuda")
    blk.forward(x, out)
    return (blk.get(nb.NITRO_T_ACT, 0), blk.get(nb.NITRO_T_REGION, 0),
            blk.get(nb.NITRO_T_ARGMAX, 0) if blk.layers[0][5] else None)


def _oracle_forward(x, w, B, h, wd, cin, cout, pool, alpha):
    """Conv, NITRO-Scaling (SF = 2^8 * 9 * cin), NITRO-ReLU and the optional
    2x2 max-pool, each step from the oracle."""
    z = O.conv3x3_fwd(x.reshape(B, h, wd, cin), w.reshape(cout, 3, 3, cin))
    _, reg, act = O.scale_relu(z, 256 * 9 * cin, alpha)
    am = None
    if pool:
        act, am = O.maxpool_fwd(act)
    return act.reshape(-1), reg.reshape(-1), None if am is None else am.reshape(-1)


def _noalloc_forward(torch, x, w, B, h, wd, cin, cout, pool, alpha, check_memory):
    oh, ow = (h // 2, wd // 2) if pool else (h, wd)
    out = torch.full((B, oh * ow * cout), 99, dtype=torch.int8, device="cuda")
    region = torch.full((B, h * wd * cout), 99, dtype=torch.int8, device="cuda")
    am = torch.full((B, oh * ow * cout), 99, dtype=torch.int8, device="cuda") if pool else None
    torch.cuda.synchronize()
    free0 = torch.cuda.mem_get_info()[0]
    st = nb.nitro_conv3x3_forward_noalloc(nb._ptr(x), nb._ptr(w), B, h, wd, cin, cout, pool, alpha,
                                          nb._ptr(out), nb._ptr(region), nb._ptr(am),
                                          nb._stream_ptr(None))
    assert st == nb.NITRO_OK, nb.status_str(st)
    torch.cuda.synchronize()
    # a call after the first takes no device memory (the first one may: the
    # driver loads the library's fixed array when its address is looked up)
    if check_memory:
        assert torch.cuda.mem_get_info()[0] == free0
    return (out.cpu().numpy().reshape(-1), region.cpu().numpy().reshape(-1),
            None if am is None else am.cpu().numpy().reshape(-1))


def _same(got, want, what):
    for name, g_, w_ in zip(("activations", "region codes", "argmax codes"), got, want):
        if w_ is None:
            assert g_ is None
        else:
            assert np.array_equal(np.asarray(g_, dtype=np.int64), np.asarray(w_, dtype=np.int64)), \
                "%s: %s differ" % (what, name)


@pytest.mark.parametrize("shape", [(16, 28, 28, 1, 32, 1, 10), (5, 7, 9, 6, 11, 1, 4),
                                   (3, 8, 8, 64, 64, 0, 10),
                                   # batch * h * w * cout = 2^21, the array's limit
                                   (32, 32, 32, 3, 64, 1, 10)])
def test_noalloc_matches_block_forward_and_oracle_on_two_calls_in_a_row(torch, shape):
    B, h, wd, cin, cout, pool, alpha = shape
    blk = nb.Block([(nb.NITRO_CONV3X3, cin, cout, h, wd, pool)], h * wd * cin, seed=3,
                   max_batch=B, alpha_inv=alpha)
    try:
        # wide weights (several int8 limbs) as well as the initial ones
        for call, scale in enumerate((1, 70001)):
            w = (blk.get(nb.NITRO_T_W, 0).astype(np.int64) * scale).astype(np.int32)
            blk.set(nb.NITRO_T_W, 0, w)
            xh = synth.images(9, call, B, (h, wd, cin)).reshape(B, -1)
            x = torch.from_numpy(xh).cuda()
            wd_dev = torch.from_numpy(w).cuda()
            got = _noalloc_forward(torch, x, wd_dev, B, h, wd, cin, cout, pool, alpha, call > 0)
            _same(got, _block_forward(torch, blk, x), "call %d vs block forward" % call)
            _same(got, _oracle_forward(xh.astype(np.int64), w.astype(np.int64), B, h, wd, cin,
                                       cout, pool, alpha), "call %d vs oracle" % call)
    finally:
        blk.close()


def test_noalloc_rejects_sizes_beyond_its_array(torch):
    # 2^21 int64 pre-activations at most: 64 x 32 x 32 x 64 = 2^22 is too large
    st = nb.nitro_conv3x3_forward_noalloc(None, None, 64, 32, 32, 64, 64, 0, 10, None, None, None,
                                          nb._stream_ptr(None))
    assert st == nb.NITRO_ERR_ARG


def test_noalloc_call_captures_into_a_cuda_graph(torch):
    # a stream capture in global mode rejects device allocation, so a call
    # that allocated (or freed) would fail to capture; replays of the captured
    # call must give the oracle's outputs for whatever input the buffer holds
    B, h, wd, cin, cout, pool, alpha = 4, 16, 16, 32, 64, 1, 10
    w = synth.int_tensor(81, (cout, 3, 3, cin), -30000, 30000, dtype=np.int32)
    wd_dev = torch.from_numpy(w.reshape(-1)).cuda()
    x = torch.empty((B, h * wd * cin), dtype=torch.int8, device="cuda")
    oh, ow = h // 2, wd // 2
    out = torch.empty((B, oh * ow * cout), dtype=torch.int8, device="cuda")
    region = torch.empty((B, h * wd * cout), dtype=torch.int8, device="cuda")
    am = torch.empty((B, oh * ow * cout), dtype=torch.int8, device="cuda")

    def call(stream):
        return nb.nitro_conv3x3_forward_noalloc(nb._ptr(x), nb._ptr(wd_dev), B, h, wd, cin, cout,
                                                pool, alpha, nb._ptr(out), nb._ptr(region),
                                                nb._ptr(am), nb._stream_ptr(stream))

    x.copy_(torch.from_numpy(synth.images(12, 0, B, (h, wd, cin)).reshape(B, -1)))
    assert call(None) == nb.NITRO_OK      # the first call looks the array's address up
    torch.cuda.synchronize()
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.stream(side):
        with torch.cuda.graph(graph, stream=side):
            st = call(side)
    torch.cuda.current_stream().wait_stream(side)
    assert st == nb.NITRO_OK, nb.status_str(st)
    for k in range(1, 3):
        xh = synth.images(12, k, B, (h, wd, cin)).reshape(B, -1)
        x.copy_(torch.from_numpy(xh))
        graph.replay()
        torch.cuda.synchronize()
        got = (out.cpu().numpy().reshape(-1), region.cpu().numpy().reshape(-1),
               am.cpu().numpy().reshape(-1))
        _same(got, _oracle_forward(xh.astype(np.int64), w.astype(np.int64), B, h, wd, cin, cout,
                                   pool, alpha), "replay %d vs oracle" % k)
