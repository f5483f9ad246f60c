"""Failure path of the bounded device waits (GPU).

Every mbarrier wait of the tensor-core kernels is bounded in time; when the
bound runs out the kernel raises the TIMEOUT status bit, the CTA's other roles
leave, TMEM is freed and the kernel returns.  nitro_block_diag_timeout queues a
CTA that waits, through the same wait code, on a barrier nothing completes, so
the bound must run out.  No GPU fault or hang is involved: the wait gives up
after the given limit and the context stays usable.
"""
import time

import pytest

from paper_2407_11698_gb300 import binding as nb
from paper_2407_11698_gb300 import synth

from netpair import NetPair

pytestmark = pytest.mark.gpu

C = nb.NITRO_CONV3X3
# conv 4 -> 64 @ 16x16 with pool, conv 64 -> 64 @ 8x8 (tensor-core layers),
# then the output block
BLOCKS = [{"layers": [(C, 4, 64, 16, 16, 1), (C, 64, 64, 8, 8, 0)], "in_features": 16 * 16 * 4},
          {"layers": [], "in_features": 8 * 8 * 64}]


@pytest.fixture(scope="module")
def torch():
    t = pytest.importorskip("torch")
    if not t.cuda.is_available():
        pytest.skip("no CUDA device")
    nb.lib()
    return t


def _step(pair, s):
    x = synth.images(13, s, pair.batch, (16, 16, 4))
    y = synth.labels(13, s, pair.batch)
    gl, ol = pair.step(x, y)
    assert gl == ol, "step %d losses gpu %s oracle %s" % (s, gl, ol)
    pair.compare("step %d" % s)


@pytest.mark.parametrize("wait_us", [1000, 20000])
def test_wait_that_never_completes_gives_up_with_timeout(torch, wait_us):
    pair = NetPair(BLOCKS, 8, seed=77)
    try:
        _step(pair, 0)
        blk = pair.gb[0]
        assert blk.status() == nb.NITRO_OK
        t0 = time.perf_counter()
        blk.diag_timeout(wait_us)
        st = blk.status()                      # synchronises the device
        elapsed = time.perf_counter() - t0
        assert st == nb.NITRO_ERR_TIMEOUT
        assert blk.status_bits() & nb.STATUS_BIT_TIMEOUT
        # the waiting warp gave up at its own short limit, and the other roles
        # left on its abort flag instead of running out their 2 s bound
        assert elapsed >= wait_us * 1e-6
        assert elapsed < 1.5
        # the other block's status word is untouched
        assert pair.gb[1].status() == nb.NITRO_OK
        # clearing returns the latched status once, then the word reads OK
        assert blk.status(clear=True) == nb.NITRO_ERR_TIMEOUT
        assert blk.status() == nb.NITRO_OK
        # the context and the block's state are intact: the next training
        # steps are still bit-exact with the oracle
        _step(pair, 1)
        _step(pair, 2)
    finally:
        pair.close()


def test_timeout_probe_rejects_out_of_range_limits(torch):
    blk = nb.Block([], 10, seed=1, max_batch=1)
    try:
        for bad in (0, -5, 2000001):
            assert nb.lib().nitro_block_diag_timeout(blk.h, bad, nb._stream_ptr(None)) == \
                nb.NITRO_ERR_ARG
    finally:
        blk.close()
    assert nb.lib().nitro_block_diag_timeout(None, 1000, nb._stream_ptr(None)) == nb.NITRO_ERR_ARG
