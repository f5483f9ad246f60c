"""GPU parity of the integer data pre-processing (App. A) against the oracle.

mu and omega must equal the oracle's exactly and x_hat element by element
(bit-exact int8), for sizes around the 16-byte vector width, every start
offset within a 16-byte boundary, input / output at matching and differing
offsets (vector and byte paths), in place, the degenerate omega = 0 case, the
dataset shapes of MNIST (60000 x 28 x 28) and CIFAR-10 (50000 x 32 x 32 x 3),
and under CUDA-graph capture.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

import oracle as O
from paper_2407_11698_gb300 import binding as nb
from paper_2407_11698_gb300 import synth


@pytest.fixture(scope="module")
def prep():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    p = nb.IntPrep()
    yield p
    p.close()


def _device_view(x, off):
    """uint8 device tensor holding x that starts `off` bytes past a 256-byte
    boundary (a slice of a larger allocation)."""
    buf = torch.zeros(x.size + off + 16, dtype=torch.uint8, device="cuda")
    v = buf[off:off + x.size]
    v.copy_(torch.from_numpy(x))
    return v


def _out_view(n, off):
    buf = torch.full((n + off + 16,), 99, dtype=torch.int8, device="cuda")
    return buf, buf[off:off + n]


def _check(prep, x, xoff=0, ooff=0):
    mu, om = O.prep_stats(x)
    want = O.prep_apply(x, mu, om)
    xd = _device_view(x, xoff)
    prep.fit(xd)
    assert prep.stats() == (mu, om)
    buf, out = _out_view(x.size, ooff)
    prep.apply(xd, out)
    torch.cuda.synchronize()
    got = out.cpu().numpy()
    assert np.array_equal(got, want), int(np.flatnonzero(got != want)[0])
    # nothing written outside the output range
    b = buf.cpu().numpy()
    assert (b[:ooff] == 99).all() and (b[ooff + x.size:] == 99).all()


@pytest.mark.parametrize("n", [1, 2, 15, 16, 17, 31, 33, 4096 + 7, (1 << 20) + 13])
@pytest.mark.parametrize("kind", ["natural", "digits", "uniform"])
def test_sizes(prep, n, kind):
    _check(prep, synth.raw_pixels(7 + n, n, kind))


@pytest.mark.parametrize("xoff", [0, 1, 7, 15])
@pytest.mark.parametrize("ooff", [0, 1, 8])
def test_offsets(prep, xoff, ooff):
    _check(prep, synth.raw_pixels(11, 100003, "natural"), xoff, ooff)


def test_constant_data_omega_zero(prep):
    x = synth.raw_pixels(0, 5000, "constant")
    _check(prep, x)
    assert prep.stats() == (77, 0)


def test_in_place(prep):
    x = synth.raw_pixels(5, (1 << 16) + 3, "digits")
    mu, om = O.prep_stats(x)
    xd = _device_view(x, 3)
    prep.fit(xd)
    prep.apply(xd, xd.view(torch.int8))
    torch.cuda.synchronize()
    assert np.array_equal(xd.view(torch.int8).cpu().numpy(), O.prep_apply(x, mu, om))


def test_test_set_uses_training_statistics(prep):
    train = synth.raw_pixels(21, 300007, "natural")
    test = synth.raw_pixels(22, 100003, "digits")
    mu, om = O.prep_stats(train)
    prep.fit(_device_view(train, 0))
    out = torch.empty(test.size, dtype=torch.int8, device="cuda")
    prep.apply(_device_view(test, 5), out)
    torch.cuda.synchronize()
    assert np.array_equal(out.cpu().numpy(), O.prep_apply(test, mu, om))


@pytest.mark.parametrize("name,shape,kind", [("mnist", (60000, 28, 28), "digits"),
                                              ("cifar10", (50000, 32, 32, 3), "natural")])
def test_full_dataset_shapes(prep, name, shape, kind):
    _check(prep, synth.raw_pixels(3, int(np.prod(shape)), kind))


def test_graph_capture(prep):
    x = synth.raw_pixels(9, (1 << 22) + 5, "natural")
    mu, om = O.prep_stats(x)
    xd = _device_view(x, 0)
    out = torch.empty(x.size, dtype=torch.int8, device="cuda")
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        prep.fit(xd, stream=s)          # warm-up outside the capture
        prep.apply(xd, out, stream=s)
    s.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        prep.fit(xd, stream=s)
        prep.apply(xd, out, stream=s)
    out.zero_()
    g.replay()
    torch.cuda.synchronize()
    assert prep.stats() == (mu, om)
    assert np.array_equal(out.cpu().numpy(), O.prep_apply(x, mu, om))


def test_kernels_ran(prep):
    n0 = nb.lib().nitro_kernel_launches()
    x = synth.raw_pixels(1, 1000, "uniform")
    xd = _device_view(x, 0)
    prep.fit(xd)
    prep.apply(xd, torch.empty(1000, dtype=torch.int8, device="cuda"))
    torch.cuda.synchronize()
    assert nb.lib().nitro_kernel_launches() - n0 == 3
