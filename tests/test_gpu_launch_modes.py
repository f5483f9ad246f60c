"""Launch modes of the library kernels against the oracle: programmatic
dependent launch inside a CUDA graph (each block on its own stream, fresh
inputs copied into the captured buffers before every replay, as a training
loop drives it), and plain stream order (NITRO_PDL=0, read once per process,
so it runs in a child process)."""
import os
import subprocess
import sys

import numpy as np
import pytest

from paper_2407_11698_gb300 import binding as nb
from paper_2407_11698_gb300 import synth
from paper_2407_11698_gb300 import workloads as WL

from netpair import NetPair

pytestmark = pytest.mark.gpu

HERE = os.path.dirname(os.path.abspath(__file__))


@pytest.fixture(scope="module")
def torch():
    t = pytest.importorskip("torch")
    if not t.cuda.is_available():
        pytest.skip("no CUDA device")
    nb.lib()
    return t


@pytest.mark.parametrize("name,batch,steps", [("cnn_32_64_b64", 64, 4),
                                              ("vgg_64_128_256_b128", 32, 6)])
def test_graph_replays_on_block_streams(torch, name, batch, steps):
    wl = WL.WORKLOADS[name]
    pair = NetPair(wl["blocks"], batch, seed=20240716, **wl.get("hyper", {}))
    try:
        B = batch
        xs = torch.empty((B, int(np.prod(wl["input_shape"]))), dtype=torch.int8, device="cuda")
        ys = torch.empty((B,), dtype=torch.int32, device="cuda")
        acts = [xs] + [torch.empty((B, g.out_features), dtype=torch.int8, device="cuda")
                       if g.layers else None for g in pair.gb]
        for i in range(1, len(acts)):
            if acts[i] is None:
                acts[i] = acts[i - 1]
        losses = torch.zeros((len(pair.gb),), dtype=torch.int64, device="cuda")
        streams = [torch.cuda.Stream() for _ in pair.gb]
        done = [torch.cuda.Event() for _ in pair.gb]

        def step():
            main = torch.cuda.current_stream()
            for i, (g, s) in enumerate(zip(pair.gb, streams)):
                s.wait_stream(main)
                if i:
                    s.wait_event(done[i - 1])
                g.forward(acts[i], acts[i + 1] if g.layers else None, stream=s)
                done[i].record(s)
                g.backward(acts[i], ys, losses[i:i + 1], stream=s)
                g.sgd(stream=s)
            for s in streams:
                main.wait_stream(s)

        def load(k):
            x = synth.images(11, k, B, wl["input_shape"])
            y = synth.labels(11, k, B)
            xs.copy_(torch.from_numpy(np.ascontiguousarray(x).reshape(B, -1)))
            ys.copy_(torch.from_numpy(y.astype(np.int32)))
            return x, y

        x, y = load(0)                            # eager step 0
        step()
        torch.cuda.synchronize()
        assert losses.cpu().tolist() == pair.step_oracle(x, y)
        pair.compare("eager step 0")
        side = torch.cuda.Stream()
        side.wait_stream(torch.cuda.current_stream())
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.stream(side):
            with torch.cuda.graph(graph, stream=side):
                step()
        torch.cuda.current_stream().wait_stream(side)
        torch.cuda.synchronize()
        for k in range(1, steps):
            x, y = load(k)
            graph.replay()
            torch.cuda.synchronize()
            assert losses.cpu().tolist() == pair.step_oracle(x, y), k
            pair.compare("replay %d" % k)
    finally:
        pair.close()


def test_stream_ordered_launch_matches_oracle(torch):
    code = ("import sys; sys.path.insert(0, %r); sys.path.insert(0, %r)\n"
            "from netpair import run_workload\n"
            "from paper_2407_11698_gb300 import workloads as WL\n"
            "run_workload(WL.WORKLOADS['cnn_32_64_b64'], steps=6, check_every=2, concurrent=True)\n"
            "run_workload(WL.WORKLOADS['vgg_64_128_256_b128'], steps=5, batch=16)\n"
            "print('ok')\n") % (HERE, os.path.dirname(HERE))
    env = dict(os.environ, NITRO_PDL="0")
    r = subprocess.run([sys.executable, "-c", code], env=env, capture_output=True, text=True,
                       timeout=900)
    assert r.returncode == 0 and r.stdout.strip().endswith("ok"), r.stdout[-2000:] + r.stderr[-4000:]
