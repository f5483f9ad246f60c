"""Run the same network on the GPU library and on the oracle, step by step,
and compare every tensor the ABI exposes (test helper)."""
import numpy as np

import oracle as O
from paper_2407_11698_gb300 import binding as nb
from paper_2407_11698_gb300 import synth


def _torch():
    import torch
    return torch


class NetPair:
    def __init__(self, blocks, batch, seed=1000, concurrent=False, fused_update=False, **hyper):
        self.batch = batch
        self.spec = blocks
        self.concurrent = concurrent   # a stream per block, as bench.py drives them
        self.fused_update = fused_update   # backward and update in one call
        self.ob = [O.OracleBlock([O.LayerDesc(*l) for l in b["layers"]],
                                 in_features=b["in_features"], seed=seed + i, **hyper)
                   for i, b in enumerate(blocks)]
        self.gb = [nb.Block(b["layers"], b["in_features"], seed=seed + i, max_batch=batch, **hyper)
                   for i, b in enumerate(blocks)]

    def close(self):
        for g in self.gb:
            g.close()

    def step_gpu(self, x, y):
        torch = _torch()
        xs = torch.from_numpy(np.ascontiguousarray(x)).cuda()
        ys = torch.from_numpy(np.ascontiguousarray(y).astype(np.int32)).cuda()
        B = xs.shape[0]
        acts = [xs.reshape(B, -1)]
        for g in self.gb:
            out = torch.empty((B, max(1, g.out_features)), dtype=torch.int8, device="cuda") \
                if g.layers else None
            acts.append(out if out is not None else acts[-1])
        losses = [torch.full((1,), -7, dtype=torch.int64, device="cuda") for _ in self.gb]
        if self.concurrent:
            # block i+1's forward waits only for block i's forward; each block's
            # backward and update run on its own stream alongside the others
            main = torch.cuda.current_stream()
            streams = [torch.cuda.Stream() for _ in self.gb]
            done = [torch.cuda.Event() for _ in self.gb]
            for i, (g, s) in enumerate(zip(self.gb, streams)):
                s.wait_stream(main)
                if i:
                    s.wait_event(done[i - 1])
                g.forward(acts[i], acts[i + 1] if g.layers else None, stream=s)
                done[i].record(s)
                if self.fused_update:
                    g.backward_update(acts[i], ys, losses[i], stream=s)
                else:
                    g.backward(acts[i], ys, losses[i], stream=s)
                    g.sgd(stream=s)
            for s in streams:
                main.wait_stream(s)
        else:
            for i, g in enumerate(self.gb):
                g.forward(acts[i], acts[i + 1] if g.layers else None)
            if self.fused_update:
                for i, g in enumerate(self.gb):
                    g.backward_update(acts[i], ys, losses[i])
            else:
                for i, g in enumerate(self.gb):
                    g.backward(acts[i], ys, losses[i])
                for g in self.gb:
                    g.sgd()
        torch.cuda.synchronize()
        return [int(l.item()) for l in losses]

    def step_oracle(self, x, y):
        return O.train_step(self.ob, x.astype(np.int64), y.astype(np.int64))

    def step(self, x, y):
        gl = self.step_gpu(x, y)
        ol = self.step_oracle(x, y)
        return gl, ol

    def compare(self, where=""):
        """Asserts bit-exact equality of every exposed tensor."""
        for bi, (o, g) in enumerate(zip(self.ob, self.gb)):
            tag = "%s block %d" % (where, bi)
            for i, L in enumerate(o.layers):
                _eq(g.get(nb.NITRO_T_W, i, check=False), o.W[i], tag + " W%d" % i)
                _eq(g.get(nb.NITRO_T_DW, i, check=False), o.dW[i], tag + " dW%d" % i)
                _eq(g.get(nb.NITRO_T_ACT, i, check=False), o.act[i], tag + " act%d" % i)
                _eq(g.get(nb.NITRO_T_REGION, i, check=False), o.region[i], tag + " region%d" % i)
                if L.pool:
                    _eq(g.get(nb.NITRO_T_ARGMAX, i, check=False), o.argmax[i], tag + " argmax%d" % i)
                _eq(g.get(nb.NITRO_T_DELTA, i, check=False), o.delta[i], tag + " delta%d" % i)
            _eq(g.get(nb.NITRO_T_WLR, 0, check=False), o.Wlr, tag + " Wlr")
            _eq(g.get(nb.NITRO_T_DWLR, 0, check=False), o.dWlr, tag + " dWlr")
            _eq(g.get(nb.NITRO_T_GRAD_L, 0, check=False), o.grad_l, tag + " grad_l")
            _eq(g.get(nb.NITRO_T_SSE, 0, check=False), np.array([o.sse]), tag + " sse")
            if getattr(o, "lr_in", None) is not None:
                _eq(g.get(nb.NITRO_T_LR_IN, 0, check=False), o.lr_in, tag + " lr_in")
                _eq(g.get(nb.NITRO_T_LR_ARGMAX, 0, check=False), o.lr_argmax, tag + " lr_argmax")
            _eq(g.get(nb.NITRO_T_STEP, 0, check=False), np.array([o.t]), tag + " step")
            assert g.status_bits() == o.status, "%s status %d vs %d" % (tag, g.status_bits(), o.status)


def _eq(got, want, what):
    want = np.asarray(want, dtype=np.int64).reshape(-1)
    got = np.asarray(got, dtype=np.int64).reshape(-1)
    assert got.shape == want.shape, "%s: shape %s vs %s" % (what, got.shape, want.shape)
    if not np.array_equal(got, want):
        bad = np.nonzero(got != want)[0]
        raise AssertionError("%s: %d of %d differ; first at %d: gpu %d oracle %d" % (
            what, bad.size, want.size, bad[0], got[bad[0]], want[bad[0]]))


def run_workload(wl, steps, seed=20240716, check_every=1, data_seed=7, concurrent=False,
                 batch=None, fused_update=False, **hyper):
    batch = batch or wl["batch"]
    hyper = dict(wl.get("hyper", {}), **hyper)
    pair = NetPair(wl["blocks"], batch, seed=seed, concurrent=concurrent,
                   fused_update=fused_update, **hyper)
    try:
        for s in range(steps):
            x = synth.images(data_seed, s, batch, wl["input_shape"])
            y = synth.labels(data_seed, s, batch)
            gl, ol = pair.step(x, y)
            assert gl == ol, "step %d losses gpu %s oracle %s" % (s, gl, ol)
            if (s + 1) % check_every == 0 or s == steps - 1:
                pair.compare("step %d" % s)
    finally:
        pair.close()
