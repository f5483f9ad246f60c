#!/usr/bin/env python
"""Benchmark of the NITRO-D integer training step on GB300.

One step = forward of every block, every block's local backward and every
IntegerSGD update (the full local-loss block step) on one batch of synthetic
int8 images resident in HBM, for the VGG-style workload (3 blocks of two 3x3
convs 64/128/256 with max-pool + an output block, batch 128, 32x32x3 inputs).

Prints ONE JSON line on rank 0.  Multi-GPU runs (torchrun) train independent
replicas, one per GPU (the step has no exchange; weak scaling).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
"""
import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "int training images/s at 1 GB300; int conv TOPS as % of dense int8 peak"
WORKLOAD = "vgg_64_128_256_b128"
L2_FLUSH_BYTES = 512 << 20          # > 129 MB L2


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=20)
    p.add_argument("--warmup", type=int, default=5)
    p.add_argument("--impl", choices=["ours", "reference"], default="ours")
    from paper_2407_11698_gb300 import workloads as WL
    p.add_argument("--workload", default=WORKLOAD, choices=sorted(WL.WORKLOADS))
    p.add_argument("--no-graph", action="store_true")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--sequential-blocks", action="store_true",
                   help="run all blocks on one stream (default: a stream per block)")
    p.add_argument("--fused-update", action="store_true",
                   help="backward and IntegerSGD in one call (nitro_block_backward_update: the "
                        "update folded into weight-gradient kernels without a K split); "
                        "default: the two calls, measured faster")
    p.add_argument("--profile-steps", type=int, default=3)
    p.add_argument("--sweep", action="store_true",
                   help="time the kernel sweep (conv contractions, integer GEMM, IntegerSGD, "
                        "pre-processing) instead")
    p.add_argument("--sweep-parts", default="conv,gemm,sgd,prep",
                   help="comma-separated subset of the sweep to run")
    return p.parse_args()


def ncu_traffic(kernel, workload=WORKLOAD):
    """Per-launch DRAM bytes of `kernel` from the committed ncu summary, or None
    when the kernel source changed since the counters were taken or the
    workload is not the one the summary covers."""
    import hashlib
    if workload != WORKLOAD:
        return None
    try:
        src = open(os.path.join(ROOT, "paper_2407_11698_gb300", "csrc", "tc_conv.cu"), "rb").read()
        sha = hashlib.sha1(src).hexdigest()[:12]
        for line in open(os.path.join(ROOT, "profiles", "tc_conv_kernels_vgg_step.md")):
            parts = line.split()
            if len(parts) == 4 and parts[0] == "traffic" and parts[1] == kernel:
                return int(parts[2]) if parts[3] == "sha1=" + sha else None
    except OSError:
        pass
    return None


def measured_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return json.load(f), "measured"
    except OSError:
        return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}, "fallback"


# ------------------------------------------------------------------ clocks
class ClockSampler:
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.proc = None
        self.lines = []

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), "--query-gpu=" + self.FIELDS,
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except OSError:
            self.proc = None
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def __exit__(self, *a):
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in self.lines:
            parts = [t.strip() for t in line.split(",")]
            if len(parts) < 7:
                continue
            try:
                sm.append(float(parts[0]))
                mx.append(float(parts[1]))
            except ValueError:
                continue
            for n, v in zip(names, parts[3:7]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


# ------------------------------------------------------------------ ranks
def max_over_ranks(ms, world, device):
    """The slowest rank's time: every rank contributes its own `ms` and gets
    back the maximum (a MAX all-reduce when world > 1)."""
    import torch
    t = torch.tensor([float(ms)], dtype=torch.float64, device=device)
    if world > 1:
        import torch.distributed as dist
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_rate(units_per_rank, world, steps, max_ms):
    """Whole-job throughput: units processed by all ranks over `steps` steps
    divided by the slowest rank's time (weak scaling: per-rank work fixed)."""
    return world * units_per_rank * steps / (max_ms / 1e3)


# ------------------------------------------------------------------ our step
class GpuNet:
    """A chain of block handles driven through the public calls.  With
    `concurrent`, every block runs on its own stream: block i+1's forward waits
    only for block i's forward, so block i's backward and update overlap the
    blocks after it (blocks exchange no gradients, Sec. 3.3)."""

    def __init__(self, wl, seed, torch, nb, concurrent=True, fused_update=False):
        self.torch, self.nb = torch, nb
        self.fused_update = fused_update
        B = wl["batch"]
        self.B = B
        self.blocks = [nb.Block(b["layers"], b["in_features"], seed=seed + i, max_batch=B,
                                **wl.get("hyper", {}))
                       for i, b in enumerate(wl["blocks"])]
        from paper_2407_11698_gb300 import synth
        x = synth.images(seed, 0, B, wl["input_shape"]).reshape(B, -1)
        y = synth.labels(seed, 0, B)
        self.x = torch.from_numpy(x).cuda()
        self.y = torch.from_numpy(y).cuda()
        self.acts = [self.x]
        for g in self.blocks:
            self.acts.append(torch.empty((B, g.out_features), dtype=torch.int8, device="cuda")
                             if g.layers else self.acts[-1])
        self.loss = torch.zeros((len(self.blocks),), dtype=torch.int64, device="cuda")
        self.in_bytes = self.x.numel() + 4 * self.y.numel()
        self.streams = [torch.cuda.Stream() for _ in self.blocks] if concurrent else None
        self.fwd_done = [torch.cuda.Event() for _ in self.blocks] if concurrent else None

    def step(self, x=None, y=None, loss=None, sequential=False):
        x = self.x if x is None else x
        y = self.y if y is None else y
        loss = self.loss if loss is None else loss
        acts = [x] + self.acts[1:]
        if not self.streams or sequential:
            for i, g in enumerate(self.blocks):
                g.forward(acts[i], acts[i + 1] if g.layers else None)
            if self.fused_update:
                for i, g in enumerate(self.blocks):
                    g.backward_update(acts[i], y, loss[i:i + 1])
                return
            for i, g in enumerate(self.blocks):
                g.backward(acts[i], y, loss[i:i + 1])
            for g in self.blocks:
                g.sgd()
            return
        main = self.torch.cuda.current_stream()
        for i, (g, s) in enumerate(zip(self.blocks, self.streams)):
            s.wait_stream(main)                      # inputs, labels
            if i:
                s.wait_event(self.fwd_done[i - 1])   # the block's input activations
            g.forward(acts[i], acts[i + 1] if g.layers else None, stream=s)
            self.fwd_done[i].record(s)
            if self.fused_update:
                g.backward_update(acts[i], y, loss[i:i + 1], stream=s)
            else:
                g.backward(acts[i], y, loss[i:i + 1], stream=s)
                g.sgd(stream=s)
        for s in self.streams:
            main.wait_stream(s)


def kernel_profile(nb):
    import ctypes
    L = nb.lib()
    out = {}
    for k in range(L.nitro_profile_kernel_count()):
        n, ms, ops, by = ctypes.c_uint64(), ctypes.c_double(), ctypes.c_double(), ctypes.c_double()
        st = L.nitro_profile_read(k, ctypes.byref(n), ctypes.byref(ms), ctypes.byref(ops), ctypes.byref(by))
        if st == 0 and n.value:
            out[L.nitro_profile_kernel_name(k).decode()] = dict(
                launches=n.value, ms=ms.value, ops=ops.value, bytes=by.value)
    return out


def _limbs(m):
    """Signed 8-bit limbs the kernels use for a tensor with max |x| = m."""
    m = int(m)
    return 1 if m <= 127 else 2 if m <= 32639 else 3 if m <= 8355711 else 4


def issued_profile(nb, net, flush, steps, torch):
    """Issued tensor work of the tcgen05 contractions over `steps` eager steps:
    each launch's algorithmic ops times the product of its operands' limb
    counts (activations 1; W and delta from the layers' max |.|, W read before
    the step, delta after it).  Launches map to layers by order: every conv's
    forward in network order, then per block, last layer first, its weight
    gradient and (above the block's first layer) its input gradient (the order
    of the separate update).  Returns {kernel: {"issued_ops", "ms"}} or None
    when the launches do not match."""
    import ctypes
    import numpy as np
    L = nb.lib()
    convs = [(bi, i) for bi, g in enumerate(net.blocks) for i, l in enumerate(g.layers)
             if l[0] == nb.NITRO_CONV3X3]
    bwd = []
    for bi, g in enumerate(net.blocks):
        for i in reversed(range(len(g.layers))):
            if g.layers[i][0] != nb.NITRO_CONV3X3:
                continue
            bwd.append(("tc_conv_wgrad", bi, i))
            if i > 0:
                bwd.append(("tc_conv_dgrad", bi, i))

    def maxabs(bi, which, i):
        return np.abs(net.blocks[bi].get(which, i, check=False).astype(np.int64)).max()

    out = {}
    for _ in range(steps):
        wl = {c: _limbs(maxabs(c[0], nb.NITRO_T_W, c[1])) for c in convs}
        L.nitro_profile_reset()
        L.nitro_profile_enable(1)
        flush.zero_()
        net.step(sequential=True)
        torch.cuda.synchronize()
        L.nitro_profile_enable(0)
        dl = {c: _limbs(maxabs(c[0], nb.NITRO_T_DELTA, c[1])) for c in convs}
        recs = []
        for r in range(L.nitro_profile_record_count()):
            k, ms, ops, by = ctypes.c_int(), ctypes.c_double(), ctypes.c_double(), ctypes.c_double()
            L.nitro_profile_record(r, ctypes.byref(k), ctypes.byref(ms), ctypes.byref(ops), ctypes.byref(by))
            recs.append((L.nitro_profile_kernel_name(k.value).decode(), ms.value, ops.value))
        L.nitro_profile_reset()
        fwd = [r for r in recs if r[0] == "tc_conv_fwd"]
        back = [r for r in recs if r[0] in ("tc_conv_wgrad", "tc_conv_dgrad")]
        if len(fwd) != len(convs) or [r[0] for r in back] != [b[0] for b in bwd]:
            return None
        for r, c in zip(fwd, convs):
            o = out.setdefault("tc_conv_fwd", {"issued_ops": 0.0, "ms": 0.0})
            o["issued_ops"] += r[2] * wl[c]
            o["ms"] += r[1]
        for r, (name, bi, i) in zip(back, bwd):
            o = out.setdefault(name, {"issued_ops": 0.0, "ms": 0.0})
            f = dl[(bi, i)] * (wl[(bi, i)] if name == "tc_conv_dgrad" else 1)
            o["issued_ops"] += r[2] * f
            o["ms"] += r[1]
    return out


def run_ours(args, rank, world, local_rank):
    import torch
    import torch.distributed as dist
    from paper_2407_11698_gb300 import binding as nb
    from paper_2407_11698_gb300 import workloads as WL

    torch.cuda.set_device(local_rank)
    nb.lib()
    wl = WL.WORKLOADS[args.workload]
    net = GpuNet(wl, 20240716 + 7 * rank, torch, nb, concurrent=not args.sequential_blocks,
                 fused_update=args.fused_update)
    stream = torch.cuda.current_stream()
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device="cuda")

    for _ in range(args.warmup):
        net.step()
    torch.cuda.synchronize()

    # launches per step (host-side counter around one eager step)
    L = nb.lib()
    c0 = L.nitro_kernel_launches()
    net.step()
    torch.cuda.synchronize()
    launches_per_step = L.nitro_kernel_launches() - c0

    graph = None
    if not args.no_graph:
        graph = torch.cuda.CUDAGraph()
        side = torch.cuda.Stream()
        side.wait_stream(stream)
        with torch.cuda.stream(side):
            with torch.cuda.graph(graph, stream=side):
                net.step()
        stream.wait_stream(side)
        for _ in range(2):
            graph.replay()
        torch.cuda.synchronize()

    def one():
        if graph is not None:
            graph.replay()
        else:
            net.step()

    # ---------------- headline timed region: K steps, L2 flushed between steps
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(args.steps)]
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    with ClockSampler(local_rank) as clocks:
        t_wall = time.perf_counter()
        for i in range(args.steps):
            flush.zero_()
            ev[i][0].record(stream)
            one()
            ev[i][1].record(stream)
        torch.cuda.synchronize()
        t_wall = time.perf_counter() - t_wall
        if t_wall < 1.0:      # keep sampling long enough for a clock reading
            time.sleep(1.0 - t_wall)
    if world > 1:
        dist.barrier()
    step_ms = [a.elapsed_time(b) for a, b in ev]
    total_ms = max_over_ranks(sum(step_ms), world, "cuda")
    value = job_rate(net.B, world, args.steps, total_ms)

    # ---------------- end to end through the public API, host buffers
    from paper_2407_11698_gb300 import synth
    xh = torch.from_numpy(synth.images(3, 0, net.B, wl["input_shape"]).reshape(net.B, -1)).pin_memory()
    yh = torch.from_numpy(synth.labels(3, 0, net.B)).pin_memory()
    lh = torch.empty((len(net.blocks),), dtype=torch.int64).pin_memory()
    xd, yd = torch.empty_like(net.x), torch.empty_like(net.y)
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(args.steps):
        xd.copy_(xh, non_blocking=True)
        yd.copy_(yh, non_blocking=True)
        net.step(xd, yd)
        lh.copy_(net.loss, non_blocking=True)
    e1.record(stream)
    torch.cuda.synchronize()
    e2e_value = job_rate(net.B, world, args.steps,
                         max_over_ranks(e0.elapsed_time(e1), world, "cuda"))

    # ---------------- per-kernel device time inside eager steps (roofline); the
    # blocks run one after another here so that no kernel shares the GPU
    L.nitro_profile_reset()
    L.nitro_profile_enable(1)
    for _ in range(args.profile_steps):
        flush.zero_()
        net.step(sequential=True)
    torch.cuda.synchronize()
    L.nitro_profile_enable(0)
    prof = kernel_profile(nb)
    L.nitro_profile_reset()
    issued = issued_profile(nb, net, flush, 1, torch) if rank == 0 else None
    int8_ref = int8_library_rate(torch) if rank == 0 else None

    if rank != 0:
        return None
    peaks, peak_src = measured_peaks()
    total_k = sum(v["ms"] for v in prof.values()) or 1.0
    dom_name, dom = max(prof.items(), key=lambda kv: kv[1]["ms"])
    per_launch_ms = dom["ms"] / dom["launches"]
    if dom["ops"] > 0:
        if dom_name.startswith("tc_"):
            # burst peak: the kernel runs for tens of microseconds inside a
            # sub-millisecond step, not in a seconds-long loop at the power cap
            bound, peak, unit = "tensor", peaks["bf16_tflops"], "TFLOP/s"
            peak_note = "bf16 dense, %s (burst): the contraction runs as exact bf16 MMAs" % peak_src
        else:
            # CUDA-core int64 MACs: 152 SMs x 64 IMAD/clk x 2 ops x 2.07 GHz
            bound, peak, unit = "alu", 152 * 64 * 2 * 2.07e9 / 1e12, "TOPS"
            peak_note = "derived: 152 SMs x 64 int32 IMAD/clk x 2 ops x 2070 MHz"
        achieved = dom["ops"] / dom["launches"] / (per_launch_ms / 1e3) / 1e12
    else:
        bound, peak, unit = "hbm", peaks["hbm_gbs"], "GB/s"
        peak_note = "HBM copy, %s" % peak_src
        achieved = dom["bytes"] / dom["launches"] / (per_launch_ms / 1e3) / 1e9
    issued_line = None
    if issued and dom_name in issued and bound == "tensor":
        it = issued[dom_name]
        iss = it["issued_ops"] / (it["ms"] / 1e3) / 1e12
        issued_line = {"kernel": dom_name, "tflops": round(iss, 2), "frac": round(iss / peak, 4),
                       "note": "bf16 MMA work actually issued: algorithmic ops x (A limbs x B limbs)"}
    conv_ops = sum(v["ops"] for k, v in prof.items() if "conv" in k)
    conv_ms = sum(v["ms"] for k, v in prof.items() if "conv" in k)
    line = {
        "metric": METRIC,
        "value": round(value, 2),
        "unit": "images/s",
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": round(total_ms / args.steps, 4),
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "int8/int32->int64",
        "data": "synthetic",
        "config": {"workload": args.workload, "batch": net.B,
                   "input": "x".join(str(v) for v in wl["input_shape"]) + " int8 uniform [-128,127]",
                   "blocks": len(wl["blocks"]), "cuda_graph": graph is not None,
                   "block_streams": "one" if args.sequential_blocks else "one per block",
                   "update": ("nitro_block_backward_update (folded into un-split weight "
                              "gradients)" if args.fused_update else "separate IntegerSGD call"),
                   "launch": ("programmatic dependent launch" if os.environ.get("NITRO_PDL", "1") != "0"
                              else "stream-ordered"),
                   "l2": "flushed (512 MiB write) between timed steps",
                   "parallelism": "replicas" if world > 1 else "single"},
        "e2e": {"value": round(e2e_value, 2), "unit": "images/s",
                "h2d_bytes_per_step": int(net.in_bytes),
                "d2h_bytes_per_step": int(8 * len(net.blocks))},
        "gpu_launches": int(launches_per_step * args.steps),
        "roofline": {"bound": bound, "kernel": dom_name, "achieved": round(achieved, 3),
                     "peak": round(peak, 2), "unit": unit, "frac": round(achieved / peak, 4),
                     "traffic": ncu_traffic(dom_name, args.workload), "peak_source": peak_note,
                     "per_launch_ms": round(per_launch_ms, 5),
                     "share_of_kernel_time": round(dom["ms"] / total_k, 4),
                     "issued": issued_line},
        "issued_tflops": ({k: round(v["issued_ops"] / (v["ms"] / 1e3) / 1e12, 2)
                           for k, v in sorted(issued.items())} if issued else None),
        "conv_tops": round(conv_ops / (conv_ms / 1e3) / 1e12, 3) if conv_ms else None,
        "int8_ref": (dict(int8_ref, conv_frac=round(conv_ops / (conv_ms / 1e3) / 1e12 / int8_ref["tops"], 4),
                          dominant_frac=(round(achieved / int8_ref["tops"], 4) if bound == "tensor" else None))
                     if int8_ref and conv_ms else None),
        "kernels": {k: {"launches": v["launches"], "ms": round(v["ms"], 4),
                        "share": round(v["ms"] / total_k, 4)} for k, v in sorted(prof.items())},
        "clocks": clocks.summary(),
    }
    return line


def int8_library_rate(torch, n=8192, reps=5):
    """Dense int8 rate of the library GEMM on this GPU: torch._int_mm (int8 x
    int8 -> int32, cuBLASLt) at n^3, best of `reps` timed calls.  The metric
    asks for a fraction of the dense int8 tensor peak; no measured int8 peak is
    recorded for this GPU and tcgen05 kind::i8 does not assemble for sm_103a, so
    this library rate is reported beside the bf16 peak as context."""
    try:
        g = torch.Generator(device="cuda")
        g.manual_seed(5)
        a = torch.randint(-128, 128, (n, n), dtype=torch.int8, device="cuda", generator=g)
        b = torch.randint(-128, 128, (n, n), dtype=torch.int8, device="cuda", generator=g).t()
        torch._int_mm(a, b)
        torch.cuda.synchronize()
        best = None
        for _ in range(reps):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            torch._int_mm(a, b)
            e1.record()
            torch.cuda.synchronize()
            ms = e0.elapsed_time(e1)
            best = ms if best is None else min(best, ms)
        del a, b
        torch.cuda.empty_cache()
    except RuntimeError:
        return None
    return {"tops": round(2.0 * n ** 3 / (best / 1e3) / 1e12, 2),
            "what": "torch._int_mm int8 %d^3 best of %d (cuBLASLt): a measured library rate, "
                    "not a hardware peak" % (n, reps)}


# ------------------------------------------------------------------ oracle (CPU)
def oracle_rate(wl_name, sample_batch, steps, warmup=0):
    """images/s of the CPU oracle training `steps` steps of the workload at a
    reduced batch (the sample); returns (value, seconds, threads)."""
    import numpy as np
    import oracle as O
    from paper_2407_11698_gb300 import synth
    from paper_2407_11698_gb300 import workloads as WL
    wl = WL.WORKLOADS[wl_name]
    blocks = [O.OracleBlock([O.LayerDesc(*l) for l in b["layers"]], in_features=b["in_features"],
                            seed=20240716 + i, **wl.get("hyper", {}))
              for i, b in enumerate(wl["blocks"])]
    for s in range(warmup + steps):
        if s == warmup:
            t0 = time.perf_counter()
        x = synth.images(1, s, sample_batch, wl["input_shape"]).astype(np.int64)
        y = synth.labels(1, s, sample_batch).astype(np.int64)
        O.train_step(blocks, x, y)
    dt = time.perf_counter() - t0
    return sample_batch * steps / dt, dt, O.num_threads()


# ------------------------------------------------------------------ kernel sweep
SWEEP_RANGES = {1: (-127, 127), 2: (-32639, 32639), 3: (-8355711, 8355711)}


def run_sweep(args):
    """One JSON line per (contraction, shape, operand limbs): device time of
    the contraction kernel alone (library events) and of the whole call
    (limb packing included), as algorithmic TOPS (2 x MACs of the integer
    contraction) and as a fraction of the measured bf16 dense peak."""
    import ctypes
    import numpy as np
    import torch
    from paper_2407_11698_gb300 import binding as nb
    from paper_2407_11698_gb300 import synth
    from paper_2407_11698_gb300 import workloads as WL
    nb.lib()
    L = nb.lib()
    peaks, src = measured_peaks()
    peak = peaks["bf16_tflops"]
    stream = torch.cuda.current_stream()

    def timed(fn, reps):
        fn()
        torch.cuda.synchronize()
        L.nitro_profile_reset()
        L.nitro_profile_enable(1)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(reps):
            fn()
        e1.record(stream)
        torch.cuda.synchronize()
        L.nitro_profile_enable(0)
        prof = kernel_profile(nb)
        L.nitro_profile_reset()
        return e0.elapsed_time(e1) / reps, prof

    def emit(kind, shape, limbs, ops, call_ms, prof, key):
        k = prof.get(key, {"ms": float("nan"), "launches": 1})
        kms = k["ms"] / max(1, k["launches"])
        passes = 1
        for v in limbs.values():
            passes *= v
        line = {"sweep": kind, "shape": shape, "limbs": limbs, "ops": ops,
                "kernel": key, "kernel_ms": round(kms, 5), "call_ms": round(call_ms, 5),
                "kernel_tops": round(ops / kms / 1e9, 2), "call_tops": round(ops / call_ms / 1e9, 2),
                "kernel_frac_bf16": round(ops / kms / 1e9 / peak, 4),
                "issued_tflops": round(ops * passes / kms / 1e9, 2),
                "issued_frac_bf16": round(ops * passes / kms / 1e9 / peak, 4), "peak": peak,
                "peak_source": "bf16 dense, %s" % src}
        print(json.dumps(line), flush=True)

    parts = set(args.sweep_parts.split(","))
    for B, hw, c in (WL.SWEEP_CONV if "conv" in parts else ()):
        a = torch.from_numpy(synth.images(51, 0, B, (hw, hw, c))).cuda()
        conv = nb.Conv3x3(B, hw, hw, c, c)
        out = torch.empty((B, hw, hw, c), dtype=torch.int64, device="cuda")
        dw = torch.empty((c, 3, 3, c), dtype=torch.int64, device="cuda")
        ops = 2.0 * B * hw * hw * c * 9 * c
        for limbs in (1, 2, 3):
            lo, hi = SWEEP_RANGES[limbs]
            W = torch.from_numpy(synth.int_tensor(52, (c, 3, 3, c), lo, hi, dtype=np.int32)).cuda()
            d = torch.from_numpy(synth.int_tensor(53, (B, hw, hw, c), lo, hi, dtype=np.int32)).cuda()
            ms, prof = timed(lambda: conv.contract(nb.NITRO_CONTRACT_FWD, a, W, out), 5)
            emit("conv_fwd", [B, hw, hw, c, c], {"W": limbs}, ops, ms, prof, "tc_conv_fwd")
            ms, prof = timed(lambda: conv.contract(nb.NITRO_CONTRACT_WGRAD, a, d, dw), 5)
            emit("conv_wgrad", [B, hw, hw, c, c], {"delta": limbs}, ops, ms, prof, "tc_conv_wgrad")
            ms, prof = timed(lambda: conv.contract(nb.NITRO_CONTRACT_DGRAD, d, W, out), 5)
            emit("conv_dgrad", [B, hw, hw, c, c], {"delta": limbs, "W": limbs}, ops, ms, prof,
                 "tc_conv_dgrad")
            del W, d
        conv.close()
        del a, out, dw
        torch.cuda.empty_cache()
    for n in (WL.SWEEP_GEMM if "gemm" in parts else ()):
        a = torch.from_numpy(synth.int_tensor(61, (n, n), -128, 127, dtype=np.int8)).cuda()
        b8 = torch.from_numpy(synth.int_tensor(62, (n, n), -128, 127, dtype=np.int8)).cuda()
        gm = nb.IntGemm(n, n, n)
        c = torch.empty((n, n), dtype=torch.int64, device="cuda")
        ops = 2.0 * n * n * n
        for limbs in (1, 2):
            lo, hi = SWEEP_RANGES[limbs]
            b = torch.from_numpy(synth.int_tensor(63, (n, n), lo, hi, dtype=np.int32)).cuda()
            ms, prof = timed(lambda: gm.run(a, b, c), 5)
            emit("gemm", [n, n, n], {"B": limbs}, ops, ms, prof, "tc_gemm")
        # library baseline: torch._int_mm (int8 x int8 -> int32, cuBLASLt)
        bt = b8.t()
        torch._int_mm(a, bt)
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(5):
            torch._int_mm(a, bt)
        e1.record(stream)
        torch.cuda.synchronize()
        ms = e0.elapsed_time(e1) / 5
        print(json.dumps({"sweep": "torch_int_mm", "shape": [n, n, n], "call_ms": round(ms, 5),
                          "call_tops": round(ops / ms / 1e9, 2),
                          "note": "int8 x int8 -> int32 library GEMM, context for the int8 tensor rate"}),
              flush=True)
        gm.close()
        del a, b8, c
        torch.cuda.empty_cache()
    # IntegerSGD alone: one linear layer of n x n weights (16 bytes per weight:
    # W read + write, dW read; + 8 for the four bf16 limb planes the update
    # writes for the tensor-core forward) and its learning layer, against the
    # measured HBM copy bandwidth
    hbm = peaks["hbm_gbs"]
    for n in ((4096, 16384) if "sgd" in parts else ()):
        blk = nb.Block([(nb.NITRO_LINEAR, n, n, 1, 1, 0)], n, seed=1, max_batch=1)
        ms, prof = timed(lambda: blk.sgd(), 5)
        k = prof.get("integersgd", {"ms": float("nan"), "launches": 1, "bytes": 0.0})
        kms = k["ms"] / max(1, k["launches"])
        params = n * n + 10 * n
        byts = k["bytes"] / max(1, k["launches"])
        print(json.dumps({"sweep": "integersgd", "params": params, "bytes": byts,
                          "kernel_ms": round(kms, 5), "call_ms": round(ms, 5),
                          "kernel_gbs": round(byts / kms / 1e6, 1),
                          "kernel_frac_hbm": round(byts / kms / 1e6 / hbm, 4), "peak": hbm,
                          "peak_source": "HBM copy, %s" % src}), flush=True)
        blk.close()
        torch.cuda.empty_cache()
    # integer data pre-processing (App. A) at the raw dataset shapes: fit
    # (byte sum, then the sum of |x - mu|: n bytes read each) and apply (n bytes
    # read, n written), against the measured HBM copy bandwidth.  The MNIST
    # set (47 MB) stays in the 129 MB L2 between repetitions; CIFAR-10 does not.
    prep = nb.IntPrep() if "prep" in parts else None
    for name, shape, kind in ((("mnist_train", (60000, 28, 28), "digits"),
                               ("cifar10_train", (50000, 32, 32, 3), "natural"))
                              if prep else ()):
        n = int(np.prod(shape))
        x = torch.from_numpy(synth.raw_pixels(3, n, kind)).cuda()
        out = torch.empty(n, dtype=torch.int8, device="cuda")
        ms_fit, prof_fit = timed(lambda: prep.fit(x), 10)
        ms_app, prof_app = timed(lambda: prep.apply(x, out), 10)
        kern = {}
        for key, prof, byts in (("prep_sum", prof_fit, n), ("prep_mad", prof_fit, n),
                                ("prep_apply", prof_app, 2 * n)):
            k = prof.get(key, {"ms": float("nan"), "launches": 1})
            kms = k["ms"] / max(1, k["launches"])
            kern[key] = {"kernel_ms": round(kms, 5), "bytes": byts,
                         "kernel_gbs": round(byts / kms / 1e6, 1),
                         "kernel_frac_hbm": round(byts / kms / 1e6 / hbm, 4)}
        print(json.dumps({"sweep": "preprocess", "dataset": name, "shape": list(shape),
                          "values": kind, "n": n, "fit_ms": round(ms_fit, 5),
                          "apply_ms": round(ms_app, 5),
                          "fit_gbs": round(2 * n / ms_fit / 1e6, 1),
                          "apply_gbs": round(2 * n / ms_app / 1e6, 1), "kernels": kern,
                          "l2_resident": n < 129e6, "peak": hbm,
                          "peak_source": "HBM copy, %s" % src}), flush=True)
        del x, out
    if prep:
        prep.close()
    torch.cuda.empty_cache()
    return 0


def main():
    args = parse()
    if args.sweep:
        return run_sweep(args)
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if args.impl == "reference":
        if rank != 0:
            return 0
        # the oracle as it stands, on the host cores, each step a bounded
        # sample (batch 8 of the workload's 128)
        sample_b = 8
        value, dt, cores = oracle_rate(args.workload, sample_b, args.steps, args.warmup)
        line = {"impl": "reference", "metric": METRIC, "value": round(value, 4), "unit": "images/s",
                "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
                "ms_per_step": round(dt / args.steps * 1e3, 2), "higher_is_better": True,
                "scaling": "weak", "vs_baseline": None, "dtype": "int64", "data": "synthetic",
                "config": {"workload": args.workload, "sample_batch": sample_b},
                "cpu_baseline": {"value": round(value, 4), "unit": "images/s", "cores": cores,
                                 "kind": "oracle",
                                 "sample": "%d training steps at batch %d of %s" % (args.steps, sample_b, args.workload)},
                "e2e": {"value": round(value, 4), "unit": "images/s", "h2d_bytes_per_step": 0,
                        "d2h_bytes_per_step": 0}}
        print(json.dumps(line), flush=True)
        return 0

    if world > 1:
        import torch
        import torch.distributed as dist
        torch.cuda.set_device(local_rank)
        dist.init_process_group("nccl")
    line = run_ours(args, rank, world, local_rank)
    if rank == 0:
        if not args.no_cpu_baseline:
            sample_b = 16
            v, dt, cores = oracle_rate(args.workload, sample_b, 1)
            line["cpu_baseline"] = {"value": round(v, 4), "unit": "images/s", "cores": cores,
                                    "kind": "oracle",
                                    "sample": "1 training step at batch %d of %s (%.1f s)" % (sample_b, args.workload, dt)}
        print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.barrier()
        dist.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
