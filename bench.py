#!/usr/bin/env python3
"""Throughput of the ShiftQuant training hot path on GB300.

One step = for every linear layer of the workload: the range pass, grouping and
quantization of the activation X (round to nearest) and of the gradient dY (stochastic),
the per-out-channel and per-in-channel quantization of W with the ShiftMM shift folded
in, and the three integer GEMMs (forward, loss propagation, weight gradient) with their
dequantizing epilogues.  Inputs are resident in HBM when the timed region starts.  Before
every timed step, outside the timed interval, L2 is flushed by writing a 256 MiB buffer and
then reading another 256 MiB buffer, so the step starts with no input in L2 and without
dirty flush data that the step would otherwise have to write back.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
                  [--workload conv3x3|wgrad_small|vit_mlp|large_linear|large_linear_8bit|vit_block|
                              large_linear_t4096]

Prints one JSON line (rank 0).  --impl reference times the plain CPU oracle of the
same definitions on the host cores instead (a bounded sample of the same workload).
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import re
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "ShiftQuant GEMM TOPS & % dense-INT8 peak; quantizer GB/s & % HBM peak"
UNIT = "TOPS"
DEFAULT_WORKLOAD = "large_linear"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
FP8_OVER_BF16 = 2.0    # nominal dense ratio (4.5 vs 2.25 PFLOP/s)
# dense tensor-core operations per SM per clock (BF16; E4M3 is twice that): the clock-derived
# peak at the sampled SM clock sits beside the measured cuBLAS peak, whose run was power-capped
# at a lower clock than these short launches see
BF16_OPS_PER_SM_CLOCK = 8192
L2_FLUSH_BYTES = 256 << 20


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD)
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-chain", action="store_true",
                    help="skip the fused-range chain measurement")
    ap.add_argument("--no-l1bn", action="store_true",
                    help="skip the L1 batch normalization measurement")
    ap.add_argument("--no-group-order", action="store_true",
                    help="skip the group-ordered contraction measurement")
    ap.add_argument("--no-pack", action="store_true",
                    help="skip the packed-storage measurement")
    ap.add_argument("--also", default="conv3x3",
                    help="second workload summarised in the same line ('none' for none)")
    return ap.parse_args()


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        d = json.load(open(p))
        return {k: float(d[k]) for k in FALLBACK_PEAKS}, "measured"
    except Exception:
        return dict(FALLBACK_PEAKS), "fallback"


# ----------------------------------------------------------------- clocks sampler
class ClockSampler:
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
    NAMES = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.path = None

    def start(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.index}", f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
            time.sleep(0.3)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        rows = []
        for line in open(self.path):
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 8:
                continue
            try:
                rows.append((float(parts[0]), float(parts[1]), parts[4:8]))
            except ValueError:
                continue
        os.unlink(self.path)
        if not rows:
            return None
        mx = max(r[1] for r in rows)
        load = [r[0] for r in rows]
        reasons = sorted({n for r in rows for n, v in zip(self.NAMES, r[2]) if v.lower() == "active"})
        return {"sm_mhz": statistics.median(load), "sm_max_mhz": mx, "reasons": reasons,
                "samples": len(rows)}


# --------------------------------------------------------------- our CUDA path
class Step:
    """All buffers and calls of one workload step (every layer)."""

    def __init__(self, wl, seed, device):
        import torch
        from paper_2411_10948_gb300 import layer as L
        from paper_2411_10948_gb300 import native as N
        from paper_2411_10948_gb300 import workloads as W
        self.torch, self.N, self.L = torch, N, L
        self.wl = wl
        self.layers, self.inputs = [], []
        for i, spec in enumerate(wl.layers):
            self.inputs.append(W.torch_layer_inputs(spec, seed, i, device))
            # transposed code copies only where the library advises them (the weight
            # gradient otherwise reads X's and dY's codes in place)
            self.layers.append(L.QuantLinear(spec.M, spec.K, spec.N, spec.bits, spec.n_groups,
                                             device, with_acc=False, use_workspace=True,
                                             transposed=None))
        self.specs = list(wl.layers)

    # (name, callable) for every library call of one step, in order
    def calls(self, step_idx):
        out = []
        N, L = self.N, self.L
        for lay, (x, w, dy) in zip(self.layers, self.inputs):
            b, G, st = lay.bits, lay.G, lay.status
            seed = 0x5EED + step_idx
            out += [
                ("calibrate", lambda lay=lay, x=x: N.shiftquant_calibrate(
                    x, N.SQ_GRAN_SHIFT, lay.G, lay.x.range, lay.x.tau0, lay.x.exp, lay.status)),
                ("quantize", lambda lay=lay, x=x: N.shiftquant_quantize(
                    x, N.SQ_GRAN_SHIFT, lay.bits, lay.G, lay.x.tau0, lay.x.exp, None,
                    N.SQ_ROUND_NEAREST_EVEN, 0, lay.x.codes, lay.x.codes_t, lay.x.scale)),
                ("calibrate", lambda lay=lay, dy=dy: N.shiftquant_calibrate(
                    dy, N.SQ_GRAN_SHIFT, lay.G, lay.g.range, lay.g.tau0, lay.g.exp, lay.status)),
                ("quantize", lambda lay=lay, dy=dy, seed=seed: N.shiftquant_quantize(
                    dy, N.SQ_GRAN_SHIFT, lay.bits, lay.G, lay.g.tau0, lay.g.exp, None,
                    N.SQ_ROUND_STOCHASTIC, seed, lay.g.codes, lay.g.codes_t, lay.g.scale)),
                ("calibrate", lambda lay=lay, w=w: N.shiftquant_calibrate_weight(
                    w, lay.wf.range, lay.wd.range, lay.status)),
                ("quantize", lambda lay=lay, w=w: N.shiftquant_quantize_weight(
                    w, lay.bits, lay.G, lay.wf.range, lay.wd.range, lay.x.exp, lay.g.exp,
                    lay.wf.codes, lay.wf.scale, lay.wd.codes, lay.wd.scale)),
                ("gemm", lay.gemms),   # forward, loss propagation, weight gradient: one launch
            ]
        return out

    def call_bytes(self):
        """(layer, tensor, algorithmic HBM bytes) of each call of calls(), in its order."""
        out = []
        for s, lay, gb in zip(self.specs, self.layers, self.gemm_bytes_per_launch()):
            cb = self.N.shiftquant_code_bytes(s.bits, s.n_groups)
            MK, MN, KN = s.M * s.K, s.M * s.N, s.K * s.N
            cx, cg = self.code_copies(lay)
            out += [(s.name, "X", 4 * MK), (s.name, "X", 4 * MK + cx * cb * MK),
                    (s.name, "dY", 4 * MN), (s.name, "dY", 4 * MN + cg * cb * MN),
                    (s.name, "W (both roles)", 4 * KN), (s.name, "W (both roles)", 4 * KN + 2 * cb * KN),
                    (s.name, "GEMMs", gb)]
        return out

    @staticmethod
    def code_copies(lay):
        """Code sets the quantizer writes for X and dY: the codes, plus the transposed copy
        where the layer keeps one."""
        return (1 + (lay.x.codes_t is not None), 1 + (lay.g.codes_t is not None))

    def group_histograms(self):
        """Channels per group of every grouped tensor (after the last step)."""
        out = {}
        for s, lay in zip(self.specs, self.layers):
            for t, q in (("X", lay.x), ("dY", lay.g)):
                e = q.exp.cpu().numpy()
                out[f"{s.name}:{t}"] = [int(c) for c in np.bincount(e, minlength=s.n_groups)]
        return out

    def launches_per_step(self) -> int:
        n = 0
        N = self.N
        for lay in self.layers:
            n += 3 + 1 + 3 + 1          # X and dY: range init, range, grouping; quantize
            n += 2 + 1                  # weight: range init, both ranges; both roles' codes
            # the three GEMMs: one launch, plus the output pass of each GEMM that splits K
            n += N.shiftquant_gemm_layer_kernel_launches(
                lay.M, lay.K, lay.N, lay.bits, lay.G,
                0 if lay.ws_layer is None else lay.ws_layer.numel() * 4)
        return n

    def gemm_ops(self) -> int:
        return sum(l.gemm_ops for l in self.layers)

    def gemm_flops_per_launch(self):
        return [3 * 2 * l.M * l.N * l.K for l in self.layers]

    def gemm_bytes_per_launch(self):
        """Algorithmic HBM bytes of each layer's GEMM launch: every GEMM's operand codes read
        once, every fp32 output written once."""
        out = []
        for s, lay in zip(self.specs, self.layers):
            cb = self.N.shiftquant_code_bytes(s.bits, s.n_groups)
            # X and dY codes twice each (forward / loss propagation, and the weight gradient,
            # in place or from the transposed copy), both weight roles
            codes = cb * (2 * s.M * s.K + 2 * s.M * s.N + 2 * s.K * s.N)
            outs = 4 * (s.M * s.N + s.M * s.K + s.K * s.N)
            out.append(codes + outs)
        return out

    def range_bytes(self) -> int:
        """Algorithmic HBM bytes of the range passes of one step (4 B read per element)."""
        return sum(4 * (s.M * s.K + s.M * s.N + s.K * s.N) for s in self.specs)

    def quantize_bytes(self) -> int:
        """Algorithmic HBM bytes of the quantize passes of one step."""
        tot = 0
        for s, lay in zip(self.specs, self.layers):
            cb = self.N.shiftquant_code_bytes(s.bits, s.n_groups)
            # X and dY: read, codes (+ the transposed copy where kept)
            for (R, C), n in zip(((s.M, s.K), (s.M, s.N)), self.code_copies(lay)):
                tot += 4 * R * C + n * cb * R * C
            tot += 4 * s.K * s.N + 2 * cb * s.K * s.N    # W: one read, both roles' codes
        return tot

    def quantizer_bytes(self) -> int:
        return self.range_bytes() + self.quantize_bytes()

    def status_ok(self) -> bool:
        return all(int(l.status.item()) == 0 for l in self.layers)


def kernel_source_hash() -> str:
    """Hash of the GEMM kernel's device code (sq_gemm.cu up to its host-side part, and the
    device helpers): a profile's DRAM traffic stays valid while this is unchanged."""
    csrc = os.path.join(ROOT, "paper_2411_10948_gb300", "csrc")
    gemm = open(os.path.join(csrc, "sq_gemm.cu"), "rb").read()
    h = hashlib.sha256()
    h.update(gemm.split(b"// " + b"-" * 71 + b" host side")[0])
    h.update(open(os.path.join(csrc, "sq_device.cuh"), "rb").read())
    return h.hexdigest()[:16]


def profiled_traffic(workload: str):
    """DRAM bytes per launch of the GEMM kernel from the committed ncu summary, or None when
    the kernel source changed after the capture."""
    p = os.path.join(ROOT, "profiles", f"shiftmm_{workload}.md")
    if not os.path.exists(p):
        return None
    txt = open(p).read()
    m = re.search(r"kernel_source_sha256_16:\s*([0-9a-f]+)", txt)
    t = re.search(r"dram_bytes_per_launch:\s*([0-9.eE+]+)", txt)
    if not m or not t or m.group(1) != kernel_source_hash():
        return None
    return float(t.group(1))


def make_l2_flush(dev):
    """A function that flushes L2 before a timed call: a 256 MiB write, then a 256 MiB read,
    so that the timed call finds neither its data nor dirty lines to write back."""
    import torch
    w = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device=dev)
    r = torch.zeros(L2_FLUSH_BYTES // 4, dtype=torch.float32, device=dev)
    sink = torch.zeros((), dtype=torch.float32, device=dev)

    def flush():
        w.zero_()
        torch.sum(r, dim=0, out=sink)
    return flush


def max_over_ranks(value: float, device) -> float:
    """The maximum of a per-rank float over all ranks (the value itself without a process
    group): the slowest replica's time is the job's time."""
    import torch
    import torch.distributed as dist
    t = torch.tensor([value], dtype=torch.float64, device=device)
    if dist.is_available() and dist.is_initialized() and dist.get_world_size() > 1:
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(ops_per_step: int, world: int, steps: int, total_ms: float) -> float:
    """Whole-job TOPS: every replica runs its own step of ops_per_step operations."""
    return ops_per_step * world * steps / (total_ms * 1e-3) / 1e12


def run_ours(args, rank, world, local_rank):
    import torch
    from paper_2411_10948_gb300 import build, native
    from paper_2411_10948_gb300 import layer as L
    from paper_2411_10948_gb300 import workloads as W
    build.build_library()
    native.load()
    dev = torch.device("cuda", local_rank)
    torch.cuda.set_device(dev)
    wl = W.workload(args.workload)
    st = Step(wl, args.seed + 1000 * rank, dev)
    flush_w = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device=dev)
    flush_r = torch.zeros(L2_FLUSH_BYTES // 4, dtype=torch.float32, device=dev)
    flush_sink = torch.zeros((), dtype=torch.float32, device=dev)

    def flush_l2():
        flush_w.zero_()
        torch.sum(flush_r, dim=0, out=flush_sink)

    stream = torch.cuda.current_stream()

    def run_step(i, events=None):
        for j, (name, fn) in enumerate(st.calls(i)):
            fn()
            if events is not None:
                events[j + 1].record(stream)

    for i in range(args.warmup):
        flush_l2()
        run_step(i)
    torch.cuda.synchronize()
    assert st.status_ok(), "device status set during warm-up"

    # the timed step is the whole step captured in one CUDA graph: per layer, the activation
    # chain, the gradient chain and the weight (both roles) each on its own stream, then the
    # layer's three GEMMs as one launch
    streams = [[torch.cuda.Stream(device=dev) for _ in range(3)] for _ in st.layers]

    # A second capture of the same step with events around each layer's GEMM call (external
    # events are recorded as graph nodes) times the GEMM launches in graph replays; the
    # headline replays run the graph without them.
    # (and an event at the start of each layer's step: the quantizer phase, as the step runs
    # its three quantizer chains side by side, is the time from it to the GEMM call)
    try:
        gemm_ev = [(torch.cuda.Event(enable_timing=True, external=True),
                    torch.cuda.Event(enable_timing=True, external=True)) for _ in st.layers]
        phase_ev = [torch.cuda.Event(enable_timing=True, external=True) for _ in st.layers]
    except TypeError:
        gemm_ev = phase_ev = None

    def run_step_concurrent(i, events=None):
        for li, (lay, (x, w, dy), ss) in enumerate(zip(st.layers, st.inputs, streams)):
            lay.step_concurrent(x, w, dy, 0x5EED + i, ss,
                                gemm_events=events[li] if events else None,
                                start_event=phase_ev[li] if events else None)

    graph = L.CapturedStep(lambda: run_step_concurrent(args.warmup))
    for i in range(args.warmup):
        flush_l2()
        graph.replay()
    torch.cuda.synchronize()

    sampler = ClockSampler(local_rank)
    sampler.start()
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    pairs = []
    for i in range(args.steps):
        flush_l2()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        graph.replay()
        b.record(stream)
        pairs.append((a, b))
    torch.cuda.synchronize()
    if world > 1:
        torch.distributed.barrier()
    step_ms = [a.elapsed_time(b) for a, b in pairs]
    ok = st.status_ok()

    graph_gemm_ms = []   # per layer and replay: the GEMM call inside a graph replay
    graph_quant_ms = []  # per replay: the layers' quantizer phases (step start to GEMM call)
    if gemm_ev:
        graph_ev = L.CapturedStep(lambda: run_step_concurrent(args.warmup, gemm_ev))
        for i in range(args.steps):
            flush_l2()
            graph_ev.replay()
            torch.cuda.synchronize()   # the events are recorded again by the next replay
            graph_gemm_ms += [e0.elapsed_time(e1) for e0, e1 in gemm_ev]
            graph_quant_ms.append(sum(p.elapsed_time(e0) for p, (e0, _) in zip(phase_ev, gemm_ev)))
        del graph_ev

    # per-call breakdown: the same calls un-graphed, queued behind a sleep kernel so the
    # GPU never waits on the host; events between consecutive calls
    names = [n for n, _ in st.calls(0)]
    ncalls = len(names)
    kind_ms = {"calibrate": 0.0, "quantize": 0.0, "gemm": 0.0}
    call_ms = [0.0] * ncalls
    gemm_launch_ms = []
    for i in range(args.steps):
        flush_l2()
        torch.cuda._sleep(20_000_000)
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(ncalls + 1)]
        ev[0].record(stream)
        run_step(args.warmup + i, ev)
        torch.cuda.synchronize()
        for j, n in enumerate(names):
            d = ev[j].elapsed_time(ev[j + 1])
            kind_ms[n] += d
            call_ms[j] += d
            if n == "gemm":
                gemm_launch_ms.append(d)
    total_ms = max_over_ranks(sum(step_ms), dev)
    ms_per_step = total_ms / args.steps

    # the quantizer passes as the step runs them, in a CUDA graph: the step's range and
    # quantize calls serial on one stream, captured once and replayed after an L2 flush,
    # timed with events around the replay (no per-launch host gap)
    qcalls = [(n, fn) for n, fn in st.calls(args.warmup) if n != "gemm"]
    q_graph = L.CapturedStep(lambda: [fn() for _, fn in qcalls])
    q_graph_ms = 0.0
    for i in range(args.warmup + args.steps):
        flush_l2()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        q_graph.replay()
        b.record(stream)
        torch.cuda.synchronize()
        if i >= args.warmup:
            q_graph_ms += a.elapsed_time(b)
    q_graph_ms = max_over_ranks(q_graph_ms, dev)
    # per tensor: a graph of its range call and one of its range and quantize calls, each
    # timed the same way (event nodes inside a graph cost microseconds each, so the calls
    # are not split by events); the quantize time is the difference
    def graph_ms(fns):
        g = L.CapturedStep(lambda: [fn() for fn in fns])
        tot = 0.0
        for i in range(args.warmup + args.steps):
            flush_l2()
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(stream)
            g.replay()
            b.record(stream)
            torch.cuda.synchronize()
            if i >= args.warmup:
                tot += a.elapsed_time(b)
        del g
        return tot
    q_call_graph_ms = []
    for j in range(0, len(qcalls), 2):
        r_ms = graph_ms([qcalls[j][1]])
        both_ms = graph_ms([qcalls[j][1], qcalls[j + 1][1]])
        q_call_graph_ms += [r_ms, max(both_ms - r_ms, 1e-6)]
    del q_graph

    # e2e: the C entry point shiftquant_layer_step_host_split (layer.HostSteps): every call
    # copies a layer's X, W and dY in from pinned host memory on the copy-in stream, runs its
    # whole step on the layer's stream and copies Y, dX and dW back on the copy-out stream;
    # two device buffer sets take the steps in turn.  Timed from the first copy in to the last
    # copy back.
    e2e = None
    if not args.no_e2e:
        host_in = [[a.cpu().pin_memory() for a in inp] for inp in st.inputs]
        slots = 2
        host_out = [[[torch.empty(o.shape, dtype=o.dtype, pin_memory=True)
                      for o in (l.y, l.dx, l.dw)] for l in st.layers] for _ in range(slots)]
        h2d = sum(a.numel() * a.element_size() for inp in host_in for a in inp)
        d2h = sum(a.numel() * a.element_size() for outs in host_out[0] for a in outs)
        pipe = L.HostSteps([(s.M, s.K, s.N) for s in st.specs], st.specs[0].bits,
                           st.specs[0].n_groups, dev, slots=slots)
        outs = lambda n: [host_out[i % slots] for i in range(n)]
        pipe.run([host_in] * args.warmup, outs(args.warmup)).synchronize()
        torch.cuda.synchronize()
        a = torch.cuda.Event(enable_timing=True)
        a.record(torch.cuda.current_stream())
        end = pipe.run([host_in] * args.steps, outs(args.steps))
        end.synchronize()
        e_total = max_over_ranks(a.elapsed_time(end), dev)
        ok = ok and pipe.status_ok()
        e2e = {"value": job_throughput(st.gemm_ops(), world, args.steps, e_total),
               "unit": UNIT, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
               "ms_per_step": e_total / args.steps,
               "api": "shiftquant_layer_step_host_split (C ABI), one call per layer and step",
               "pipeline": "one copy-in and one copy-out stream for all calls, a stream per "
                           "layer for the steps, two device buffer sets taking the steps in "
                           "turn: copies in, compute and copies back of successive steps "
                           "overlap",
               "l2": "not flushed: each step copies %.0f MB of inputs in from host memory "
                     "(L2 is 126 MB)" % (h2d / 1e6)}
        del pipe
    clocks = sampler.stop()

    # quantizer throughput per tensor: range pass, quantize pass and both, from the calls
    # inside the quantizer graph (else from the un-graphed breakdown)
    per_tensor = []
    cbytes = st.call_bytes()
    qcbytes = [c for c, n in zip(cbytes, names) if n != "gemm"]
    q_per_call = q_call_graph_ms
    per_tensor_src = ("per tensor, one graph of its range call and one of its range and quantize "
                      "calls, each replayed after an L2 flush; quantize = the difference")
    for j in range(0, len(qcbytes), 2):
        (lname, tname, rb), (_, _, qb) = qcbytes[j], qcbytes[j + 1]
        rms, qms = q_per_call[j] / args.steps, q_per_call[j + 1] / args.steps
        per_tensor.append({"layer": lname, "tensor": tname,
                           "range_us": round(rms * 1e3, 2), "quantize_us": round(qms * 1e3, 2),
                           "range_gbs": round(rb / (rms * 1e-3) / 1e9, 1),
                           "quantize_gbs": round(qb / (qms * 1e-3) / 1e9, 1),
                           "both_gbs": round((rb + qb) / ((rms + qms) * 1e-3) / 1e9, 1)})
    peaks, peak_src = load_peaks()
    spec0 = wl.layers[0]
    fp8 = native.shiftquant_code_type(spec0.bits, spec0.n_groups) == native.SQ_CODE_E4M3
    tensor_peak = peaks["bf16_tflops"] * (FP8_OVER_BF16 if fp8 else 1.0)
    flops = st.gemm_flops_per_launch() * args.steps
    # the GEMM launch time: from graph replays with events around the GEMM call when such
    # events can be captured, else from the breakdown pass
    gemm_src = "graph replays" if graph_gemm_ms else "breakdown pass"
    if graph_gemm_ms:
        gemm_launch_ms = graph_gemm_ms
    gemm_tflops = sum(flops) / (sum(gemm_launch_ms) * 1e-3) / 1e12
    q_bytes = st.quantizer_bytes() * args.steps
    q_ms_ungraphed = kind_ms["calibrate"] + kind_ms["quantize"]
    q_gbs_ungraphed = q_bytes / (q_ms_ungraphed * 1e-3) / 1e9
    q_ms = q_graph_ms
    q_gbs = q_bytes / (q_ms * 1e-3) / 1e9
    # The layer GEMM launch is bound by the tensor cores or by HBM depending on its
    # arithmetic intensity (operations per algorithmic byte) against the ridge point
    # peak_tensor / peak_hbm; the roofline reports the binding one.
    g_bytes = sum(st.gemm_bytes_per_launch()) * args.steps
    g_s = sum(gemm_launch_ms) * 1e-3
    intensity = sum(flops) / g_bytes
    ridge = tensor_peak * 1e12 / (peaks["hbm_gbs"] * 1e9)
    kernel_name = ("shiftmm_kernel<%d, *> (one launch = forward + loss propagation + weight "
                   "gradient of a layer)" % (1 if fp8 else 0))
    tensor_src = f"{peak_src} bf16 burst" + (" x 2 (nominal FP8/BF16)" if fp8 else "")
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    clock_mhz = (clocks or {}).get("sm_mhz") or 0.0
    clock_peak = (sms * BF16_OPS_PER_SM_CLOCK * (FP8_OVER_BF16 if fp8 else 1.0) * clock_mhz * 1e6
                  / 1e12) if clock_mhz else None
    gemm_tensor = {"bound": "tensor", "achieved": gemm_tflops, "peak": tensor_peak,
                   "unit": "TFLOP/s", "frac": gemm_tflops / tensor_peak,
                   "clock_peak": clock_peak,
                   "frac_of_clock_peak": gemm_tflops / clock_peak if clock_peak else None,
                   "clock_peak_source": "%d SMs x %d dense ops/clock x median sampled SM clock"
                                        % (sms, BF16_OPS_PER_SM_CLOCK * (2 if fp8 else 1)),
                   "traffic": profiled_traffic(args.workload), "kernel": kernel_name,
                   "launch_time_source": gemm_src,
                   "peak_source": tensor_src}
    gemm_gbs = g_bytes / g_s / 1e9
    gemm_hbm = {"bound": "hbm", "achieved": gemm_gbs, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                "frac": gemm_gbs / peaks["hbm_gbs"], "traffic": profiled_traffic(args.workload),
                "kernel": kernel_name, "peak_source": f"{peak_src} copy bandwidth",
                "launch_time_source": gemm_src,
                "algorithmic_bytes_per_launch": sum(st.gemm_bytes_per_launch()) / len(st.layers)}
    gemm_roof = dict(gemm_tensor if intensity >= ridge else gemm_hbm,
                     intensity_ops_per_byte=intensity, ridge_ops_per_byte=ridge)
    quant_roof = {"bound": "hbm", "achieved": q_gbs, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                  "frac": q_gbs / peaks["hbm_gbs"], "kernel": "calibrate + quantize",
                  "peak_source": f"{peak_src} copy bandwidth",
                  "timing": "every range and quantize call of a step, serial on one stream, "
                            "in one CUDA-graph replay after an L2 flush",
                  "ms_per_step": q_ms / args.steps,
                  "ungraphed": {"achieved": q_gbs_ungraphed,
                                "frac": q_gbs_ungraphed / peaks["hbm_gbs"],
                                "ms_per_step": q_ms_ungraphed / args.steps,
                                "timing": "the same calls launched one by one from the host, "
                                          "queued behind a sleep kernel, events between them"}}
    if graph_quant_ms:
        qs_ms = statistics.median(graph_quant_ms)
        qs_gbs = st.quantizer_bytes() / (qs_ms * 1e-3) / 1e9
        quant_roof["in_step"] = {
            "achieved": qs_gbs, "frac": qs_gbs / peaks["hbm_gbs"], "ms_per_step": qs_ms,
            "timing": "the quantizer phases of the step as it runs them (each layer's "
                      "activation, gradient and weight chains side by side on their own "
                      "streams): event nodes from the start of each layer's step to its "
                      "GEMM call, in a graph replay after an L2 flush, median over replays"}
    # the dominant kernel: the kernel class (range pass, quantize, layer GEMM launch) of the
    # single launch with the most device time in the step
    def hbm_roof(nbytes, ms, name):
        gbs = nbytes * args.steps / (ms * 1e-3) / 1e9
        return {"bound": "hbm", "achieved": gbs, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                "frac": gbs / peaks["hbm_gbs"], "traffic": None, "kernel": name,
                "peak_source": f"{peak_src} copy bandwidth"}
    cands = [(kind_ms["gemm"], gemm_roof),
             (kind_ms["calibrate"], hbm_roof(st.range_bytes(), kind_ms["calibrate"],
                                             "calib_init_kernel + colmax_kernel / rowmax_kernel "
                                             "(range pass with grouping)")),
             (kind_ms["quantize"], hbm_roof(st.quantize_bytes(), kind_ms["quantize"],
                                            "quantize_kernel"))]
    longest = {k: max([v for n, v in zip(names, call_ms) if n == k] or [0.0])
               for k in ("gemm", "calibrate", "quantize")}
    dominant = max(zip(("gemm", "calibrate", "quantize"), cands),
                   key=lambda kc: longest[kc[0]])[1][1]

    result = {
        "metric": METRIC,
        "value": job_throughput(st.gemm_ops(), world, args.steps, total_ms),
        "unit": UNIT,
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": ms_per_step,
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "e4m3" if fp8 else "bf16",
        "data": "synthetic",
        "config": {"workload": args.workload, "description": wl.description,
                   "layers": [[s.name, s.M, s.K, s.N] for s in wl.layers],
                   "bits": spec0.bits, "n_groups": spec0.n_groups,
                   "l2": "flushed before every timed step, outside the timed interval: 256 MiB "
                         "write, then a 256 MiB read so no dirty line is left",
                   "parallelism": f"replica x{world}" if world > 1 else "single GPU"},
        "roofline": dominant,
        "gemm": dict(gemm_tensor, tops_step=st.gemm_ops() / (ms_per_step * 1e-3) / 1e12,
                     hbm_gbs=gemm_gbs, hbm_frac=gemm_gbs / peaks["hbm_gbs"],
                     intensity_ops_per_byte=intensity, ridge_ops_per_byte=ridge,
                     int8_peak="none: sm_103a has no integer MMA (tcgen05 kind::i8 does not "
                               "assemble); exact integers run on the E4M3/BF16 tensor cores"),
        "quantizer": dict(quant_roof, bytes_per_step=st.quantizer_bytes(),
                          nominal_hbm_gbs=7900.0, frac_nominal=q_gbs / 7900.0,
                          transposed_copies={s.name: lay.x.codes_t is not None
                                             for s, lay in zip(st.specs, st.layers)}),
        "breakdown_ms_per_step": {k: v / args.steps for k, v in kind_ms.items()},
        "calls_ms_per_step": [[f"{n}", round(v / args.steps, 5)] for n, v in zip(names, call_ms)],
        "quantizer_per_tensor": per_tensor,
        "quantizer_per_tensor_source": per_tensor_src,
        "group_histograms": st.group_histograms(),
        "timing": "CUDA events around one CUDA-graph replay of the whole step (per layer: "
                  "activation chain, gradient chain and the weight (both roles) on three streams, "
                  "then the three GEMMs as one launch); breakdown from un-graphed serial "
                  "calls (one launch per GEMM) queued behind a sleep kernel",
        "gpu_launches": st.launches_per_step() * args.steps,
        "clocks": clocks,
        "status_ok": ok,
    }
    if e2e is not None:
        result["e2e"] = e2e
    return result, st


def run_chain(args, dev, flush_steps=None):
    """The range pass fused into the producer's epilogue, measured: vit_mlp's fc1 and fc2
    trained as a chain (fc2's X = fc1's Y, fc1's dY = fc2's dX; nothing between the layers),
    forward then backward, each variant captured as one CUDA graph and replayed after an L2
    flush.  fused: the inner activation's and gradient's ranges come from the GEMM epilogues
    (shiftquant_gemm_layer's y_range / dx_range); separate: the usual range passes."""
    import torch
    from paper_2411_10948_gb300 import layer as L
    from paper_2411_10948_gb300 import workloads as W
    wl = W.workload("vit_mlp")
    s1, s2 = wl.layers
    M, dims, bits, G = s1.M, (s1.K, s1.N, s2.N), s1.bits, s1.n_groups
    x0, w1, _ = W.torch_layer_inputs(s1, args.seed, 0, dev)
    _, w2, dy = W.torch_layer_inputs(s2, args.seed, 1, dev)
    flush_w = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device=dev)
    flush_r = torch.zeros(L2_FLUSH_BYTES // 4, dtype=torch.float32, device=dev)
    sink = torch.zeros((), dtype=torch.float32, device=dev)
    out = {}
    steps = flush_steps or max(5, min(args.steps, 20))
    for fused in (True, False):
        ch = L.LinearChain(M, dims, bits, G, dev, fused_ranges=fused)
        g = L.CapturedStep(lambda: ch.step(x0, [w1, w2], dy, 0x5EED))
        for _ in range(3):
            g.replay()
        torch.cuda.synchronize()
        ms = []
        for _ in range(steps):
            flush_w.zero_()
            torch.sum(flush_r, dim=0, out=sink)
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record()
            g.replay()
            b.record()
            b.synchronize()
            ms.append(a.elapsed_time(b))
        assert ch.status_ok(), "device status set in the chain"
        out["fused_ms" if fused else "separate_ms"] = statistics.median(ms)
        del g, ch
    out.update({"workload": "vit_mlp fc1 -> fc2 as a chain (M=%d, %d -> %d -> %d, %d-bit), "
                            "forward then backward, one graph per variant" % (M, *dims, bits),
                "range_bytes_removed": 4 * M * dims[1] * 2,
                "steps": steps, "statistic": "median of graph replays after an L2 flush"})
    out["saved_frac"] = 1.0 - out["fused_ms"] / out["separate_ms"]
    return out


L1BN_SHAPES = (("resnet_stage1", 64 * 56 * 56, 64), ("resnet_stage3", 64 * 14 * 14, 256))
# HBM bytes per element of the passes (fp32 in / out, 1-byte codes): forward = range pass 4,
# quantize + code sums 4 + 1, deviation sums 1, output 1 + 4; backward = range pass 4,
# quantize + sums 4 + 1 (x codes) + 1 (gradient codes), output 1 + 1 + 4
L1BN_FWD_BYTES, L1BN_BWD_BYTES = 15, 16


def run_l1bn(args, dev):
    """The fully-quantized L1 batch normalization (8-bit, N_G = 4) on ResNet-shaped
    activations: forward and backward each captured in a CUDA graph and timed with CUDA
    events around a replay after an L2 flush (median), against HBM."""
    import torch
    from paper_2411_10948_gb300 import layer as L
    from paper_2411_10948_gb300 import native as N
    from paper_2411_10948_gb300 import workloads as W
    peaks, src = load_peaks()
    flush_l2 = make_l2_flush(dev)
    out = []
    steps = max(5, min(args.steps, 20))
    for name, R, C in L1BN_SHAPES:
        x = W.torch_tensor(("normal_outlier", 0.02, 50.0), R, C, args.seed + 1, dev)
        dy = W.torch_tensor(("grad", "laplace", 2.0, 0.0, 1.0), R, C, args.seed + 2, dev)
        gamma = torch.ones(C, device=dev) + 0.1 * torch.randn(C, device=dev)
        beta = 0.1 * torch.randn(C, device=dev)
        y, dx = torch.empty_like(x), torch.empty_like(x)
        dg, db = torch.empty(C, device=dev), torch.empty(C, device=dev)
        st = torch.zeros(1, dtype=torch.int32, device=dev)
        state = torch.zeros(N.shiftquant_l1bn_state_bytes(R, C), dtype=torch.uint8, device=dev)
        fwd_call = lambda: N.shiftquant_l1bn_forward(x, gamma, beta, 8, 4, y, state, st)
        bwd_call = lambda: N.shiftquant_l1bn_backward(dy, 8, 4, 0x5EED, state, dx, dg, db, st)
        fwd_graph, bwd_graph = L.CapturedStep(fwd_call), L.CapturedStep(bwd_call)
        fwd, bwd = fwd_graph.replay, bwd_graph.replay
        for _ in range(3):
            fwd()
            bwd()
        times = {"fwd": [], "bwd": []}
        for _ in range(steps):
            for k, fn in (("fwd", fwd), ("bwd", bwd)):
                flush_l2()
                a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                a.record()
                fn()
                b.record()
                b.synchronize()
                times[k].append(a.elapsed_time(b))
        assert st.item() == 0, "device status set in the L1 batch normalization"
        fm, bm = statistics.median(times["fwd"]), statistics.median(times["bwd"])
        fg = L1BN_FWD_BYTES * R * C / (fm * 1e-3) / 1e9
        bg = L1BN_BWD_BYTES * R * C / (bm * 1e-3) / 1e9
        launches = {"fwd": N.shiftquant_l1bn_kernel_launches(C),
                    "bwd": N.shiftquant_l1bn_kernel_launches(C, True)}
        out.append({"shape": name, "rows": R, "channels": C, "fwd_ms": fm, "bwd_ms": bm,
                    "fwd_gbs": fg, "bwd_gbs": bg, "fwd_frac": fg / peaks["hbm_gbs"],
                    "bwd_frac": bg / peaks["hbm_gbs"], "launches": launches})
    return {"bits": 8, "n_groups": 4, "bytes_per_element": {"fwd": L1BN_FWD_BYTES,
                                                           "bwd": L1BN_BWD_BYTES},
            "peak": peaks["hbm_gbs"], "peak_source": f"{src} copy bandwidth",
            "statistic": "median over graph replays after an L2 flush", "shapes": out}


def run_group_order(args, dev):
    """The group-ordered contraction against the folded layout, on the 8-bit large_linear
    layers (16384 tokens, 4096 <-> 11008): each layer's GEMM launch timed alone (median of
    CUDA-event timings after an L2 flush), on the workload's own data and on 'flat' data whose
    channels all fall in the top group (N(0,1) activations and gradients: every range within a
    factor 2 of the largest), where the folded layout's chunks are shortest."""
    import torch
    from paper_2411_10948_gb300 import layer as L
    from paper_2411_10948_gb300 import workloads as W
    peaks, src = load_peaks()
    wl = W.workload("large_linear_8bit")
    flush_l2 = make_l2_flush(dev)
    steps = max(3, min(args.steps, 10))
    rows = []
    for data in ("workload", "flat"):
        for grouped in (False, True):
            ms_tot, flops = 0.0, 0
            for li, spec in enumerate(wl.layers):
                x, w, dy = W.torch_layer_inputs(spec, args.seed, li, dev)
                if data == "flat":
                    x = torch.randn_like(x)
                    dy = torch.randn_like(dy)
                lay = L.QuantLinear(spec.M, spec.K, spec.N, spec.bits, spec.n_groups, dev,
                                    grouped=grouped)
                lay.quantize_activation(x)
                lay.quantize_gradient(dy, 7)
                lay.quantize_weights(w)
                for _ in range(2):
                    lay.gemms()
                ts = []
                for _ in range(steps):
                    flush_l2()
                    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                    a.record()
                    lay.gemms()
                    b.record()
                    b.synchronize()
                    ts.append(a.elapsed_time(b))
                assert lay.status.item() == 0, "device status set"
                hist = [int(v) for v in torch.bincount(lay.x.exp.long(), minlength=spec.n_groups).cpu()]
                ms_tot += statistics.median(ts)
                flops += lay.gemm_ops
                del lay, x, w, dy
            tf = flops / (ms_tot * 1e-3) / 1e12
            rows.append({"data": data, "layout": "group-ordered" if grouped else "folded",
                         "gemm_ms": ms_tot, "tflops": tf, "frac": tf / peaks["bf16_tflops"],
                         "x_group_histogram_last_layer": hist})
    return {"workload": "large_linear_8bit layers (16384 x 4096 x 11008, 16384 x 11008 x 4096)",
            "peak": peaks["bf16_tflops"], "peak_source": f"{src} bf16 burst",
            "statistic": "sum over the two layers of the median layer-launch time", "rows": rows}


def run_pack(args, dev):
    """Packed sub-byte storage of the 4-bit conv3x3 activation codes (X [12544, 2304], and its
    transposed copy [2304, 12544], the layout a group-ordered layer's weight gradient reads):
    pack (1 byte read + 0.5 written per code) and
    unpack (0.5 + 1), each captured in a CUDA graph and timed with CUDA events around a
    replay after an L2 flush (median), against HBM."""
    import torch
    from paper_2411_10948_gb300 import layer as L
    from paper_2411_10948_gb300 import native as N
    from paper_2411_10948_gb300 import workloads as W
    peaks, src = load_peaks()
    spec = W.workload("conv3x3").layers[0]
    bits, G = spec.bits, spec.n_groups
    x = W.torch_tensor(spec.act, spec.M, spec.K, args.seed + 3, dev)
    q = L.ShiftTensor.alloc(spec.M, spec.K, bits, G, dev)
    st = torch.zeros(1, dtype=torch.int32, device=dev)
    L.shift_quantize(x, q, bits, G, N.SQ_ROUND_NEAREST_EVEN, 0, st)
    flush_l2 = make_l2_flush(dev)
    steps = max(5, min(args.steps, 20))
    out = []
    for name, codes in (("X codes", q.codes), ("X codes transposed", q.codes_t)):
        R, C = codes.shape
        packed = torch.zeros((R, (C + 15) // 16 * 8), dtype=torch.uint8, device=dev)
        back = L.empty_codes(R, C, bits, G, dev)
        graphs = {"pack": L.CapturedStep(lambda: N.shiftquant_pack_codes(codes, bits, G, packed, st)),
                  "unpack": L.CapturedStep(lambda: N.shiftquant_unpack_codes(packed, C, bits, G, back))}
        fns = {k: g.replay for k, g in graphs.items()}
        row = {"tensor": name, "rows": R, "cols": C, "bytes_codes": R * C,
               "bytes_packed": R * ((C + 1) // 2)}
        for k, fn in fns.items():
            fn()
            ts = []
            for _ in range(steps):
                flush_l2()
                a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                a.record()
                fn()
                b.record()
                b.synchronize()
                ts.append(a.elapsed_time(b))
            ms = statistics.median(ts)
            gbs = 1.5 * R * C / (ms * 1e-3) / 1e9
            row.update({f"{k}_ms": ms, f"{k}_gbs": gbs, f"{k}_frac": gbs / peaks["hbm_gbs"]})
        assert torch.equal(back.view(torch.uint8), codes.view(torch.uint8)), "round trip"
        out.append(row)
    assert st.item() == 0
    return {"bits": bits, "n_groups": G, "bytes_per_code": 1.5, "peak": peaks["hbm_gbs"],
            "peak_source": f"{src} copy bandwidth",
            "statistic": "median over graph replays after an L2 flush", "tensors": out}


def oracle_sample_step(wl, rows_per_layer, seed):
    """One bounded oracle step: the quantizer chain and the three GEMMs on the first rows."""
    import oracle as O
    from paper_2411_10948_gb300 import workloads as W
    data = [W.np_layer_inputs(s, seed, i, rows=r) for i, (s, r) in
            enumerate(zip(wl.layers, rows_per_layer))]

    def run(step_idx):
        t0 = time.perf_counter()
        for s, (x, w, dy) in zip(wl.layers, data):
            G = s.n_groups
            ox = O.shiftquant_tensor(x, s.bits, G, 0)
            og = O.shiftquant_tensor(dy, s.bits, G, 1, 0x5EED + step_idx)
            wf = O.channel_tensor(w, s.bits, 0)
            wd = O.channel_tensor(w, s.bits, 1)
            T = O.gemm_fwd(ox["codes"], ox["exp"], wf["codes"], G)
            O.dequant(T, ox["scale"], 1.0, G - 1, wf["scale"])
            T = O.gemm_dgrad(og["codes"], og["exp"], wd["codes"], G)
            O.dequant(T, og["scale"], 1.0, G - 1, wd["scale"])
            T = O.gemm_wgrad(ox["codes"], ox["exp"], og["codes"], og["exp"], G)
            O.dequant(T, ox["scale"], og["scale"], 2 * (G - 1))
        return time.perf_counter() - t0
    ops = sum(3 * 2 * r * s.N * s.K for s, r in zip(wl.layers, rows_per_layer))
    return run, ops


def choose_rows(wl, target_s, seed):
    """Rows per layer so that one oracle step takes about target_s seconds."""
    probe = [min(s.M, 256) for s in wl.layers]
    run, ops = oracle_sample_step(wl, probe, seed)
    run(0)
    dt = max(run(0), 1e-3)
    scale = target_s / dt
    return [max(1, min(s.M, int(p * scale))) for s, p in zip(wl.layers, probe)]


def cpu_baseline(wl, seed, target_s=12.0):
    import oracle as O
    rows = choose_rows(wl, target_s, seed)
    run, ops = oracle_sample_step(wl, rows, seed)
    dt = run(0)
    full_ops = sum(3 * 2 * s.M * s.N * s.K for s in wl.layers)
    sampled = any(r < s.M for s, r in zip(wl.layers, rows))
    return {"value": ops / dt / 1e12, "unit": UNIT, "cores": O.max_threads(), "kind": "oracle",
            "sample": (f"first {rows} token rows of the {[s.M for s in wl.layers]} of each layer: "
                       "range+grouping+quantization of X, dY and W (both roles) and the three "
                       f"GEMMs over those rows, one step, {dt:.1f} s"),
            "extrapolated": sampled,
            "full_step_seconds_extrapolated": full_ops / (ops / dt) if sampled else dt,
            "seconds": dt}


def run_reference(args):
    import oracle as O
    from paper_2411_10948_gb300 import workloads as W
    O.build()
    wl = W.workload(args.workload)
    rows = choose_rows(wl, 4.0, args.seed)
    run, ops = oracle_sample_step(wl, rows, args.seed)
    for i in range(args.warmup):
        run(i)
    times = [run(args.warmup + i) for i in range(args.steps)]
    total = sum(times)
    value = ops * args.steps / total / 1e12
    sample = (f"first {rows} token rows of the {[s.M for s in wl.layers]} of each layer per step: "
              "range+grouping+quantization of X, dY and W and the three GEMMs over those rows")
    return {
        "impl": "reference",
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": total / args.steps * 1e3,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "int64",
        "data": "synthetic",
        "config": {"workload": args.workload, "description": wl.description,
                   "layers": [[s.name, s.M, s.K, s.N] for s in wl.layers]},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": O.max_threads(), "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }


def main():
    args = parse_args()
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if args.impl == "reference":
        if rank == 0:
            print(json.dumps(run_reference(args)), flush=True)
        return
    if world > 1:
        import torch
        import torch.distributed as dist
        torch.cuda.set_device(local_rank)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local_rank))
    result, _ = run_ours(args, rank, world, local_rank)
    if rank == 0:
        if world == 1 and args.also not in ("", "none", args.workload):
            # a second workload (by default the 4-bit conv3x3 layer) summarised in the same line
            sub = argparse.Namespace(**vars(args))
            sub.workload, sub.no_e2e, sub.steps = args.also, True, max(3, min(args.steps, 10))
            other, _ = run_ours(sub, rank, world, local_rank)
            result["also"] = {k: other[k] for k in ("value", "unit", "ms_per_step", "dtype")}
            result["also"].update({"config": {"workload": args.also,
                                              "description": other["config"]["description"]},
                                   "roofline": other["roofline"],
                                   "gemm": {k: other["gemm"][k] for k in ("achieved", "peak", "unit", "frac",
                                                                          "frac_of_clock_peak", "hbm_gbs",
                                                                          "hbm_frac")},
                                   "quantizer": {k: other["quantizer"][k] for k in ("achieved", "peak", "unit", "frac", "in_step")
                                                 if k in other["quantizer"]},
                                   "clocks": other["clocks"]})
        if world == 1 and not args.no_chain:
            result["fused_range_chain"] = run_chain(args, f"cuda:{local_rank}")
        if world == 1 and not args.no_l1bn:
            result["l1bn"] = run_l1bn(args, f"cuda:{local_rank}")
        if world == 1 and not args.no_group_order:
            result["group_order"] = run_group_order(args, f"cuda:{local_rank}")
        if world == 1 and not args.no_pack:
            result["packed_storage"] = run_pack(args, f"cuda:{local_rank}")
        if world == 1 and not args.no_cpu_baseline:
            from paper_2411_10948_gb300 import workloads as W
            result["cpu_baseline"] = cpu_baseline(W.workload(args.workload), args.seed)
        print(json.dumps(result), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.barrier()
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
