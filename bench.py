#!/usr/bin/env python3
"""Benchmark of the structured-pruned CONV forward path on GB300.

One step = the whole path over one batch of every layer of the workload:
sadmm_project_groups (group norms + exact top-k) -> sadmm_pack -> sadmm_conv_fwd
(implicit GEMM on the kept filters and columns, bias + ReLU, zero planes).

Default workload: AlexNet CONV1-5 at batch 128 (bf16 inputs, fp32 output),
filter-wise plus shape-wise pruning at retained fractions 1.0/0.5/0.25/0.2/0.2
(each applied to filters and columns), seeded synthetic tensors.

Metric: TFLOP/s on retained MACs (2 * M * F' * K' per layer) over the step,
plus the fraction of the measured bf16 tensor peak and the speedup over the
same step at 0% sparsity.  Timing: CUDA events on the launching stream, L2
flushed (256 MiB write) before every timed step, outside the timed window; a
short device sleep before each step's start event lets the host enqueue ahead,
so the window holds only GPU work.

Usage: python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reference]
                       [--workload alexnet|single2d|c3d|resnet50|sweep]
                       [--out-dtype fp32|bf16]
Under torchrun (N > 1) every rank runs its own batch (weak scaling, no
collective on the data path); rank 0 prints one JSON line.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import workloads as wl  # noqa: E402

METRIC = "pruned-conv TFLOP/s (retained MACs) & % bf16 peak; speedup vs dense"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(p) as fh:
            d = json.load(fh)
        return {k: float(d[k]) for k in FALLBACK_PEAKS}, "measured"
    except Exception:
        return dict(FALLBACK_PEAKS), "fallback"


def dist_env():
    from paper_1807_11091_gb300 import ranks
    return ranks.dist_env()


def check_gpus(gpus, world_size):
    """None when --gpus matches the launch, else the error to print: one process
    per GPU, so N > 1 GPUs need N ranks (torchrun sets WORLD_SIZE)."""
    if gpus == world_size:
        return None
    return (f"bench.py: --gpus {gpus} but {world_size} rank(s) running; launch N > 1 GPUs as "
            f"python -m torch.distributed.run --nproc-per-node N bench.py --gpus N")


def workload_name(name, layers, out_dtype):
    desc = {
        "alexnet": "AlexNet CONV1-5, batch 128, filter-wise + shape-wise pruning, retained 1.0/0.5/0.25/0.2/0.2",
        "single2d": "single 2-D CONV N8 C64 32x32 F64 3x3, shape-wise 50%",
        "c3d": "C3D layer N8 C128 T8 28x28 F256 3x3x3, shape-wise 30%",
        "resnet50": "ResNet-50 bottleneck CONV layers, batch 64, filter-wise 50% + channel-wise 50%",
        "sweep": "N128 C256 28x28 F512 3x3, shape-wise {1,.5,.25,.1,.05} x filter-wise {1,.5}",
    }[name]
    return f"{desc} ({out_dtype} output)"


def workload_config(args, layers):
    """The config keys that name the workload, the same in both arms."""
    return {"workload": workload_name(args.workload, layers, args.out_dtype),
            "layers": [L.name for L in layers],
            "out_dtype": args.out_dtype,
            "parallelism": "one replica per GPU, batch per GPU fixed, no collective"}


# --------------------------------------------------------------------------
# Reference arm: the CPU oracle as it stands
# --------------------------------------------------------------------------

def oracle_sample_step(layers, tensors, nimg):
    """The path through the oracle on images 0..nimg-1 of every layer; returns
    the retained FLOPs of that sample."""
    import oracle
    flops = 0.0
    for L, t in zip(layers, tensors):
        s = L.shape
        rows, cols, _, _ = oracle.project(t["W"], s.taps, L.k_filters, L.colkind, L.k_cols)
        d = s.with_batch(int(t["x"].shape[0])).desc16()
        oracle.pruned_conv(t["x"], t["W"], t["bias"], d, s.taps, rows, L.colkind, cols,
                           relu=True, n0=0, n1=nimg)
        flops += L.retained_flops() * nimg / s.n
    return flops


def oracle_threads():
    try:
        import oracle
        lib = oracle._load()
        import ctypes
        omp = ctypes.CDLL(lib._name)
        f = getattr(omp, "omp_get_max_threads", None)
        if f is not None:
            return int(f())
    except Exception:
        pass
    return os.cpu_count() or 1


def cpu_baseline(layers, tensors, target_s=10.0):
    """Times the oracle on a bounded sample: images 0..n-1 of every layer,
    repeated until about target_s seconds of CPU work (capped at the batch)."""
    t0 = time.perf_counter()
    f1 = oracle_sample_step(layers, tensors, 1)
    dt1 = time.perf_counter() - t0
    batch = min(int(t["x"].shape[0]) for t in tensors)
    nimg = max(1, min(batch, int(target_s / max(dt1, 1e-3))))
    f, dt, passes = 0.0, 0.0, 0
    while dt < target_s * 0.8 and passes < 16:
        t0 = time.perf_counter()
        f += oracle_sample_step(layers, tensors, nimg)
        dt += time.perf_counter() - t0
        passes += 1
    return {"value": f / dt / 1e12, "unit": "TFLOP/s", "cores": oracle_threads(), "kind": "oracle",
            "sample": f"images 0..{nimg - 1} of every layer, {passes} pass(es), through oracle.project + "
                      f"oracle.pruned_conv (fp64 direct convolution over the full masked weights), {dt:.1f} s"}


def run_reference(args):
    from paper_1807_11091_gb300 import ranks
    ws, rank, _ = dist_env()
    if not ranks.reports(rank):
        return 0  # the oracle runs on rank 0 only; the other ranks exit without work
    layers = wl.get(args.workload)
    tensors = [wl.gen_tensors(L.shape.with_batch(1), seed=L.seed) for L in layers]
    # each step is one image of every layer (a bounded sample of the workload)
    for _ in range(args.warmup):
        oracle_sample_step(layers, tensors, 1)
    times, flops = [], 0.0
    for _ in range(args.steps):
        t0 = time.perf_counter()
        flops = oracle_sample_step(layers, tensors, 1)
        times.append(time.perf_counter() - t0)
    tot = sum(times)
    value = flops * args.steps / tot / 1e12
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "TFLOP/s",
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": tot / args.steps * 1e3, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": workload_config(args, layers),
        "cpu_baseline": {"value": value, "unit": "TFLOP/s", "cores": oracle_threads(), "kind": "oracle",
                         "sample": "image 0 of every layer per step, through oracle.project + "
                                   "oracle.pruned_conv (fp64 direct convolution over the full masked weights)"},
        "e2e": {"value": value, "unit": "TFLOP/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
        "gpu_launches": 0,
    }
    print(json.dumps(line), flush=True)
    return 0


# --------------------------------------------------------------------------
# GPU arm
# --------------------------------------------------------------------------

class LayerRun:
    """Device buffers and raw-pointer arguments of one layer's path."""

    def __init__(self, L, t, dev, out_dtype, dense=False, max_ctas=0):
        import torch
        from paper_1807_11091_gb300 import sadmm
        self.L = L
        s = L.shape
        self.s = s
        self.dense = dense
        self.k_filters = s.f if dense else L.k_filters
        self.colkind = L.colkind
        G = s.cg if L.colkind == wl.COL_CHANNEL else s.k
        self.k_cols = (G if dense else L.k_cols) if L.colkind != wl.COL_NONE else 0
        self.n_cg = self.k_cols if L.colkind != wl.COL_NONE else s.k
        self.W = t["W"].to(dev)
        self.x = t["x"].to(dev)
        self.bias = t["bias"].to(dev)
        self.desc = sadmm.make_desc(s.desc16())
        self.ws_bytes = sadmm.sadmm_workspace_size(self.desc, self.colkind)
        self.ws = torch.empty(self.ws_bytes, dtype=torch.uint8, device=dev)
        self.fi = torch.empty(max(s.f, 1), dtype=torch.int32, device=dev)
        self.ci = torch.empty(max(G, 1), dtype=torch.int32, device=dev)
        st, self.plan = sadmm.sadmm_plan_init_ctas(self.desc, self.k_filters, self.colkind, self.n_cg, max_ctas)
        assert st == 0, st
        self.buf = torch.empty(self.plan.dev_bytes, dtype=torch.uint8, device=dev)
        self.ydt = sadmm.SADMM_BF16 if out_dtype == "bf16" else sadmm.SADMM_FP32
        ytype = torch.bfloat16 if out_dtype == "bf16" else torch.float32
        self.y = torch.empty(s.y_shape(), dtype=ytype, device=dev)
        self.out_bytes = 2 if out_dtype == "bf16" else 4
        # projection (filter keys, whose launch also writes the lists of kinds kept
        # whole; the row select; column keys + select), pack (meta + rows, the
        # slab-ordered rows in the same launch), conv (+ split-K finalize, or after
        # the input-slab path's space-to-depth pass)
        rows_all = self.k_filters == s.f
        cols_all = self.colkind != wl.COL_NONE and self.k_cols == G
        self.launches = (1 + (0 if rows_all else 1)
                         + (2 if self.colkind != wl.COL_NONE and not cols_all else 0) + 2
                         + (2 if self.plan.splits > 1 or self.plan.xs_mode else 1))

    def flops(self):
        s = self.s
        return 2.0 * s.m * self.k_filters * (self.k_cols * (s.taps if self.colkind == wl.COL_CHANNEL else 1)
                                            if self.colkind != wl.COL_NONE else s.k)

    def conv_bytes(self):
        """Algorithmic HBM bytes of one conv launch: x once, packed weights once,
        the full output once, the bias."""
        s = self.s
        kc = self.flops() / (2.0 * s.m * max(self.k_filters, 1)) if self.k_filters else 0
        return (s.n * s.c * s.t * s.h * s.w * 2 + self.k_filters * kc * 2
                + s.n * s.f * s.plane * self.out_bytes + s.f * 4)

    def project(self, stream):
        from paper_1807_11091_gb300 import sadmm
        st = sadmm.sadmm_project_groups(self.desc, self.W.data_ptr(), None, sadmm.SADMM_BF16, self.k_filters,
                                        self.colkind, self.k_cols, self.fi.data_ptr(),
                                        self.ci.data_ptr() if self.colkind != wl.COL_NONE else None, None,
                                        self.ws.data_ptr(), self.ws_bytes, stream)
        assert st == 0, st

    def pack(self, stream):
        from paper_1807_11091_gb300 import sadmm
        st = sadmm.sadmm_pack(self.plan, self.W.data_ptr(), sadmm.SADMM_BF16,
                              self.fi.data_ptr() if self.k_filters < self.s.f else None,
                              self.ci.data_ptr() if self.colkind != wl.COL_NONE else None,
                              self.buf.data_ptr(), self.plan.dev_bytes, stream)
        assert st == 0, st

    def conv(self, stream, phase=0):
        """sadmm_conv_fwd, or one phase of it (sadmm_conv_fwd_phase)."""
        from paper_1807_11091_gb300 import sadmm
        st = sadmm.sadmm_conv_fwd_phase(self.plan, self.x.data_ptr(), self.bias.data_ptr(), 1, self.y.data_ptr(),
                                        self.ydt, phase, stream)
        assert st == 0, st

    @property
    def early_input(self):
        """The forward's input pass reads only x: it can run before the pack."""
        return bool(self.plan.xs_mode) and self.colkind != wl.COL_CHANNEL


class FirstLayerChunks:
    """The first layer's forward over n_chunks equal slices of its batch, with a
    plan of its own for the slice (the same projection lists, packed again for
    that plan).  Used by the end-to-end step only: the first slice's output can
    go back to the host while the later slices' inputs still upload, instead of
    after the whole first input has crossed the link.  Every image's output is
    the one the whole-batch plan gives."""

    def __init__(self, r, n_chunks, dev, max_ctas=0):
        import torch
        from paper_1807_11091_gb300 import sadmm
        s = r.s
        assert n_chunks > 1 and s.n % n_chunks == 0
        self.r = r
        self.n_chunks = n_chunks
        self.nb = s.n // n_chunks
        d16 = s.desc16()
        d16[0] = self.nb
        self.desc = sadmm.make_desc(d16)
        st, self.plan = sadmm.sadmm_plan_init_ctas(self.desc, r.k_filters, r.colkind, r.n_cg, max_ctas)
        assert st == 0, st
        self.buf = torch.empty(self.plan.dev_bytes, dtype=torch.uint8, device=dev)
        self.x_bytes = self.nb * s.c * s.t * s.h * s.w * 2
        self.y_bytes = self.nb * s.f * s.plane * r.out_bytes

    def pack(self, stream):
        from paper_1807_11091_gb300 import sadmm
        r = self.r
        st = sadmm.sadmm_pack(self.plan, r.W.data_ptr(), sadmm.SADMM_BF16,
                              r.fi.data_ptr() if r.k_filters < r.s.f else None,
                              r.ci.data_ptr() if r.colkind != wl.COL_NONE else None,
                              self.buf.data_ptr(), self.plan.dev_bytes, stream)
        assert st == 0, st

    def conv(self, stream, j, phase=0):
        from paper_1807_11091_gb300 import sadmm
        r = self.r
        st = sadmm.sadmm_conv_fwd_phase(self.plan, r.x.data_ptr() + j * self.x_bytes, r.bias.data_ptr(), 1,
                                        r.y.data_ptr() + j * self.y_bytes, r.ydt, phase, stream)
        assert st == 0, st

    @property
    def early_input(self):
        return bool(self.plan.xs_mode) and self.r.colkind != wl.COL_CHANNEL

    @staticmethod
    def plan_whole_tiles(plan):
        """Every output tile summed by one CTA in K' order (no split-K, no stream-K)."""
        return plan.splits == 1 and plan.sk_len == 0

    def whole_tiles(self):
        return self.plan_whole_tiles(self.plan)

    def rows(self, j):
        return slice(j * self.nb, (j + 1) * self.nb)


class StepStreams:
    """One side stream per layer: each layer's projection and pack run on its own
    stream (the layers are independent), forked from and joined back to the main
    stream (high priority), where the convolutions run back to back.  The first
    layer's side stream has the main stream's priority (its pack gates the first conv); the first
    conv's plan leaves a few SMs free so the other layers' projection and pack
    run beside it instead of after it."""

    def __init__(self, n):
        import torch
        self.main = torch.cuda.current_stream()
        self.side = [torch.cuda.Stream(priority=-1 if i == 0 else 0) for i in range(n)]
        self.fork = torch.cuda.Event()
        self.done = [torch.cuda.Event() for _ in range(n)]


def enqueue_step(runs, ss, conv_events=None):
    """One step.  An input-slab layer without channel pruning (the first
    layer) runs its forward's input pass on the main stream at once, beside its
    projection and pack, then the rest after them.  With conv_events (the
    per-layer breakdown) every forward runs as one call between its events."""
    import torch
    from paper_1807_11091_gb300 import sadmm
    ss.fork.record(ss.main)
    for r, side, done in zip(runs, ss.side, ss.done):
        side.wait_event(ss.fork)
        sp = int(side.cuda_stream)
        r.project(sp)
        r.pack(sp)
        done.record(side)
    mp = int(ss.main.cuda_stream)
    split = conv_events is None
    for r in runs:
        if split and r.early_input:
            r.conv(mp, sadmm.SADMM_FWD_INPUT)
    for i, (r, done) in enumerate(zip(runs, ss.done)):
        # The later layers' packs finish beside the first conv; waiting for all
        # of them before the second conv leaves the later convs back to back in
        # the stream, so each is launched while the one before it drains
        # (programmatic dependent launch; a wait between two kernels prevents it).
        if i == 0:
            ss.main.wait_event(done)
        elif i == 1:
            for d in ss.done[1:]:
                ss.main.wait_event(d)
        if conv_events is not None:
            conv_events[i][0].record(ss.main)
        r.conv(mp, sadmm.SADMM_FWD_REST if split and r.early_input else sadmm.SADMM_FWD_ALL)
        if conv_events is not None:
            conv_events[i][1].record(ss.main)


def enqueue_step_e2e(runs, ss, copy_stream, h_x, h_w, h_b, h_y, up_stream, first=None):
    """The step with its host transfers overlapped.  The inputs go host -> device
    on one upload stream, the layers' weights and biases first (small: every
    projection and pack can start), then x layer by layer, so the first conv's
    input arrives at the link's full rate; each output goes device -> host on
    `copy_stream` as soon as its conv has run, while the later inputs still
    upload (the link carries both directions at once).  With `first` (a
    FirstLayerChunks) the first layer's input, forward and output go slice by
    slice, so its first output slice starts back while the rest still uploads.
    The main stream joins the copy stream at the end, so an event recorded
    after this call covers every copy."""
    import torch
    from paper_1807_11091_gb300 import sadmm
    ss.fork.record(ss.main)
    up_stream.wait_event(ss.fork)
    w_ready, x_ready, xc_ready = [], [], []
    with torch.cuda.stream(up_stream):
        for r, b, c in zip(runs, h_w, h_b):
            r.W.copy_(b, non_blocking=True)
            r.bias.copy_(c, non_blocking=True)
            ev = torch.cuda.Event()
            ev.record(up_stream)
            w_ready.append(ev)
        for i, (r, a) in enumerate(zip(runs, h_x)):
            if i == 0 and first is not None:
                for j in range(first.n_chunks):
                    r.x[first.rows(j)].copy_(a[first.rows(j)], non_blocking=True)
                    ev = torch.cuda.Event()
                    ev.record(up_stream)
                    xc_ready.append(ev)
                x_ready.append(xc_ready[-1])
                continue
            r.x.copy_(a, non_blocking=True)
            ev = torch.cuda.Event()
            ev.record(up_stream)
            x_ready.append(ev)
    for i, (r, side, done, wr) in enumerate(zip(runs, ss.side, ss.done, w_ready)):
        side.wait_event(wr)
        sp = int(side.cuda_stream)
        r.project(sp)
        (first if i == 0 and first is not None else r).pack(sp)
        done.record(side)
    mp = int(ss.main.cuda_stream)

    def copy_back(hy, y):
        ev = torch.cuda.Event()
        ev.record(ss.main)
        copy_stream.wait_event(ev)
        with torch.cuda.stream(copy_stream):
            hy.copy_(y, non_blocking=True)

    if first is not None:
        early = first.early_input
        for j in range(first.n_chunks):
            ss.main.wait_event(xc_ready[j])
            if early:
                first.conv(mp, j, sadmm.SADMM_FWD_INPUT)
            if j == 0:
                ss.main.wait_event(ss.done[0])
            first.conv(mp, j, sadmm.SADMM_FWD_REST if early else sadmm.SADMM_FWD_ALL)
            copy_back(h_y[0][first.rows(j)], runs[0].y[first.rows(j)])
    else:
        early = runs[0].early_input
        if early:
            ss.main.wait_event(x_ready[0])
            runs[0].conv(mp, sadmm.SADMM_FWD_INPUT)
    for i, (r, done, hy, xr) in enumerate(zip(runs, ss.done, h_y, x_ready)):
        if i == 0 and first is not None:
            continue
        ss.main.wait_event(done)
        ss.main.wait_event(xr)
        r.conv(mp, sadmm.SADMM_FWD_REST if (i == 0 and early) else sadmm.SADMM_FWD_ALL)
        copy_back(hy, r.y)
    end = torch.cuda.Event()
    end.record(copy_stream)
    ss.main.wait_event(end)


class ClockSampler:
    """nvidia-smi sampling of SM clock, power and throttle reasons."""

    FIELDS = ("timestamp,index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index, path=None):
        self.index = index
        self.proc = None
        self.lines = []
        self.path = path

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits", "-i",
                 str(self.index), "-lms", "100"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except Exception:
            self.proc.kill()
            out, _ = self.proc.communicate()
        self.lines = [ln for ln in out.splitlines() if ln.strip()]
        if self.path:
            try:
                with open(self.path, "w") as fh:
                    fh.write(self.FIELDS + "\n" + "\n".join(self.lines) + "\n")
            except Exception:
                pass

    def summary(self):
        sm, mx, reasons, power = [], None, set(), []
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            f = [x.strip() for x in ln.split(",")]
            if len(f) < 10:
                continue
            try:
                clk = float(f[2])
                mx = float(f[3])
            except ValueError:
                continue
            try:
                power.append(float(f[4]))
            except ValueError:
                pass
            sm.append(clk)
            for nm, v in zip(names, f[6:10]):
                if v.lower().startswith("active"):
                    reasons.add(nm)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        # under load: samples drawing at least half the peak power seen (all of them when
        # the power column was unreadable); the sampler also runs a little before and after
        # the timed steps, where the GPU idles
        if len(power) == len(sm):
            top = max(power)
            loaded = [c for c, p in zip(sm, power) if p >= 0.5 * top]
        else:
            loaded = sm
        return {"sm_mhz": statistics.median(loaded), "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(sm), "power_w_max": max(power) if power else None}


TRAFFIC_FILE = os.path.join(ROOT, "profiles", "conv_fwd_alexnet_b128_dram.txt")
# the forward kernels' sources: the gathered kernel, the input-slab kernels and what they share
CONV_SRCS = [os.path.join(ROOT, "paper_1807_11091_gb300", "csrc", f)
             for f in ("conv_fwd.cu", "conv_slab.cu", "conv_common.cuh", "common.cuh")]


def conv_source_sha1():
    """sha1 over the forward kernels' source files, in CONV_SRCS order."""
    import hashlib
    h = hashlib.sha1()
    for f in CONV_SRCS:
        with open(f, "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()


def conv_traffic(workload, out_dtype):
    """DRAM bytes per sadmm_conv_fwd call (read + write of every kernel it
    launches, averaged over the step's calls) from the committed ncu summary, or
    None when that summary is for another workload or the kernel sources changed
    since it was taken."""
    if workload != "alexnet" or out_dtype != "fp32":
        return None
    try:
        fields = {}
        with open(TRAFFIC_FILE) as fh:
            for ln in fh:
                if ":" in ln and not ln.startswith("#"):
                    k, v = ln.split(":", 1)
                    fields[k.strip()] = v.strip()
        if fields.get("kernel_source_sha1") != conv_source_sha1():
            return None
        return float(fields["dram_bytes_per_call_avg"])
    except Exception:
        return None


def capture_step(rs, ss):
    """The step of the layers `rs` captured once (after warm-up) into a CUDA
    graph: the same launches, streams' dependencies and programmatic launches,
    replayed with one graph launch per step instead of one host call per
    kernel."""
    import torch
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=ss.main):
        enqueue_step(rs, ss)
    torch.cuda.synchronize()
    return g


def time_steps(rs, ss, flush, k, with_conv_events, graph=None):
    """k steps of the layers `rs`, L2 flushed before each (outside the window):
    the step times (ms) and, with events around each forward call, the per-call
    times.  With `graph` (capture_step) each step without per-call events is
    one replay of it."""
    import torch
    step_ms, conv_ms = [], [[] for _ in rs]
    for _ in range(k):
        flush.fill_(1)
        torch.cuda._sleep(3_000_000)  # ~1.5-2 ms: host enqueues the step meanwhile
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in rs] \
            if with_conv_events else None
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record()
        if graph is not None and not with_conv_events:
            graph.replay()
        else:
            enqueue_step(rs, ss, ev)
        e1.record()
        torch.cuda.synchronize()
        step_ms.append(e0.elapsed_time(e1))
        if ev:
            for i, (a, b) in enumerate(ev):
                conv_ms[i].append(a.elapsed_time(b))
    return step_ms, conv_ms


def calls_report(runs, flush, reps=50, warmup=10):
    """sadmm_conv_fwd alone, per layer (the plans packed by the steps before):
    10 warm-up calls, then the median of `reps` calls with the L2 flushed before
    each (outside the window) and of `reps` back-to-back calls with a warm L2."""
    import torch
    sp = int(torch.cuda.current_stream().cuda_stream)
    out = {}
    for r in runs:
        for _ in range(warmup):
            r.conv(sp)
        res = {}
        for mode in ("flushed", "warm"):
            evs = []
            for _ in range(reps):
                if mode == "flushed":
                    flush.fill_(1)
                e0 = torch.cuda.Event(enable_timing=True)
                e1 = torch.cuda.Event(enable_timing=True)
                e0.record()
                r.conv(sp)
                e1.record()
                evs.append((e0, e1))
            torch.cuda.synchronize()
            us = statistics.median(a.elapsed_time(b) for a, b in evs) * 1e3
            res[f"{mode}_us"] = us
            res[f"{mode}_tflops"] = r.flops() / (us * 1e-6) / 1e12
        out[r.L.name] = res
    return {"what": f"sadmm_conv_fwd alone per layer: {warmup} warm-up calls, median of {reps} calls with the L2 "
                    f"flushed before each and of {reps} back-to-back calls (warm L2)", "layers": out}


def forward_roofline(runs, t_conv_s, peaks):
    """Roofline of the forward calls of a step: the binding roof (HBM bytes or
    bf16 tensor flops, algorithmic) and the fraction of it reached."""
    nbytes = sum(r.conv_bytes() for r in runs)
    flops = sum(r.flops() for r in runs)
    t_mem = nbytes / (peaks["hbm_gbs"] * 1e9)
    t_cmp = flops / (peaks["bf16_tflops"] * 1e12)
    if t_mem >= t_cmp:
        a = nbytes / t_conv_s / 1e9
        roof = {"bound": "hbm", "achieved": a, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                "frac": a / peaks["hbm_gbs"]}
    else:
        a = flops / t_conv_s / 1e12
        roof = {"bound": "tensor", "achieved": a, "peak": peaks["bf16_tflops"], "unit": "TFLOP/s",
                "frac": a / peaks["bf16_tflops"]}
    roof["combined_roofline_frac"] = max(t_mem, t_cmp) / t_conv_s
    return roof


WORKLOAD_LABELS = {
    "c3d": "C3D layer N8 C128 T8 28x28 F256 3x3x3 p1, shape-wise 30%",
    "resnet50": "ResNet-50 bottleneck CONV layers (16), batch 64, filter-wise 50% x channel-wise 50%",
    "single2d": "single 2-D CONV N8 C64 32x32 F64 3x3 p1, shape-wise 50%",
}


def configs_report(dev, out_dtype, peaks, steps=10, names=("c3d", "resnet50", "single2d"), graphs=True):
    """The other workloads through the same step as the headline line
    (projection + pack + forward of every layer, L2 flushed before each step):
    TFLOP/s on retained MACs, the forward calls' roofline (whichever of HBM and
    the bf16 tensor peak binds) and the speedup over the same step at 0%
    sparsity."""
    import torch
    out = {}
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    for name in names:
        layers = wl.get(name)
        tensors = [wl.gen_tensors(L.shape, seed=L.seed) for L in layers]
        runs = [LayerRun(L, t, dev, out_dtype) for L, t in zip(layers, tensors)]
        dense = [LayerRun(L, t, dev, out_dtype, dense=True) for L, t in zip(layers, tensors)]
        ss = StepStreams(len(runs))
        for _ in range(3):
            enqueue_step(runs, ss)
            enqueue_step(dense, ss)
        torch.cuda.synchronize()
        g_runs = capture_step(runs, ss) if graphs else None
        g_dense = capture_step(dense, ss) if graphs else None
        step_ms, _ = time_steps(runs, ss, flush, steps, False, g_runs)
        _, conv_ms = time_steps(runs, ss, flush, steps, True)
        dense_ms, _ = time_steps(dense, ss, flush, steps, False, g_dense)
        _, dconv_ms = time_steps(dense, ss, flush, steps, True)
        del g_runs, g_dense
        from paper_1807_11091_gb300 import sadmm
        if sadmm.sadmm_last_device_status(int(torch.cuda.current_stream().cuda_stream)) != 0:
            raise RuntimeError(f"device status set after the {name} steps")
        flops = sum(r.flops() for r in runs)
        t_step = statistics.median(step_ms)
        t_conv = sum(statistics.median(c) for c in conv_ms)
        t_dconv = sum(statistics.median(c) for c in dconv_ms)
        tf = flops / (t_step * 1e-3) / 1e12
        out[name] = {
            "workload": WORKLOAD_LABELS[name], "layers": len(runs), "ms_per_step": t_step,
            "tflops_retained": tf, "pct_bf16_peak": tf / peaks["bf16_tflops"],
            "conv_us": t_conv * 1e3, "conv_tflops": flops / (t_conv * 1e-3) / 1e12,
            "speedup_vs_dense": statistics.median(dense_ms) / t_step,
            "conv_speedup_vs_dense": t_dconv / t_conv,
            "roofline": forward_roofline(runs, t_conv * 1e-3, peaks),
        }
        del runs, dense, tensors, ss
        torch.cuda.empty_cache()
    del flush
    torch.cuda.empty_cache()
    return out


def sweep_report(dev, out_dtype, reps=5, peak_tflops=None):
    """sadmm_conv_fwd alone on the large sweep layer (N128 C256 28x28 F512 3x3)
    at every retained fraction, against the same kernel at 0% sparsity."""
    import torch
    layers = wl.sweep()
    s = layers[0].shape
    t = wl.gen_tensors(s, seed=layers[0].seed)
    dense = wl.Layer("sweep_dense", s, 1.0, wl.COL_SHAPE, 1.0, seed=layers[0].seed)
    runs = [LayerRun(L, t, dev, out_dtype) for L in [dense] + layers]
    for r in runs[1:]:  # one input and output buffer for all variants
        r.x, r.y = runs[0].x, runs[0].y
    sp = int(torch.cuda.current_stream().cuda_stream)
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    for r in runs:
        r.project(sp)
        r.pack(sp)
        r.conv(sp)
    torch.cuda.synchronize()
    times = []
    for r in runs:
        ms = []
        for _ in range(reps):
            flush.fill_(1)
            torch.cuda._sleep(1_000_000)
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record()
            r.conv(sp)
            e1.record()
            torch.cuda.synchronize()
            ms.append(e0.elapsed_time(e1))
        times.append(statistics.median(ms))
    dense_us = times[0] * 1e3
    out = {"layer": "N128 C256 28x28 F512 3x3 p1, shape-wise x filter-wise", "dense_conv_us": dense_us,
           "dense_tflops": runs[0].flops() / (times[0] * 1e-3) / 1e12, "variants": []}
    if peak_tflops:
        out["dense_pct_bf16_peak"] = out["dense_tflops"] / peak_tflops
    for L, r, ms in zip(layers, runs[1:], times[1:]):
        out["variants"].append({"filters": L.filt_frac, "columns": L.col_frac, "conv_us": ms * 1e3,
                                "tflops_retained": r.flops() / (ms * 1e-3) / 1e12,
                                "speedup_vs_dense": times[0] / ms,
                                "retained_fraction": r.flops() / runs[0].flops()})
        if peak_tflops:
            out["variants"][-1]["pct_bf16_peak"] = out["variants"][-1]["tflops_retained"] / peak_tflops
    del runs, flush
    torch.cuda.empty_cache()
    return out


def sparse_report(dev, out_dtype, sweep, reps=3, densities=(0.5, 0.25, 0.1, 0.05)):
    """The paper's non-structured comparison (Sec. 5) on this GPU: the sweep
    layer pruned element by element (sadmm_project_elements keeps the largest
    |W|) and run by the sparse forward (sadmm_sparse_conv_fwd, CSR rows on the
    CUDA cores), beside the structured kernel at the same retained fraction
    (filters kept, that fraction of the columns) and the dense run."""
    import torch
    from paper_1807_11091_gb300 import sadmm
    L0 = wl.sweep()[0]
    s = L0.shape
    t = wl.gen_tensors(s, seed=L0.seed)
    W, x, b = t["W"].to(dev), t["x"].to(dev), t["bias"].to(dev)
    ytype = torch.bfloat16 if out_dtype == "bf16" else torch.float32
    y = torch.empty(s.y_shape(), dtype=ytype, device=dev)
    ydt = sadmm.SADMM_BF16 if out_dtype == "bf16" else sadmm.SADMM_FP32
    desc = sadmm.make_desc(s.desc16())
    sp = int(torch.cuda.current_stream().cuda_stream)
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    structured = {(v["filters"], v["columns"]): v for v in sweep["variants"]}
    out = {"what": "sweep layer N128 C256 28x28 F512 3x3 pruned element by element (largest |W| kept), "
                   "sadmm_sparse_conv_fwd (CSR rows, CUDA cores) vs sadmm_conv_fwd at the same retained "
                   "fraction, L2 flushed, median of " + str(reps), "variants": []}
    for d in densities:
        k = wl.retained(d, s.f * s.k)
        keep = sadmm.project_elements(s.desc16(), W, k)
        nbytes = sadmm.sadmm_sparse_plan_size(desc, k)
        plan = torch.empty(nbytes, dtype=torch.uint8, device=dev)
        st = sadmm.sadmm_sparse_pack(desc, W.data_ptr(), sadmm.SADMM_BF16, keep.data_ptr(), k, plan.data_ptr(),
                                     nbytes, sp)
        assert st == 0, st
        ms = []
        for _ in range(reps + 1):
            flush.fill_(1)
            torch.cuda._sleep(1_000_000)
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record()
            st = sadmm.sadmm_sparse_conv_fwd(desc, plan.data_ptr(), x.data_ptr(), b.data_ptr(), 1, y.data_ptr(),
                                             ydt, sp)
            e1.record()
            torch.cuda.synchronize()
            assert st == 0, st
            ms.append(e0.elapsed_time(e1))
        t_ms = statistics.median(ms[1:])
        fl = 2.0 * s.m * k
        v = {"density": d, "sparse_us": t_ms * 1e3, "sparse_tflops_retained": fl / (t_ms * 1e-3) / 1e12,
             "sparse_speedup_vs_dense": sweep["dense_conv_us"] / (t_ms * 1e3)}
        st_v = structured.get((1.0, d))
        if st_v:
            v["structured_us"] = st_v["conv_us"]
            v["structured_over_sparse"] = t_ms * 1e3 / st_v["conv_us"]
        out["variants"].append(v)
        del keep, plan
    if sadmm.sadmm_last_device_status(sp) != 0:
        raise RuntimeError("device status set after the sparse forwards")
    del flush, y, W, x, b
    torch.cuda.empty_cache()
    return out


def projection_batch_report(dev, peak_gbs, reps=5):
    """The projection of every ResNet-50 bottleneck layer (16 layers, bf16 W,
    filter-wise 50 % + channel-wise 50 %, Sec. 4) as one
    sadmm_project_groups_batch call, against the same 16 projections as
    separate sadmm_project_groups calls back to back; L2 flushed before each.
    Algorithmic bytes: W read once per key family (filter keys over all rows,
    column keys over the kept rows) plus the keys and index lists."""
    import torch
    from paper_1807_11091_gb300 import sadmm
    layers = wl.resnet50()
    Ws = [wl.gen_tensors(L.shape.with_batch(1), seed=L.seed)["W"].to(dev) for L in layers]
    args = [(L.shape.desc16(), W, L.k_filters, L.colkind, L.k_cols, None) for L, W in zip(layers, Ws)]
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    nbytes = 0
    for L in layers:
        s = L.shape
        G = s.cg if L.colkind == wl.COL_CHANNEL else s.k
        nbytes += 2 * s.f * s.k + 2 * L.k_filters * s.k + 8 * (s.f + G) + 4 * (L.k_filters + L.k_cols)

    def timed(fn):
        fn()
        torch.cuda.synchronize()
        ms = []
        for _ in range(reps):
            flush.fill_(1)
            torch.cuda._sleep(2_000_000)  # the host enqueues the calls meanwhile
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record()
            fn()
            e1.record()
            torch.cuda.synchronize()
            ms.append(e0.elapsed_time(e1))
        return statistics.median(ms)

    pb = sadmm.ProjectBatch(args)
    singles = [sadmm.ProjectBatch([a]) for a in args]  # the same work as 16 separate calls
    t_batch = timed(lambda: pb())
    t_each = timed(lambda: [p() for p in singles])
    # the 16 packs (sadmm_pack_batch vs 16 sadmm_pack calls) of the lists just
    # made; algorithmic bytes: the kept weights read, the packed matrices written
    convs, pbytes = [], 0
    for L, W, (fi, ci, _) in zip(layers, Ws, pb.outs):
        s = L.shape
        pc = sadmm.PrunedConv(s.desc16(), W, fi, L.colkind, ci, L.k_filters, L.k_cols)
        convs.append((pc, W, fi, ci))
        pbytes += 2 * L.k_filters * pc.plan.n_cols + 2 * s.groups * pc.plan.n_pad * pc.plan.k_pad
    t_pack = timed(lambda: sadmm.pack_batch(convs))
    t_pack_each = timed(lambda: [pc.repack(W, fi, ci) for pc, W, fi, ci in convs])
    if sadmm.device_status() != 0:
        raise RuntimeError("device status set after the projections and packs")
    del flush, Ws, pb, singles, convs
    torch.cuda.empty_cache()
    gbs = nbytes / (t_batch * 1e-3) / 1e9
    pgbs = pbytes / (t_pack * 1e-3) / 1e9
    return {"what": "projection of the 16 ResNet-50 bottleneck layers (bf16 W), one batched call vs 16 calls",
            "batch_us": t_batch * 1e3, "separate_us": t_each * 1e3, "bytes": nbytes, "batch_gbs": gbs,
            "batch_hbm_frac": gbs / peak_gbs if peak_gbs else None,
            "pack": {"what": "sadmm_pack of the same 16 layers: one sadmm_pack_batch call vs 16 sadmm_pack calls",
                     "batch_us": t_pack * 1e3, "separate_us": t_pack_each * 1e3, "bytes": pbytes,
                     "batch_gbs": pgbs, "batch_hbm_frac": pgbs / peak_gbs if peak_gbs else None}}


def batch1_report(dev, out_dtype, reps=7):
    """The paper's timing setting (Sec. 5): every AlexNet CONV layer at batch 1,
    sadmm_conv_fwd alone (projection and pack done once), against the same
    kernel at 0% sparsity.  Small layers split K' over several CTAs per output
    tile (plan.splits).  Then the five forwards back to back, captured once in a
    CUDA graph and replayed (launch overhead amortised, as a batch-1 serving
    loop would run them)."""
    import torch
    out = {"what": "AlexNet CONV1-5 at batch 1, sadmm_conv_fwd alone, L2 flushed, median of "
                   f"{reps}", "layers": {}}
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    sp = int(torch.cuda.current_stream().cuda_stream)
    tot_p = tot_d = 0.0
    all_runs = []
    for L in wl.alexnet():
        L1 = wl.subset_layer(L, 1)
        t = wl.gen_tensors(L1.shape, seed=L.seed)
        runs = [LayerRun(L1, t, dev, out_dtype), LayerRun(L1, t, dev, out_dtype, dense=True)]
        all_runs.append(runs)
        times = []
        for r in runs:
            r.project(sp)
            r.pack(sp)
            r.conv(sp)
            torch.cuda.synchronize()
            ms = []
            for _ in range(reps):
                flush.fill_(1)
                torch.cuda._sleep(200_000)
                e0 = torch.cuda.Event(enable_timing=True)
                e1 = torch.cuda.Event(enable_timing=True)
                e0.record()
                r.conv(sp)
                e1.record()
                torch.cuda.synchronize()
                ms.append(e0.elapsed_time(e1))
            times.append(statistics.median(ms))
        tot_p += times[0]
        tot_d += times[1]
        out["layers"][L.name] = {"pruned_us": times[0] * 1e3, "dense_us": times[1] * 1e3,
                                 "speedup_vs_dense": times[1] / times[0],
                                 "tflops_retained": runs[0].flops() / (times[0] * 1e-3) / 1e12,
                                 "splits": int(runs[0].plan.splits)}
    out["total_pruned_us"] = tot_p * 1e3
    out["total_dense_us"] = tot_d * 1e3
    out["speedup_vs_dense"] = tot_d / tot_p
    try:
        graph_us = []
        for k in (0, 1):
            g = torch.cuda.CUDAGraph()
            cap = torch.cuda.Stream()
            cap.wait_stream(torch.cuda.current_stream())
            with torch.cuda.stream(cap):
                with torch.cuda.graph(g, stream=cap):
                    cs = int(torch.cuda.current_stream().cuda_stream)
                    for runs in all_runs:
                        runs[k].conv(cs)
            torch.cuda.current_stream().wait_stream(cap)
            ms = []
            for _ in range(reps):
                flush.fill_(1)
                torch.cuda._sleep(200_000)
                e0 = torch.cuda.Event(enable_timing=True)
                e1 = torch.cuda.Event(enable_timing=True)
                e0.record()
                g.replay()
                e1.record()
                torch.cuda.synchronize()
                ms.append(e0.elapsed_time(e1))
            graph_us.append(statistics.median(ms) * 1e3)
            del g
        from paper_1807_11091_gb300 import sadmm
        if sadmm.sadmm_last_device_status(sp) != 0:
            raise RuntimeError("device status set after the graph replays")
        out["graph"] = {"what": "the five batch-1 forwards in one CUDA graph, replayed (L2 flushed before each)",
                        "pruned_us": graph_us[0], "dense_us": graph_us[1],
                        "speedup_vs_dense": graph_us[1] / graph_us[0]}
    except Exception as e:  # the per-layer figures above stand on their own
        out["graph"] = {"error": f"{type(e).__name__}: {e}"[:200]}
    del flush, all_runs
    torch.cuda.empty_cache()
    return out


def backward_report(dev, out_dtype, reps=3):
    """Masked-retraining backward (sadmm_conv_bwd over the kept weights) of every
    AlexNet CONV layer at batch 128, L2 flushed, median of `reps`: dW and db of
    every layer, dx of conv2-5 (conv1's input is the image, whose gradient
    training never uses).  TFLOP/s counts the retained contractions run: weight
    and input gradient (4 * M * F' * K'), the weight gradient alone on conv1."""
    import torch
    from paper_1807_11091_gb300 import sadmm
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    out = {"what": "sadmm_conv_bwd per AlexNet CONV layer at batch 128 (dW and db; dx for conv2-5: conv1's input "
                   "is the image), L2 flushed", "layers": {}}
    tot_ms = tot_fl = 0.0
    for li, L in enumerate(wl.alexnet()):
        s = L.shape
        want_dx = li > 0
        t = wl.gen_tensors(s, seed=L.seed)
        r = LayerRun(L, t, dev, "fp32")
        sp = int(torch.cuda.current_stream().cuda_stream)
        r.project(sp)
        r.pack(sp)
        r.conv(sp)
        g = torch.Generator().manual_seed(L.seed + 1)
        dy = torch.randn(s.y_shape(), generator=g).to(torch.bfloat16).to(dev)
        dW = torch.empty((s.f, s.k), dtype=torch.float32, device=dev)
        db = torch.empty(s.f, dtype=torch.float32, device=dev)
        dx = torch.empty(r.x.shape, dtype=torch.float32, device=dev) if want_dx else None
        ws_bytes = sadmm.sadmm_conv_bwd_workspace_size(r.plan)
        ws = torch.empty(ws_bytes + 1024, dtype=torch.uint8, device=dev)
        wptr = (ws.data_ptr() + 1023) // 1024 * 1024
        ms = []
        for _ in range(reps + 1):
            flush.fill_(1)
            torch.cuda._sleep(200_000)
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record()
            st = sadmm.sadmm_conv_bwd(r.plan, r.x.data_ptr(), dy.data_ptr(), r.y.data_ptr(), sadmm.SADMM_FP32, 1,
                                      dW.data_ptr(), db.data_ptr(), dx.data_ptr() if want_dx else None, wptr,
                                      ws_bytes, sp)
            e1.record()
            torch.cuda.synchronize()
            assert st == 0, st
            ms.append(e0.elapsed_time(e1))
        t_ms = statistics.median(ms[1:])
        fl = (2.0 if want_dx else 1.0) * r.flops()
        tot_ms += t_ms
        tot_fl += fl
        out["layers"][L.name] = {"us": t_ms * 1e3, "tflops_retained": fl / (t_ms * 1e-3) / 1e12, "dx": want_dx}
        del r, dy, dW, db, dx, ws
    out["total_us"] = tot_ms * 1e3
    out["tflops_retained"] = tot_fl / (tot_ms * 1e-3) / 1e12
    del flush
    torch.cuda.empty_cache()
    return out


def admm_report(dev, peak_gbs, reps=5):
    """sadmm_admm_update (the ADMM Z- and U-update, Sec. 4) on every AlexNet
    CONV layer with fp32 W and U resident in HBM, L2 flushed before each
    timed pass over the five layers.  Algorithmic bytes per layer: W and U read
    once, Z and U written once (16 B per weight)."""
    import torch
    from paper_1807_11091_gb300 import sadmm
    layers = wl.alexnet()
    steps, bufs = [], []
    for L in layers:
        s = L.shape
        st = wl.gen_admm_state(s, L.seed)
        W, U = st["W"].to(dev), st["U"].to(dev)
        bufs.append((W, U, torch.empty_like(W)))
        steps.append(sadmm.AdmmStep(s.desc16(), L.k_filters, L.colkind, L.k_cols, dev))
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    for step, (W, U, Z) in zip(steps, bufs):
        step(W, U, Z)
    torch.cuda.synchronize()
    per = [[] for _ in layers]
    for _ in range(reps):
        for i, (step, (W, U, Z)) in enumerate(zip(steps, bufs)):
            flush.fill_(1)
            torch.cuda._sleep(200_000)
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record()
            step(W, U, Z)
            e1.record()
            torch.cuda.synchronize()
            per[i].append(e0.elapsed_time(e1))
    out = {"what": "sadmm_admm_update per AlexNet CONV layer, fp32 W/U/Z, L2 flushed", "layers": {}}
    tot_ms = tot_bytes = 0.0
    for L, ms in zip(layers, per):
        t = statistics.median(ms)
        nbytes = 16.0 * L.shape.f * L.shape.k
        tot_ms += t
        tot_bytes += nbytes
        out["layers"][L.name] = {"us": t * 1e3, "gbs": nbytes / (t * 1e-3) / 1e9}
    out["total_us"] = tot_ms * 1e3
    out["gbs"] = tot_bytes / (tot_ms * 1e-3) / 1e9
    out["hbm_frac"] = out["gbs"] / peak_gbs if peak_gbs else None
    # the five updates as one sadmm_admm_update_batch call (one launch per phase for all layers)
    batch = sadmm.AdmmBatch([(L.shape.desc16(), L.k_filters, L.colkind, L.k_cols) for L in layers], dev)
    Ws, Us, Zs = [b[0] for b in bufs], [b[1] for b in bufs], [b[2] for b in bufs]
    batch(Ws, Us, Zs)
    torch.cuda.synchronize()
    ms = []
    for _ in range(reps):
        flush.fill_(1)
        torch.cuda._sleep(1_000_000)
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record()
        batch(Ws, Us, Zs)
        e1.record()
        torch.cuda.synchronize()
        ms.append(e0.elapsed_time(e1))
    tb = statistics.median(ms)
    out["batch"] = {"what": "the five layers' updates in one sadmm_admm_update_batch call", "us": tb * 1e3,
                    "gbs": tot_bytes / (tb * 1e-3) / 1e9,
                    "hbm_frac": tot_bytes / (tb * 1e-3) / 1e9 / peak_gbs if peak_gbs else None}
    del bufs, steps, flush, batch
    torch.cuda.empty_cache()
    return out


def run_gpu(args):
    import torch
    ws, rank, local = dist_env()
    if ws > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    from paper_1807_11091_gb300 import sadmm
    sadmm.load()
    # The forwards run on a high-priority stream: the projections and packs on
    # the side streams then take the SMs only when the critical path leaves
    # them (first layer's input pass, the four SMs the first conv leaves free).
    torch.cuda.set_stream(torch.cuda.Stream(priority=-1))
    stream = torch.cuda.current_stream()
    sp = int(stream.cuda_stream)

    layers = wl.get(args.workload)
    from paper_1807_11091_gb300 import ranks
    tensors = [wl.gen_tensors(L.shape, seed=ranks.shard_seed(L.seed, rank)) for L in layers]
    n_sm = torch.cuda.get_device_properties(dev).multi_processor_count
    first_ctas = max(1, n_sm - args.reserve_sms) if args.reserve_sms > 0 else 0
    runs = [LayerRun(L, t, dev, args.out_dtype, max_ctas=first_ctas if i == 0 else 0)
            for i, (L, t) in enumerate(zip(layers, tensors))]
    dense = [LayerRun(L, t, dev, args.out_dtype, dense=True, max_ctas=first_ctas if i == 0 else 0)
             for i, (L, t) in enumerate(zip(layers, tensors))]
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    ss = StepStreams(len(runs))
    peaks, peak_src = load_peaks()

    graphs = {}

    def timed_steps(rs, k, with_conv_events):
        return time_steps(rs, ss, flush, k, with_conv_events, graphs.get(id(rs)))

    # warm-up (also the first-call setup of every kernel)
    for _ in range(max(args.warmup, 3)):
        enqueue_step(runs, ss)
        enqueue_step(dense, ss)
    torch.cuda.synchronize()
    st = sadmm.sadmm_last_device_status(sp)
    if st != 0:
        raise RuntimeError(f"device status {st} after warm-up")
    if not args.eager:
        # each step one replay of the step captured here (the per-call breakdown stays eager)
        graphs[id(runs)] = capture_step(runs, ss)
        graphs[id(dense)] = capture_step(dense, ss)

    log_dir = args.log_dir if os.path.isabs(args.log_dir) else os.path.join(ROOT, args.log_dir)
    os.makedirs(log_dir, exist_ok=True)
    clocks = ClockSampler(local, os.path.join(log_dir, f"bench_clocks_rank{rank}.csv"))
    clocks.start()
    # clock soak: the same steps, untimed, so the sampler sees the load before the window
    t_end = time.time() + 1.0
    while time.time() < t_end:
        enqueue_step(runs, ss)
        torch.cuda.synchronize()

    if ws > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    # the timed steps carry no events between their kernels (an event recorded
    # between two back-to-back launches keeps the second from starting early);
    # the per-conv breakdown comes from separate steps with events around each conv
    step_ms, _ = timed_steps(runs, args.steps, False)
    torch.cuda.synchronize()
    if ws > 1:
        torch.distributed.barrier()
    clocks.stop()
    n_aux = max(3, min(args.steps, 10))
    _, conv_ms = timed_steps(runs, n_aux, True)
    dense_ms, _ = timed_steps(dense, n_aux, False)
    _, dense_conv_ms = timed_steps(dense, n_aux, True)
    calls = calls_report(runs, flush) if rank == 0 else None

    # end to end through the C ABI with host buffers: pinned H2D of every input,
    # the step, D2H of every output
    h_x = [r.x.cpu().pin_memory() for r in runs]
    h_w = [r.W.cpu().pin_memory() for r in runs]
    h_b = [r.bias.cpu().pin_memory() for r in runs]
    h_y = [torch.empty(r.y.shape, dtype=r.y.dtype).pin_memory() for r in runs]
    h2d = sum(a.numel() * a.element_size() for a in h_x + h_w + h_b)
    d2h = sum(a.numel() * a.element_size() for a in h_y)
    copy_stream = torch.cuda.Stream()
    up_stream = torch.cuda.Stream()
    # the first layer in slices of its batch (its output is the largest and
    # the first to go back); the device step's output checks the host's copy
    nc = args.e2e_chunks
    first = (FirstLayerChunks(runs[0], nc, dev, first_ctas)
             if nc > 1 and runs[0].s.n % nc == 0 else None)
    if first is not None and not (first.whole_tiles() and FirstLayerChunks.plan_whole_tiles(runs[0].plan)):
        first = None  # split or stream-K sums: a slice's output need not match the whole batch's bit for bit
    y_first = runs[0].y.cpu()
    e2e_ms = []
    for _ in range(max(2, min(args.steps, 10))):
        flush.fill_(1)
        torch.cuda._sleep(3_000_000)
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record()
        enqueue_step_e2e(runs, ss, copy_stream, h_x, h_w, h_b, h_y, up_stream, first)
        e1.record()
        torch.cuda.synchronize()
        e2e_ms.append(e0.elapsed_time(e1))
    st = sadmm.sadmm_last_device_status(sp)
    if st != 0:
        raise RuntimeError(f"device status {st} after the timed steps")
    if not torch.equal(h_y[0], y_first):
        raise RuntimeError("the end-to-end step's first output differs from the device step's")
    e2e_slices = first.n_chunks if first is not None else 1
    del first

    # max over ranks of the timed totals
    tot_ms = ranks.max_over_ranks(sum(step_ms), device=dev)

    flops_step = sum(r.flops() for r in runs)
    value = ranks.job_throughput(flops_step, ws, args.steps, tot_ms) / 1e12
    ms_per_step = tot_ms / args.steps
    dense_step = statistics.median(dense_ms)
    pruned_step_med = statistics.median(step_ms)
    conv_avg = [statistics.mean(c) for c in conv_ms]
    dense_conv_avg = [statistics.mean(c) for c in dense_conv_ms]

    # roofline of the dominant call (sadmm_conv_fwd over the step's five calls)
    conv_bytes = [r.conv_bytes() for r in runs]
    conv_flops = [r.flops() for r in runs]
    t_conv = sum(conv_avg) * 1e-3
    t_mem = sum(conv_bytes) / (peaks["hbm_gbs"] * 1e9)
    t_cmp = sum(conv_flops) / (peaks["bf16_tflops"] * 1e12)
    if t_mem >= t_cmp:
        achieved = sum(conv_bytes) / len(runs) / (t_conv / len(runs)) / 1e9
        roof = {"bound": "hbm", "achieved": achieved, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                "frac": achieved / peaks["hbm_gbs"]}
    else:
        achieved = sum(conv_flops) / t_conv / 1e12
        roof = {"bound": "tensor", "achieved": achieved, "peak": peaks["bf16_tflops"], "unit": "TFLOP/s",
                "frac": achieved / peaks["bf16_tflops"]}
    roof["traffic"] = conv_traffic(args.workload, args.out_dtype)
    roof["peak_source"] = f"{peak_src} (MEASURED_PEAKS.json)" if peak_src == "measured" else "fallback"
    roof["kernel"] = ("sadmm_conv_fwd (k_conv_fwd; CONV1: k_slab_input + k_conv_slab), "
                      "averaged over the step's five calls")
    roof["combined_roofline_frac"] = max(t_mem, t_cmp) / t_conv

    e2e_med = ranks.max_over_ranks(statistics.median(e2e_ms), device=dev)
    e2e_value = ranks.job_throughput(flops_step, ws, 1, e2e_med) / 1e12

    line = {
        "metric": METRIC, "value": value, "unit": "TFLOP/s", "n_gpus": ws, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {**workload_config(args, layers),
                   "l2": "flushed before every timed step (256 MiB write, outside the timed window)",
                   "schedule": f"projection+pack of each layer on its own stream; convs back to back on the "
                               f"main stream (high priority); first conv on {first_ctas or n_sm} of {n_sm} SMs, its input-slab "
                               f"space-to-depth pass issued at the step's start beside the projections and packs",
                   "launch": ("eager: one host call per kernel" if args.eager else
                              "the step (every projection, pack and forward call and their streams) captured once "
                              "after warm-up into a CUDA graph, one replay per timed step"),
                   "breakdown": "per-conv times from separate eager steps with CUDA events around each whole "
                                "forward call"},
        "pct_bf16_peak": value / peaks["bf16_tflops"],
        "speedup_vs_dense": dense_step / pruned_step_med,
        "conv_speedup_vs_dense": sum(dense_conv_avg) / sum(conv_avg),
        "conv_tflops": sum(conv_flops) / t_conv / 1e12,
        "breakdown_us": {L.name: {"conv": c * 1e3, "dense_conv": d * 1e3}
                         for L, c, d in zip(layers, conv_avg, dense_conv_avg)},
        "roofline": roof,
        "e2e": {"value": e2e_value, "unit": "TFLOP/s", "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                "transfers": "pinned host buffers; inputs uploaded on one stream (weights and biases first, then "
                             "x layer by layer), each output copied back as soon as its conv has run (overlapped "
                             "with the later uploads and convs)" +
                             (f"; the first layer in {e2e_slices} slices of its batch (a plan for the slice), each "
                              "slice's output copied back as soon as it is written" if e2e_slices > 1 else ""),
                "ms_per_step": e2e_med},
        "gpu_launches": sum(r.launches for r in runs) * args.steps,
        "clocks": clocks.summary(),
    }
    if calls is not None:
        line["calls"] = calls
    if rank == 0 and not args.no_configs and args.workload == "alexnet":
        line["configs"] = configs_report(dev, args.out_dtype, peaks, graphs=not args.eager)
    if rank == 0 and not args.no_sweep:
        line["sweep"] = sweep_report(dev, args.out_dtype, peak_tflops=peaks["bf16_tflops"])
        if not args.no_sparse:
            line["non_structured"] = sparse_report(dev, args.out_dtype, line["sweep"])
    if rank == 0 and not args.no_batch1:
        line["batch1"] = batch1_report(dev, args.out_dtype)
    if rank == 0 and not args.no_backward:
        line["backward"] = backward_report(dev, args.out_dtype)
    if rank == 0 and not args.no_admm:
        line["admm"] = admm_report(dev, peaks.get("hbm_gbs"))
        line["projection_batch"] = projection_batch_report(dev, peaks.get("hbm_gbs"))
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(layers, [wl.gen_tensors(L.shape.with_batch(64), seed=L.seed)
                                                     for L in layers])
    if rank == 0:
        print(json.dumps(line), flush=True)
    if ws > 1:
        torch.distributed.destroy_process_group()
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--log-dir", default="bench_logs",
                    help="directory (relative to the repo root unless absolute) for the raw clock samples")
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="alexnet", choices=sorted(wl.WORKLOADS))
    ap.add_argument("--out-dtype", default="fp32", choices=["fp32", "bf16"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-sweep", action="store_true")
    ap.add_argument("--no-sparse", action="store_true",
                    help="skip the element-wise (non-structured) sparse forward beside the sweep")
    ap.add_argument("--no-configs", action="store_true",
                    help="skip the C3D, ResNet-50 and single 2-D steps reported beside the headline")
    ap.add_argument("--no-admm", action="store_true")
    ap.add_argument("--no-batch1", action="store_true")
    ap.add_argument("--no-backward", action="store_true")
    ap.add_argument("--eager", action="store_true",
                    help="time each step as host calls per kernel instead of replaying the step's CUDA graph")
    ap.add_argument("--e2e-chunks", type=int, default=4,
                    help="end-to-end step: the first layer's batch in this many slices (1: whole)")
    ap.add_argument("--reserve-sms", type=int, default=4,
                    help="SMs the first conv leaves to the other layers' projection and pack (0: none)")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    err = check_gpus(args.gpus, dist_env()[0])
    if err:
        print(err, file=sys.stderr, flush=True)
        return 2
    if args.impl == "reference":
        return run_reference(args)
    return run_gpu(args)


if __name__ == "__main__":
    sys.exit(main())
