"""Runs one pruned layer of a seeded workload through the C ABI and times it.

    python -m paper_1807_11091_gb300.run_layer --workload sweep --layer 0 --reps 3

Projection and pack run once; sadmm_conv_fwd runs `reps` times, each timed with
CUDA events on the launching stream (after a device-side sleep, so the host's
launch latency stays outside the timed interval).  Prints one line per run: time, TFLOP/s on
retained MACs and the plan's tile sizes.  This is the program the per-kernel
profiles run under ncu.
"""
from __future__ import annotations

import argparse
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def main(argv=None) -> int:
    import torch

    import workloads as wl
    from paper_1807_11091_gb300 import sadmm

    ap = argparse.ArgumentParser()
    ap.add_argument("--workload", default="alexnet", choices=sorted(wl.WORKLOADS))
    ap.add_argument("--layer", type=int, default=0)
    ap.add_argument("--batch", type=int, default=0, help="override the workload's batch")
    ap.add_argument("--reps", type=int, default=3)
    ap.add_argument("--out-dtype", default="fp32", choices=["fp32", "bf16"])
    ap.add_argument("--dense", action="store_true", help="keep every filter and column")
    ap.add_argument("--admm", action="store_true",
                    help="time sadmm_admm_update on fp32 W/U of the layer instead of the forward call")
    ap.add_argument("--elements", type=float, default=0.0,
                    help="time the non-structured ADMM update keeping this fraction of the weights")
    ap.add_argument("--backward", action="store_true", help="time sadmm_conv_bwd (dW, db, dx) after one forward")
    ap.add_argument("--batch-all", action="store_true",
                    help="with --admm: one sadmm_admm_update_batch over every layer of the workload; alone: one "
                         "sadmm_project_groups_batch over every layer (bf16 W)")
    ap.add_argument("--pack-all", action="store_true",
                    help="sadmm_pack of every layer of the workload (after one batched projection), `reps` times "
                         "as separate calls and as one sadmm_pack_batch call")
    ap.add_argument("--sparse", type=float, default=0.0,
                    help="time sadmm_sparse_conv_fwd with the layer pruned element by element to this density")
    args = ap.parse_args(argv)
    if args.pack_all:
        return run_pack_all(args)
    if args.batch_all:
        return run_batch_all(args)
    if args.sparse > 0:
        return run_sparse(args)
    if args.admm:
        return run_admm(args)
    if args.elements > 0:
        return run_elements(args)

    L = wl.get(args.workload)[args.layer]
    s = L.shape if args.batch == 0 else L.shape.with_batch(args.batch)
    t = wl.gen_tensors(s, seed=L.seed, device="cuda")
    kf = s.f if args.dense else L.k_filters
    G = s.cg if L.colkind == wl.COL_CHANNEL else s.k
    kc = (G if args.dense else L.k_cols) if L.colkind != wl.COL_NONE else 0
    fi, ci, _ = sadmm.project_groups(s.desc16(), t["W"], kf, L.colkind, kc)
    pc = sadmm.PrunedConv(s.desc16(), t["W"], fi if kf < s.f else None, L.colkind, ci, kf,
                          kc if L.colkind != wl.COL_NONE else s.k)
    ydt = torch.bfloat16 if args.out_dtype == "bf16" else torch.float32
    y = torch.empty(pc.out_shape(), dtype=ydt, device="cuda")
    flops = 2.0 * s.m * kf * pc.plan.n_cols
    if args.backward:
        pc.forward(t["x"], t["bias"], out=y)
        g = torch.Generator().manual_seed(L.seed + 1)
        dy = torch.randn(y.shape, generator=g).to(torch.bfloat16).cuda()
        for i in range(args.reps):
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            torch.cuda._sleep(200_000)
            e0.record()
            pc.backward(t["x"], dy, y=y)
            e1.record()
            torch.cuda.synchronize()
            ms = e0.elapsed_time(e1)
            print(f"{L.name} N={s.n} backward run {i}: {ms * 1e3:.1f} us  {2 * flops / ms / 1e9:.1f} TFLOP/s "
                  "(dW and dx contractions)")
        return 1 if sadmm.device_status() != 0 else 0
    for i in range(args.reps):
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        # a short device-side sleep first, so the host finishes enqueueing the
        # forward call before the start event is reached on the GPU
        torch.cuda._sleep(200_000)
        e0.record()
        pc.forward(t["x"], t["bias"], out=y)
        e1.record()
        torch.cuda.synchronize()
        ms = e0.elapsed_time(e1)
        print(f"{L.name} N={s.n} run {i}: {ms * 1e3:.1f} us  {flops / ms / 1e9:.1f} TFLOP/s  "
              f"bn={pc.plan.bn} n_tiles={pc.plan.n_tiles} k_pad={pc.plan.k_pad}")
    st = sadmm.device_status()
    if st != 0:
        print(f"device status {st}")
        return 1
    return 0


def run_elements(args) -> int:
    """sadmm_admm_update_elements `reps` times on the layer's fp32 ADMM state."""
    import torch

    import workloads as wl
    from paper_1807_11091_gb300 import sadmm

    L = wl.get(args.workload)[args.layer]
    s = L.shape
    st = wl.gen_admm_state(s, L.seed)
    W, U = st["W"].cuda(), st["U"].cuda()
    Z = torch.empty_like(W)
    k = int(args.elements * s.f * s.k)
    ws = torch.empty(sadmm.sadmm_elements_workspace_size(sadmm.make_desc(s.desc16())), dtype=torch.uint8,
                     device="cuda")
    nbytes = 16.0 * s.f * s.k
    for i in range(args.reps):
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        torch.cuda._sleep(200_000)
        e0.record()
        sadmm.admm_update_elements(s.desc16(), W, U, Z, k, workspace=ws)
        e1.record()
        torch.cuda.synchronize()
        ms = e0.elapsed_time(e1)
        print(f"{L.name} elements {args.elements} run {i}: {ms * 1e3:.1f} us  {nbytes / ms / 1e6:.1f} GB/s "
              "(16 B per weight)")
    return 1 if sadmm.device_status() != 0 else 0


def run_batch_all(args) -> int:
    """One batched projection (or, with --admm, ADMM update on fp32 state) of
    every layer of the workload, `reps` times."""
    import torch

    import workloads as wl
    from paper_1807_11091_gb300 import sadmm

    layers = wl.get(args.workload)
    dev = torch.device("cuda", 0)
    if args.admm:
        states = [wl.gen_admm_state(L.shape, L.seed) for L in layers]
        Ws = [st["W"].to(dev) for st in states]
        Us = [st["U"].to(dev) for st in states]
        Zs = [torch.empty_like(w) for w in Ws]
        batch = sadmm.AdmmBatch([(L.shape.desc16(), L.k_filters, L.colkind, L.k_cols) for L in layers], dev)
        fn = lambda: batch(Ws, Us, Zs)  # noqa: E731
        what = "admm batch"
    else:
        Ws = [wl.gen_tensors(L.shape.with_batch(1), seed=L.seed)["W"].to(dev) for L in layers]
        pb = sadmm.ProjectBatch([(L.shape.desc16(), W, L.k_filters, L.colkind, L.k_cols, None)
                                 for L, W in zip(layers, Ws)])
        fn = pb
        what = "projection batch"
    for i in range(args.reps):
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        torch.cuda._sleep(1_000_000)
        e0.record()
        fn()
        e1.record()
        torch.cuda.synchronize()
        print(f"{args.workload} {what} of {len(layers)} layers run {i}: {e0.elapsed_time(e1) * 1e3:.1f} us")
    return 1 if sadmm.device_status() != 0 else 0


def run_pack_all(args) -> int:
    """sadmm_pack of every layer of the workload (bf16 W; the index lists from one
    batched projection), `reps` times as separate calls, then `reps` times as one
    sadmm_pack_batch call; prints the time of all packs and their algorithmic
    bytes (the kept weights read, the packed matrices written)."""
    import torch

    import workloads as wl
    from paper_1807_11091_gb300 import sadmm

    layers = wl.get(args.workload)
    dev = torch.device("cuda", 0)
    Ws = [wl.gen_tensors(L.shape.with_batch(1), seed=L.seed)["W"].to(dev) for L in layers]
    pb = sadmm.ProjectBatch([(L.shape.desc16(), W, L.k_filters, L.colkind, L.k_cols, None)
                             for L, W in zip(layers, Ws)])
    lists = pb()
    pcs = []
    nbytes = 0
    for L, W, (fi, ci, _) in zip(layers, Ws, lists):
        s = L.shape
        pc = sadmm.PrunedConv(s.desc16(), W, fi if L.k_filters < s.f else None, L.colkind,
                              ci if L.colkind != wl.COL_NONE else None, L.k_filters,
                              L.k_cols if L.colkind != wl.COL_NONE else s.k)
        pcs.append((pc, W, fi if L.k_filters < s.f else None, ci if L.colkind != wl.COL_NONE else None))
        kc = pc.plan.n_cols
        nbytes += L.k_filters * kc * 2 + s.groups * pc.plan.n_pad * pc.plan.k_pad * 2
    torch.cuda.synchronize()
    for what, fn in (("separate calls", lambda: [pc.repack(W, fi, ci) for pc, W, fi, ci in pcs]),
                     ("one batched call", lambda: sadmm.pack_batch(pcs))):
        for i in range(args.reps):
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            torch.cuda._sleep(1_000_000)
            e0.record()
            fn()
            e1.record()
            torch.cuda.synchronize()
            us = e0.elapsed_time(e1) * 1e3
            print(f"{args.workload} pack of {len(layers)} layers, {what}, run {i}: {us:.1f} us, "
                  f"{nbytes / 1e6:.2f} MB ({nbytes / us / 1e3:.0f} GB/s)")
    return 1 if sadmm.device_status() != 0 else 0


def run_sparse(args) -> int:
    """sadmm_sparse_conv_fwd `reps` times with the layer pruned element by
    element (sadmm_project_elements keeps the largest |W|)."""
    import torch

    import workloads as wl
    from paper_1807_11091_gb300 import sadmm

    L = wl.get(args.workload)[args.layer]
    s = L.shape if args.batch == 0 else L.shape.with_batch(args.batch)
    t = wl.gen_tensors(s, seed=L.seed, device="cuda")
    k = wl.retained(args.sparse, s.f * s.k)
    keep = sadmm.project_elements(s.desc16(), t["W"], k)
    desc = sadmm.make_desc(s.desc16())
    nbytes = sadmm.sadmm_sparse_plan_size(desc, k)
    plan = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
    sp = int(torch.cuda.current_stream().cuda_stream)
    assert sadmm.sadmm_sparse_pack(desc, t["W"].data_ptr(), sadmm.SADMM_BF16, keep.data_ptr(), k, plan.data_ptr(),
                                   nbytes, sp) == 0
    y = torch.empty(s.y_shape(), dtype=torch.float32, device="cuda")
    for i in range(args.reps):
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        torch.cuda._sleep(200_000)
        e0.record()
        assert sadmm.sadmm_sparse_conv_fwd(desc, plan.data_ptr(), t["x"].data_ptr(), t["bias"].data_ptr(), 1,
                                           y.data_ptr(), sadmm.SADMM_FP32, sp) == 0
        e1.record()
        torch.cuda.synchronize()
        ms = e0.elapsed_time(e1)
        print(f"{L.name} N={s.n} sparse {args.sparse} run {i}: {ms * 1e3:.1f} us  "
              f"{2.0 * s.m * k / ms / 1e9:.2f} TFLOP/s")
    return 1 if sadmm.device_status() != 0 else 0


def run_admm(args) -> int:
    """sadmm_admm_update `reps` times on the layer's seeded fp32 ADMM state."""
    import torch

    import workloads as wl
    from paper_1807_11091_gb300 import sadmm

    L = wl.get(args.workload)[args.layer]
    s = L.shape
    st = wl.gen_admm_state(s, L.seed)
    W, U = st["W"].cuda(), st["U"].cuda()
    Z = torch.empty_like(W)
    step = sadmm.AdmmStep(s.desc16(), L.k_filters, L.colkind, L.k_cols, W.device)
    nbytes = 16.0 * s.f * s.k
    for i in range(args.reps):
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        torch.cuda._sleep(200_000)
        e0.record()
        step(W, U, Z)
        e1.record()
        torch.cuda.synchronize()
        ms = e0.elapsed_time(e1)
        print(f"{L.name} admm run {i}: {ms * 1e3:.1f} us  {nbytes / ms / 1e6:.1f} GB/s (16 B per weight)")
    return 1 if sadmm.device_status() != 0 else 0


if __name__ == "__main__":
    sys.exit(main())
