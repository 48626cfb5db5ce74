"""GPU parity at the benchmark sizes, through the calls bench.py times.

Every layer of every workload runs at its full batch through
sadmm_project_groups -> sadmm_pack -> sadmm_conv_fwd.  Index lists are compared
with the oracle's in full (bit-exact); the output is compared element by element
on the first and last image of the batch (the oracle's fp64 direct convolution
of those images), and on the whole tensor through properties that hold at any
size: every element written and finite, every pruned filter's plane exactly zero,
ReLU outputs non-negative.
"""
import numpy as np
import pytest
import torch

import oracle
import workloads as wl

from _helpers import assert_close, pruned_filters

pytestmark = pytest.mark.gpu

LAYERS = (wl.single2d() + wl.alexnet() + wl.resnet50() + wl.c3d()
          + wl.sweep(col_fracs=(1.0, 0.25, 0.05), filt_fracs=(1.0, 0.5)))


def _run_full(layer):
    from paper_1807_11091_gb300 import sadmm
    s = layer.shape
    t = wl.gen_tensors(s, seed=layer.seed)
    dev = torch.device("cuda", 0)
    W, x, bias = t["W"].to(dev), t["x"].to(dev), t["bias"].to(dev)
    fi, ci, _ = sadmm.project_groups(s.desc16(), W, layer.k_filters, layer.colkind, layer.k_cols)
    pc = sadmm.PrunedConv(s.desc16(), W, fi if layer.k_filters < s.f else None, layer.colkind, ci,
                          layer.k_filters, layer.k_cols if layer.colkind != wl.COL_NONE else s.k)
    y = torch.full(pc.out_shape(), float("nan"), dtype=torch.float32, device=dev)
    pc.forward(x, bias, relu=True, out=y)
    assert sadmm.device_status() == 0
    return t, fi.cpu().numpy().astype(np.int64), ci.cpu().numpy().astype(np.int64), y


@pytest.mark.parametrize("layer", LAYERS, ids=lambda l: l.name)
def test_full_size_layer(layer):
    s = layer.shape
    t, fi, ci, y = _run_full(layer)
    rows, cols, _, _ = oracle.project(t["W"], s.taps, layer.k_filters, layer.colkind, layer.k_cols)
    assert np.array_equal(fi, rows), "filter index list"
    assert np.array_equal(ci, cols), "column index list"
    # whole-tensor properties
    assert bool(torch.isfinite(y).all()), "unwritten or non-finite outputs"
    assert bool((y >= 0).all()), "ReLU output below zero"
    pr = torch.as_tensor(pruned_filters(s.f, rows), device=y.device)
    if pr.numel():
        assert bool((y.index_select(1, pr) == 0).all()), "pruned planes not zero"
    # element by element on the first and last image
    for n in sorted({0, s.n - 1}):
        ref = oracle.pruned_conv(t["x"], t["W"], t["bias"], s.desc16(), s.taps, rows, layer.colkind, cols,
                                 relu=True, n0=n, n1=n + 1)
        assert_close(y[n:n + 1].cpu().numpy(), ref, what=f"{layer.name} image {n}")


BF16_LAYERS = [wl.alexnet()[0], wl.alexnet()[1], wl.alexnet()[4], wl.c3d()[0],
               wl.sweep(col_fracs=(0.25,), filt_fracs=(0.5,))[0]]


@pytest.mark.parametrize("layer", BF16_LAYERS, ids=lambda l: l.name)
def test_full_size_layer_bf16_output(layer):
    """The bf16-output forward at full size: within one bf16 ulp of the oracle
    rounded to bf16 on the first and last image; every element written; pruned
    planes exactly zero over the whole tensor."""
    from paper_1807_11091_gb300 import sadmm
    s = layer.shape
    t = wl.gen_tensors(s, seed=layer.seed)
    dev = torch.device("cuda", 0)
    W, x, bias = t["W"].to(dev), t["x"].to(dev), t["bias"].to(dev)
    fi, ci, _ = sadmm.project_groups(s.desc16(), W, layer.k_filters, layer.colkind, layer.k_cols)
    pc = sadmm.PrunedConv(s.desc16(), W, fi if layer.k_filters < s.f else None, layer.colkind, ci,
                          layer.k_filters, layer.k_cols if layer.colkind != wl.COL_NONE else s.k)
    y = torch.full(pc.out_shape(), float("nan"), dtype=torch.bfloat16, device=dev)
    pc.forward(x, bias, relu=True, out=y)
    assert sadmm.device_status() == 0
    rows = fi.cpu().numpy().astype(np.int64)
    cols = ci.cpu().numpy().astype(np.int64)
    assert bool(torch.isfinite(y).all()), "unwritten or non-finite outputs"
    pr = torch.as_tensor(pruned_filters(s.f, rows), device=dev)
    if pr.numel():
        assert bool((y.index_select(1, pr) == 0).all()), "pruned planes not zero"
    for n in sorted({0, s.n - 1}):
        ref = oracle.pruned_conv(t["x"], t["W"], t["bias"], s.desc16(), s.taps, rows, layer.colkind, cols,
                                 relu=True, n0=n, n1=n + 1)
        ref_b = torch.from_numpy(ref).to(torch.bfloat16).float().numpy()
        got = y[n:n + 1].float().cpu().numpy().reshape(ref.shape)
        ulp = np.abs(ref_b) * 2.0 ** -7 + 1e-30
        assert np.all(np.abs(got - ref_b) <= ulp + 1e-6 * np.abs(ref).max()), f"{layer.name} image {n}"
