"""Batch-1 layers (the paper's timing setting, Sec. 5): few output tiles, so
the plan splits K' over several CTAs per tile and a second kernel adds the
partial sums.  Parity with the oracle as for every other layer (indices
bit-exact, output within 2e-3 * max|y|), and the split must really engage on a
GPU with more SMs than tiles."""
import numpy as np
import pytest
import torch

import oracle
import workloads as wl
from workloads import ConvShape

from _helpers import assert_close, pruned_filters

pytestmark = pytest.mark.gpu

BATCH1 = ([L for L in wl.alexnet()] + [wl.resnet50()[i] for i in (3, 7, 15)] + wl.c3d()
          + [wl.sweep(col_fracs=(0.5,), filt_fracs=(1.0,))[0]])


def _run(layer, n, out_dtype=torch.float32, relu=True):
    from paper_1807_11091_gb300 import sadmm
    s = layer.shape.with_batch(n)
    t = wl.gen_tensors(s, seed=layer.seed)
    dev = torch.device("cuda", 0)
    W, x, bias = t["W"].to(dev), t["x"].to(dev), t["bias"].to(dev)
    fi, ci, _ = sadmm.project_groups(s.desc16(), W, layer.k_filters, layer.colkind, layer.k_cols)
    pc = sadmm.PrunedConv(s.desc16(), W, fi if layer.k_filters < s.f else None, layer.colkind, ci,
                          layer.k_filters, layer.k_cols if layer.colkind != wl.COL_NONE else s.k)
    y = torch.full(pc.out_shape(), float("nan"), dtype=out_dtype, device=dev)
    pc.forward(x, bias, relu=relu, out=y)
    assert sadmm.device_status() == 0
    return s, t, fi.cpu().numpy(), ci.cpu().numpy() if ci is not None else None, y.float().cpu().numpy(), pc


@pytest.mark.parametrize("layer", BATCH1, ids=lambda l: l.name)
def test_batch1_layer(layer):
    s, t, fi, ci, y, pc = _run(layer, 1)
    rows, cols, _, _ = oracle.project(t["W"], s.taps, layer.k_filters, layer.colkind, layer.k_cols)
    assert np.array_equal(fi, rows)
    ref = oracle.pruned_conv(t["x"], t["W"], t["bias"], s.desc16(), s.taps, rows, layer.colkind, cols, relu=True)
    assert_close(y, ref, what=f"{layer.name} batch 1")
    assert np.all(y[:, pruned_filters(s.f, rows)] == 0.0)


def test_split_engages_on_small_layers():
    n_sm = torch.cuda.get_device_properties(0).multi_processor_count
    _, _, _, _, _, pc = _run(wl.alexnet()[2], 1)  # conv3: 2 pixel tiles, 9 stages
    assert n_sm > 2 and pc.plan.splits > 1
    assert pc.plan.splits * pc.plan.stages_per_split >= pc.plan.k_pad // 64
    _, _, _, _, _, pc = _run(wl.alexnet()[2], 128)  # 169 tiles: no split
    assert pc.plan.splits == 1


def test_batch1_bf16_output_and_no_relu():
    L = wl.alexnet()[1]
    s, t, fi, ci, y, pc = _run(L, 1, out_dtype=torch.bfloat16, relu=False)
    assert pc.plan.splits > 1
    ref = oracle.pruned_conv(t["x"], t["W"], t["bias"], s.desc16(), s.taps, fi, L.colkind, ci, relu=False)
    ref_b = torch.from_numpy(ref).to(torch.bfloat16).float().numpy()
    assert np.all(np.abs(y - ref_b) <= np.abs(ref_b) * 2.0 ** -7 + 1e-6 * np.abs(ref).max() + 2e-3 * np.abs(ref).max())
    assert (y < 0).any()


@pytest.mark.parametrize("case", [
    ("ragged_tile", ConvShape(n=1, c=40, h=15, w=17, f=70, kh=3, kw=3, ph=1, pw=1), 0.8, 0.9),
    # 41 pixel tiles, 10 stages: splits of 3, 3, 3 and 1 stages on a 152-SM GPU
    ("uneven_split", ConvShape(n=1, c=70, h=72, w=72, f=32, kh=3, kw=3, ph=1, pw=1), 1.0, 1.0),
], ids=lambda c: c[0])
def test_ragged_small_layer_split(case):
    name, s, ff, cf = case
    L = wl.Layer(name, s, ff, wl.COL_SHAPE, cf, seed=5)
    s2, t, fi, ci, y, pc = _run(L, 1)
    assert pc.plan.splits > 1
    ref = oracle.pruned_conv(t["x"], t["W"], t["bias"], s.desc16(), s.taps, fi, L.colkind, ci, relu=True)
    assert_close(y, ref, what=name)
