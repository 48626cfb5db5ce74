"""Tail balance (stream-K): when a layer's output tiles do not spread evenly
over the SMs, each CTA takes an equal run of 64-column stages, and a tile cut
between two CTAs is finished by whichever of them arrives second (fp32 partial
sums of both pieces, added in K' order).  Parity with the oracle over the whole
output (indices bit-exact, output within 2e-3 * max|y|), every pruned plane
zero, the tail split really engaged, and repeated launches on one plan
bit-identical (the arrival counters return to zero after each launch)."""
import numpy as np
import pytest
import torch

import oracle
import workloads as wl
from workloads import ConvShape

from _helpers import assert_close, pruned_filters

pytestmark = pytest.mark.gpu


def _n_sm():
    return torch.cuda.get_device_properties(0).multi_processor_count


def _expect_streamk(plan, shape):
    """The plan's rule: whole tiles leave the busiest CTA with ceil(units/SMs)
    tiles; an even run of stages must be at least a tile long and shorten that
    by 1/8 or more, with two accumulator sets in TMEM and K' >= 4 * bn."""
    n_sm = _n_sm()
    nks = plan.k_pad // 64
    nacc = 2 if plan.n_tiles >= 2 else 1
    upairs = -(-plan.n_tiles // nacc)
    units = -(-shape.n * shape.ot * shape.oh * shape.ow // 128) * shape.groups * upairs
    if plan.splits > 1 or units < n_sm:
        return False
    if 2 * nacc * (-(-plan.bn // 32) * 32) > 512 or plan.k_pad < 4 * plan.bn:
        return False
    dp = -(-units // n_sm) * nks
    L = -(-units * nks // n_sm)
    return L >= nks and (dp - L) * 8 >= dp


def _plan_layer(layer, n=None):
    from paper_1807_11091_gb300 import sadmm
    s = layer.shape if n is None else layer.shape.with_batch(n)
    t = wl.gen_tensors(s, seed=layer.seed)
    dev = torch.device("cuda", 0)
    W, x, bias = t["W"].to(dev), t["x"].to(dev), t["bias"].to(dev)
    fi, ci, _ = sadmm.project_groups(s.desc16(), W, layer.k_filters, layer.colkind, layer.k_cols)
    pc = sadmm.PrunedConv(s.desc16(), W, fi if layer.k_filters < s.f else None, layer.colkind, ci,
                          layer.k_filters, layer.k_cols if layer.colkind != wl.COL_NONE else s.k)
    fi = fi.cpu().numpy().astype(np.int64)[:layer.k_filters]
    ci = ci.cpu().numpy().astype(np.int64) if ci is not None else np.arange(s.k)
    return s, t, x, bias, fi, ci, pc


def _forward(pc, x, bias, relu=True, out_dtype=torch.float32):
    from paper_1807_11091_gb300 import sadmm
    y = torch.full(pc.out_shape(), float("nan"), dtype=out_dtype, device=x.device)
    pc.forward(x, bias, relu=relu, out=y)
    assert sadmm.device_status() == 0
    return y


def _check(layer, n=None, relu=True, out_dtype=torch.float32, repeats=1):
    s, t, x, bias, fi, ci, pc = _plan_layer(layer, n)
    assert _expect_streamk(pc.plan, s), "test shape does not call for the tail split on this GPU"
    assert pc.plan.sk_len >= pc.plan.k_pad // 64 and pc.plan.sk_grid >= 2, "tail split not engaged"
    rows, cols, _, _ = oracle.project(t["W"], s.taps, layer.k_filters, layer.colkind, layer.k_cols)
    assert np.array_equal(fi, rows) and np.array_equal(ci, cols)
    ref = oracle.pruned_conv(t["x"], t["W"], t["bias"], s.desc16(), s.taps, rows, layer.colkind, cols, relu=relu)
    first = None
    for _ in range(repeats):
        y = _forward(pc, x, bias, relu=relu, out_dtype=out_dtype).float().cpu().numpy()
        if first is None:
            first = y
        else:
            assert np.array_equal(y, first), "repeated launch on one plan differs"
    if out_dtype == torch.float32:
        assert_close(first, ref, what=layer.name)
    else:
        ref_b = torch.from_numpy(ref).to(torch.bfloat16).float().numpy()
        scale = np.abs(ref).max()
        assert np.all(np.abs(first - ref_b) <= np.abs(ref_b) * 2.0 ** -7 + 2e-3 * scale), layer.name
    assert np.all(first[:, pruned_filters(s.f, rows)] == 0.0)
    return pc


@pytest.mark.parametrize("li", [2, 3, 4], ids=lambda i: f"conv{i + 1}")
def test_alexnet_tail_layers_full_output(li):
    """AlexNet conv3-5 at batch 128 (169 and 338 tiles): every output element."""
    L = wl.alexnet()[li]
    s, t, x, bias, fi, ci, pc = _plan_layer(L)
    if not _expect_streamk(pc.plan, s):
        pytest.skip("this GPU's SM count spreads the tiles evenly")
    _check(L, repeats=2)


def _constructed():
    n_sm = _n_sm()
    return [
        # one tile past the SM count and a ragged last tile; 3 stages per tile
        wl.Layer("extra_tile_ragged", ConvShape(n=1, c=24, h=n_sm + 1, w=131, f=48, kh=3, kw=3, ph=1, pw=1),
                 0.75, wl.COL_SHAPE, 0.6, seed=11),
        # a full 128-row filter tile and 9 stages per tile, every column kept
        wl.Layer("wide_tile", ConvShape(n=1, c=64, h=n_sm + n_sm // 8, w=127, f=128, kh=3, kw=3, ph=1, pw=1),
                 1.0, wl.COL_NONE, 1.0, seed=12),
        # two conv groups, channel-wise pruning, pruned filters' planes zero-filled by the first piece
        wl.Layer("groups2_channel", ConvShape(n=1, c=32, h=n_sm // 2 + n_sm // 16 + 1, w=125, f=64, kh=3, kw=3,
                                              ph=1, pw=1, groups=2), 0.5, wl.COL_CHANNEL, 0.5, seed=13),
        # stride 2, 5x5, several images
        # (OH = -(-n_sm * 128 * 1.15 // 345) rows of 115 pixels per image: about 1.15 tiles per SM)
        wl.Layer("strided_batch", ConvShape(n=3, c=12, h=2 * (-(-n_sm * 1472 // 3450) - 1) + 1, w=229, f=40, kh=5,
                                            kw=5, sh=2, sw=2, ph=2, pw=2), 0.6, wl.COL_SHAPE, 0.7, seed=14),
    ]


@pytest.mark.parametrize("idx", range(4), ids=["extra_tile_ragged", "wide_tile", "groups2_channel",
                                               "strided_batch"])
def test_constructed_tail_split(idx):
    _check(_constructed()[idx], repeats=3)


def test_tail_split_bf16_no_relu():
    L = _constructed()[0]
    _check(L, relu=False, out_dtype=torch.bfloat16, repeats=2)


def test_no_tail_split_where_it_does_not_pay():
    """Two filter tiles per unit (one accumulator set) or a short K' keep whole tiles."""
    n_sm = _n_sm()
    for L in (wl.Layer("two_tiles", ConvShape(n=1, c=16, h=n_sm + n_sm // 8, w=127, f=320, kh=3, kw=3, ph=1, pw=1),
                       1.0, wl.COL_SHAPE, 0.5, seed=15),
              wl.Layer("short_k", ConvShape(n=1, c=8, h=n_sm + n_sm // 8, w=127, f=64, kh=3, kw=3, ph=1, pw=1),
                       1.0, wl.COL_SHAPE, 1.0, seed=16)):
        s, t, x, bias, fi, ci, pc = _plan_layer(L)
        assert pc.plan.sk_len == 0 and not _expect_streamk(pc.plan, s), L.name
