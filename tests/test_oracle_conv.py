"""Pins for the oracle's convolution and masking (no GPU).

The oracle's direct convolution is checked against what fixes it from outside:
a library convolution at 0% sparsity (torch conv2d / conv3d in fp64, a textbook
special case), the delta-input probe, and the invariants the masking semantics
imply (100% filter pruning gives zero; channel-wise equals shape-wise pruning of
all the channel's columns).
"""
import itertools

import numpy as np
import pytest
import torch
import torch.nn.functional as Fnn

import oracle
import workloads as wl
from workloads import ConvShape

CASES_2D = [
    ConvShape(n=2, c=3, h=9, w=11, f=4, kh=3, kw=3, ph=1, pw=1),
    ConvShape(n=1, c=4, h=10, w=7, f=6, kh=3, kw=2, sh=2, sw=1, ph=0, pw=1),
    ConvShape(n=2, c=4, h=8, w=8, f=6, kh=5, kw=5, ph=2, pw=2, groups=2),
    ConvShape(n=1, c=3, h=23, w=19, f=5, kh=11, kw=11, sh=4, sw=4),
    ConvShape(n=3, c=5, h=6, w=6, f=7, kh=1, kw=1),
    ConvShape(n=1, c=6, h=7, w=9, f=9, kh=3, kw=3, ph=1, pw=1, groups=3),
]

CASES_3D = [
    ConvShape(n=2, c=3, t=5, h=6, w=7, f=4, kt=3, kh=3, kw=3, pt=1, ph=1, pw=1),
    ConvShape(n=1, c=4, t=4, h=5, w=5, f=4, kt=2, kh=3, kw=1, st=2, sh=1, sw=1, pt=0, ph=1, pw=0, groups=2),
]


def _torch_conv(x, W, b, s: ConvShape, relu: bool):
    xd, Wd = x.to(torch.float64), W.to(torch.float64)
    bd = None if b is None else b.to(torch.float64)
    if s.is3d:
        y = Fnn.conv3d(xd, Wd, bd, stride=(s.st, s.sh, s.sw), padding=(s.pt, s.ph, s.pw), groups=s.groups)
    else:
        y = Fnn.conv2d(xd, Wd, bd, stride=(s.sh, s.sw), padding=(s.ph, s.pw), groups=s.groups)
    return torch.relu(y) if relu else y


@pytest.mark.parametrize("s", CASES_2D + CASES_3D, ids=lambda s: f"{s.x_shape()}-{s.w_shape()}-g{s.groups}")
@pytest.mark.parametrize("relu", [False, True])
def test_conv_equals_library_conv_at_zero_sparsity(s, relu):
    t = wl.gen_tensors(s, seed=11)
    y = oracle.conv(t["x"], t["W"], t["bias"], s.desc16(), relu=relu)
    ref = _torch_conv(t["x"], t["W"], t["bias"], s, relu).numpy()
    assert y.shape == ref.shape
    scale = max(1.0, float(np.abs(ref).max()))
    assert np.abs(y - ref).max() <= 1e-12 * scale


def test_conv_image_range_matches_full_run():
    s = CASES_2D[0]
    t = wl.gen_tensors(s, seed=3)
    full = oracle.conv(t["x"], t["W"], t["bias"], s.desc16())
    part = oracle.conv(t["x"], t["W"], t["bias"], s.desc16(), n0=1, n1=2)
    assert np.array_equal(full[1:2], part)


@pytest.mark.parametrize("s", [CASES_2D[1], CASES_2D[2], CASES_2D[3], CASES_3D[0]],
                         ids=["stride", "groups", "alex_conv1_like", "3d"])
def test_delta_probe_reproduces_weights(s):
    """x = one-hot at (n, c, t, ih, iw), bias 0, no ReLU: every output equals the
    weight tap that lines the input up with that output, or zero."""
    t = wl.gen_tensors(s, seed=5)
    W = t["W"].to(torch.float64).reshape(s.f, s.cg, s.kt, s.kh, s.kw).numpy()
    rng = np.random.default_rng(0)
    for _ in range(4):
        n = int(rng.integers(s.n)); c = int(rng.integers(s.c))
        it = int(rng.integers(s.t)); ih = int(rng.integers(s.h)); iw = int(rng.integers(s.w))
        x = torch.zeros(s.x_shape(), dtype=torch.bfloat16)
        x.view(s.n, s.c, s.t, s.h, s.w)[n, c, it, ih, iw] = 1.0
        y = oracle.conv(x, t["W"], None, s.desc16(), relu=False).reshape(s.n, s.f, s.ot, s.oh, s.ow)
        g = c // s.cg
        expect = np.zeros_like(y)
        for f in range(g * s.fg, (g + 1) * s.fg):
            for ot, oh, ow in itertools.product(range(s.ot), range(s.oh), range(s.ow)):
                kt = it - (ot * s.st - s.pt); kh = ih - (oh * s.sh - s.ph); kw = iw - (ow * s.sw - s.pw)
                if 0 <= kt < s.kt and 0 <= kh < s.kh and 0 <= kw < s.kw:
                    expect[n, f, ot, oh, ow] = W[f, c - g * s.cg, kt, kh, kw]
        assert np.array_equal(y, expect)


def test_full_filter_pruning_gives_zero_output():
    s = CASES_2D[2]
    t = wl.gen_tensors(s, seed=8)
    for relu in (False, True):
        y = oracle.pruned_conv(t["x"], t["W"], t["bias"], s.desc16(), s.taps,
                               filt_idx=np.array([], dtype=np.int32), colkind=oracle.COL_SHAPE,
                               col_idx=np.arange(s.k), relu=relu)
        assert np.all(y == 0.0)


def test_zero_sparsity_equals_dense_conv():
    s = CASES_2D[0]
    t = wl.gen_tensors(s, seed=9)
    rows, cols, _, _ = oracle.project(t["W"], s.taps, s.f, oracle.COL_SHAPE, s.k)
    assert np.array_equal(rows, np.arange(s.f)) and np.array_equal(cols, np.arange(s.k))
    y = oracle.pruned_conv(t["x"], t["W"], t["bias"], s.desc16(), s.taps, rows, oracle.COL_SHAPE, cols)
    ref = _torch_conv(t["x"], t["W"], t["bias"], s, True).numpy()
    assert np.abs(y - ref).max() <= 1e-12 * max(1.0, float(np.abs(ref).max()))


@pytest.mark.parametrize("s", [CASES_2D[0], CASES_2D[2], CASES_3D[0]], ids=["2d", "groups", "3d"])
def test_channel_pruning_equals_shape_pruning_of_its_columns(s):
    t = wl.gen_tensors(s, seed=21)
    rng = np.random.default_rng(1)
    chans = np.sort(rng.choice(s.cg, size=max(1, s.cg // 2), replace=False)).astype(np.int32)
    cols = oracle.expand_columns(oracle.COL_CHANNEL, chans, s.taps, s.k)
    rows = np.arange(s.f, dtype=np.int32)
    y_ch = oracle.pruned_conv(t["x"], t["W"], t["bias"], s.desc16(), s.taps, rows, oracle.COL_CHANNEL, chans)
    y_sh = oracle.pruned_conv(t["x"], t["W"], t["bias"], s.desc16(), s.taps, rows, oracle.COL_SHAPE, cols)
    assert np.array_equal(y_ch, y_sh)


def test_masked_conv_equals_library_conv_of_masked_weights():
    """Masking (rows + columns) then convolving equals torch conv of the masked tensor."""
    s = CASES_2D[2]
    t = wl.gen_tensors(s, seed=4)
    rows = np.array([0, 2, 5], dtype=np.int32)
    cols = np.array([0, 3, 7, 24, 30, 49], dtype=np.int32)
    Wm = oracle.masked_weights(t["W"], rows, oracle.COL_SHAPE, cols, s.taps)
    bm = oracle.masked_bias(t["bias"], s.f, rows)
    y = oracle.pruned_conv(t["x"], t["W"], t["bias"], s.desc16(), s.taps, rows, oracle.COL_SHAPE, cols)
    ref = _torch_conv(t["x"], torch.from_numpy(Wm), torch.from_numpy(bm), s, True).numpy()
    assert np.abs(y - ref).max() <= 1e-12 * max(1.0, float(np.abs(ref).max()))
    # pruned filters' planes are exactly zero
    pruned = np.setdiff1d(np.arange(s.f), rows)
    assert np.all(y[:, pruned] == 0.0)
