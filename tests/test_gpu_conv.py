"""GPU parity of the whole path (project -> pack -> conv_fwd) against the oracle.

Every output is pre-filled with NaN, so an element the kernel fails to write
fails the finiteness check.  Tolerance: max|gpu - oracle| <= 2e-3 * max|oracle|
per layer for fp32 output (bf16 inputs, fp32 accumulation); bf16 output within
one bf16 ulp of the oracle rounded to bf16.
"""
import numpy as np
import pytest
import torch

import oracle
import workloads as wl
from workloads import ConvShape

from _helpers import assert_close, gpu_layer, oracle_layer, pruned_filters

pytestmark = pytest.mark.gpu

# (shape, filter fraction, column kind, column fraction)
SMALL = [
    ("single2d", wl.single2d()[0].shape, 1.0, wl.COL_SHAPE, 0.5),
    ("ragged", ConvShape(n=3, c=5, h=11, w=13, f=37, kh=3, kw=3, ph=1, pw=1), 0.7, wl.COL_SHAPE, 0.4),
    ("multi_stage", ConvShape(n=2, c=40, h=20, w=21, f=200, kh=3, kw=3, ph=1, pw=1), 1.0, wl.COL_SHAPE, 0.6),
    ("two_filter_tiles", ConvShape(n=2, c=16, h=10, w=10, f=300, kh=3, kw=3, ph=1, pw=1), 1.0, wl.COL_SHAPE, 1.0),
    ("groups2_5x5", ConvShape(n=2, c=8, h=9, w=9, f=12, kh=5, kw=5, ph=2, pw=2, groups=2), 0.5, wl.COL_SHAPE, 0.5),
    ("stride4_11x11", ConvShape(n=2, c=3, h=35, w=35, f=16, kh=11, kw=11, sh=4, sw=4), 1.0, wl.COL_SHAPE, 0.8),
    ("c3d", ConvShape(n=2, c=4, t=5, h=6, w=7, f=20, kt=3, kh=3, kw=3, pt=1, ph=1, pw=1), 1.0, wl.COL_SHAPE, 0.3),
    # 45 taps: the split tap-mask form (row bits kt*KH + kh, kw bits apart), frames and rows clipped
    ("c3d_45_taps", ConvShape(n=2, c=4, t=6, h=7, w=8, f=16, kt=3, kh=3, kw=5, pt=1, ph=1, pw=2), 0.75, wl.COL_SHAPE,
     0.4),
    ("channel_1x1", ConvShape(n=2, c=32, h=8, w=8, f=48, kh=1, kw=1), 0.5, wl.COL_CHANNEL, 0.5),
    ("channel_3x3", ConvShape(n=2, c=24, h=9, w=9, f=40, kh=3, kw=3, ph=1, pw=1), 0.5, wl.COL_CHANNEL, 0.5),
    ("no_col_pruning", ConvShape(n=1, c=12, h=7, w=7, f=33, kh=3, kw=3, ph=1, pw=1, groups=3), 0.6, wl.COL_NONE, 1.0),
    ("stride2_rect", ConvShape(n=2, c=6, h=13, w=10, f=24, kh=3, kw=2, sh=2, sw=1, ph=1, pw=0), 0.75, wl.COL_SHAPE, 0.7),
]


def _k(s, ff, ck, cf):
    G = s.cg if ck == wl.COL_CHANNEL else s.k
    return wl.retained(ff, s.f), (wl.retained(cf, G) if ck != wl.COL_NONE else 0)


@pytest.mark.parametrize("case", SMALL, ids=lambda c: c[0])
def test_small_layers_fp32(case):
    name, s, ff, ck, cf = case
    kf, kc = _k(s, ff, ck, cf)
    t = wl.gen_tensors(s, seed=123)
    fi, ci, y, _ = gpu_layer(s, t, kf, ck, kc)
    rows, cols, _, _ = oracle.project(t["W"], s.taps, kf, ck, kc)
    assert np.array_equal(fi, rows)
    if ck != wl.COL_NONE:
        assert np.array_equal(ci, cols)
    ref = oracle_layer(s, t, rows, ck, cols)
    assert_close(y, ref, what=name)
    assert np.all(y[:, pruned_filters(s.f, rows)] == 0.0)


@pytest.mark.parametrize("case", [SMALL[1], SMALL[4], SMALL[6]], ids=lambda c: c[0])
def test_bf16_output_within_one_ulp(case):
    name, s, ff, ck, cf = case
    kf, kc = _k(s, ff, ck, cf)
    t = wl.gen_tensors(s, seed=7)
    fi, ci, y, _ = gpu_layer(s, t, kf, ck, kc, out_dtype=torch.bfloat16)
    ref = oracle_layer(s, t, fi, ck, ci if ck != wl.COL_NONE else None)
    ref_b = torch.from_numpy(ref).to(torch.bfloat16).float().numpy()
    # one bf16 ulp at the reference magnitude
    ulp = np.abs(ref_b) * 2.0 ** -7 + 1e-30
    assert np.all(np.abs(y - ref_b) <= ulp + 1e-6 * np.abs(ref).max())


def test_no_relu_no_bias():
    _, s, ff, ck, cf = SMALL[1]
    kf, kc = _k(s, ff, ck, cf)
    t = wl.gen_tensors(s, seed=99)
    fi, ci, y, _ = gpu_layer(s, t, kf, ck, kc, relu=False, use_bias=False)
    ref = oracle_layer(s, t, fi, ck, ci, relu=False, use_bias=False)
    assert_close(y, ref, what="no relu")
    assert (y < 0).any()


def test_all_filters_pruned_gives_zeros():
    _, s, _, ck, cf = SMALL[4]
    t = wl.gen_tensors(s, seed=1)
    fi, ci, y, _ = gpu_layer(s, t, 0, ck, _k(s, 1, ck, cf)[1])
    assert np.all(y == 0.0)


def test_all_columns_pruned_gives_bias():
    _, s, _, ck, _ = SMALL[1]
    t = wl.gen_tensors(s, seed=2)
    kf = 20
    fi, ci, y, _ = gpu_layer(s, t, kf, ck, 0)
    ref = oracle_layer(s, t, fi, ck, np.array([], np.int64))
    assert_close(y, ref, what="K'=0")
    keep = np.zeros(s.f, bool); keep[fi] = True
    b = np.maximum(t["bias"].numpy(), 0)
    assert np.allclose(y[:, keep], b[keep][None, :, None, None])


def test_dense_equals_library_conv():
    s = ConvShape(n=2, c=16, h=12, w=12, f=64, kh=3, kw=3, ph=1, pw=1)
    t = wl.gen_tensors(s, seed=4)
    fi, ci, y, _ = gpu_layer(s, t, s.f, wl.COL_NONE, 0)
    ref = torch.relu(torch.nn.functional.conv2d(t["x"].double(), t["W"].double(), t["bias"].double(),
                                                padding=1)).numpy()
    assert_close(y, ref, what="dense")


@pytest.mark.parametrize("case", [SMALL[2], SMALL[5], SMALL[6]], ids=lambda c: c[0])
def test_delta_probe_reads_packed_weights(case):
    """x = one-hot at (n, c, t, ih, iw), bias 0, no ReLU: the output equals the kept
    weight taps that line that input up with each output (exact in bf16 x 1)."""
    name, s, ff, ck, cf = case
    kf, kc = _k(s, ff, ck, cf)
    t = wl.gen_tensors(s, seed=17)
    rng = np.random.default_rng(3)
    for _ in range(2):
        n, c = int(rng.integers(s.n)), int(rng.integers(s.c))
        it, ih, iw = int(rng.integers(s.t)), int(rng.integers(s.h)), int(rng.integers(s.w))
        x = torch.zeros(s.x_shape(), dtype=torch.bfloat16)
        x.view(s.n, s.c, s.t, s.h, s.w)[n, c, it, ih, iw] = 1.0
        td = dict(t, x=x)
        fi, ci, y, _ = gpu_layer(s, td, kf, ck, kc, relu=False, use_bias=False)
        ref = oracle_layer(s, td, fi, ck, ci, relu=False, use_bias=False)
        assert np.array_equal(y.astype(np.float64), ref), name


def test_repeated_calls_reuse_the_plan():
    _, s, ff, ck, cf = SMALL[2]
    kf, kc = _k(s, ff, ck, cf)
    t = wl.gen_tensors(s, seed=31)
    fi, ci, y1, pc = gpu_layer(s, t, kf, ck, kc)
    x = t["x"].cuda()
    b = t["bias"].cuda()
    for _ in range(3):
        y2 = pc.forward(x, b).cpu().numpy()
        assert np.array_equal(y1, y2)


def test_status_word_clear_after_runs():
    from paper_1807_11091_gb300 import sadmm
    assert sadmm.device_status() == 0


def test_slab_and_direct_stages_in_one_launch():
    """Wide input rows make each slab slot large, so stages whose columns span
    many channels take the direct gather while the others read the slab."""
    s = ConvShape(n=2, c=16, h=227, w=227, f=24, kh=11, kw=11, sh=4, sw=4)
    t = wl.gen_tensors(s, seed=61)
    cols = list(range(0, 121)) + [c * 121 + (7 * c) % 121 for c in range(1, 16)] + list(range(15 * 121, 15 * 121 + 40))
    cols = np.array(sorted(set(cols)), dtype=np.int64)
    rows = np.array([0, 3, 4, 9, 10, 11, 20, 23], dtype=np.int64)
    fi, ci, y, _ = gpu_layer(s, t, len(rows), wl.COL_SHAPE, len(cols), project=False, filt_idx=rows, col_idx=cols)
    ref = oracle_layer(s, t, rows, wl.COL_SHAPE, cols)
    assert_close(y, ref, what="mixed stages")
    assert np.all(y[:, pruned_filters(s.f, rows)] == 0.0)


@pytest.mark.parametrize("case", [
    ("odd_plane_3x3", ConvShape(n=3, c=20, h=13, w=13, f=40, kh=3, kw=3, ph=1, pw=1), 0.5, wl.COL_SHAPE, 0.3),
    ("tiny_plane_7x7", ConvShape(n=5, c=16, h=7, w=7, f=32, kh=3, kw=3, ph=1, pw=1), 1.0, wl.COL_CHANNEL, 0.5),
    ("c3d_two_slices", ConvShape(n=2, c=6, t=4, h=12, w=12, f=16, kt=3, kh=3, kw=3, pt=1, ph=1, pw=1), 1.0,
     wl.COL_SHAPE, 0.5),
], ids=lambda c: c[0])
def test_slab_tiling_edge_planes(case):
    """Planes smaller than or not a multiple of a 128-pixel tile (ragged last tile
    of every slice), and 3-D slices."""
    name, s, ff, ck, cf = case
    kf, kc = _k(s, ff, ck, cf)
    t = wl.gen_tensors(s, seed=71)
    fi, ci, y, _ = gpu_layer(s, t, kf, ck, kc)
    ref = oracle_layer(s, t, fi, ck, ci)
    assert_close(y, ref, what=name)
