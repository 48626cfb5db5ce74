"""GPU parity of sadmm_project_groups against the oracle (index lists bit-exact,
keys to fp64 rounding)."""
import numpy as np
import pytest
import torch

import oracle
import workloads as wl
from workloads import ConvShape

from _helpers import gpu_project

pytestmark = pytest.mark.gpu

TINY = [
    ConvShape(n=1, c=3, h=4, w=4, f=6, kh=2, kw=2),
    ConvShape(n=1, c=4, h=4, w=4, f=4, kh=3, kw=1, groups=2),
    ConvShape(n=1, c=2, t=3, h=3, w=3, f=5, kt=2, kh=1, kw=3),
    ConvShape(n=1, c=33, h=5, w=5, f=70, kh=3, kw=3, ph=1, pw=1),
]


def _check(shape, W, kf, ck, kc, U=None):
    fi, ci, keys = gpu_project(shape, W.cuda(), kf, ck, kc, U=None if U is None else U.cuda())
    rows, cols, fk, ckeys = oracle.project(W, shape.taps, kf, ck, kc, U=U)
    assert np.array_equal(fi, rows), "filter index list"
    if ck != wl.COL_NONE:
        assert np.array_equal(ci, cols), "column index list"
    F = shape.f
    assert np.allclose(keys[:F], fk, rtol=1e-12, atol=0), "filter keys"
    if ckeys is not None:
        assert np.allclose(keys[F:], ckeys, rtol=1e-12, atol=1e-300), "column keys"


@pytest.mark.parametrize("si", range(len(TINY)))
@pytest.mark.parametrize("ck", [wl.COL_NONE, wl.COL_SHAPE, wl.COL_CHANNEL])
def test_tiny_all_k(si, ck):
    s = TINY[si]
    t = wl.gen_tensors(s, seed=40 + si)
    G = s.k if ck == wl.COL_SHAPE else s.cg
    for kf in sorted({0, 1, s.f // 2, s.f}):
        for kc in sorted({0, 1, G // 3, G}):
            _check(s, t["W"], kf, ck, kc if ck != wl.COL_NONE else 0)


@pytest.mark.parametrize("si", range(len(TINY)))
@pytest.mark.parametrize("ck", [wl.COL_NONE, wl.COL_SHAPE, wl.COL_CHANNEL])
def test_tiny_all_k_without_keys(si, ck):
    """No keys requested: a kind kept whole skips its keys and select (its list
    is 0..G-1); the lists must equal the oracle's for every mix of kept counts."""
    s = TINY[si]
    t = wl.gen_tensors(s, seed=60 + si)
    G = s.k if ck == wl.COL_SHAPE else s.cg
    for kf in sorted({0, 1, s.f // 2, s.f}):
        for kc in sorted({0, 1, G // 3, G}):
            kc = kc if ck != wl.COL_NONE else 0
            fi, ci, keys = gpu_project(s, t["W"].cuda(), kf, ck, kc, with_keys=False)
            rows, cols, _, _ = oracle.project(t["W"], s.taps, kf, ck, kc)
            assert keys is None
            assert np.array_equal(fi, rows), (kf, kc)
            if ck != wl.COL_NONE:
                assert np.array_equal(ci, cols), (kf, kc)


def test_dual_and_fp32_weights():
    s = TINY[3]
    t = wl.gen_tensors(s, seed=3)
    U = wl.gen_dual(s, seed=3, scale=0.05)
    _check(s, t["W"], 35, wl.COL_SHAPE, 100, U=U)
    W32 = t["W"].float() * 1.37
    _check(s, W32, 20, wl.COL_CHANNEL, 9)


def test_ties_resolved_by_index():
    """Integer weights: every key is an exact small integer on both sides, so
    equal keys are common and the lower index must win."""
    s = ConvShape(n=1, c=40, h=5, w=5, f=300, kh=3, kw=3, ph=1, pw=1)
    W = wl.gen_integer_weights(s, seed=5, lo=-1, hi=1)
    for kf, kc in ((150, 100), (7, 359), (299, 1)):
        _check(s, W, kf, wl.COL_SHAPE, kc)
        _check(s, W, kf, wl.COL_CHANNEL, min(kc, s.cg))
    Wz = torch.zeros(s.w_shape(), dtype=torch.bfloat16)
    _check(s, Wz, 10, wl.COL_SHAPE, 17)  # all keys zero: lowest indices


ALL = wl.single2d() + wl.alexnet() + wl.resnet50() + wl.c3d() + wl.sweep()


@pytest.mark.parametrize("layer", ALL, ids=lambda l: l.name)
def test_workload_layers(layer):
    s = layer.shape
    t = wl.gen_tensors(s.with_batch(1), seed=layer.seed)
    _check(s, t["W"], layer.k_filters, layer.colkind, layer.k_cols)


def test_large_group_count():
    """More groups than one block pass of the select (several compaction chunks)."""
    s = ConvShape(n=1, c=512, h=3, w=3, f=1500, kh=3, kw=3, ph=1, pw=1)
    t = wl.gen_tensors(s, seed=77)
    _check(s, t["W"], 1499, wl.COL_SHAPE, 2345)
    _check(s, t["W"], 1, wl.COL_SHAPE, s.k - 1)


def _scaled(shape, seed, dtype):
    """Random weights whose rows and columns span fp32's magnitudes: a per-row
    power of two from 2^-70 to 2^70 times a per-column one from 2^-8 to 2^8,
    plus 5 % exact zeros."""
    g = torch.Generator().manual_seed(seed)
    F = shape.f
    W = torch.randn(shape.w_shape(), generator=g, dtype=torch.float64).reshape(F, -1)
    K = W.shape[1]
    er = torch.randint(-70, 71, (F, 1), generator=g).double()
    ec = torch.randint(-8, 9, (1, K), generator=g).double()
    W = W * torch.pow(2.0, er + ec)
    W[torch.rand(W.shape, generator=g) < 0.05] = 0.0
    return W.reshape(shape.w_shape()).to(dtype)


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16], ids=["fp32", "bf16"])
def test_keys_across_the_fp32_range(dtype):
    """Groups whose elements span fp32's range, about 2^-85 to 2^79 (squares far
    outside fp32's): keys within 1e-12 of the oracle's fp64 keys and index lists
    exact, with and without U (U cancelling W exactly in some entries, tiny next
    to W in others)."""
    s = ConvShape(n=1, c=48, h=5, w=5, f=96, kh=3, kw=3, ph=1, pw=1)
    W = _scaled(s, 11, dtype)
    for kf, kc in ((48, 200), (95, 7), (3, 431)):
        _check(s, W, kf, wl.COL_SHAPE, kc)
        _check(s, W, kf, wl.COL_CHANNEL, min(kc, s.cg - 1))
    g = torch.Generator().manual_seed(12)
    U = (W.double() * torch.randn(W.shape, generator=g, dtype=torch.float64) * 2.0 ** -30).to(dtype)
    flat = U.reshape(-1)
    idx = torch.randperm(flat.numel(), generator=g)[: flat.numel() // 10]
    flat[idx] = -W.reshape(-1)[idx]
    _check(s, W, 40, wl.COL_SHAPE, 150, U=U)
    _check(s, W, 70, wl.COL_CHANNEL, 20, U=U)


def test_keys_of_long_rows_fp32_with_dual():
    """36864 columns (144 elements per thread in the filter-key pass): the
    partial sums keep the keys within 1e-12 of the oracle's sequential sums."""
    s = ConvShape(n=1, c=4096, h=3, w=3, f=24, kh=3, kw=3, ph=1, pw=1)
    t = wl.gen_tensors(s, seed=13)
    W = t["W"].float() * 0.731
    U = wl.gen_dual(s, seed=13, scale=0.3).float()
    _check(s, W, 12, wl.COL_SHAPE, 9000, U=U)
    _check(s, W, 23, wl.COL_CHANNEL, 1000, U=U)
