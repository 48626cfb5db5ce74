"""Pins for the oracle's masked-retraining backward (no GPU): its gradients
match central finite differences of the oracle's own forward (the C direct
convolution), masked weights get zero gradient, and dy = 0 gives zero."""
import numpy as np
import pytest
import torch

import oracle
import workloads as wl
from workloads import ConvShape

CASES = [
    ("2d_groups", ConvShape(n=2, c=4, h=5, w=6, f=6, kh=3, kw=2, ph=1, pw=0, groups=2), 0.67, wl.COL_SHAPE, 0.6),
    ("3d_stride", ConvShape(n=1, c=3, t=4, h=5, w=5, f=4, kt=2, kh=3, kw=3, st=2, sh=2, sw=1, pt=1, ph=1, pw=1),
     0.75, wl.COL_CHANNEL, 0.67),
]


def _loss(s, x, W, bias, rows, ck, cols, dy, relu):
    y = oracle.pruned_conv(x, W, bias, s.desc16(), s.taps, rows, ck, cols, relu=relu)
    return float((y * dy).sum())


@pytest.mark.parametrize("case", CASES, ids=lambda c: c[0])
@pytest.mark.parametrize("relu", [True, False])
def test_gradients_match_finite_differences(case, relu):
    name, s, ff, ck, cf = case
    G = s.cg if ck == wl.COL_CHANNEL else s.k
    kf, kc = wl.retained(ff, s.f), wl.retained(cf, G)
    t = wl.gen_tensors(s, seed=21)
    x = t["x"].double() - 0.3  # both signs, so the ReLU mask is non-trivial
    W, bias = t["W"].double(), t["bias"].double()
    rows, cols, _, _ = oracle.project(t["W"], s.taps, kf, ck, kc)
    rng = np.random.default_rng(4)
    dy = rng.standard_normal((s.n, s.f) + ((s.ot,) if s.t > 1 else ()) + (s.oh, s.ow))
    dx, dW, db = oracle.pruned_conv_backward(x, W, bias, s.desc16(), s.taps, rows, ck, cols, dy, relu=relu)
    eps = 1e-6
    keepW = oracle.masked_weights(np.ones(W.shape), rows, ck, cols, s.taps) != 0
    # weights: kept entries by central differences, masked entries exactly zero
    flat = np.flatnonzero(keepW.reshape(-1))
    for e in rng.choice(flat, 6, replace=False):
        Wp, Wmn = W.clone().reshape(-1), W.clone().reshape(-1)
        Wp[e] += eps
        Wmn[e] -= eps
        num = (_loss(s, x, Wp.reshape(W.shape), bias, rows, ck, cols, dy, relu)
               - _loss(s, x, Wmn.reshape(W.shape), bias, rows, ck, cols, dy, relu)) / (2 * eps)
        assert abs(num - dW.reshape(-1)[e]) <= 1e-6 * max(1.0, abs(num))
    assert np.all(dW[~keepW] == 0.0)
    # inputs
    for e in rng.choice(x.numel(), 6, replace=False):
        xp, xm = x.clone().reshape(-1), x.clone().reshape(-1)
        xp[e] += eps
        xm[e] -= eps
        num = (_loss(s, xp.reshape(x.shape), W, bias, rows, ck, cols, dy, relu)
               - _loss(s, xm.reshape(x.shape), W, bias, rows, ck, cols, dy, relu)) / (2 * eps)
        assert abs(num - dx.reshape(-1)[e]) <= 1e-6 * max(1.0, abs(num))
    # bias of a kept and of a pruned filter
    for f in (int(rows[0]), int(np.setdiff1d(np.arange(s.f), rows)[0])):
        bp, bmn = bias.clone(), bias.clone()
        bp[f] += eps
        bmn[f] -= eps
        num = (_loss(s, x, W, bp, rows, ck, cols, dy, relu) - _loss(s, x, W, bmn, rows, ck, cols, dy, relu)) / (2 * eps)
        expect = num if f in set(rows.tolist()) else 0.0
        assert abs(expect - db[f]) <= 1e-6 * max(1.0, abs(num))


def test_zero_upstream_gradient():
    name, s, ff, ck, cf = CASES[0]
    t = wl.gen_tensors(s, seed=2)
    rows, cols, _, _ = oracle.project(t["W"], s.taps, 4, ck, 5)
    dy = np.zeros((s.n, s.f, s.oh, s.ow))
    dx, dW, db = oracle.pruned_conv_backward(t["x"], t["W"], t["bias"], s.desc16(), s.taps, rows, ck, cols, dy)
    assert not dx.any() and not dW.any() and not db.any()
