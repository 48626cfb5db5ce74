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


@pytest.mark.parametrize("stride", [1, 2])
def test_pointwise_layer_reduces_to_matrix_products(stride):
    """A 1x1 conv without ReLU is y[:, p] = Wm x[:, q(p)] + bm at every output
    pixel p (input pixel q(p) = stride * p), so its gradients are matrix
    products: dW = (dY X^T) on the kept entries, dX[:, q(p)] = Wm^T dY[:, p]
    (zero at the input pixels the stride skips), db = the sum of dY over the
    pixels and the batch for kept filters.  Checked to 1e-12 relative."""
    s = ConvShape(n=3, c=7, h=6, w=8, f=9, kh=1, kw=1, sh=stride, sw=stride)
    t = wl.gen_tensors(s, seed=31)
    x, W, bias = t["x"].double(), t["W"].double(), t["bias"].double()
    rows, cols, _, _ = oracle.project(t["W"], s.taps, 6, wl.COL_CHANNEL, 4)
    rng = np.random.default_rng(8)
    dy = rng.standard_normal((s.n, s.f, s.oh, s.ow))
    dx, dW, db = oracle.pruned_conv_backward(x, W, bias, s.desc16(), s.taps, rows, wl.COL_CHANNEL, cols, dy,
                                             relu=False)
    Wm = oracle.masked_weights(W, rows, wl.COL_CHANNEL, cols, s.taps).reshape(s.f, s.c)
    keep = oracle.masked_weights(np.ones(W.shape), rows, wl.COL_CHANNEL, cols, s.taps).reshape(s.f, s.c) != 0
    xs = x.numpy()[:, :, ::stride, ::stride][:, :, :s.oh, :s.ow]      # [n][c][oh][ow]
    X = xs.transpose(1, 0, 2, 3).reshape(s.c, -1)                      # [c][n*oh*ow]
    D = dy.transpose(1, 0, 2, 3).reshape(s.f, -1)                      # [f][n*oh*ow]
    dW_ref = (D @ X.T) * keep
    assert np.allclose(dW.reshape(s.f, s.c), dW_ref, rtol=1e-12, atol=1e-12 * np.abs(dW_ref).max())
    dx_ref = np.zeros(x.shape)
    dx_ref[:, :, ::stride, ::stride][:, :, :s.oh, :s.ow] = (Wm.T @ D).reshape(s.c, s.n, s.oh, s.ow).transpose(1, 0, 2, 3)
    assert np.allclose(dx, dx_ref, rtol=1e-12, atol=1e-12 * np.abs(dx_ref).max())
    bkeep = np.isin(np.arange(s.f), rows)
    assert np.allclose(db, D.sum(axis=1) * bkeep, rtol=1e-12, atol=1e-12)
    assert np.all(db[~bkeep] == 0.0) and np.all(dW.reshape(s.f, s.c)[~keep] == 0.0)
