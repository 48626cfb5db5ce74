"""Independent pins for the oracle's mask builders (no GPU).

Every conv parity check rests on ``oracle.masked_weights`` and
``oracle.masked_bias``: the weight tensor with the pruned GEMM rows (filters)
and columns ((c, kt, kh, kw) taps, or whole channels) set to zero, and the bias
with every pruned filter's entry zero (Sec. 3, "Combination of structured
sparsities": filter-wise sparsity removes rows of the lowered matrix,
channel- and shape-wise sparsity removes columns).

The expected tensors here are written from scratch, one element at a time: a
kept column index j is decoded into (c, kt, kh, kw) from the OIDHW strides
(j = ((c*KT + kt)*KH + kh)*KW + kw), a kept channel b expands to every
(kt, kh, kw) in explicit loops, and nothing calls ``masked_weights``,
``masked_bias`` or ``expand_columns``.  A delta-input probe then runs the whole
pruned layer (``oracle.pruned_conv``): a one-hot input with bias 0 and ReLU off
must give the kept weight at every kept (filter, channel, tap) and an exact
zero at every pruned one.  The last test plants wrong column decodes into the
oracle (monkeypatched, on the CPU) and checks that these pins catch each one.
"""
import itertools

import numpy as np
import pytest
import torch

import oracle
import workloads as wl
from workloads import ConvShape

SHAPES = {
    "2d": ConvShape(n=2, c=5, h=7, w=8, f=6, kh=3, kw=3, ph=1, pw=1),
    "rect": ConvShape(n=1, c=4, h=9, w=6, f=5, kh=3, kw=2, sh=2, sw=1, ph=1, pw=0),
    "groups": ConvShape(n=2, c=6, h=6, w=6, f=8, kh=3, kw=3, ph=1, pw=1, groups=2),
    "3d": ConvShape(n=1, c=3, t=4, h=5, w=5, f=4, kt=3, kh=2, kw=3, pt=1, ph=0, pw=1),
    "3d_groups": ConvShape(n=1, c=4, t=3, h=4, w=4, f=6, kt=2, kh=2, kw=2, st=1, pt=1, ph=1, pw=0, groups=2),
}


def _decode(j: int, s: ConvShape):
    """(c, kt, kh, kw) of GEMM column j: j = ((c*KT + kt)*KH + kh)*KW + kw."""
    kw = j % s.kw
    r = j // s.kw
    kh = r % s.kh
    r //= s.kh
    kt = r % s.kt
    c = r // s.kt
    return c, kt, kh, kw


def _kept_taps(s: ConvShape, colkind: int, cols):
    """The set of kept (c, kt, kh, kw), built without the oracle's column expansion."""
    kept = set()
    if colkind == oracle.COL_NONE:
        for c, kt, kh, kw in itertools.product(range(s.cg), range(s.kt), range(s.kh), range(s.kw)):
            kept.add((c, kt, kh, kw))
    elif colkind == oracle.COL_CHANNEL:
        for b in cols:
            for kt, kh, kw in itertools.product(range(s.kt), range(s.kh), range(s.kw)):
                kept.add((int(b), kt, kh, kw))
    else:
        for j in cols:
            kept.add(_decode(int(j), s))
    return kept


def _expected_mask(W5: np.ndarray, s: ConvShape, rows, colkind: int, cols) -> np.ndarray:
    """W with pruned rows and columns zeroed, element by element ([F][Cg][KT][KH][KW])."""
    kept = _kept_taps(s, colkind, cols)
    rows = set(int(f) for f in rows)
    E = np.zeros_like(W5)
    for f in range(s.f):
        for c, kt, kh, kw in itertools.product(range(s.cg), range(s.kt), range(s.kh), range(s.kw)):
            if f in rows and (c, kt, kh, kw) in kept:
                E[f, c, kt, kh, kw] = W5[f, c, kt, kh, kw]
    return E


def _cases(s: ConvShape, rng):
    """(name, rows, colkind, cols) cases: shape, channel, combined, none, empty."""
    rows_all = np.arange(s.f, dtype=np.int32)
    rows_half = np.sort(rng.choice(s.f, size=max(1, s.f // 2), replace=False)).astype(np.int32)
    cols_shape = np.sort(rng.choice(s.k, size=max(1, (2 * s.k) // 5), replace=False)).astype(np.int32)
    chans = np.sort(rng.choice(s.cg, size=max(1, s.cg // 2), replace=False)).astype(np.int32)
    return [
        ("shape", rows_all, oracle.COL_SHAPE, cols_shape),
        ("channel", rows_all, oracle.COL_CHANNEL, chans),
        ("rows+shape", rows_half, oracle.COL_SHAPE, cols_shape),
        ("rows+channel", rows_half, oracle.COL_CHANNEL, chans),
        ("rows only", rows_half, oracle.COL_NONE, None),
        ("no columns", rows_half, oracle.COL_SHAPE, np.array([], dtype=np.int32)),
        ("first and last column", rows_all, oracle.COL_SHAPE, np.array([0, s.k - 1], dtype=np.int32)),
    ]


def _w5(t, s: ConvShape) -> np.ndarray:
    return t["W"].to(torch.float64).reshape(s.f, s.cg, s.kt, s.kh, s.kw).numpy()


@pytest.mark.parametrize("name", sorted(SHAPES))
def test_masked_weights_match_elementwise_mask(name):
    s = SHAPES[name]
    t = wl.gen_tensors(s, seed=31)
    W5 = _w5(t, s)
    rng = np.random.default_rng(7)
    for case, rows, colkind, cols in _cases(s, rng):
        got = oracle.masked_weights(t["W"], rows, colkind, cols, s.taps).reshape(W5.shape)
        exp = _expected_mask(W5, s, rows, colkind, cols)
        assert np.array_equal(got, exp), f"{name}/{case}"


def test_masked_bias_on_partial_filter_sets():
    F = 9
    bias = torch.tensor([0.5 * (i + 1) * (-1) ** i for i in range(F)], dtype=torch.float32)
    for rows in ([], [0], [8], [1, 4, 5], list(range(F))):
        got = oracle.masked_bias(bias, F, np.array(rows, dtype=np.int32))
        exp = np.array([float(bias[f]) if f in rows else 0.0 for f in range(F)])
        assert np.array_equal(got, exp), rows
    # no bias at all: zeros whatever is kept
    assert np.array_equal(oracle.masked_bias(None, 4, np.array([1, 2], dtype=np.int32)), np.zeros(4))


def _probe(s: ConvShape, t, rows, colkind, cols, rng, n_probes=3):
    """One-hot inputs through oracle.pruned_conv; the expected output is built
    from the kept (filter, channel, tap) sets directly."""
    W5 = _w5(t, s)
    kept = _kept_taps(s, colkind, cols)
    rows_set = set(int(f) for f in rows)
    for _ in range(n_probes):
        n = int(rng.integers(s.n)); c = int(rng.integers(s.c))
        it = int(rng.integers(s.t)); ih = int(rng.integers(s.h)); iw = int(rng.integers(s.w))
        x = torch.zeros(s.x_shape(), dtype=torch.bfloat16)
        x.view(s.n, s.c, s.t, s.h, s.w)[n, c, it, ih, iw] = 1.0
        y = oracle.pruned_conv(x, t["W"], torch.zeros(s.f), s.desc16(), s.taps, rows, colkind, cols,
                               relu=False).reshape(s.n, s.f, s.ot, s.oh, s.ow)
        g = c // s.cg
        cl = c - g * s.cg
        expect = np.zeros_like(y)
        for f in range(g * s.fg, (g + 1) * s.fg):
            if f not in rows_set:
                continue
            for ot, oh, ow in itertools.product(range(s.ot), range(s.oh), range(s.ow)):
                kt = it - (ot * s.st - s.pt); kh = ih - (oh * s.sh - s.ph); kw = iw - (ow * s.sw - s.pw)
                if 0 <= kt < s.kt and 0 <= kh < s.kh and 0 <= kw < s.kw and (cl, kt, kh, kw) in kept:
                    expect[n, f, ot, oh, ow] = W5[f, cl, kt, kh, kw]
        if not np.array_equal(y, expect):
            return False
    return True


@pytest.mark.parametrize("name", ["2d", "rect", "groups", "3d"])
def test_delta_probe_through_pruned_conv(name):
    """x one-hot, bias 0, ReLU off: y holds the kept weight taps and exact zeros elsewhere."""
    s = SHAPES[name]
    t = wl.gen_tensors(s, seed=41)
    rng = np.random.default_rng(3)
    for case, rows, colkind, cols in _cases(s, rng):
        assert _probe(s, t, rows, colkind, cols, rng), f"{name}/{case}"


def test_pins_catch_planted_mask_errors(monkeypatch):
    """Wrong column expansions planted in the oracle fail both pins."""
    s = SHAPES["groups"]
    t = wl.gen_tensors(s, seed=51)
    W5 = _w5(t, s)
    rows = np.array([0, 3, 4, 7], dtype=np.int32)
    cols = np.array([1, 5, 9, 13, 20, 26], dtype=np.int32)
    chans = np.array([0, 2], dtype=np.int32)
    real = oracle.expand_columns

    def shifted(colkind, c, taps, K):  # every kept column moved one to the right
        return np.minimum(real(colkind, c, taps, K) + 1, K - 1)

    def transposed(colkind, c, taps, K):  # channel-major read as tap-major
        j = real(colkind, c, taps, K)
        cg = K // taps
        return (j % taps) * cg + j // taps

    def channel_strided(colkind, c, taps, K):  # channel b read as columns b, b+Cg, ...
        if colkind != oracle.COL_CHANNEL:
            return real(colkind, c, taps, K)
        cg = K // taps
        return (np.asarray(c)[:, None] + cg * np.arange(taps)[None, :]).reshape(-1)

    for bad in (shifted, transposed, channel_strided):
        monkeypatch.setattr(oracle, "expand_columns", bad)
        for colkind, cl in ((oracle.COL_SHAPE, cols), (oracle.COL_CHANNEL, chans)):
            if bad is channel_strided and colkind == oracle.COL_SHAPE:
                continue
            got = oracle.masked_weights(t["W"], rows, colkind, cl, s.taps).reshape(W5.shape)
            assert not np.array_equal(got, _expected_mask(W5, s, rows, colkind, cl)), bad.__name__
            assert not _probe(s, t, rows, colkind, cl, np.random.default_rng(5), n_probes=12), bad.__name__
        monkeypatch.setattr(oracle, "expand_columns", real)
    # a bias mask that keeps the complement is caught too
    bias = t["bias"]
    wrong = oracle.masked_bias(bias, s.f, np.setdiff1d(np.arange(s.f), rows))
    exp = np.array([float(bias[f]) if f in set(rows.tolist()) else 0.0 for f in range(s.f)])
    assert not np.array_equal(wrong, exp)
