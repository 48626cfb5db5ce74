"""Pins for the oracle's group keys and Euclidean projection (no GPU).

The projection is pinned to its definition (Sec. 4, Eq. 4): among all tensors Z
in the structured-sparsity set, the one closest to V in Frobenius norm.  Brute
force over every support set of k groups on tiny tensors computes that distance
element by element (not from the keys) and must pick the oracle's set.  The keys
are pinned by the sum invariant (every grouping partitions the elements of V).
"""
import itertools
import math

import numpy as np
import pytest
import torch

import oracle
import workloads as wl
from workloads import ConvShape

TINY = [
    ConvShape(n=1, c=3, h=4, w=4, f=6, kh=2, kw=2),            # F=6, K=12, Cg=3
    ConvShape(n=1, c=4, h=4, w=4, f=4, kh=3, kw=1, groups=2),  # F=4, K=6, Cg=2
    ConvShape(n=1, c=2, t=3, h=3, w=3, f=5, kt=2, kh=1, kw=3),  # 3-D, K=12
]


def _V(s, seed, U=False):
    t = wl.gen_tensors(s, seed=seed)
    u = wl.gen_dual(s, seed=seed, scale=0.05) if U else None
    return t["W"], u


def _groups(kind, s):
    """Element masks of every group of the [F, K] matrix (row/column/channel)."""
    F, K, taps = s.f, s.k, s.taps
    out = []
    if kind == "filter":
        for a in range(F):
            m = np.zeros((F, K), bool); m[a, :] = True; out.append(m)
    elif kind == "shape":
        for j in range(K):
            m = np.zeros((F, K), bool); m[:, j] = True; out.append(m)
    else:
        for b in range(K // taps):
            m = np.zeros((F, K), bool); m[:, b * taps:(b + 1) * taps] = True; out.append(m)
    return out


def _best_subsets(V, groups, k, within=None):
    """All k-subsets minimising ||V - Z||_F^2 where Z keeps the subset's groups
    (intersected with `within` when given); distance summed element by element."""
    base = np.ones_like(V, bool) if within is None else within
    best, arg = None, []
    for sub in itertools.combinations(range(len(groups)), k):
        keep = np.zeros_like(V, bool)
        for g in sub:
            keep |= groups[g]
        Z = np.where(keep & base, V, 0.0)
        d = float(((V - Z) ** 2).sum())
        if best is None or d < best - 1e-15:
            best, arg = d, [sub]
        elif abs(d - best) <= 1e-15:
            arg.append(sub)
    return best, arg


def _oracle_select(kind, s, W, k, U=None):
    if kind == "filter":
        rows, _, _, _ = oracle.project(W, s.taps, k, oracle.COL_NONE, 0, U=U)
        return tuple(int(i) for i in rows)
    ck = oracle.COL_SHAPE if kind == "shape" else oracle.COL_CHANNEL
    _, cols, _, _ = oracle.project(W, s.taps, s.f, ck, k, U=U)
    return tuple(int(i) for i in cols)


@pytest.mark.parametrize("kind", ["filter", "shape", "channel"])
@pytest.mark.parametrize("si", range(len(TINY)))
@pytest.mark.parametrize("with_u", [False, True])
def test_projection_is_the_brute_force_nearest_point(kind, si, with_u):
    s = TINY[si]
    W, U = _V(s, seed=31 + si, U=with_u)
    V = oracle.as_matrix(W, U)
    groups = _groups(kind, s)
    G = len(groups)
    for k in sorted({0, 1, G // 2, G - 1, G}):
        _, arg = _best_subsets(V, groups, k)
        assert len(arg) == 1, "continuous data should give a unique nearest point"
        assert _oracle_select(kind, s, W, k, U) == arg[0]


def test_ties_go_to_the_lower_index():
    """Integer weights with planted equal groups: the oracle's set is a nearest
    point, and among the tied groups it holds the lowest indices."""
    s = ConvShape(n=1, c=2, h=3, w=3, f=8, kh=2, kw=2)
    W = torch.zeros(s.w_shape(), dtype=torch.bfloat16)
    # filters 1, 3, 4, 6 share norm^2 = 8; filter 5 has 18; others 2
    pattern = {0: 1, 1: 2, 2: 1, 3: 2, 4: 2, 5: 3, 6: 2, 7: 1}
    for a, v in pattern.items():
        W[a, 0, 0, 0] = v
        W[a, 1, 1, 1] = -v
    V = oracle.as_matrix(W)
    groups = _groups("filter", s)
    for k in range(0, 9):
        best, arg = _best_subsets(V, groups, k)
        got = _oracle_select("filter", s, W, k)
        assert got in arg
        # among all nearest points, the oracle's is lexicographically smallest
        assert got == min(arg)


def test_ties_in_columns_integer_weights():
    s = ConvShape(n=1, c=3, h=4, w=4, f=4, kh=2, kw=2)
    W = wl.gen_integer_weights(s, seed=2, lo=-1, hi=1)
    V = oracle.as_matrix(W)
    for kind in ("shape", "channel"):
        groups = _groups(kind, s)
        for k in range(len(groups) + 1):
            _, arg = _best_subsets(V, groups, k)
            got = _oracle_select(kind, s, W, k)
            assert got == min(arg)


@pytest.mark.parametrize("si", range(len(TINY)))
def test_key_sums_partition_the_tensor(si):
    """Every grouping partitions the elements: each key family sums to ||V||^2,
    and a channel key is the sum of its columns' keys."""
    s = TINY[si]
    W, U = _V(s, seed=50 + si, U=True)
    V = oracle.as_matrix(W, U)
    total = math.fsum((V.reshape(-1) ** 2).tolist())
    fk = oracle.filter_keys(V)
    sk = oracle.shape_keys(V)
    ck = oracle.channel_keys(V, s.taps)
    for keys in (fk, sk, ck):
        assert abs(math.fsum(keys.tolist()) - total) <= 1e-13 * total
    per_chan = sk.reshape(-1, s.taps).sum(axis=1)
    assert np.allclose(per_chan, ck, rtol=1e-14, atol=0)
    # restricted to a subset of rows: the sums are the squared norm of those rows
    rows = np.array([0, s.f - 1])
    sub = math.fsum((V[rows].reshape(-1) ** 2).tolist())
    assert abs(math.fsum(oracle.shape_keys(V, rows).tolist()) - sub) <= 1e-13 * sub
    assert abs(math.fsum(oracle.channel_keys(V, s.taps, rows).tolist()) - sub) <= 1e-13 * sub


def test_keys_single_element_groups():
    """Closed form: with one filter and a 1x1 kernel the shape keys are the squares."""
    s = ConvShape(n=1, c=7, h=2, w=2, f=1, kh=1, kw=1)
    W, _ = _V(s, seed=3)
    V = oracle.as_matrix(W)
    assert np.array_equal(oracle.shape_keys(V), V[0] ** 2)
    assert oracle.filter_keys(V)[0] == math.fsum((V[0] ** 2).tolist()) or \
        abs(oracle.filter_keys(V)[0] - math.fsum((V[0] ** 2).tolist())) <= 1e-15


@pytest.mark.parametrize("si", [0, 2])
def test_combined_rows_then_columns(si):
    """Columns chosen over the kept rows are the nearest point given those rows."""
    s = TINY[si]
    W, _ = _V(s, seed=70 + si)
    V = oracle.as_matrix(W)
    kf = s.f // 2
    cgroups = _groups("shape", s)
    joint_differs = 0
    for kc in (1, len(cgroups) // 2, len(cgroups) - 1):
        rows, cols, _, _ = oracle.project(W, s.taps, kf, oracle.COL_SHAPE, kc)
        rmask = np.zeros_like(V, bool); rmask[rows, :] = True
        _, arg = _best_subsets(V, cgroups, kc, within=rmask)
        assert len(arg) == 1 and tuple(int(c) for c in cols) == arg[0]
        # the rows themselves are the filter-wise nearest point on the full tensor
        _, rarg = _best_subsets(V, _groups("filter", s), kf)
        assert tuple(int(r) for r in rows) == rarg[0]
        # report (not assert) whether a joint search over rows x columns differs
        best_joint = None
        for rs in itertools.combinations(range(s.f), kf):
            rm = np.zeros_like(V, bool); rm[list(rs), :] = True
            d, _ = _best_subsets(V, cgroups, kc, within=rm)
            best_joint = d if best_joint is None else min(best_joint, d)
        keep = np.zeros_like(V, bool); keep[np.ix_(rows, cols)] = True
        d_seq = float(((V - np.where(keep, V, 0.0)) ** 2).sum())
        joint_differs += int(d_seq > best_joint + 1e-15)
    print(f"sequential rows-then-columns differed from the joint optimum in {joint_differs}/3 cases")


def test_topk_bounds_and_closed_forms():
    keys = np.array([3.0, 1.0, 2.0, 2.0, 0.0])
    assert oracle.topk(keys, 0).tolist() == []
    assert oracle.topk(keys, 5).tolist() == [0, 1, 2, 3, 4]
    assert oracle.topk(keys, 2).tolist() == [0, 2]
    assert oracle.topk(keys, 3).tolist() == [0, 2, 3]
    with pytest.raises(ValueError):
        oracle.topk(keys, 6)
    with pytest.raises(ValueError):
        oracle.topk(keys, -1)


def test_topk_matches_library_sort():
    rng = np.random.default_rng(7)
    for G in (1, 2, 17, 1000):
        keys = rng.random(G) ** 3
        keys[rng.integers(G, size=G // 4)] = 0.5  # planted ties
        order = np.lexsort((np.arange(G), -keys))
        for k in (0, 1, G // 3, G):
            assert oracle.topk(keys, k).tolist() == sorted(order[:k].tolist())


ALL_LAYERS = (wl.single2d() + wl.alexnet() + wl.resnet50() + wl.c3d()
              + wl.sweep(filt_fracs=(1.0, 0.5)))


@pytest.mark.parametrize("layer", ALL_LAYERS, ids=lambda l: l.name)
def test_seeded_layers_have_a_clear_selection_margin(layer):
    """The GPU sums keys in another order; fp64 error there is below 1e-12
    relative, so a margin above 1e-11 between kept and dropped keys fixes the
    same index sets on both sides."""
    s = layer.shape
    t = wl.gen_tensors(s.with_batch(1), seed=layer.seed)
    rows, cols, fk, ck = oracle.project(t["W"], s.taps, layer.k_filters, layer.colkind, layer.k_cols)
    assert len(rows) == layer.k_filters and len(cols) == layer.k_cols
    assert oracle.select_margin(fk, layer.k_filters) > 1e-11
    if ck is not None:
        assert oracle.select_margin(ck, layer.k_cols) > 1e-11
