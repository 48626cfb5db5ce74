"""Pins for the oracle's ADMM Z- and U-update (no GPU).

Sec. 4: Z^{k+1} is the Euclidean projection of V = W^{k+1} + U^k onto the
structured-sparsity set, and U^{k+1} = U^k + W^{k+1} - Z^{k+1}.  Z is pinned to
brute force (the nearest point over every support set, distance summed element
by element), U^{k+1} to the dual update computed in exact arithmetic on
integer-valued tensors, and both to the fixed point (V already in the set) and
to one rounding of V into the tensors' precision.
"""
import itertools

import numpy as np
import pytest
import torch

import oracle
import workloads as wl
from workloads import ConvShape

TINY = [
    ConvShape(n=1, c=3, h=4, w=4, f=5, kh=2, kw=2),            # F=5, K=12, Cg=3
    ConvShape(n=1, c=4, h=4, w=4, f=4, kh=3, kw=1, groups=2),  # F=4, K=6, Cg=2
]


def _group_masks(kind, s):
    F, K, taps = s.f, s.k, s.taps
    if kind == "filter":
        return [np.outer(np.arange(F) == a, np.ones(K, bool)) for a in range(F)]
    if kind == "shape":
        return [np.outer(np.ones(F, bool), np.arange(K) == j) for j in range(K)]
    return [np.outer(np.ones(F, bool), (np.arange(K) // taps) == b) for b in range(K // taps)]


def _nearest(V, masks, k):
    """The point of the k-group set closest to V (ties: the first subset in
    lexicographic order), by brute force over every support set."""
    best, Zb = None, None
    for sub in itertools.combinations(range(len(masks)), k):
        keep = np.zeros_like(V, bool)
        for g in sub:
            keep |= masks[g]
        Z = np.where(keep, V, 0.0)
        dist = float(((V - Z) ** 2).sum())
        if best is None or dist < best:
            best, Zb = dist, Z
    return Zb


def _state(s, seed, dtype=torch.float32):
    st = wl.gen_admm_state(s, seed, dtype)
    return st["W"], st["U"]


@pytest.mark.parametrize("kind", ["filter", "shape", "channel"])
@pytest.mark.parametrize("si", range(len(TINY)))
def test_z_is_the_nearest_point_and_u_the_residual(kind, si):
    s = TINY[si]
    W, U = _state(s, 10 + si)
    V = W.double().numpy().reshape(s.f, -1) + U.double().numpy().reshape(s.f, -1)
    G = {"filter": s.f, "shape": s.k, "channel": s.cg}[kind]
    for k in (0, 1, G // 2, G - 1, G):
        if kind == "filter":
            args = (k, oracle.COL_NONE, 0)
        else:
            args = (s.f, oracle.COL_SHAPE if kind == "shape" else oracle.COL_CHANNEL, k)
        _, _, Z, Un = oracle.admm_update(W, U, s.taps, *args)
        Zbf = _nearest(V, _group_masks(kind, s), k)
        assert torch.equal(Z.reshape(s.f, -1), torch.from_numpy(Zbf).float()), (kind, k)
        assert torch.equal(Un.reshape(s.f, -1), torch.from_numpy(V - Zbf).float()), (kind, k)


def test_combined_rows_then_columns():
    s = TINY[0]
    W, U = _state(s, 3)
    rows, cols, Z, Un = oracle.admm_update(W, U, s.taps, 3, oracle.COL_SHAPE, 5)
    Zm = Z.reshape(s.f, -1).numpy()
    nz_rows = np.flatnonzero(np.abs(Zm).sum(1) > 0)
    nz_cols = np.flatnonzero(np.abs(Zm).sum(0) > 0)
    assert set(nz_rows) <= set(rows.tolist()) and len(rows) == 3
    assert set(nz_cols) <= set(cols.tolist()) and len(cols) == 5
    # Z + U_next reproduces V wherever one of them is zero (always)
    V = (W.double() + U.double()).float().reshape(s.f, -1)
    assert torch.equal(torch.where(Z.reshape(s.f, -1) != 0, Z.reshape(s.f, -1), Un.reshape(s.f, -1)), V)
    assert not bool(((Z != 0) & (Un != 0)).any())


def test_dual_update_in_exact_arithmetic():
    """Integer-valued W and U: every sum is exact, so U_next must equal
    U + W - Z computed directly, with Z in the set."""
    s = TINY[0]
    g = torch.Generator().manual_seed(5)
    W = torch.randint(-4, 5, s.w_shape(), generator=g).float()
    U = torch.randint(-2, 3, s.w_shape(), generator=g).float()
    for args in ((2, oracle.COL_NONE, 0), (s.f, oracle.COL_SHAPE, 4), (3, oracle.COL_CHANNEL, 2)):
        rows, cols, Z, Un = oracle.admm_update(W, U, s.taps, *args)
        assert torch.equal(Un, U + W - Z)
        Zm = Z.reshape(s.f, -1)
        assert int((Zm.abs().sum(1) > 0).sum()) <= len(rows)


def test_fixed_point_when_v_is_already_in_the_set():
    s = TINY[0]
    W, _ = _state(s, 8)
    W = W.clone()
    W[[1, 3]] = 0.0  # 3 nonzero filters, k = 3
    U = torch.zeros_like(W)
    rows, _, Z, Un = oracle.admm_update(W, U, s.taps, 3, oracle.COL_NONE, 0)
    assert rows.tolist() == [0, 2, 4]
    assert torch.equal(Z, W) and not bool(Un.any())
    # the next update from (W, U_next) lands on the same point
    _, _, Z2, Un2 = oracle.admm_update(W, Un, s.taps, 3, oracle.COL_NONE, 0)
    assert torch.equal(Z2, W) and not bool(Un2.any())


def test_bf16_rounds_v_once():
    """bf16 tensors: V = W + U is rounded once to bf16 (nearest even)."""
    s = ConvShape(n=1, c=1, h=2, w=2, f=2, kh=1, kw=1)  # F=2, K=1
    W = torch.tensor([1.0, 0.125], dtype=torch.bfloat16).reshape(s.w_shape())
    U = torch.tensor([2.0 ** -9, 2.0 ** -12], dtype=torch.bfloat16).reshape(s.w_shape())
    rows, _, Z, Un = oracle.admm_update(W, U, s.taps, 1, oracle.COL_NONE, 0)
    assert rows.tolist() == [0]
    assert Z.dtype == torch.bfloat16
    assert Z.flatten().tolist() == [1.0, 0.0]       # 1 + 2^-9 rounds to 1 in bf16
    assert Un.flatten().tolist() == [0.0, 0.125]    # 0.125 + 2^-12 rounds to 0.125
    U2 = torch.tensor([3 * 2.0 ** -9, 0.0], dtype=torch.bfloat16).reshape(s.w_shape())
    _, _, Z2, _ = oracle.admm_update(W, U2, s.taps, 1, oracle.COL_NONE, 0)
    assert Z2.flatten().tolist()[0] == 1.0 + 2.0 ** -7  # 1 + 3*2^-9 rounds up to the next bf16
