"""Pins for the oracle's non-structured projection (Sec. 4): among all tensors
with at most k nonzero entries, the one nearest to V keeps the k largest |V|.
Pinned by brute force over every support set (distance summed element by
element), planted ties (equal magnitudes of either sign go to the lower flat
index), and the ADMM dual update in exact arithmetic."""
import itertools

import numpy as np
import pytest
import torch

import oracle
import workloads as wl
from workloads import ConvShape

TINY = ConvShape(n=1, c=2, h=3, w=3, f=3, kh=2, kw=1)  # F=3, K=4: 12 entries


def test_nearest_k_sparse_point_by_brute_force():
    st = wl.gen_admm_state(TINY, 3)
    W, U = st["W"], st["U"]
    V = (W.double() + U.double()).numpy().reshape(-1)
    for k in range(0, V.size + 1):
        keep = oracle.project_elements(W, k, U=U).reshape(-1)
        best, arg = None, None
        for sub in itertools.combinations(range(V.size), k):
            Z = np.zeros_like(V)
            Z[list(sub)] = V[list(sub)]
            d = float(((V - Z) ** 2).sum())
            if best is None or d < best:
                best, arg = d, set(sub)
        assert set(np.flatnonzero(keep)) == arg, k


def test_ties_go_to_the_lower_flat_index():
    W = torch.tensor([[1.0, -3.0, 2.0, 3.0], [-3.0, 0.5, 3.0, -2.0], [0.0, 2.0, -1.0, 1.0]])
    W = W.reshape(TINY.w_shape())
    keep = oracle.project_elements(W, 3).reshape(-1)
    assert np.flatnonzero(keep).tolist() == [1, 3, 4]  # four entries of magnitude 3; the first three
    keep = oracle.project_elements(W, 6).reshape(-1)
    assert np.flatnonzero(keep).tolist() == [1, 2, 3, 4, 6, 7]  # all 3s, then the first two 2s by index


def test_admm_elements_dual_update_exact():
    g = torch.Generator().manual_seed(9)
    W = torch.randint(-5, 6, TINY.w_shape(), generator=g).float()
    U = torch.randint(-2, 3, TINY.w_shape(), generator=g).float()
    for k in (0, 4, 7, 12):
        keep, Z, Un = oracle.admm_update_elements(W, U, k)
        assert torch.equal(Un, U + W - Z)
        assert int((Z != 0).sum()) <= k
        assert int(keep.sum()) == k
