"""GPU parity of the non-structured projection and its ADMM update with the
oracle: keep masks, Z and U bit for bit (|V| compared exactly in fp64, ties to
the lower flat index, including ties spread over many 4096-entry chunks)."""
import numpy as np
import pytest
import torch

import oracle
import workloads as wl
from workloads import ConvShape

pytestmark = pytest.mark.gpu


def _keep(s, W, k, U=None):
    from paper_1807_11091_gb300 import sadmm
    dev = torch.device("cuda", 0)
    keep = sadmm.project_elements(s.desc16(), W.to(dev), k, U=None if U is None else U.to(dev))
    assert sadmm.device_status() == 0
    return keep.cpu().numpy().astype(bool)


@pytest.mark.parametrize("layer", wl.alexnet() + [wl.sweep()[0]], ids=lambda l: l.name)
def test_keep_mask_matches_oracle(layer):
    s = layer.shape
    st = wl.gen_admm_state(s, layer.seed)
    N = s.f * s.k
    for frac in (0.1, 0.5):
        k = int(frac * N)
        got = _keep(s, st["W"], k, U=st["U"])
        ref = oracle.project_elements(st["W"], k, U=st["U"])
        assert np.array_equal(got, ref), (layer.name, frac)


def test_bf16_weights_and_edge_counts():
    s = wl.alexnet()[1].shape
    W = wl.gen_tensors(s, seed=3)["W"]  # bf16: many exactly equal magnitudes
    N = s.f * s.k
    for k in (0, 1, N // 3, N - 1, N):
        got = _keep(s, W, k)
        ref = oracle.project_elements(W, k)
        assert np.array_equal(got, ref), k
        assert int(got.sum()) == k


def test_ties_across_chunks():
    """Integer weights in -3..3: huge groups of equal magnitudes, ranked by flat
    index across every chunk."""
    s = ConvShape(n=1, c=64, h=3, w=3, f=256, kh=3, kw=3)
    W = wl.gen_integer_weights(s, seed=8)
    N = s.f * s.k
    for k in (N // 7, N // 2, N - 5):
        assert np.array_equal(_keep(s, W, k), oracle.project_elements(W, k)), k


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16], ids=["fp32", "bf16"])
def test_admm_update_elements(dtype):
    from paper_1807_11091_gb300 import sadmm
    L = wl.alexnet()[2]
    s = L.shape
    st = wl.gen_admm_state(s, L.seed, dtype)
    W, U = st["W"], st["U"]
    k = int(0.2 * s.f * s.k)
    dev = torch.device("cuda", 0)
    Wd, Ud = W.to(dev), U.to(dev).clone()
    Z = torch.full_like(Wd, float("nan"))
    sadmm.admm_update_elements(s.desc16(), Wd, Ud, Z, k)
    assert sadmm.device_status() == 0
    keep, Zo, Uo = oracle.admm_update_elements(W, U, k)
    iv = torch.int16 if dtype == torch.bfloat16 else torch.int32
    assert torch.equal(Z.cpu().view(iv), Zo.view(iv))
    assert torch.equal(Ud.cpu().view(iv), Uo.view(iv))
