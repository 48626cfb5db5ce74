"""GPU parity of sadmm_admm_update (Sec. 4 Z- and U-update) with the oracle.

Index lists, Z and U^{k+1} must match bit for bit: the keys are exact fp64
sums of exact squares (the selection is exact once the margin test of the
projection holds), and Z and U^{k+1} are V = W + U rounded once to the
tensors' precision on both sides.
"""
import numpy as np
import pytest
import torch

import oracle
import workloads as wl
from workloads import ConvShape

pytestmark = pytest.mark.gpu

LAYERS = (wl.alexnet() + [wl.resnet50()[i] for i in (0, 3, 7, 12, 15)] + wl.c3d()
          + [wl.sweep(col_fracs=(0.25,), filt_fracs=(0.5,))[0]])

SMALL = [
    ("ragged_shape", ConvShape(n=1, c=5, h=11, w=13, f=37, kh=3, kw=3), 0.7, wl.COL_SHAPE, 0.4),
    ("grouped_channel", ConvShape(n=1, c=12, h=7, w=7, f=30, kh=3, kw=3, groups=3), 0.5, wl.COL_CHANNEL, 0.5),
    ("filters_only", ConvShape(n=1, c=7, h=5, w=5, f=41, kh=2, kw=2), 0.3, wl.COL_NONE, 1.0),
    ("wide_rows", ConvShape(n=1, c=600, h=3, w=3, f=9, kh=3, kw=3), 1.0, wl.COL_SHAPE, 0.1),
]


def _run(s, W, U, kf, ck, kc):
    from paper_1807_11091_gb300 import sadmm
    dev = torch.device("cuda", 0)
    step = sadmm.AdmmStep(s.desc16(), kf, ck, kc, dev)
    Wd, Ud = W.to(dev), U.to(dev).clone()
    Z = torch.full_like(Wd, float("nan"))
    fi, ci = step(Wd, Ud, Z)
    assert sadmm.device_status() == 0
    return fi.cpu().numpy(), (ci.cpu().numpy() if ci is not None else None), Z.cpu(), Ud.cpu()


def _check(s, W, U, kf, ck, kc, what):
    fi, ci, Z, Un = _run(s, W, U, kf, ck, kc)
    rows, cols, Zo, Uo = oracle.admm_update(W, U, s.taps, kf, ck, kc)
    assert np.array_equal(fi, rows), f"{what}: filter list"
    if ck != wl.COL_NONE:
        assert np.array_equal(ci, cols), f"{what}: column list"
    assert torch.equal(Z.view(torch.int16 if Z.dtype == torch.bfloat16 else torch.int32),
                       Zo.view(torch.int16 if Zo.dtype == torch.bfloat16 else torch.int32)), f"{what}: Z"
    assert torch.equal(Un.view(torch.int16 if Un.dtype == torch.bfloat16 else torch.int32),
                       Uo.view(torch.int16 if Uo.dtype == torch.bfloat16 else torch.int32)), f"{what}: U"


@pytest.mark.parametrize("layer", LAYERS, ids=lambda l: l.name)
def test_admm_update_fp32_layers(layer):
    s = layer.shape
    st = wl.gen_admm_state(s, layer.seed)
    _check(s, st["W"], st["U"], layer.k_filters, layer.colkind, layer.k_cols, layer.name)


@pytest.mark.parametrize("case", SMALL, ids=lambda c: c[0])
@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16], ids=["fp32", "bf16"])
def test_admm_update_small(case, dtype):
    name, s, ff, ck, cf = case
    G = s.cg if ck == wl.COL_CHANNEL else s.k
    kf, kc = wl.retained(ff, s.f), (wl.retained(cf, G) if ck != wl.COL_NONE else 0)
    st = wl.gen_admm_state(s, 77, dtype)
    _check(s, st["W"], st["U"], kf, ck, kc, name)


def test_admm_keep_all_and_keep_none():
    s = SMALL[0][1]
    st = wl.gen_admm_state(s, 5)
    W, U = st["W"], st["U"]
    _, _, Z, Un = _run(s, W, U, s.f, wl.COL_SHAPE, s.k)
    assert torch.equal(Z, W + U) and not bool(Un.any())
    _, _, Z, Un = _run(s, W, U, 0, wl.COL_SHAPE, s.k)
    assert not bool(Z.any()) and torch.equal(Un, W + U)
    _check(s, W, U, 0, wl.COL_SHAPE, 0, "nothing kept")


def test_admm_iterations_track_the_oracle():
    """Three ADMM rounds with a new W each round and U carried over: the GPU
    and the oracle each carry their own U, which must stay bit-identical."""
    from paper_1807_11091_gb300 import sadmm
    L = wl.alexnet()[2]
    s = L.shape
    dev = torch.device("cuda", 0)
    step = sadmm.AdmmStep(s.desc16(), L.k_filters, L.colkind, L.k_cols, dev)
    U_gpu = torch.zeros(s.w_shape(), device=dev)
    U_cpu = torch.zeros(s.w_shape())
    for it in range(3):
        W = wl.gen_admm_state(s, 1000 + it)["W"]
        Z = torch.empty_like(U_gpu)
        fi, ci = step(W.to(dev), U_gpu, Z)
        rows, cols, Zo, U_cpu = oracle.admm_update(W, U_cpu, s.taps, L.k_filters, L.colkind, L.k_cols)
        assert np.array_equal(fi.cpu().numpy(), rows) and np.array_equal(ci.cpu().numpy(), cols)
        assert torch.equal(Z.cpu(), Zo) and torch.equal(U_gpu.cpu(), U_cpu), f"iteration {it}"
