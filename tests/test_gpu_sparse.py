"""GPU parity of the non-structured sparse forward (sadmm_sparse_pack +
sadmm_sparse_conv_fwd): the layer with W pruned element by element, against the
oracle's fp64 direct convolution of W times the keep mask (Sec. 4,
non-structured sparsity; the kept set is the oracle's element projection, the
largest |W| entries).  Outputs within 2e-3 * max|oracle|, every element
written; a plan whose capacity is too small comes out empty and raises the
status word."""
import numpy as np
import pytest
import torch

import oracle
import workloads as wl
from workloads import ConvShape

from _helpers import assert_close

pytestmark = pytest.mark.gpu

CASES = [
    ("pad_3x3", ConvShape(n=2, c=5, h=11, w=13, f=37, kh=3, kw=3, ph=1, pw=1), 0.3),
    ("groups2_5x5", ConvShape(n=2, c=8, h=9, w=9, f=12, kh=5, kw=5, ph=2, pw=2, groups=2), 0.5),
    ("stride4_11x11", ConvShape(n=1, c=3, h=35, w=35, f=16, kh=11, kw=11, sh=4, sw=4), 0.2),
    ("c3d", ConvShape(n=2, c=4, t=5, h=6, w=7, f=20, kt=3, kh=3, kw=3, pt=1, ph=1, pw=1), 0.1),
    ("1x1", ConvShape(n=3, c=24, h=7, w=7, f=40, kh=1, kw=1), 0.05),
    ("7x7_split_mask", ConvShape(n=1, c=6, h=15, w=12, f=8, kh=7, kw=7, sh=2, sw=2, ph=3, pw=3), 0.4),
]


def _sparse(s, t, keep, capacity=None, out_dtype=torch.float32, relu=True):
    from paper_1807_11091_gb300 import sadmm
    dev = torch.device("cuda", 0)
    desc = sadmm.make_desc(s.desc16())
    cap = int(keep.sum()) if capacity is None else capacity
    nbytes = sadmm.sadmm_sparse_plan_size(desc, cap)
    assert nbytes > 0
    plan = torch.empty(nbytes, dtype=torch.uint8, device=dev)
    W = t["W"].to(dev)
    kd = torch.as_tensor(keep.reshape(s.f, -1).astype(np.uint8), device=dev)
    stream = int(torch.cuda.current_stream().cuda_stream)
    st = sadmm.sadmm_sparse_pack(desc, W.data_ptr(), sadmm.SADMM_BF16, kd.data_ptr(), cap, plan.data_ptr(), nbytes,
                                 stream)
    assert st == 0
    y = torch.full(s.y_shape(), float("nan"), dtype=out_dtype, device=dev)
    x, b = t["x"].to(dev), t["bias"].to(dev)
    st = sadmm.sadmm_sparse_conv_fwd(desc, plan.data_ptr(), x.data_ptr(), b.data_ptr(), 1 if relu else 0, y.data_ptr(),
                                     sadmm.SADMM_BF16 if out_dtype == torch.bfloat16 else sadmm.SADMM_FP32, stream)
    assert st == 0
    return y, sadmm.sadmm_last_device_status(stream)


def _oracle(s, t, keep, relu=True, n0=0, n1=None):
    Wm = t["W"].to(torch.float64).numpy() * keep.reshape(t["W"].shape)
    return oracle.conv(t["x"], Wm, t["bias"], s.desc16(), relu=relu, n0=n0, n1=n1)


@pytest.mark.parametrize("case", CASES, ids=lambda c: c[0])
@pytest.mark.parametrize("relu", [True, False])
def test_sparse_forward_matches_oracle(case, relu):
    name, s, density = case
    t = wl.gen_tensors(s, seed=23)
    keep = oracle.project_elements(t["W"], wl.retained(density, s.f * s.k))
    y, st = _sparse(s, t, keep, relu=relu)
    assert st == 0
    assert bool(torch.isfinite(y).all())
    assert_close(y.cpu().numpy(), _oracle(s, t, keep, relu=relu), what=f"sparse {name}")


def test_sparse_forward_empty_and_full_masks():
    s = CASES[1][1]
    t = wl.gen_tensors(s, seed=3)
    for keep in (np.zeros(t["W"].shape, bool), np.ones(t["W"].shape, bool)):
        y, st = _sparse(s, t, keep)
        assert st == 0
        assert_close(y.cpu().numpy(), _oracle(s, t, keep), what=f"mask of {int(keep.sum())}")


def test_sparse_capacity_overflow_gives_empty_plan():
    from paper_1807_11091_gb300 import sadmm
    s = CASES[0][1]
    t = wl.gen_tensors(s, seed=4)
    keep = oracle.project_elements(t["W"], wl.retained(0.3, s.f * s.k))
    y, st = _sparse(s, t, keep, capacity=int(keep.sum()) - 1)
    assert st == sadmm.SADMM_EINVAL
    b = np.maximum(t["bias"].numpy(), 0.0)
    assert np.array_equal(y.cpu().numpy(), np.broadcast_to(b[None, :, None, None], y.shape).astype(np.float32))


def test_sparse_bf16_output():
    s = CASES[0][1]
    t = wl.gen_tensors(s, seed=5)
    keep = oracle.project_elements(t["W"], wl.retained(0.4, s.f * s.k))
    y, st = _sparse(s, t, keep, out_dtype=torch.bfloat16)
    assert st == 0
    ref = _oracle(s, t, keep)
    ref_b = torch.from_numpy(ref).to(torch.bfloat16).float().numpy()
    ulp = np.abs(ref_b) * 2.0 ** -7 + 1e-30
    assert np.all(np.abs(y.float().cpu().numpy() - ref_b) <= ulp + 1e-6 * np.abs(ref).max())


def test_sparse_full_size_sweep_layer():
    """The sweep layer (N128 C256 28x28 F512 3x3) at 10% element density, the
    kept set from the oracle's projection: first and last image element by
    element, every element written."""
    s = wl.sweep()[0].shape
    t = wl.gen_tensors(s, seed=wl.sweep()[0].seed)
    keep = oracle.project_elements(t["W"], wl.retained(0.1, s.f * s.k))
    y, st = _sparse(s, t, keep)
    assert st == 0
    assert bool(torch.isfinite(y).all())
    for n in (0, s.n - 1):
        assert_close(y[n:n + 1].cpu().numpy(), _oracle(s, t, keep, n0=n, n1=n + 1), what=f"image {n}")
