"""Failure detection, tested without faulting or hanging the GPU.

* Bad index lists are injected from the host into sadmm_pack: a filter or
  column list that is not strictly ascending, or holds an index out of range.
  The pack kernel's own checks must turn them into an all-zero plan (every
  filter pruned, every column dropped), raise the device status word (read
  back as SADMM_EINVAL), and leave the library usable: a repack with good lists
  gives the oracle's output again.
* A bounded wait is made to run out: the library's self-test runs the same
  mbarrier wait the pipelined kernels use, with a limit of a few milliseconds,
  on a barrier nothing arrives on.  The kernel must return, the status word must
  read SADMM_ETIMEOUT, and the context must stay usable (a real forward runs
  and matches the oracle afterwards).
"""
import numpy as np
import pytest
import torch

import oracle
import workloads as wl
from workloads import ConvShape

pytestmark = pytest.mark.gpu

KF, KC = 6, 40


def _good_lists(s, t):
    rows, cols, _, _ = oracle.project(t["W"], s.taps, KF, wl.COL_SHAPE, KC)
    return rows.astype(np.int32), cols.astype(np.int32)


def _corrupt(rows, cols, kind, s):
    rows, cols = rows.copy(), cols.copy()
    if kind == "filters_descending":
        rows[[1, 2]] = rows[[2, 1]]
    elif kind == "filter_repeated":
        rows[3] = rows[2]
    elif kind == "filter_out_of_range":
        rows[-1] = s.f
    elif kind == "columns_descending":
        cols[[0, 5]] = cols[[5, 0]]
    elif kind == "column_out_of_range":
        cols[-1] = s.k + 3
    elif kind == "column_negative":
        cols[0] = -1
    return rows, cols


def _forward(pc, x, bias):
    y = torch.full(pc.out_shape(), float("nan"), dtype=torch.float32, device=x.device)
    pc.forward(x, bias, relu=True, out=y)
    return y


@pytest.mark.parametrize("n", [2, 32], ids=["split_k", "whole_tiles"])
@pytest.mark.parametrize("kind", ["filters_descending", "filter_repeated", "filter_out_of_range",
                                  "columns_descending", "column_out_of_range", "column_negative"])
def test_bad_index_lists_give_zero_plan_and_einval(kind, n):
    from paper_1807_11091_gb300 import sadmm
    s = ConvShape(n=n, c=8, h=16, w=16, f=12, kh=3, kw=3, ph=1, pw=1)
    t = wl.gen_tensors(s, seed=61)
    dev = torch.device("cuda", 0)
    W, x, bias = t["W"].to(dev), t["x"].to(dev), t["bias"].to(dev)
    rows, cols = _good_lists(s, t)
    bad_r, bad_c = _corrupt(rows, cols, kind, s)
    assert sadmm.device_status() == 0
    pc = sadmm.PrunedConv(s.desc16(), W, torch.as_tensor(bad_r, device=dev), wl.COL_SHAPE,
                          torch.as_tensor(bad_c, device=dev), KF, KC)
    assert sadmm.device_status() == sadmm.SADMM_EINVAL  # raised by the pack kernel, then cleared
    y = _forward(pc, x, bias)
    assert sadmm.device_status() == 0
    assert torch.all(y == 0), "a rejected plan must write an all-zero output"
    # the same plan buffer, repacked with good lists, is correct again
    pc.repack(W, torch.as_tensor(rows, device=dev), torch.as_tensor(cols, device=dev))
    y = _forward(pc, x, bias)
    assert sadmm.device_status() == 0
    n1 = min(n, 2)
    ref = oracle.pruned_conv(t["x"], t["W"], t["bias"], s.desc16(), s.taps, rows, wl.COL_SHAPE, cols, n1=n1)
    got = y[:n1].cpu().numpy()
    assert np.abs(got - ref).max() <= 2e-3 * np.abs(ref).max()


def test_bounded_wait_runs_out_and_reports_timeout():
    from paper_1807_11091_gb300 import sadmm
    stream = torch.cuda.current_stream().cuda_stream
    res = torch.full((1,), -1, dtype=torch.int32, device="cuda")
    assert sadmm.sadmm_last_device_status(stream) == 0
    # nothing arrives: the wait gives up after 3 ms and the kernel returns
    assert sadmm.sadmm_selftest_wait(3000, 0, res.data_ptr(), stream) == 0
    assert sadmm.sadmm_last_device_status(stream) == sadmm.SADMM_ETIMEOUT
    assert int(res.item()) == 0
    assert sadmm.sadmm_last_device_status(stream) == 0  # reading the word cleared it
    # the barrier completes: the same wait succeeds and raises nothing
    assert sadmm.sadmm_selftest_wait(3000, 1, res.data_ptr(), stream) == 0
    assert sadmm.sadmm_last_device_status(stream) == 0
    assert int(res.item()) == 1
    # the context is still usable: a pruned forward matches the oracle
    layer = wl.single2d()[0]
    s = layer.shape
    t = wl.gen_tensors(s, seed=layer.seed)
    dev = torch.device("cuda", 0)
    W = t["W"].to(dev)
    fi, ci, _ = sadmm.project_groups(s.desc16(), W, layer.k_filters, layer.colkind, layer.k_cols)
    pc = sadmm.PrunedConv(s.desc16(), W, None, layer.colkind, ci, layer.k_filters, layer.k_cols)
    y = _forward(pc, t["x"].to(dev), t["bias"].to(dev))
    assert sadmm.device_status() == 0
    rows, cols, _, _ = oracle.project(t["W"], s.taps, layer.k_filters, layer.colkind, layer.k_cols)
    ref = oracle.pruned_conv(t["x"], t["W"], t["bias"], s.desc16(), s.taps, rows, layer.colkind, cols)
    assert np.abs(y.cpu().numpy() - ref).max() <= 2e-3 * np.abs(ref).max()
