"""Shared helpers of the GPU parity tests: run one pruned layer through the C ABI
and through the oracle on the same seeded tensors."""
from __future__ import annotations

import numpy as np
import torch

import oracle
import workloads as wl

TOL_REL = 2e-3  # max|gpu - oracle| <= 2e-3 * max|oracle|, per layer (fp32 output)


def gpu_project(shape: wl.ConvShape, W, k_filters, colkind, k_cols, U=None, with_keys=True):
    from paper_1807_11091_gb300 import sadmm
    fi, ci, keys = sadmm.project_groups(shape.desc16(), W, k_filters, colkind, k_cols, U=U, with_keys=with_keys)
    torch.cuda.synchronize()
    fi = fi.cpu().numpy().astype(np.int64)
    ci = ci.cpu().numpy().astype(np.int64) if ci is not None else None
    keys = keys.cpu().numpy() if keys is not None else None
    return fi, ci, keys


def n_colgroups(colkind, k_cols, shape):
    return shape.k if colkind == wl.COL_NONE else k_cols


def gpu_layer(shape: wl.ConvShape, t, k_filters, colkind, k_cols, relu=True, out_dtype=torch.float32,
              use_bias=True, project=True, filt_idx=None, col_idx=None, max_ctas=0):
    """Projection (unless index lists are given), pack and forward on cuda:0
    (max_ctas > 0: a plan for at most that many SMs).
    Returns (filt_idx, col_idx, y on the host, the PrunedConv)."""
    from paper_1807_11091_gb300 import sadmm
    dev = torch.device("cuda", 0)
    W = t["W"].to(dev)
    x = t["x"].to(dev)
    bias = t["bias"].to(dev) if use_bias else None
    if project:
        fi_d, ci_d, _ = sadmm.project_groups(shape.desc16(), W, k_filters, colkind, k_cols)
    else:
        fi_d = torch.as_tensor(np.asarray(filt_idx, dtype=np.int32), device=dev)
        ci_d = None if col_idx is None else torch.as_tensor(np.asarray(col_idx, dtype=np.int32), device=dev)
    pc = sadmm.PrunedConv(shape.desc16(), W, fi_d if k_filters < shape.f else None, colkind,
                          ci_d if colkind != wl.COL_NONE else None, k_filters, n_colgroups(colkind, k_cols, shape),
                          max_ctas=max_ctas)
    y = torch.full(pc.out_shape(), float("nan"), dtype=out_dtype, device=dev)
    pc.forward(x, bias, relu=relu, out=y)
    st = sadmm.device_status()
    assert st == 0, f"device status {st}"
    fi = fi_d.cpu().numpy().astype(np.int64)[:k_filters]
    ci = ci_d.cpu().numpy().astype(np.int64) if ci_d is not None else np.arange(shape.k)
    return fi, ci, y.float().cpu().numpy() if out_dtype != torch.float32 else y.cpu().numpy(), pc


def oracle_layer(shape: wl.ConvShape, t, filt_idx, colkind, col_idx, relu=True, use_bias=True, n0=0, n1=None):
    return oracle.pruned_conv(t["x"], t["W"], t["bias"] if use_bias else None, shape.desc16(), shape.taps,
                              filt_idx, colkind, col_idx, relu=relu, n0=n0, n1=n1)


def assert_close(y_gpu, y_ref, tol=TOL_REL, what=""):
    assert y_gpu.shape == y_ref.shape, (y_gpu.shape, y_ref.shape)
    assert np.all(np.isfinite(y_gpu)), f"{what}: non-finite outputs (unwritten?)"
    scale = float(np.abs(y_ref).max())
    err = float(np.abs(y_gpu.astype(np.float64) - y_ref).max())
    assert err <= tol * max(scale, 1e-30), f"{what}: max err {err:.3e} vs {tol} * {scale:.3e}"
    return err, scale


def pruned_filters(F, filt_idx):
    keep = np.zeros(F, bool)
    keep[np.asarray(filt_idx, dtype=np.int64)] = True
    return np.nonzero(~keep)[0]
