"""CPU oracle for the structured-pruned CONV forward path (StructADMM, arXiv 1807.11091).

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may import this package.  It shares no code
with the CUDA library (``paper_1807_11091_gb300``) and neither imports the
other.  All arithmetic is fp64 in plain C loops (``sadmm_oracle.c``); this file
only marshals numpy arrays and composes the steps in the paper's order.

What it computes, with the passage each step follows:

* ``group_keys`` -- squared Frobenius norms O_g of the filter, channel or
  shape groups of V = W (+U) (Sec. 4, solution of the Z-subproblem, Eq. 4).
* ``topk`` -- keep the k largest O_g; equal keys go to the lower index
  (a reading: the paper does not say how ties break).
* ``project`` -- the Euclidean projection onto the structured-sparsity set
  (Sec. 4); combined row + column pruning (Table 2) takes rows first on the
  full tensor, then column keys over the kept rows only (a reading: the paper
  gives no rule for the combination).
* ``masked_weights`` / ``masked_bias`` -- W with the pruned rows and columns
  of the GEMM matrix set to zero (Sec. 3, "Combination of structured
  sparsities"); the bias of a pruned filter is zero (a reading).
* ``admm_update`` -- the ADMM Z-update (projection of W + U) and the dual
  update U <- U + W - Z (Sec. 4), in the tensors' precision.
* ``project_elements`` / ``admm_update_elements`` -- the non-structured case
  (Sec. 4): keep the largest |V| entries.
* ``conv`` -- direct convolution over the full masked tensor (fp64).
* ``pruned_conv_backward`` -- gradients for masked retraining (Sec. 4).

Parity pins: every function here is checked in ``tests/test_oracle_*.py``
against brute force, a library convolution, closed forms and invariants.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from typing import Optional, Tuple

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "sadmm_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "libsadmm_oracle.so")

COL_NONE, COL_SHAPE, COL_CHANNEL = 0, 1, 2

_lib = None


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (-O2, OpenMP).  Returns the library path."""
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    os.makedirs(_BUILD, exist_ok=True)
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fopenmp", _SRC, "-o", tmp]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    if _lib is None:
        lib = ctypes.CDLL(build())
        dp = ctypes.POINTER(ctypes.c_double)
        ip = ctypes.POINTER(ctypes.c_int)
        up = ctypes.POINTER(ctypes.c_ubyte)
        lib.oracle_filter_keys.argtypes = [ctypes.c_int, ctypes.c_int, dp, dp]
        lib.oracle_shape_keys.argtypes = [ctypes.c_int, ctypes.c_int, dp, up, dp]
        lib.oracle_channel_keys.argtypes = [ctypes.c_int, ctypes.c_int, ctypes.c_int, dp, up, dp]
        lib.oracle_topk.argtypes = [ctypes.c_int, dp, ctypes.c_int, ip]
        lib.oracle_topk.restype = ctypes.c_int
        lib.oracle_conv.argtypes = [ip, dp, dp, dp, ctypes.c_int, ctypes.c_int, ctypes.c_int, dp]
        _lib = lib
    return _lib


def _dptr(a: np.ndarray):
    return a.ctypes.data_as(ctypes.POINTER(ctypes.c_double))


def _as_f64(a) -> np.ndarray:
    """Exact widening of a bf16/fp32/fp64 torch tensor or numpy array to fp64."""
    try:
        import torch
        if isinstance(a, torch.Tensor):
            return np.ascontiguousarray(a.detach().cpu().to(torch.float64).numpy())
    except ImportError:  # pragma: no cover
        pass
    return np.ascontiguousarray(np.asarray(a, dtype=np.float64))


def _rows_mask(F: int, rows) -> Optional[np.ndarray]:
    if rows is None:
        return None
    m = np.zeros(F, dtype=np.uint8)
    m[np.asarray(rows, dtype=np.int64)] = 1
    return m


# ---------------------------------------------------------------------------
# Group keys and selection
# ---------------------------------------------------------------------------

def filter_keys(V2: np.ndarray) -> np.ndarray:
    """O_a = ||V[a,:]||^2 for every row a of the [F, K] GEMM matrix."""
    V2 = np.ascontiguousarray(V2, dtype=np.float64)
    F, K = V2.shape
    out = np.empty(F, dtype=np.float64)
    _load().oracle_filter_keys(F, K, _dptr(V2), _dptr(out))
    return out


def shape_keys(V2: np.ndarray, rows=None) -> np.ndarray:
    """O_j = ||V[rows, j]||^2 for every column j (rows: kept filter indices or None)."""
    V2 = np.ascontiguousarray(V2, dtype=np.float64)
    F, K = V2.shape
    out = np.empty(K, dtype=np.float64)
    m = _rows_mask(F, rows)
    mp = m.ctypes.data_as(ctypes.POINTER(ctypes.c_ubyte)) if m is not None else None
    _load().oracle_shape_keys(F, K, _dptr(V2), mp, _dptr(out))
    return out


def channel_keys(V2: np.ndarray, taps: int, rows=None) -> np.ndarray:
    """O_b = ||V[rows, b*taps:(b+1)*taps]||^2 for every channel b of a group."""
    V2 = np.ascontiguousarray(V2, dtype=np.float64)
    F, K = V2.shape
    assert K % taps == 0
    Cg = K // taps
    out = np.empty(Cg, dtype=np.float64)
    m = _rows_mask(F, rows)
    mp = m.ctypes.data_as(ctypes.POINTER(ctypes.c_ubyte)) if m is not None else None
    _load().oracle_channel_keys(F, Cg, taps, _dptr(V2), mp, _dptr(out))
    return out


def topk(keys: np.ndarray, k: int) -> np.ndarray:
    """Ascending indices of the k largest keys; equal keys go to the lower index."""
    keys = np.ascontiguousarray(keys, dtype=np.float64)
    G = keys.shape[0]
    out = np.empty(max(k, 1), dtype=np.int32)
    r = _load().oracle_topk(G, _dptr(keys), int(k), out.ctypes.data_as(ctypes.POINTER(ctypes.c_int)))
    if r < 0:
        raise ValueError(f"k={k} out of range for {G} groups")
    return out[:k].copy()


def select_margin(keys: np.ndarray, k: int) -> float:
    """Relative gap (key_k - key_{k+1}) / key_k between the last kept and first
    dropped key (sorted descending); inf when nothing is dropped or kept."""
    if k <= 0 or k >= len(keys):
        return float("inf")
    s = np.sort(np.asarray(keys, dtype=np.float64))[::-1]
    if s[k - 1] == 0.0:
        return 0.0
    return float((s[k - 1] - s[k]) / s[k - 1])


def as_matrix(W, U=None) -> np.ndarray:
    """V = W (+U), widened exactly to fp64 and viewed as the [F, K] GEMM matrix."""
    V = _as_f64(W)
    if U is not None:
        V = V + _as_f64(U)
    return V.reshape(V.shape[0], -1)


def project(W, taps: int, k_filters: int, colkind: int, k_cols: int, U=None):
    """Euclidean projection onto the structured-sparsity set (Sec. 4).

    Returns (filt_idx, col_idx, filter_keys, column_keys).  col_idx holds
    column indices (shape-wise), channel indices (channel-wise) or every column
    (no column pruning).  Rows are chosen first; column keys are taken over the
    kept rows only.
    """
    V = as_matrix(W, U)
    F, K = V.shape
    fk = filter_keys(V)
    rows = topk(fk, k_filters)
    row_sel = None if k_filters == F else rows
    if colkind == COL_SHAPE:
        ck = shape_keys(V, row_sel)
        cols = topk(ck, k_cols)
    elif colkind == COL_CHANNEL:
        ck = channel_keys(V, taps, row_sel)
        cols = topk(ck, k_cols)
    elif colkind == COL_NONE:
        ck = None
        cols = np.arange(K, dtype=np.int32)
    else:
        raise ValueError(f"bad colkind {colkind}")
    return rows, cols, fk, ck


def expand_columns(colkind: int, cols, taps: int, K: int) -> np.ndarray:
    """GEMM column indices kept: channel b keeps columns b*taps .. b*taps+taps-1."""
    if colkind == COL_NONE:
        return np.arange(K, dtype=np.int64)
    cols = np.asarray(cols, dtype=np.int64)
    if colkind == COL_CHANNEL:
        return (cols[:, None] * taps + np.arange(taps)[None, :]).reshape(-1)
    return cols


def masked_weights(W, filt_idx, colkind: int, col_idx, taps: int) -> np.ndarray:
    """W in fp64 with pruned GEMM rows and columns set to zero (original shape)."""
    Wd = _as_f64(W)
    shape = Wd.shape
    V = Wd.reshape(shape[0], -1).copy()
    F, K = V.shape
    rmask = np.zeros(F, dtype=bool)
    rmask[np.asarray(filt_idx, dtype=np.int64)] = True
    cmask = np.zeros(K, dtype=bool)
    cmask[expand_columns(colkind, col_idx, taps, K)] = True
    V[~rmask, :] = 0.0
    V[:, ~cmask] = 0.0
    return V.reshape(shape)


def masked_bias(bias, F: int, filt_idx) -> np.ndarray:
    """Bias in fp64 with the bias of every pruned filter set to zero."""
    b = np.zeros(F, dtype=np.float64) if bias is None else _as_f64(bias).reshape(-1).copy()
    keep = np.zeros(F, dtype=bool)
    keep[np.asarray(filt_idx, dtype=np.int64)] = True
    b[~keep] = 0.0
    return b


def admm_update(W, U, taps: int, k_filters: int, colkind: int, k_cols: int):
    """One ADMM Z- and U-update (Sec. 4).

    The Z-subproblem's optimum is the Euclidean projection of
    V = W^{k+1} + U^k onto the structured-sparsity set (``project``), and the
    scaled dual becomes U^{k+1} = U^k + W^{k+1} - Z^{k+1} = V - Z^{k+1}.
    W and U are torch tensors of one dtype (bf16 or fp32).  V is formed
    exactly in fp64 and rounded once to that dtype for Z and U^{k+1} (a
    reading: the paper works in real arithmetic, the tensors keep their
    precision), so Z is V on the kept (row, column) pairs and 0 elsewhere and
    U^{k+1} is 0 on the kept pairs and V elsewhere.

    Returns (filt_idx, col_idx, Z, U_next); Z and U_next have W's dtype and shape.
    """
    import torch
    rows, cols, _, _ = project(W, taps, k_filters, colkind, k_cols, U=U)
    V = as_matrix(W, U)
    F, K = V.shape
    rkeep = np.zeros(F, dtype=bool)
    rkeep[np.asarray(rows, dtype=np.int64)] = True
    ckeep = np.zeros(K, dtype=bool)
    ckeep[expand_columns(colkind, cols, taps, K)] = True
    keep = rkeep[:, None] & ckeep[None, :]
    Z64 = np.where(keep, V, 0.0)
    U64 = V - Z64
    Z = torch.from_numpy(Z64).to(W.dtype).reshape(W.shape)
    Un = torch.from_numpy(U64).to(W.dtype).reshape(W.shape)
    return rows, cols, Z, Un


def project_elements(W, k_elems: int, U=None) -> np.ndarray:
    """Non-structured projection (Sec. 4): keep the k_elems entries of
    V = W (+U) with the largest |V| (V exact in fp64), equal magnitudes to the
    lower flat index.  Returns a bool mask of W's shape."""
    V = as_matrix(W, U)
    flat = np.abs(V).reshape(-1)
    keep = np.zeros(flat.shape[0], dtype=bool)
    keep[topk(flat, int(k_elems))] = True
    return keep.reshape(_as_f64(W).shape)


def admm_update_elements(W, U, k_elems: int):
    """ADMM Z- and U-update for non-structured sparsity: Z = V on the kept
    entries (V rounded once to the tensors' dtype), U_next = V - Z."""
    import torch
    keep = project_elements(W, k_elems, U=U)
    V = _as_f64(W) + _as_f64(U)
    Z64 = np.where(keep, V, 0.0)
    U64 = V - Z64
    return keep, torch.from_numpy(Z64).to(W.dtype), torch.from_numpy(U64).to(W.dtype)


# ---------------------------------------------------------------------------
# Convolution
# ---------------------------------------------------------------------------

def conv(x, Wm, bm, desc16, relu: bool = True, n0: int = 0, n1: Optional[int] = None) -> np.ndarray:
    """Direct convolution in fp64 of images n0..n1-1.

    x: [N, C, (T,) H, W]; Wm: [F, Cg, (KT,) KH, KW]; bm: [F] or None;
    desc16: n c t h w f groups kt kh kw st sh sw pt ph pw.
    Returns y: [n1-n0, F, (OT,) OH, OW] (the T axis only when x has one).
    """
    d = [int(v) for v in desc16]
    N, C, T, H, Wd, F, G, KT, KH, KW, ST, SH, SW, PT, PH, PW = d
    if n1 is None:
        n1 = N
    xd = _as_f64(x)
    wd = _as_f64(Wm)
    bd = np.zeros(F, dtype=np.float64) if bm is None else _as_f64(bm).reshape(-1)
    assert xd.size == N * C * T * H * Wd, "x does not match the descriptor"
    assert wd.size == F * (C // G) * KT * KH * KW, "W does not match the descriptor"
    OT = (T + 2 * PT - KT) // ST + 1
    OH = (H + 2 * PH - KH) // SH + 1
    OW = (Wd + 2 * PW - KW) // SW + 1
    y = np.empty((n1 - n0, F, OT, OH, OW), dtype=np.float64)
    darr = (ctypes.c_int * 16)(*d)
    _load().oracle_conv(darr, _dptr(np.ascontiguousarray(xd.reshape(-1))),
                        _dptr(np.ascontiguousarray(wd.reshape(-1))), _dptr(np.ascontiguousarray(bd)),
                        1 if relu else 0, int(n0), int(n1), _dptr(y))
    if xd.ndim == 4:
        y = y.reshape(n1 - n0, F, OH, OW)
    return y


def pruned_conv(x, W, bias, desc16, taps: int, filt_idx, colkind: int, col_idx,
                relu: bool = True, n0: int = 0, n1: Optional[int] = None) -> np.ndarray:
    """The pruned layer's output: conv over the masked W with the masked bias."""
    Wm = masked_weights(W, filt_idx, colkind, col_idx, taps)
    bm = masked_bias(bias, int(desc16[5]), filt_idx)
    return conv(x, Wm, bm, desc16, relu=relu, n0=n0, n1=n1)


# ---------------------------------------------------------------------------
# Backward for masked retraining
# ---------------------------------------------------------------------------

def pruned_conv_backward(x, W, bias, desc16, taps: int, filt_idx, colkind: int, col_idx, dy, relu: bool = True,
                         y=None):
    """Gradients of the pruned layer for masked retraining (Sec. 4: the zero
    weights stay masked, only kept weights learn), in fp64.

    y = ReLU(conv(x, Wm) + bm) with Wm, bm the masked weights and bias.
    Returns (dx, dW, db) for the upstream gradient dy: dW and db are the
    gradients with respect to the kept entries (zero on masked entries), dx the
    input gradient.  The derivative is taken by torch's autograd in fp64 (a
    library routine serving as the differentiation step); the tests pin it to
    finite differences of ``pruned_conv``.  When ``y`` (a given forward
    output) is passed, the ReLU derivative is [y > 0] from it, so that a
    comparison takes the ReLU decision on the same values.
    """
    import torch
    d = [int(v) for v in desc16]
    N, C, T, H, Wd, F, G, KT, KH, KW, ST, SH, SW, PT, PH, PW = d
    Wm = torch.from_numpy(masked_weights(W, filt_idx, colkind, col_idx, taps)).requires_grad_(True)
    bm = torch.from_numpy(masked_bias(bias, F, filt_idx)).requires_grad_(True)
    xd = torch.from_numpy(_as_f64(x)).requires_grad_(True)
    if T == 1 and KT == 1 and xd.dim() == 4:
        z = torch.nn.functional.conv2d(xd, Wm.reshape(F, C // G, KH, KW), bm, stride=(SH, SW), padding=(PH, PW),
                                       groups=G)
    else:
        z = torch.nn.functional.conv3d(xd.reshape(N, C, T, H, Wd), Wm.reshape(F, C // G, KT, KH, KW), bm,
                                       stride=(ST, SH, SW), padding=(PT, PH, PW), groups=G)
    g = torch.from_numpy(_as_f64(dy)).reshape(z.shape)
    if relu:
        on = (torch.from_numpy(_as_f64(y)).reshape(z.shape) > 0) if y is not None else (z.detach() > 0)
        g = g * on.to(g.dtype)
    z.backward(g)
    keep = masked_weights(np.ones(_as_f64(W).shape), filt_idx, colkind, col_idx, taps) != 0
    dW = Wm.grad.numpy() * keep
    bkeep = np.zeros(F, dtype=bool)
    bkeep[np.asarray(filt_idx, dtype=np.int64)] = True
    db = bm.grad.numpy() * bkeep
    return xd.grad.numpy().reshape(_as_f64(x).shape), dW, db
