"""ctypes binding of libsadmm (include/sadmm.h).

The functions named like the C entry points (``sadmm_*``) marshal arguments and
nothing else: every step of the path runs in the CUDA library.  The torch
helpers at the end (``project_groups``, ``PrunedConv``) only allocate device
memory with torch and pass raw pointers and the current stream through.

There is no CPU fallback: when the library cannot be built or loaded, every
call raises.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional, Sequence, Tuple

from . import build as _build

SADMM_OK, SADMM_EINVAL, SADMM_ECUDA, SADMM_ETIMEOUT, SADMM_EUNSUPPORTED, SADMM_EBOUNDS = 0, -1, -2, -3, -4, -5
SADMM_BF16, SADMM_FP32 = 0, 1
SADMM_COL_NONE, SADMM_COL_SHAPE, SADMM_COL_CHANNEL = 0, 1, 2
SADMM_FWD_ALL, SADMM_FWD_INPUT, SADMM_FWD_REST = 0, 1, 2

SADMM_NOALLOC_SCRATCH_BYTES = 256 * 1024  # include/sadmm.h

DESC_FIELDS = ("n", "c", "t", "h", "w", "f", "groups", "kt", "kh", "kw", "st", "sh", "sw", "pt", "ph", "pw")


class SadmmError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {status_string(status)} ({status})")


class ConvDesc(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int) for n in DESC_FIELDS]


class ProjectItem(ctypes.Structure):
    """sadmm_project_item: one layer of sadmm_project_groups_batch."""
    _fields_ = [("desc", ConvDesc), ("W", ctypes.c_void_p), ("U", ctypes.c_void_p),
                ("k_filters", ctypes.c_int), ("colkind", ctypes.c_int), ("k_cols", ctypes.c_int),
                ("filt_idx", ctypes.c_void_p), ("col_idx", ctypes.c_void_p), ("keys_out", ctypes.c_void_p),
                ("workspace", ctypes.c_void_p), ("ws_bytes", ctypes.c_size_t)]


class AdmmItem(ctypes.Structure):
    """sadmm_admm_item: one layer of sadmm_admm_update_batch."""
    _fields_ = [("desc", ConvDesc), ("W", ctypes.c_void_p), ("U", ctypes.c_void_p), ("Z", ctypes.c_void_p),
                ("k_filters", ctypes.c_int), ("colkind", ctypes.c_int), ("k_cols", ctypes.c_int),
                ("filt_idx", ctypes.c_void_p), ("col_idx", ctypes.c_void_p), ("keys_out", ctypes.c_void_p),
                ("workspace", ctypes.c_void_p), ("ws_bytes", ctypes.c_size_t)]


SADMM_MAX_BATCH = 64  # include/sadmm.h


class Plan(ctypes.Structure):
    _fields_ = [
        ("desc", ConvDesc),
        ("n_filt", ctypes.c_int),
        ("colkind", ctypes.c_int),
        ("n_colgroups", ctypes.c_int),
        ("n_cols", ctypes.c_int),
        ("k_pad", ctypes.c_int),
        ("bn", ctypes.c_int),
        ("n_tiles", ctypes.c_int),
        ("n_pad", ctypes.c_int),
        ("dev_bytes", ctypes.c_size_t),
        ("dev", ctypes.c_void_p),
        ("off_wp", ctypes.c_size_t),
        ("off_gather", ctypes.c_size_t),
        ("off_rowmap", ctypes.c_size_t),
        ("off_zeromap", ctypes.c_size_t),
        ("off_counts", ctypes.c_size_t),
        ("off_colidx", ctypes.c_size_t),
        ("off_partial", ctypes.c_size_t),
        ("splits", ctypes.c_int),
        ("stages_per_split", ctypes.c_int),
        ("off_sk", ctypes.c_size_t),
        ("sk_len", ctypes.c_int),
        ("sk_grid", ctypes.c_int),
        ("ctas", ctypes.c_int),
        ("xs_mode", ctypes.c_int),
        ("xs_r", ctypes.c_int),
        ("xs_q", ctypes.c_int),
        ("xs_cs", ctypes.c_int),
        ("xs_hb", ctypes.c_int),
        ("xs_wb", ctypes.c_int),
        ("xs_pimg", ctypes.c_int),
        ("xs_sp", ctypes.c_int),
        ("xs_kpad", ctypes.c_int),
        ("off_xs", ctypes.c_size_t),
        ("off_wps", ctypes.c_size_t),
        ("off_scol", ctypes.c_size_t),
        ("tmap", ctypes.c_uint64 * 16),
        ("tmap_ws", ctypes.c_uint64 * 16),
        ("tmap_xs", ctypes.c_uint64 * 16),
    ]


class PackItem(ctypes.Structure):
    """sadmm_pack_item: one layer of sadmm_pack_batch."""
    _fields_ = [("plan", ctypes.POINTER(Plan)), ("W", ctypes.c_void_p), ("filt_idx", ctypes.c_void_p),
                ("col_idx", ctypes.c_void_p), ("dev", ctypes.c_void_p), ("dev_bytes", ctypes.c_size_t)]


_lib = None


def library_path() -> str:
    """The library load() uses: the debug build when SADMM_DEBUG=1 is set."""
    return _build.DEBUG_LIB if _build.debug_requested() else _build.LIB


def load():
    """Loads libsadmm.so, building it first when it is missing or stale."""
    global _lib
    if _lib is not None:
        return _lib
    path = _build.build()
    lib = ctypes.CDLL(path)
    vp, sz, ci = ctypes.c_void_p, ctypes.c_size_t, ctypes.c_int
    P = ctypes.POINTER
    lib.sadmm_abi_version.restype = ci
    lib.sadmm_abi_version.argtypes = []
    lib.sadmm_plan_struct_size.restype = sz
    lib.sadmm_plan_struct_size.argtypes = []
    lib.sadmm_status_string.restype = ctypes.c_char_p
    lib.sadmm_status_string.argtypes = [ci]
    lib.sadmm_workspace_size.restype = sz
    lib.sadmm_workspace_size.argtypes = [P(ConvDesc), ci]
    lib.sadmm_project_groups.restype = ci
    lib.sadmm_project_groups.argtypes = [P(ConvDesc), vp, vp, ci, ci, ci, ci, vp, vp, vp, vp, sz, vp]
    lib.sadmm_plan_init.restype = ci
    lib.sadmm_plan_init.argtypes = [P(Plan), P(ConvDesc), ci, ci, ci]
    lib.sadmm_plan_init_ctas.restype = ci
    lib.sadmm_plan_init_ctas.argtypes = [P(Plan), P(ConvDesc), ci, ci, ci, ci]
    lib.sadmm_pack.restype = ci
    lib.sadmm_pack.argtypes = [P(Plan), vp, ci, vp, vp, vp, sz, vp]
    lib.sadmm_pack_batch.restype = ci
    lib.sadmm_pack_batch.argtypes = [P(PackItem), ci, ci, vp]
    lib.sadmm_conv_fwd_phase.restype = ci
    lib.sadmm_conv_fwd_phase.argtypes = [P(Plan), vp, vp, ci, vp, ci, ci, vp]
    lib.sadmm_conv_fwd.restype = ci
    lib.sadmm_conv_fwd.argtypes = [P(Plan), vp, vp, ci, vp, ci, vp]
    lib.sadmm_admm_workspace_size.restype = sz
    lib.sadmm_admm_workspace_size.argtypes = [P(ConvDesc), ci]
    lib.sadmm_admm_update.restype = ci
    lib.sadmm_admm_update.argtypes = [P(ConvDesc), vp, vp, vp, ci, ci, ci, ci, vp, vp, vp, vp, sz, vp]
    ll = ctypes.c_longlong
    lib.sadmm_elements_workspace_size.restype = sz
    lib.sadmm_elements_workspace_size.argtypes = [P(ConvDesc)]
    lib.sadmm_project_elements.restype = ci
    lib.sadmm_project_elements.argtypes = [P(ConvDesc), vp, vp, ci, ll, vp, vp, sz, vp]
    lib.sadmm_admm_update_elements.restype = ci
    lib.sadmm_admm_update_elements.argtypes = [P(ConvDesc), vp, vp, vp, ci, ll, vp, sz, vp]
    lib.sadmm_conv_bwd_workspace_size.restype = sz
    lib.sadmm_conv_bwd_workspace_size.argtypes = [P(Plan)]
    lib.sadmm_conv_bwd_workspace_size_chunk.restype = sz
    lib.sadmm_conv_bwd_workspace_size_chunk.argtypes = [P(Plan), ll]
    lib.sadmm_conv_bwd.restype = ci
    lib.sadmm_conv_bwd.argtypes = [P(Plan), vp, vp, vp, ci, ci, vp, vp, vp, vp, sz, vp]
    lib.sadmm_gemm_bf16.restype = ci
    lib.sadmm_gemm_bf16.argtypes = [vp, vp, vp, ll, ll, ll, ll, ci, vp]
    lib.sadmm_last_device_status.restype = ci
    lib.sadmm_last_device_status.argtypes = [vp]
    lib.sadmm_project_groups_batch.restype = ci
    lib.sadmm_project_groups_batch.argtypes = [P(ProjectItem), ci, ci, vp]
    lib.sadmm_admm_update_batch.restype = ci
    lib.sadmm_admm_update_batch.argtypes = [P(AdmmItem), ci, ci, vp]
    lib.sadmm_sparse_plan_size.restype = sz
    lib.sadmm_sparse_plan_size.argtypes = [P(ConvDesc), ll]
    lib.sadmm_sparse_pack.restype = ci
    lib.sadmm_sparse_pack.argtypes = [P(ConvDesc), vp, ci, vp, ll, vp, sz, vp]
    lib.sadmm_sparse_conv_fwd.restype = ci
    lib.sadmm_sparse_conv_fwd.argtypes = [P(ConvDesc), vp, vp, vp, ci, vp, ci, vp]
    lib.sadmm_selftest_wait.restype = ci
    lib.sadmm_selftest_wait.argtypes = [ctypes.c_uint, ci, vp, vp]
    lib.sadmm_project_groups_noalloc.restype = ci
    lib.sadmm_project_groups_noalloc.argtypes = [P(ConvDesc), vp, vp, ci, ci, ci, ci, vp, vp, vp, vp]
    if lib.sadmm_plan_struct_size() != ctypes.sizeof(Plan):
        raise RuntimeError("sadmm_plan layout differs between the library and this binding")
    _lib = lib
    return lib


def _check(status: int, where: str) -> None:
    if status != SADMM_OK:
        raise SadmmError(status, where)


def status_string(status: int) -> str:
    try:
        return load().sadmm_status_string(int(status)).decode()
    except Exception:  # pragma: no cover - only when the library is absent
        return "status"


def make_desc(values: Sequence[int]) -> ConvDesc:
    """ConvDesc from the 16 fields n c t h w f groups kt kh kw st sh sw pt ph pw."""
    return ConvDesc(*[int(v) for v in values])


# --------------------------------------------------------------------------
# C entry points (argument marshalling only; pointers are plain ints)
# --------------------------------------------------------------------------

def sadmm_abi_version() -> int:
    return load().sadmm_abi_version()


def sadmm_plan_struct_size() -> int:
    return load().sadmm_plan_struct_size()


def sadmm_status_string(status: int) -> str:
    return status_string(status)


def sadmm_workspace_size(desc: ConvDesc, colkind: int) -> int:
    return load().sadmm_workspace_size(ctypes.byref(desc), int(colkind))


def sadmm_project_groups(desc: ConvDesc, W: int, U: Optional[int], wdt: int, k_filters: int, colkind: int,
                         k_cols: int, filt_idx: int, col_idx: Optional[int], keys_out: Optional[int],
                         workspace: int, ws_bytes: int, stream: Optional[int]) -> int:
    return load().sadmm_project_groups(ctypes.byref(desc), W, U, int(wdt), int(k_filters), int(colkind),
                                       int(k_cols), filt_idx, col_idx, keys_out, workspace, int(ws_bytes),
                                       stream)


def sadmm_project_groups_noalloc(desc: ConvDesc, W: int, U: Optional[int], wdt: int, k_filters: int,
                                 colkind: int, k_cols: int, filt_idx: int, col_idx: Optional[int],
                                 keys_out: Optional[int], stream: Optional[int]) -> int:
    """The projection for callers that cannot pass device scratch memory: the
    keys live in a fixed array inside the library (see include/sadmm.h)."""
    return load().sadmm_project_groups_noalloc(ctypes.byref(desc), W, U, int(wdt), int(k_filters),
                                               int(colkind), int(k_cols), filt_idx, col_idx, keys_out, stream)


def sadmm_admm_workspace_size(desc: ConvDesc, colkind: int) -> int:
    return load().sadmm_admm_workspace_size(ctypes.byref(desc), int(colkind))


def sadmm_admm_update(desc: ConvDesc, W: int, U: int, Z: int, wdt: int, k_filters: int, colkind: int, k_cols: int,
                      filt_idx: int, col_idx: Optional[int], keys_out: Optional[int], workspace: int,
                      ws_bytes: int, stream: Optional[int]) -> int:
    return load().sadmm_admm_update(ctypes.byref(desc), W, U, Z, int(wdt), int(k_filters), int(colkind),
                                    int(k_cols), filt_idx, col_idx, keys_out, workspace, int(ws_bytes), stream)


def sadmm_elements_workspace_size(desc: ConvDesc) -> int:
    return load().sadmm_elements_workspace_size(ctypes.byref(desc))


def sadmm_project_elements(desc: ConvDesc, W: int, U: Optional[int], wdt: int, k_elems: int, keep_out: int,
                           workspace: int, ws_bytes: int, stream: Optional[int]) -> int:
    return load().sadmm_project_elements(ctypes.byref(desc), W, U, int(wdt), int(k_elems), keep_out, workspace,
                                         int(ws_bytes), stream)


def sadmm_admm_update_elements(desc: ConvDesc, W: int, U: int, Z: int, wdt: int, k_elems: int, workspace: int,
                               ws_bytes: int, stream: Optional[int]) -> int:
    return load().sadmm_admm_update_elements(ctypes.byref(desc), W, U, Z, int(wdt), int(k_elems), workspace,
                                             int(ws_bytes), stream)


def sadmm_plan_init(desc: ConvDesc, n_filt: int, colkind: int, n_colgroups: int) -> Tuple[int, Plan]:
    plan = Plan()
    st = load().sadmm_plan_init(ctypes.byref(plan), ctypes.byref(desc), int(n_filt), int(colkind),
                                int(n_colgroups))
    return st, plan


def sadmm_plan_init_ctas(desc: ConvDesc, n_filt: int, colkind: int, n_colgroups: int,
                         max_ctas: int) -> Tuple[int, Plan]:
    plan = Plan()
    st = load().sadmm_plan_init_ctas(ctypes.byref(plan), ctypes.byref(desc), int(n_filt), int(colkind),
                                     int(n_colgroups), int(max_ctas))
    return st, plan


def sadmm_pack(plan: Plan, W: int, wdt: int, filt_idx: Optional[int], col_idx: Optional[int], dev: int,
               dev_bytes: int, stream: Optional[int]) -> int:
    return load().sadmm_pack(ctypes.byref(plan), W, int(wdt), filt_idx, col_idx, dev, int(dev_bytes), stream)


def sadmm_conv_fwd(plan: Plan, x: int, bias: Optional[int], relu: int, y: int, ydt: int,
                   stream: Optional[int]) -> int:
    return load().sadmm_conv_fwd(ctypes.byref(plan), x, bias, int(relu), y, int(ydt), stream)


def sadmm_conv_fwd_phase(plan: Plan, x: Optional[int], bias: Optional[int], relu: int, y: Optional[int], ydt: int,
                         phase: int, stream: Optional[int]) -> int:
    return load().sadmm_conv_fwd_phase(ctypes.byref(plan), x, bias, int(relu), y, int(ydt), int(phase), stream)


def sadmm_conv_bwd_workspace_size(plan: Plan) -> int:
    return load().sadmm_conv_bwd_workspace_size(ctypes.byref(plan))


def sadmm_conv_bwd_workspace_size_chunk(plan: Plan, chunk_pixels: int) -> int:
    return load().sadmm_conv_bwd_workspace_size_chunk(ctypes.byref(plan), int(chunk_pixels))


def sadmm_conv_bwd(plan: Plan, x: Optional[int], dy: int, y: Optional[int], ydt: int, relu: int, dW: Optional[int],
                   db: Optional[int], dx: Optional[int], workspace: int, ws_bytes: int, stream: Optional[int]) -> int:
    return load().sadmm_conv_bwd(ctypes.byref(plan), x, dy, y, int(ydt), int(relu), dW, db, dx, workspace,
                                 int(ws_bytes), stream)


def sadmm_gemm_bf16(A: int, B: int, C: int, M: int, N: int, K: int, ldc: int, accumulate: int,
                    stream: Optional[int]) -> int:
    return load().sadmm_gemm_bf16(A, B, C, int(M), int(N), int(K), int(ldc), int(accumulate), stream)


def sadmm_last_device_status(stream: Optional[int]) -> int:
    return load().sadmm_last_device_status(stream)


def sadmm_project_groups_batch(items: Sequence[ProjectItem], wdt: int, stream: Optional[int]) -> int:
    arr = (ProjectItem * len(items))(*items)
    return load().sadmm_project_groups_batch(arr, len(items), int(wdt), stream)


def sadmm_pack_batch(items: Sequence[PackItem], wdt: int, stream: Optional[int]) -> int:
    arr = (PackItem * len(items))(*items)
    return load().sadmm_pack_batch(arr, len(items), int(wdt), stream)


def sadmm_admm_update_batch(items: Sequence[AdmmItem], wdt: int, stream: Optional[int]) -> int:
    arr = (AdmmItem * len(items))(*items)
    return load().sadmm_admm_update_batch(arr, len(items), int(wdt), stream)


def sadmm_sparse_plan_size(desc: ConvDesc, capacity: int) -> int:
    return load().sadmm_sparse_plan_size(ctypes.byref(desc), int(capacity))


def sadmm_sparse_pack(desc: ConvDesc, W: int, wdt: int, keep: int, capacity: int, plan: int, plan_bytes: int,
                      stream: Optional[int]) -> int:
    return load().sadmm_sparse_pack(ctypes.byref(desc), W, int(wdt), keep, int(capacity), plan, int(plan_bytes),
                                    stream)


def sadmm_sparse_conv_fwd(desc: ConvDesc, plan: int, x: int, bias: Optional[int], relu: int, y: int, ydt: int,
                          stream: Optional[int]) -> int:
    return load().sadmm_sparse_conv_fwd(ctypes.byref(desc), plan, x, bias, int(relu), y, int(ydt), stream)


def sadmm_selftest_wait(limit_us: int, arrive: int, result: Optional[int], stream: Optional[int]) -> int:
    return load().sadmm_selftest_wait(int(limit_us), int(arrive), result, stream)


# --------------------------------------------------------------------------
# torch helpers: device memory and streams only
# --------------------------------------------------------------------------

def _torch():
    import torch
    return torch


def _ptr(t) -> Optional[int]:
    return None if t is None else int(t.data_ptr())


def _stream(stream=None) -> int:
    torch = _torch()
    s = stream if stream is not None else torch.cuda.current_stream()
    return int(s.cuda_stream)


def _wdt(t) -> int:
    torch = _torch()
    if t.dtype == torch.bfloat16:
        return SADMM_BF16
    if t.dtype == torch.float32:
        return SADMM_FP32
    raise TypeError(f"weights must be bf16 or fp32, got {t.dtype}")


def project_groups(desc16: Sequence[int], W, k_filters: int, colkind: int, k_cols: int, U=None,
                   with_keys: bool = False, stream=None, workspace=None):
    """Runs sadmm_project_groups; returns (filt_idx, col_idx, keys or None) as device tensors."""
    torch = _torch()
    desc = make_desc(desc16)
    dev = W.device
    ws_bytes = sadmm_workspace_size(desc, colkind)
    if ws_bytes == 0:
        raise SadmmError(SADMM_EINVAL, "sadmm_workspace_size")
    if workspace is None or workspace.numel() < ws_bytes:
        workspace = torch.empty(ws_bytes, dtype=torch.uint8, device=dev)
    f = int(desc16[5])
    cg = int(desc16[1]) // int(desc16[6])
    taps = int(desc16[7]) * int(desc16[8]) * int(desc16[9])
    G = 0 if colkind == SADMM_COL_NONE else (cg * taps if colkind == SADMM_COL_SHAPE else cg)
    filt_idx = torch.empty(max(k_filters, 1), dtype=torch.int32, device=dev)
    col_idx = torch.empty(max(k_cols, 1), dtype=torch.int32, device=dev) if colkind != SADMM_COL_NONE else None
    keys = torch.empty(f + G, dtype=torch.float64, device=dev) if with_keys else None
    st = sadmm_project_groups(desc, _ptr(W), _ptr(U), _wdt(W), k_filters, colkind, k_cols, _ptr(filt_idx),
                              _ptr(col_idx), _ptr(keys), _ptr(workspace), ws_bytes, _stream(stream))
    _check(st, "sadmm_project_groups")
    fi = filt_idx[:k_filters]
    ci = col_idx[:k_cols] if col_idx is not None else None
    return fi, ci, keys


def project_elements(desc16: Sequence[int], W, k_elems: int, U=None, stream=None):
    """Runs sadmm_project_elements; returns the keep flags as a uint8 device tensor of W's shape."""
    torch = _torch()
    desc = make_desc(desc16)
    ws_bytes = sadmm_elements_workspace_size(desc)
    ws = torch.empty(ws_bytes, dtype=torch.uint8, device=W.device)
    keep = torch.empty(W.shape, dtype=torch.uint8, device=W.device)
    st = sadmm_project_elements(desc, _ptr(W), _ptr(U), _wdt(W), k_elems, _ptr(keep), _ptr(ws), ws_bytes,
                                _stream(stream))
    _check(st, "sadmm_project_elements")
    return keep


def admm_update_elements(desc16: Sequence[int], W, U, Z, k_elems: int, stream=None, workspace=None):
    """Z <- the k_elems largest-magnitude entries of W + U; U <- (W + U) - Z."""
    torch = _torch()
    desc = make_desc(desc16)
    ws_bytes = sadmm_elements_workspace_size(desc)
    if workspace is None or workspace.numel() < ws_bytes:
        workspace = torch.empty(ws_bytes, dtype=torch.uint8, device=W.device)
    st = sadmm_admm_update_elements(desc, _ptr(W), _ptr(U), _ptr(Z), _wdt(W), k_elems, _ptr(workspace), ws_bytes,
                                    _stream(stream))
    _check(st, "sadmm_admm_update_elements")


class ProjectBatch:
    """Repeated sadmm_project_groups_batch calls over fixed layers: the index
    lists, keys and workspaces are allocated once and the item array is built
    once, so a call is one C entry point and nothing else."""

    def __init__(self, layers, with_keys: bool = False):
        """layers: (desc16, W, k_filters, colkind, k_cols, U or None) per layer."""
        torch = _torch()
        items, self.outs, self._keep = [], [], []
        self.wdt = None
        for desc16, W, k_filters, colkind, k_cols, U in layers:
            desc = make_desc(desc16)
            dev = W.device
            self.wdt = _wdt(W) if self.wdt is None else self.wdt
            ws_bytes = sadmm_workspace_size(desc, colkind)
            if ws_bytes == 0:
                raise SadmmError(SADMM_EINVAL, "sadmm_workspace_size")
            ws = torch.empty(ws_bytes, dtype=torch.uint8, device=dev)
            f = int(desc16[5])
            cg = int(desc16[1]) // int(desc16[6])
            taps = int(desc16[7]) * int(desc16[8]) * int(desc16[9])
            G = 0 if colkind == SADMM_COL_NONE else (cg * taps if colkind == SADMM_COL_SHAPE else cg)
            fi = torch.empty(max(k_filters, 1), dtype=torch.int32, device=dev)
            ci = torch.empty(max(k_cols, 1), dtype=torch.int32, device=dev) if colkind != SADMM_COL_NONE else None
            keys = torch.empty(f + G, dtype=torch.float64, device=dev) if with_keys else None
            items.append(ProjectItem(desc, _ptr(W), _ptr(U), int(k_filters), int(colkind), int(k_cols), _ptr(fi),
                                     _ptr(ci), _ptr(keys), _ptr(ws), ws_bytes))
            self._keep += [W, U, ws]
            self.outs.append((fi[:k_filters], ci[:k_cols] if ci is not None else None, keys))
        self.n = len(items)
        self.arr = (ProjectItem * self.n)(*items)

    def __call__(self, stream=None):
        """Projects every layer; returns [(filt_idx, col_idx, keys or None)]."""
        _check(load().sadmm_project_groups_batch(self.arr, self.n, int(self.wdt), _stream(stream)),
               "sadmm_project_groups_batch")
        return self.outs


def project_groups_batch(layers, with_keys: bool = False, stream=None):
    """Runs sadmm_project_groups_batch over layers given as (desc16, W,
    k_filters, colkind, k_cols, U or None); returns [(filt_idx, col_idx, keys
    or None)] per layer, device tensors."""
    torch = _torch()
    items, outs, keep = [], [], []
    wdt = None
    for desc16, W, k_filters, colkind, k_cols, U in layers:
        desc = make_desc(desc16)
        dev = W.device
        wdt = _wdt(W) if wdt is None else wdt
        ws_bytes = sadmm_workspace_size(desc, colkind)
        if ws_bytes == 0:
            raise SadmmError(SADMM_EINVAL, "sadmm_workspace_size")
        ws = torch.empty(ws_bytes, dtype=torch.uint8, device=dev)
        f = int(desc16[5])
        cg = int(desc16[1]) // int(desc16[6])
        taps = int(desc16[7]) * int(desc16[8]) * int(desc16[9])
        G = 0 if colkind == SADMM_COL_NONE else (cg * taps if colkind == SADMM_COL_SHAPE else cg)
        fi = torch.empty(max(k_filters, 1), dtype=torch.int32, device=dev)
        ci = torch.empty(max(k_cols, 1), dtype=torch.int32, device=dev) if colkind != SADMM_COL_NONE else None
        keys = torch.empty(f + G, dtype=torch.float64, device=dev) if with_keys else None
        items.append(ProjectItem(desc, _ptr(W), _ptr(U), int(k_filters), int(colkind), int(k_cols), _ptr(fi),
                                 _ptr(ci), _ptr(keys), _ptr(ws), ws_bytes))
        keep.append(ws)
        outs.append((fi[:k_filters], ci[:k_cols] if ci is not None else None, keys))
    _check(sadmm_project_groups_batch(items, wdt, _stream(stream)), "sadmm_project_groups_batch")
    return outs


class AdmmStep:
    """Device buffers for repeated sadmm_admm_update calls on one layer: the
    kept index lists, the optional keys and the workspace."""

    def __init__(self, desc16: Sequence[int], k_filters: int, colkind: int, k_cols: int, device,
                 with_keys: bool = False):
        torch = _torch()
        self.desc16 = [int(v) for v in desc16]
        self.desc = make_desc(self.desc16)
        self.k_filters, self.colkind, self.k_cols = int(k_filters), int(colkind), int(k_cols)
        self.ws_bytes = sadmm_admm_workspace_size(self.desc, colkind)
        if self.ws_bytes == 0:
            raise SadmmError(SADMM_EINVAL, "sadmm_admm_workspace_size")
        self.workspace = torch.empty(self.ws_bytes, dtype=torch.uint8, device=device)
        f = self.desc16[5]
        cg = self.desc16[1] // self.desc16[6]
        taps = self.desc16[7] * self.desc16[8] * self.desc16[9]
        G = 0 if colkind == SADMM_COL_NONE else (cg * taps if colkind == SADMM_COL_SHAPE else cg)
        self.filt_idx = torch.empty(max(k_filters, 1), dtype=torch.int32, device=device)
        self.col_idx = (torch.empty(max(k_cols, 1), dtype=torch.int32, device=device)
                        if colkind != SADMM_COL_NONE else None)
        self.keys = torch.empty(f + G, dtype=torch.float64, device=device) if with_keys else None

    def __call__(self, W, U, Z, stream=None):
        """Z <- Proj_S(W + U); U <- (W + U) - Z.  Returns (filt_idx, col_idx)."""
        st = sadmm_admm_update(self.desc, _ptr(W), _ptr(U), _ptr(Z), _wdt(W), self.k_filters, self.colkind,
                               self.k_cols, _ptr(self.filt_idx), _ptr(self.col_idx), _ptr(self.keys),
                               _ptr(self.workspace), self.ws_bytes, _stream(stream))
        _check(st, "sadmm_admm_update")
        ci = self.col_idx[:self.k_cols] if self.col_idx is not None else None
        return self.filt_idx[:self.k_filters], ci


class AdmmBatch:
    """Repeated sadmm_admm_update_batch calls over a list of layers: one
    AdmmStep's buffers per layer, one call for all of them."""

    def __init__(self, layers, device, with_keys: bool = False):
        """layers: (desc16, k_filters, colkind, k_cols) per layer."""
        self.steps = [AdmmStep(d, kf, ck, kc, device, with_keys=with_keys) for d, kf, ck, kc in layers]

    def __call__(self, Ws, Us, Zs, stream=None):
        """Z_l <- Proj_S(W_l + U_l); U_l <- (W_l + U_l) - Z_l for every layer.
        Returns [(filt_idx, col_idx)] per layer.  The item array is built once
        per set of tensor addresses."""
        key = tuple(_ptr(t) for t in list(Ws) + list(Us) + list(Zs))
        if getattr(self, "_key", None) != key:
            items = []
            for st, W, U, Z in zip(self.steps, Ws, Us, Zs):
                items.append(AdmmItem(st.desc, _ptr(W), _ptr(U), _ptr(Z), st.k_filters, st.colkind, st.k_cols,
                                      _ptr(st.filt_idx), _ptr(st.col_idx), _ptr(st.keys), _ptr(st.workspace),
                                      st.ws_bytes))
            self._arr = (AdmmItem * len(items))(*items)
            self._wdt = _wdt(Ws[0])
            self._key = key
        _check(load().sadmm_admm_update_batch(self._arr, len(self.steps), int(self._wdt), _stream(stream)),
               "sadmm_admm_update_batch")
        out = []
        for st in self.steps:
            ci = st.col_idx[:st.k_cols] if st.col_idx is not None else None
            out.append((st.filt_idx[:st.k_filters], ci))
        return out


class PrunedConv:
    """A packed pruned layer: plan plus its device buffer (sadmm_plan_init + sadmm_pack)."""

    def __init__(self, desc16: Sequence[int], W, filt_idx, colkind: int, col_idx, n_filt: int,
                 n_colgroups: int, stream=None, max_ctas: int = 0):
        torch = _torch()
        self.desc16 = [int(v) for v in desc16]
        desc = make_desc(self.desc16)
        st, plan = sadmm_plan_init_ctas(desc, n_filt, colkind, n_colgroups, max_ctas)
        _check(st, "sadmm_plan_init_ctas")
        self.plan = plan
        self.buf = torch.empty(plan.dev_bytes, dtype=torch.uint8, device=W.device)
        self.W = W
        self.repack(W, filt_idx, col_idx, stream)

    def repack(self, W, filt_idx, col_idx, stream=None):
        st = sadmm_pack(self.plan, _ptr(W), _wdt(W), _ptr(filt_idx), _ptr(col_idx), _ptr(self.buf),
                        self.plan.dev_bytes, _stream(stream))
        _check(st, "sadmm_pack")

    def backward(self, x, dy, y=None, relu=True, want_dw=True, want_db=True, want_dx=True, stream=None,
                 chunk_pixels=0):
        """Runs sadmm_conv_bwd; returns (dW, db, dx) fp32 device tensors (None where not requested).
        chunk_pixels > 0 sizes the workspace for chunks of that many output pixels
        (default: chunks of up to 32768 pixels)."""
        torch = _torch()
        n, c, t, h, w, f, g, kt, kh, kw = self.desc16[:10]
        dev = dy.device
        dW = torch.empty((f, (c // g) * kt * kh * kw), dtype=torch.float32, device=dev) if want_dw else None
        db = torch.empty(f, dtype=torch.float32, device=dev) if want_db else None
        dx = torch.empty(x.shape, dtype=torch.float32, device=dev) if want_dx else None
        ws_bytes = (sadmm_conv_bwd_workspace_size_chunk(self.plan, chunk_pixels) if chunk_pixels > 0
                    else sadmm_conv_bwd_workspace_size(self.plan))
        ws = torch.empty(ws_bytes + 1024, dtype=torch.uint8, device=dev)
        wptr = (_ptr(ws) + 1023) // 1024 * 1024
        ydt = SADMM_BF16 if (y is not None and y.dtype == torch.bfloat16) else SADMM_FP32
        st = sadmm_conv_bwd(self.plan, _ptr(x), _ptr(dy), _ptr(y), ydt, 1 if relu else 0, _ptr(dW), _ptr(db),
                            _ptr(dx), wptr, ws_bytes, _stream(stream))
        _check(st, "sadmm_conv_bwd")
        return dW, db, dx

    def out_shape(self):
        n, c, t, h, w, f, g, kt, kh, kw, st_, sh, sw, pt, ph, pw = self.desc16
        ot = (t + 2 * pt - kt) // st_ + 1
        oh = (h + 2 * ph - kh) // sh + 1
        ow = (w + 2 * pw - kw) // sw + 1
        if t == 1 and kt == 1:
            return (n, f, oh, ow)
        return (n, f, ot, oh, ow)

    def forward(self, x, bias=None, relu: bool = True, out_dtype=None, out=None, stream=None):
        torch = _torch()
        if x.dtype != torch.bfloat16 or not x.is_contiguous():
            raise TypeError("x must be a contiguous bf16 tensor")
        if out is None:
            out_dtype = out_dtype or torch.float32
            out = torch.empty(self.out_shape(), dtype=out_dtype, device=x.device)
        ydt = SADMM_BF16 if out.dtype == torch.bfloat16 else SADMM_FP32
        if bias is not None and (bias.dtype != torch.float32 or not bias.is_contiguous()):
            raise TypeError("bias must be a contiguous fp32 tensor")
        st = sadmm_conv_fwd(self.plan, _ptr(x), _ptr(bias), 1 if relu else 0, _ptr(out), ydt, _stream(stream))
        _check(st, "sadmm_conv_fwd")
        return out


def pack_batch(convs, stream=None) -> None:
    """Repacks PrunedConv layers with one sadmm_pack_batch call: convs is a
    sequence of (PrunedConv, W, filt_idx or None, col_idx or None), every W of
    one dtype."""
    items = [PackItem(ctypes.pointer(pc.plan), _ptr(W), _ptr(fi), _ptr(ci), _ptr(pc.buf), pc.plan.dev_bytes)
             for pc, W, fi, ci in convs]
    _check(sadmm_pack_batch(items, _wdt(convs[0][1]), _stream(stream)), "sadmm_pack_batch")


def device_status(stream=None) -> int:
    """Synchronises the stream and returns (and clears) the device status word."""
    return sadmm_last_device_status(_stream(stream))
