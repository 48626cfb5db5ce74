"""The C ABI without a GPU: the library builds for sm_103a, loads, exports every
entry point include/*.h declares, and rejects bad arguments on the host before
any launch."""
import ctypes
import glob
import os
import re

import pytest

from paper_1807_11091_gb300 import sadmm
import workloads as wl

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared():
    names = set()
    for h in glob.glob(os.path.join(ROOT, "include", "*.h")):
        text = open(h).read()
        text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
        for m in re.finditer(r"\b(sadmm_[a-z0-9_]+)\s*\(", text):
            names.add(m.group(1))
    return sorted(names)


def test_library_exports_every_declared_entry_point():
    lib = sadmm.load()
    names = _declared()
    assert {"sadmm_project_groups", "sadmm_pack", "sadmm_conv_fwd"} <= set(names)
    for n in names:
        assert hasattr(lib, n), f"{n} not exported"


def test_struct_layout_and_version():
    assert sadmm.sadmm_abi_version() == 6
    assert sadmm.sadmm_plan_struct_size() == ctypes.sizeof(sadmm.Plan)
    assert sadmm.sadmm_status_string(-1) == "invalid argument"


def test_plan_sizes():
    L = wl.alexnet()[3]  # conv4: groups 2, 77 filters, 346 columns
    st, p = sadmm.sadmm_plan_init(sadmm.make_desc(L.shape.desc16()), L.k_filters, wl.COL_SHAPE, L.k_cols)
    assert st == 0
    assert p.n_cols == 346 and p.k_pad == 384
    assert p.bn % 16 == 0 and p.bn <= 256 and p.n_pad == p.bn * p.n_tiles >= 77
    assert p.dev_bytes >= 2 * p.n_pad * p.k_pad * 2
    # channel-wise expands to taps columns per channel
    st, p = sadmm.sadmm_plan_init(sadmm.make_desc(L.shape.desc16()), 10, wl.COL_CHANNEL, 7)
    assert st == 0 and p.n_cols == 7 * 9
    # more than 256 kept rows per group -> several filter tiles
    s = wl.sweep()[0].shape
    st, p = sadmm.sadmm_plan_init(sadmm.make_desc(s.desc16()), 512, wl.COL_SHAPE, 2304)
    assert st == 0 and p.n_tiles == 2 and p.bn == 256 and p.k_pad == 2304


@pytest.mark.parametrize("field,value", [("n", 0), ("groups", 3), ("kh", 40), ("st", 0), ("ph", -1)])
def test_bad_descriptors_rejected(field, value):
    d = wl.single2d()[0].shape.desc16()
    d[sadmm.DESC_FIELDS.index(field)] = value
    st, _ = sadmm.sadmm_plan_init(sadmm.make_desc(d), 10, wl.COL_SHAPE, 10)
    assert st in (sadmm.SADMM_EINVAL, sadmm.SADMM_EUNSUPPORTED)


def test_bad_counts_rejected_on_host():
    s = wl.single2d()[0].shape
    d = sadmm.make_desc(s.desc16())
    assert sadmm.sadmm_plan_init(d, s.f + 1, wl.COL_SHAPE, 1)[0] == sadmm.SADMM_EINVAL
    assert sadmm.sadmm_plan_init(d, 1, wl.COL_SHAPE, s.k + 1)[0] == sadmm.SADMM_EINVAL
    assert sadmm.sadmm_plan_init(d, 1, wl.COL_CHANNEL, s.cg + 1)[0] == sadmm.SADMM_EINVAL
    assert sadmm.sadmm_plan_init(d, 1, 7, 1)[0] == sadmm.SADMM_EINVAL
    ws = sadmm.sadmm_workspace_size(d, wl.COL_SHAPE)
    assert ws > 0
    fake = 1 << 20  # never dereferenced: validation fails first
    args = dict(W=fake, U=None, wdt=0, k_filters=1, colkind=wl.COL_SHAPE, k_cols=1, filt_idx=fake,
                col_idx=fake, keys_out=None, workspace=fake, ws_bytes=ws, stream=None)
    for bad in (dict(k_filters=-1), dict(k_filters=s.f + 1), dict(k_cols=s.k + 1), dict(wdt=5),
                dict(ws_bytes=ws - 1), dict(W=None), dict(col_idx=None), dict(colkind=9)):
        a = dict(args, **bad)
        assert sadmm.sadmm_project_groups(d, **a) == sadmm.SADMM_EINVAL, bad


def test_conv_rejects_unbound_plan_and_nulls():
    s = wl.single2d()[0].shape
    st, p = sadmm.sadmm_plan_init(sadmm.make_desc(s.desc16()), s.f, wl.COL_SHAPE, 100)
    assert st == 0
    fake = 1 << 20
    # plan never packed: no device buffer
    assert sadmm.sadmm_conv_fwd(p, fake, None, 1, fake, 1, None) == sadmm.SADMM_EINVAL
    p.dev = fake
    assert sadmm.sadmm_conv_fwd(p, None, None, 1, fake, 1, None) == sadmm.SADMM_EINVAL
    assert sadmm.sadmm_conv_fwd(p, fake, None, 1, None, 1, None) == sadmm.SADMM_EINVAL
    assert sadmm.sadmm_conv_fwd(p, fake + 1, None, 1, fake, 1, None) == sadmm.SADMM_EINVAL
    assert sadmm.sadmm_conv_fwd(p, fake, None, 1, fake, 7, None) == sadmm.SADMM_EINVAL
    assert sadmm.sadmm_pack(p, fake, 0, None, fake, fake, p.dev_bytes - 1, None) == sadmm.SADMM_EINVAL
    assert sadmm.sadmm_pack(p, fake, 0, None, fake, fake + 8, p.dev_bytes, None) == sadmm.SADMM_EINVAL


def test_admm_update_rejects_bad_arguments_on_host():
    s = wl.single2d()[0].shape
    d = sadmm.make_desc(s.desc16())
    ws = sadmm.sadmm_admm_workspace_size(d, wl.COL_SHAPE)
    assert ws >= sadmm.sadmm_workspace_size(d, wl.COL_SHAPE) + s.f + s.k
    nbytes = s.f * s.k * 4
    W, U, Z, ws_ptr = 1 << 24, (1 << 24) + (1 << 22), (1 << 24) + (2 << 22), 1 << 30  # never dereferenced
    args = dict(W=W, U=U, Z=Z, wdt=sadmm.SADMM_FP32, k_filters=1, colkind=wl.COL_SHAPE, k_cols=1, filt_idx=W,
                col_idx=W, keys_out=None, workspace=ws_ptr, ws_bytes=ws, stream=None)
    for bad in (dict(U=None), dict(Z=None), dict(W=None), dict(workspace=None), dict(ws_bytes=ws - 1),
                dict(workspace=ws_ptr + 16), dict(k_filters=s.f + 1), dict(k_cols=s.k + 1), dict(wdt=4),
                dict(colkind=5), dict(Z=U), dict(Z=U + nbytes - 4), dict(U=W + 4), dict(W=W + 2),
                dict(keys_out=ws_ptr + 4)):
        a = dict(args, **bad)
        assert sadmm.sadmm_admm_update(d, **a) == sadmm.SADMM_EINVAL, bad


def test_elements_reject_bad_arguments_on_host():
    s = wl.single2d()[0].shape
    d = sadmm.make_desc(s.desc16())
    ws = sadmm.sadmm_elements_workspace_size(d)
    assert ws >= 2048 * 4
    fake, ws_ptr = 1 << 24, 1 << 30
    N = s.f * s.k
    args = dict(W=fake, U=None, wdt=sadmm.SADMM_BF16, k_elems=10, keep_out=fake, workspace=ws_ptr, ws_bytes=ws,
                stream=None)
    for bad in (dict(W=None), dict(keep_out=None), dict(k_elems=-1), dict(k_elems=N + 1), dict(wdt=3),
                dict(ws_bytes=ws - 1), dict(workspace=ws_ptr + 8), dict(W=fake + 1)):
        assert sadmm.sadmm_project_elements(d, **dict(args, **bad)) == sadmm.SADMM_EINVAL, bad
    Z = fake + (1 << 22)
    assert sadmm.sadmm_admm_update_elements(d, fake, fake, Z, sadmm.SADMM_FP32, 5, ws_ptr, ws, None) == sadmm.SADMM_EINVAL
    assert sadmm.sadmm_admm_update_elements(d, fake, None, Z, sadmm.SADMM_FP32, 5, ws_ptr, ws, None) == sadmm.SADMM_EINVAL


def test_plan_cta_cap_on_host():
    """sadmm_plan_init_ctas records the cap, ignores 0 and caps above the SM
    count, rejects a negative cap, and sizes split-K for the capped count."""
    L = wl.alexnet()[2]
    d = sadmm.make_desc(L.shape.with_batch(1).desc16())
    st, full = sadmm.sadmm_plan_init(d, L.k_filters, L.colkind, L.k_cols)
    assert st == 0 and full.ctas >= 1
    st, same = sadmm.sadmm_plan_init_ctas(d, L.k_filters, L.colkind, L.k_cols, 0)
    assert st == 0 and same.ctas == full.ctas and same.dev_bytes == full.dev_bytes
    st, big = sadmm.sadmm_plan_init_ctas(d, L.k_filters, L.colkind, L.k_cols, 1 << 20)
    assert st == 0 and big.ctas == full.ctas
    st, capped = sadmm.sadmm_plan_init_ctas(d, L.k_filters, L.colkind, L.k_cols, 1)
    assert st == 0 and capped.ctas == 1 and capped.splits == 1 and capped.sk_len == 0
    st, _ = sadmm.sadmm_plan_init_ctas(d, L.k_filters, L.colkind, L.k_cols, -1)
    assert st == sadmm.SADMM_EINVAL


def test_slab_plan_rule_host():
    """The plan takes the input-slab path for AlexNet CONV1 (kept whole) with the
    space-to-depth geometry of a stride-4 11x11 kernel over 3 channels, and
    declines it for shape-wise pruned columns, two conv groups, more than 64
    slab channels, a slab GEMM over twice as wide as K', more than 256 kept
    filters and a single block tap (1 x 1, or 2 x 2 at stride 2)."""
    from workloads import ConvShape
    L = wl.alexnet()[0]
    st, p = sadmm.sadmm_plan_init(sadmm.make_desc(L.shape.desc16()), L.k_filters, wl.COL_SHAPE, L.k_cols)
    assert st == 0 and p.xs_mode == 1
    # 3 channels x 4 x 4 phases = 48 slab channels; ceil(11/4) = 3 block taps;
    # 55 + 3 - 1 = 57 block rows and columns; 128 + 2*57 + 2 = 244 -> 248 slab pixels
    assert (p.xs_cs, p.xs_r, p.xs_q, p.xs_hb, p.xs_wb, p.xs_sp) == (48, 3, 3, 57, 57, 248)
    assert p.xs_pimg == 3256 and p.xs_kpad == 448 and p.splits == 1 and p.sk_len == 0
    assert p.off_xs + 128 * 6 * 3256 * 16 <= p.dev_bytes
    declined = [
        (ConvShape(n=1, c=3, h=35, w=35, f=16, kh=11, kw=11, sh=4, sw=4), wl.COL_SHAPE, 300),
        (ConvShape(n=1, c=8, h=9, w=9, f=16, kh=3, kw=3, ph=1, pw=1, groups=2), wl.COL_NONE, 0),
        (ConvShape(n=1, c=5, h=35, w=35, f=16, kh=11, kw=11, sh=4, sw=4), wl.COL_NONE, 0),
        (ConvShape(n=1, c=3, h=9, w=9, f=16, kh=3, kw=3, ph=1, pw=1), wl.COL_NONE, 0),
        (ConvShape(n=1, c=3, h=9, w=9, f=300, kh=3, kw=3, sh=2, sw=2), wl.COL_NONE, 0),
        (ConvShape(n=1, c=32, h=8, w=8, f=48, kh=1, kw=1), wl.COL_CHANNEL, 16),
        (ConvShape(n=1, c=4, h=8, w=8, f=48, kh=2, kw=2, sh=2, sw=2), wl.COL_NONE, 0),
    ]
    for s, ck, kc in declined:
        st, p = sadmm.sadmm_plan_init(sadmm.make_desc(s.desc16()), s.f, ck, s.k if ck == wl.COL_NONE else kc)
        assert st == 0 and p.xs_mode == 0, s


def test_conv_fwd_phase_argument_checks_host():
    """sadmm_conv_fwd_phase rejects on the host, before any device call: an
    unknown phase, the rest of a gathered plan without x (it reads x itself),
    and the input phase without x.  (The plan's buffer pointer is set to a
    dummy: nothing is enqueued.)"""
    import ctypes
    from workloads import ConvShape
    s = ConvShape(n=1, c=8, h=9, w=9, f=16, kh=3, kw=3, ph=1, pw=1)
    st, p = sadmm.sadmm_plan_init(sadmm.make_desc(s.desc16()), s.f, wl.COL_SHAPE, 36)
    assert st == 0 and p.xs_mode == 0
    p.dev = ctypes.c_void_p(1 << 20)
    y = 1 << 21
    assert sadmm.sadmm_conv_fwd_phase(p, 1 << 22, None, 1, y, sadmm.SADMM_FP32, 7, None) == sadmm.SADMM_EINVAL
    assert sadmm.sadmm_conv_fwd_phase(p, None, None, 1, y, sadmm.SADMM_FP32, sadmm.SADMM_FWD_REST,
                                      None) == sadmm.SADMM_EINVAL
    assert sadmm.sadmm_conv_fwd_phase(p, None, None, 1, None, sadmm.SADMM_FP32, sadmm.SADMM_FWD_INPUT,
                                      None) == sadmm.SADMM_EINVAL
    assert sadmm.sadmm_conv_fwd_phase(p, 1 << 22, None, 1, None, sadmm.SADMM_FP32, sadmm.SADMM_FWD_ALL,
                                      None) == sadmm.SADMM_EINVAL


def test_noalloc_array_size_matches_header():
    """The binding's copy of SADMM_NOALLOC_SCRATCH_BYTES equals the header's #define."""
    import re
    with open(os.path.join(ROOT, "include", "sadmm.h")) as fh:
        m = re.search(r"#define\s+SADMM_NOALLOC_SCRATCH_BYTES\s+\(([^)]*)\)", fh.read())
    assert m, "define not found"
    assert eval(m.group(1), {"__builtins__": {}}) == sadmm.SADMM_NOALLOC_SCRATCH_BYTES


def test_noalloc_size_rule_host():
    """The fit rule the header states (round_up(F, 32) + round_up(K, 32) <= 16352)
    is exactly where the projection's workspace reaches the fixed array."""
    limit = sadmm.SADMM_NOALLOC_SCRATCH_BYTES
    r32 = lambda v: (v + 31) // 32 * 32
    for f, c in ((192, 16160), (193, 16160), (16320, 32), (16321, 32), (16384, 1), (1, 16352), (64, 16288)):
        desc = sadmm.make_desc([1, c, 1, 1, 1, f, 1, 1, 1, 1, 1, 1, 1, 0, 0, 0])
        for ck in (0, 1, 2):
            fits = sadmm.sadmm_workspace_size(desc, ck) <= limit
            assert fits == (r32(f) + r32(c) <= 16352), (f, c, ck)


def test_selftest_wait_rejects_bad_arguments_on_host():
    assert sadmm.sadmm_selftest_wait(0, 0, None, None) == sadmm.SADMM_EINVAL
    assert sadmm.sadmm_selftest_wait(1000001, 0, None, None) == sadmm.SADMM_EINVAL
    assert sadmm.sadmm_selftest_wait(1000, 0, (1 << 20) + 2, None) == sadmm.SADMM_EINVAL


def test_sparse_entry_points_reject_bad_arguments_on_host():
    desc = sadmm.make_desc([1, 4, 1, 6, 6, 8, 1, 1, 3, 3, 1, 1, 1, 0, 1, 1])
    full = 8 * 36
    assert sadmm.sadmm_sparse_plan_size(desc, full) == 256 + full * 16
    assert sadmm.sadmm_sparse_plan_size(desc, full + 1) == 0
    assert sadmm.sadmm_sparse_plan_size(desc, -1) == 0
    fake = 1 << 20
    nb = sadmm.sadmm_sparse_plan_size(desc, 10)
    assert sadmm.sadmm_sparse_pack(desc, fake, sadmm.SADMM_BF16, fake, 10, fake, nb - 1, None) == sadmm.SADMM_EINVAL
    assert sadmm.sadmm_sparse_pack(desc, fake, sadmm.SADMM_BF16, fake, 10, fake + 16, nb, None) == sadmm.SADMM_EINVAL
    assert sadmm.sadmm_sparse_pack(desc, fake, 7, fake, 10, fake, nb, None) == sadmm.SADMM_EINVAL
    assert sadmm.sadmm_sparse_pack(desc, None, sadmm.SADMM_BF16, fake, 10, fake, nb, None) == sadmm.SADMM_EINVAL
    assert sadmm.sadmm_sparse_conv_fwd(desc, fake, fake, None, 1, fake, 9, None) == sadmm.SADMM_EINVAL
    assert sadmm.sadmm_sparse_conv_fwd(desc, fake + 16, fake, None, 1, fake, 1, None) == sadmm.SADMM_EINVAL
    assert sadmm.sadmm_sparse_conv_fwd(desc, fake, fake, None, 1, fake + 2, 1, None) == sadmm.SADMM_EINVAL


def test_pack_batch_rejects_bad_items_on_host():
    s = wl.single2d()[0].shape
    st, p = sadmm.sadmm_plan_init(sadmm.make_desc(s.desc16()), s.f, wl.COL_SHAPE, 100)
    assert st == 0
    st, q = sadmm.sadmm_plan_init(sadmm.make_desc(s.desc16()), s.f, wl.COL_SHAPE, 100)
    fake = 1 << 20

    def item(plan, W=fake, col=fake, dev=fake, nbytes=None):
        return sadmm.PackItem(ctypes.pointer(plan), W, None, col, dev, plan.dev_bytes if nbytes is None else nbytes)

    assert sadmm.sadmm_pack_batch([], 0, None) == sadmm.SADMM_EINVAL
    assert sadmm.sadmm_pack_batch([item(p)], 7, None) == sadmm.SADMM_EINVAL  # no such weight type
    assert sadmm.sadmm_pack_batch([item(p), item(p)], 0, None) == sadmm.SADMM_EINVAL  # one plan twice
    assert sadmm.sadmm_pack_batch([item(p), item(q, W=None)], 0, None) == sadmm.SADMM_EINVAL
    assert sadmm.sadmm_pack_batch([item(p), item(q, col=None)], 0, None) == sadmm.SADMM_EINVAL
    assert sadmm.sadmm_pack_batch([item(p), item(q, dev=fake + 8)], 0, None) == sadmm.SADMM_EINVAL
    assert sadmm.sadmm_pack_batch([item(p), item(q, nbytes=q.dev_bytes - 1)], 0, None) == sadmm.SADMM_EINVAL
    plans = [sadmm.sadmm_plan_init(sadmm.make_desc(s.desc16()), s.f, wl.COL_SHAPE, 100)[1]
             for _ in range(sadmm.SADMM_MAX_BATCH + 1)]
    assert sadmm.sadmm_pack_batch([item(pl) for pl in plans], 0, None) == sadmm.SADMM_EINVAL
    # nothing was bound: every rejected call enqueues nothing
    assert not p.dev and not q.dev
