"""GPU checks of sadmm_pack: the packed matrix is the exact bf16 copy of the kept
rows and columns, and the per-group filter lists and gather table are the ones
the index lists fix (compared bit-exactly)."""
import numpy as np
import pytest
import torch

import oracle
import workloads as wl
from workloads import ConvShape

pytestmark = pytest.mark.gpu


def _pack(shape, W, fi, ck, ci, k_filters, n_cg):
    from paper_1807_11091_gb300 import sadmm
    dev = torch.device("cuda", 0)
    fi_d = torch.as_tensor(np.asarray(fi, np.int32), device=dev) if k_filters < shape.f else None
    ci_d = torch.as_tensor(np.asarray(ci, np.int32), device=dev) if ck != wl.COL_NONE else None
    pc = sadmm.PrunedConv(shape.desc16(), W.to(dev), fi_d, ck, ci_d, k_filters, n_cg)
    torch.cuda.synchronize()
    return pc


def _view(pc, off, nbytes, dtype):
    return pc.buf[off:off + nbytes].view(dtype).cpu()


CASES = [
    (ConvShape(n=1, c=8, h=6, w=6, f=12, kh=3, kw=3, ph=1, pw=1, groups=2), 5, wl.COL_SHAPE, 30),
    (ConvShape(n=1, c=16, h=6, w=6, f=300, kh=3, kw=3, ph=1, pw=1), 300, wl.COL_SHAPE, 100),
    (ConvShape(n=1, c=6, t=4, h=5, w=5, f=40, kt=3, kh=3, kw=3, pt=1, ph=1, pw=1), 17, wl.COL_CHANNEL, 4),
    (ConvShape(n=1, c=3, h=30, w=30, f=96, kh=11, kw=11, sh=4, sw=4), 60, wl.COL_SHAPE, 200),
    (ConvShape(n=1, c=12, h=5, w=5, f=20, kh=1, kw=1, groups=4), 9, wl.COL_NONE, 0),
]


@pytest.mark.parametrize("case", CASES, ids=lambda c: f"{c[0].w_shape()}-g{c[0].groups}-ck{c[2]}")
@pytest.mark.parametrize("wdtype", [torch.bfloat16, torch.float32])
def test_pack_matches_index_lists(case, wdtype):
    s, kf, ck, kc = case
    t = wl.gen_tensors(s, seed=13)
    W = t["W"].to(torch.float32) * 1.3 if wdtype == torch.float32 else t["W"]
    rows, cols, _, _ = oracle.project(W.float(), s.taps, kf, ck, kc)
    n_cg = s.k if ck == wl.COL_NONE else kc
    pc = _pack(s, W, rows, ck, cols, kf, n_cg)
    p = pc.plan
    G, n_pad, k_pad = s.groups, p.n_pad, p.k_pad
    kcols = oracle.expand_columns(ck, cols, s.taps, s.k)
    assert p.n_cols == len(kcols)
    wp = _view(pc, p.off_wp, G * n_pad * k_pad * 2, torch.bfloat16).reshape(G, n_pad, k_pad)
    Wb = W.reshape(s.f, -1).to(torch.bfloat16)
    expect = torch.zeros_like(wp)
    counts = _view(pc, p.off_counts, G * 8, torch.int32).numpy().reshape(G, 2)
    rowmap = _view(pc, p.off_rowmap, G * n_pad * 4, torch.int32).numpy().reshape(G, n_pad)
    zeromap = _view(pc, p.off_zeromap, s.f * 4, torch.int32).numpy().reshape(G, s.fg)
    for g in range(G):
        kept = [int(f) for f in rows if g * s.fg <= f < (g + 1) * s.fg]
        pruned = [f for f in range(g * s.fg, (g + 1) * s.fg) if f not in kept]
        assert counts[g].tolist() == [len(kept), len(pruned)]
        assert rowmap[g, :len(kept)].tolist() == kept
        assert np.all(rowmap[g, len(kept):] == -1)
        assert zeromap[g, :len(pruned)].tolist() == pruned
        for i, f in enumerate(kept):
            expect[g, i, :len(kcols)] = Wb[f, torch.as_tensor(kcols)]
    assert torch.equal(wp.view(torch.int16), expect.view(torch.int16)), "packed weights differ"
    gt = _view(pc, p.off_gather, k_pad * 8, torch.int32).numpy().reshape(k_pad, 2).view(np.uint32)
    for j in range(k_pad):
        if j >= len(kcols):
            assert int(gt[j, 1]) == 1 << 31
            continue
        col = int(kcols[j])
        c, r = divmod(col, s.taps)
        kt, rem = divmod(r, s.kh * s.kw)
        kh, kw = divmod(rem, s.kw)
        assert gt[j, 0] == c * s.t * s.h * s.w + kt * s.h * s.w + kh * s.w + kw
        if s.taps <= 31:
            assert int(gt[j, 1]) == (1 << r)
        else:
            assert int(gt[j, 1]) == (1 << (kt * s.kh + kh)) | (1 << (16 + kw))
