"""Host check of the input-slab decomposition (no GPU): with the plan's slab
geometry (xs_r, xs_q, xs_cs, xs_hb, xs_wb, xs_sp as sadmm_plan_init sets them),
the space-to-depth rewrite of x and the GEMM of 128-row tiles against shifted
slabs, written out in numpy as the header defines them, reproduce the oracle's
pruned convolution exactly (same fp64 sums, another order), for strided,
padded, rectangular and channel-pruned layers; and rows past the output read
only the zeroed padding or real block pixels (never past the tile's slab)."""
import numpy as np
import pytest

import oracle
import workloads as wl
from workloads import ConvShape


def slab_forward(s, t, rows, colkind, cols, p):
    x = t["x"].double().numpy()
    W = t["W"].double().numpy().reshape(s.f, -1)
    b = t["bias"].double().numpy()
    C, H, Wd = s.c, s.h, s.w
    nck = len(cols) if colkind == wl.COL_CHANNEL else C
    chan = [int(c) for c in cols] if colkind == wl.COL_CHANNEL else list(range(C))
    cs, R, Q, Hb, Wb, sp = p.xs_cs, p.xs_r, p.xs_q, p.xs_hb, p.xs_wb, p.xs_sp
    OH = (s.h + 2 * s.ph - s.kh) // s.sh + 1
    OW = (s.w + 2 * s.pw - s.kw) // s.sw + 1
    assert Hb == OH + R - 1 and Wb == OW + Q - 1 and sp >= 128 + (R - 1) * Wb + Q - 1
    # space-to-depth input, zero padding pixels up to pimg (and beyond: the TMA's zero fill)
    xs = np.zeros((s.n, cs, p.xs_pimg + sp), np.float64)
    for cc in range(nck * s.sh * s.sw):
        ci, a, bb = cc // (s.sh * s.sw), (cc // s.sw) % s.sh, cc % s.sw
        for hb in range(Hb):
            ih = hb * s.sh + a - s.ph
            if not 0 <= ih < H:
                continue
            iw = np.arange(Wb) * s.sw + bb - s.pw
            ok = (iw >= 0) & (iw < Wd)
            xs[:, cc, hb * Wb + np.nonzero(ok)[0]] = x[:, chan[ci], ih, iw[ok]]
    # slab-ordered weights: column (tap, cc) -> GEMM column, zero past the kernel
    Ws = np.zeros((len(rows), R * Q * cs))
    for tap in range(R * Q):
        r, q = divmod(tap, Q)
        for cc in range(nck * s.sh * s.sw):
            ci, a, bb = cc // (s.sh * s.sw), (cc // s.sw) % s.sh, cc % s.sw
            kh, kw = r * s.sh + a, q * s.sw + bb
            if kh < s.kh and kw < s.kw:
                Ws[:, tap * cs + cc] = W[rows, chan[ci] * s.taps + kh * s.kw + kw]
    y = np.zeros((s.n, s.f, OH, OW))
    mt = -(-(OH * Wb) // 128)
    for n in range(s.n):
        for t_ in range(mt):
            slab = xs[n, :, t_ * 128:t_ * 128 + sp]          # [cs][sp]: the tile's one slab
            acc = np.zeros((128, len(rows)))
            for tap in range(R * Q):
                r, q = divmod(tap, Q)
                shift = r * Wb + q
                assert shift + 128 <= sp
                acc += slab[:, shift:shift + 128].T @ Ws[:, tap * cs:(tap + 1) * cs].T
            for i in range(128):
                pix = t_ * 128 + i
                oh, ow = divmod(pix, Wb)
                if oh < OH and ow < OW:
                    y[n, rows, oh, ow] = np.maximum(acc[i] + b[rows], 0.0)
    return y


CASES = [
    ("stride4_11x11", ConvShape(n=2, c=3, h=35, w=35, f=16, kh=11, kw=11, sh=4, sw=4), 0.75, wl.COL_NONE, 1.0),
    ("stem_7x7_s2_p3", ConvShape(n=1, c=3, h=21, w=19, f=8, kh=7, kw=7, sh=2, sw=2, ph=3, pw=3), 1.0, wl.COL_NONE,
     1.0),
    ("rect_stride_kernel", ConvShape(n=2, c=6, h=13, w=10, f=12, kh=3, kw=2, sh=2, sw=1, ph=1, pw=0), 0.75,
     wl.COL_NONE, 1.0),
    ("channel_3x3", ConvShape(n=1, c=24, h=9, w=9, f=10, kh=3, kw=3, ph=1, pw=1), 0.5, wl.COL_CHANNEL, 0.5),
]


@pytest.mark.parametrize("case", CASES, ids=lambda c: c[0])
def test_slab_decomposition_reproduces_the_oracle(case):
    from paper_1807_11091_gb300 import sadmm
    name, s, ff, ck, cf = case
    G = s.cg if ck == wl.COL_CHANNEL else s.k
    kf, kc = wl.retained(ff, s.f), (wl.retained(cf, G) if ck != wl.COL_NONE else 0)
    st, p = sadmm.sadmm_plan_init(sadmm.make_desc(s.desc16()), kf, ck, kc if ck != wl.COL_NONE else s.k)
    assert st == 0 and p.xs_mode == 1, name
    t = wl.gen_tensors(s, seed=41)
    rows, cols, _, _ = oracle.project(t["W"], s.taps, kf, ck, kc)
    ref = oracle.pruned_conv(t["x"], t["W"], t["bias"], s.desc16(), s.taps, rows, ck, cols, relu=True)
    got = slab_forward(s, t, np.asarray(rows), ck, np.asarray(cols), p)
    assert np.abs(got - ref).max() <= 1e-12 * max(np.abs(ref).max(), 1.0), name
