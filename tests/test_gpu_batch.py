"""GPU checks of the batched projection and ADMM update: sadmm_project_groups_batch
and sadmm_admm_update_batch over a list of layers give, bit for bit, what one
call per layer gives (index lists, keys, Z and U), for batches that mix layer
shapes, column kinds, kinds kept whole and requested keys.  The per-layer calls
are themselves checked against the oracle in test_gpu_project.py and
test_gpu_admm.py; the batched ADMM update is also checked against the oracle
directly on AlexNet CONV1-5."""
import numpy as np
import pytest
import torch

import oracle
import workloads as wl

pytestmark = pytest.mark.gpu


def _layers(name):
    if name == "alexnet":
        return wl.alexnet()
    if name == "resnet50":
        return wl.resnet50()
    # a mix: shape-wise, channel-wise, filters only, kept whole, 3-D
    return [wl.alexnet()[2], wl.resnet50()[3], wl.c3d()[0], wl.single2d()[0],
            wl.Layer("filters_only", wl.alexnet()[4].shape, 0.3, wl.COL_NONE, 1.0, seed=3),
            wl.Layer("whole", wl.alexnet()[3].shape, 1.0, wl.COL_SHAPE, 1.0, seed=4)]


@pytest.mark.parametrize("name", ["alexnet", "resnet50", "mixed"])
@pytest.mark.parametrize("with_keys", [False, True])
@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
def test_batched_projection_equals_per_layer_calls(name, with_keys, dtype):
    from paper_1807_11091_gb300 import sadmm
    layers = _layers(name)
    dev = torch.device("cuda", 0)
    Ws = [wl.gen_tensors(L.shape.with_batch(1), seed=L.seed)["W"].to(dtype).to(dev) for L in layers]
    args = [(L.shape.desc16(), W, L.k_filters, L.colkind, L.k_cols, None) for L, W in zip(layers, Ws)]
    got = sadmm.project_groups_batch(args, with_keys=with_keys)
    for (d, W, kf, ck, kc, U), (fi, ci, keys) in zip(args, got):
        fi1, ci1, keys1 = sadmm.project_groups(d, W, kf, ck, kc, with_keys=with_keys)
        assert torch.equal(fi, fi1)
        assert (ci is None) == (ci1 is None) and (ci is None or torch.equal(ci, ci1))
        if with_keys:
            assert torch.equal(keys, keys1)
    assert sadmm.device_status() == 0


def _bits(t):
    return t.view(torch.int16 if t.dtype == torch.bfloat16 else torch.int32)


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
def test_batched_admm_update_equals_per_layer_and_oracle(dtype):
    from paper_1807_11091_gb300 import sadmm
    layers = _layers("alexnet") + [wl.resnet50()[15]]
    dev = torch.device("cuda", 0)
    states = [wl.gen_admm_state(L.shape, L.seed) for L in layers]
    W = [st["W"].to(dtype).to(dev) for st in states]
    U0 = [st["U"].to(dtype).to(dev) for st in states]
    spec = [(L.shape.desc16(), L.k_filters, L.colkind, L.k_cols) for L in layers]
    batch = sadmm.AdmmBatch(spec, dev)
    steps = [sadmm.AdmmStep(d, kf, ck, kc, dev) for d, kf, ck, kc in spec]
    Ub = [u.clone() for u in U0]
    Us = [u.clone() for u in U0]
    for it in range(2):  # twice in a row: the second update starts from the first one's U
        Zb = [torch.full_like(w, float("nan")) for w in W]
        Zs = [torch.full_like(w, float("nan")) for w in W]
        outs = batch(W, Ub, Zb)
        for step, w, u, z, (fi, ci) in zip(steps, W, Us, Zs, outs):
            fi1, ci1 = step(w, u, z)
            assert torch.equal(fi, fi1) and ((ci is None and ci1 is None) or torch.equal(ci, ci1))
        for ub, zb, us, zs in zip(Ub, Zb, Us, Zs):
            assert torch.equal(_bits(ub), _bits(us)) and torch.equal(_bits(zb), _bits(zs))
        if it == 0:
            # the first update against the oracle
            for L, st, (fi, ci), ub, zb in zip(layers, states, outs, Ub, Zb):
                s = L.shape
                rows, cols, Zo, Uo = oracle.admm_update(st["W"].to(dtype), st["U"].to(dtype), s.taps, L.k_filters,
                                                        L.colkind, L.k_cols)
                assert np.array_equal(fi.cpu().numpy(), rows)
                if ci is not None:
                    assert np.array_equal(ci.cpu().numpy(), cols)
                assert torch.equal(_bits(zb.cpu()), _bits(Zo.reshape(zb.shape)))
                assert torch.equal(_bits(ub.cpu()), _bits(Uo.reshape(ub.shape)))
    assert sadmm.device_status() == 0


def test_batch_rejects_bad_items():
    from paper_1807_11091_gb300 import sadmm
    L = wl.alexnet()[2]
    dev = torch.device("cuda", 0)
    W = wl.gen_tensors(L.shape.with_batch(1), seed=L.seed)["W"].to(dev)
    good = (L.shape.desc16(), W, L.k_filters, L.colkind, L.k_cols, None)
    bad = (L.shape.desc16(), W, L.shape.f + 1, L.colkind, L.k_cols, None)
    with pytest.raises(sadmm.SadmmError):
        sadmm.project_groups_batch([good, bad])
    with pytest.raises(sadmm.SadmmError):
        sadmm.project_groups_batch([good] * (sadmm.SADMM_MAX_BATCH + 1))


def _pack_layers():
    """Plans of every kind: gathered shape-wise, channel-wise, grouped, 3-D,
    filters only, kept whole on the input-slab path, split K' (batch 1) and
    stream-K (AlexNet CONV3 at batch 128)."""
    return [wl.Layer("first", wl.alexnet()[0].shape.with_batch(2), 1.0, wl.COL_SHAPE, 1.0, seed=100),
            wl.Layer("conv2_b3", wl.alexnet()[1].shape.with_batch(3), 0.5, wl.COL_SHAPE, 0.5, seed=101),
            wl.alexnet()[2],
            wl.Layer("conv4_b1", wl.alexnet()[3].shape.with_batch(1), 0.2, wl.COL_SHAPE, 0.2, seed=103),
            wl.resnet50()[3], wl.resnet50()[6], wl.c3d()[0], wl.single2d()[0],
            wl.Layer("filters_only", wl.alexnet()[4].shape.with_batch(4), 0.3, wl.COL_NONE, 1.0, seed=3)]


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
def test_batched_pack_equals_per_layer_packs(dtype):
    """sadmm_pack_batch gives each plan the packed weights, tables and forward
    output that its own sadmm_pack gives, bit for bit."""
    from paper_1807_11091_gb300 import sadmm
    dev = torch.device("cuda", 0)
    layers = _pack_layers()
    one, batch, tensors = [], [], []
    for L in layers:
        s = L.shape
        t = wl.gen_tensors(s, seed=L.seed)
        W = t["W"].to(dev).to(dtype)
        fi, ci, _ = sadmm.project_groups(s.desc16(), W, L.k_filters, L.colkind, L.k_cols)
        fi = fi if L.k_filters < s.f else None
        ci = ci if L.colkind != wl.COL_NONE else None
        ncg = L.k_cols if L.colkind != wl.COL_NONE else s.k
        one.append(sadmm.PrunedConv(s.desc16(), W, fi, L.colkind, ci, L.k_filters, ncg))
        pc = sadmm.PrunedConv(s.desc16(), W, fi, L.colkind, ci, L.k_filters, ncg)
        pc.buf.zero_()
        batch.append((pc, W, fi, ci))
        tensors.append(t)
    kinds = {(pc.plan.xs_mode, pc.plan.splits > 1, pc.plan.sk_len > 0) for pc, _, _, _ in batch}
    assert (1, False, False) in kinds and any(k[1] for k in kinds) and any(k[2] for k in kinds), kinds
    sadmm.pack_batch(batch)
    for L, a, (b, _, _, _), t in zip(layers, one, batch, tensors):
        pa, pb = a.plan, b.plan
        end = pa.off_wp + pa.desc.groups * pa.n_pad * pa.k_pad * 2
        for lo, hi in ((pa.off_wp, end), (pa.off_gather, pa.off_gather + pa.k_pad * 8),
                       (pa.off_rowmap, pa.off_rowmap + pa.desc.groups * pa.n_pad * 4),
                       (pa.off_counts, pa.off_counts + pa.desc.groups * 8),
                       (pa.off_wps, pa.off_wps + (pa.bn * pa.xs_kpad * 2 if pa.xs_mode else 0))):
            assert torch.equal(a.buf[lo:hi], b.buf[lo:hi]), (L.name, lo, hi)
        x, bias = t["x"].to(dev), t["bias"].to(dev)
        assert torch.equal(a.forward(x, bias), b.forward(x, bias)), L.name
    assert sadmm.device_status() == 0


@pytest.mark.parametrize("case", [
    # input-slab plan (stride 4, kept whole) and a gathered whole-tile plan (shape-wise, grouped)
    ("slab_stride4", wl.ConvShape(n=8, c=3, h=67, w=67, f=32, kh=11, kw=11, sh=4, sw=4), 1.0, wl.COL_NONE, 1.0),
    ("gathered_groups", wl.ConvShape(n=8, c=32, h=27, w=27, f=64, kh=5, kw=5, ph=2, pw=2, groups=2), 0.5,
     wl.COL_SHAPE, 0.5),
], ids=lambda c: c[0])
def test_batch_slices_match_the_whole_batch(case):
    """A plan for a quarter of the batch, run on each quarter of x (the same
    projection lists), writes each image's output bit for bit as the
    whole-batch plan does, when both plans sum every tile in one CTA (no split
    K', no stream-K) -- the property the end-to-end benchmark's sliced first
    layer relies on."""
    from paper_1807_11091_gb300 import sadmm
    name, s, ff, ck, cf = case
    dev = torch.device("cuda", 0)
    t = wl.gen_tensors(s, seed=77)
    kf = wl.retained(ff, s.f)
    kc = wl.retained(cf, s.k) if ck != wl.COL_NONE else 0
    W, x, bias = t["W"].to(dev), t["x"].to(dev), t["bias"].to(dev)
    fi, ci, _ = sadmm.project_groups(s.desc16(), W, kf, ck, kc)
    ncg = kc if ck != wl.COL_NONE else s.k
    nb = s.n // 4

    def ctas(n):
        # a gathered plan on exactly as many CTAs as it has units neither splits K' nor runs stream-K
        return 0 if name.startswith("slab") else s.groups * -(-(n * s.oh * s.ow) // 128)

    whole = sadmm.PrunedConv(s.desc16(), W, fi if kf < s.f else None, ck, ci if ck != wl.COL_NONE else None, kf, ncg,
                             max_ctas=ctas(s.n))
    d16 = s.desc16()
    d16[0] = nb
    part = sadmm.PrunedConv(d16, W, fi if kf < s.f else None, ck, ci if ck != wl.COL_NONE else None, kf, ncg,
                            max_ctas=ctas(nb))
    for pc in (whole, part):
        assert pc.plan.splits == 1 and pc.plan.sk_len == 0, name
    assert whole.plan.xs_mode == part.plan.xs_mode == (1 if name.startswith("slab") else 0)
    y = whole.forward(x, bias)
    y4 = torch.full_like(y, float("nan"))
    for j in range(4):
        part.forward(x[j * nb:(j + 1) * nb].contiguous(), bias, out=y4[j * nb:(j + 1) * nb])
    assert sadmm.device_status() == sadmm.SADMM_OK
    assert torch.equal(y, y4), name
