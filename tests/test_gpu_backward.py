"""GPU parity of the masked-retraining backward (sadmm_conv_bwd) and of the
tensor-core GEMM it uses.

The GEMM is compared with a plain PyTorch fp64 product of the same bf16
operands.  The backward is compared with the oracle's fp64 gradients: dW, db
and dx within 2e-3 * max|reference| per tensor, masked weight entries and
pruned filters' bias gradients exactly zero, every output element written.
The ReLU derivative comes from the oracle's own forward output on both sides
(passed in as y), so the two take the same ReLU decisions.
"""
import numpy as np
import pytest
import torch

import oracle
import workloads as wl
from workloads import ConvShape

from _helpers import assert_close

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("shape", [(128, 256, 64), (384, 160, 640), (256, 48, 192)])
@pytest.mark.parametrize("accumulate", [0, 1])
def test_gemm_matches_torch(shape, accumulate):
    from paper_1807_11091_gb300 import sadmm
    M, N, K = shape
    g = torch.Generator().manual_seed(M + N + K)
    A = torch.randn(M, K, generator=g).to(torch.bfloat16)
    B = torch.randn(N, K, generator=g).to(torch.bfloat16)
    C0 = torch.randn(M, N, generator=g)
    dev = torch.device("cuda", 0)
    Ad, Bd, Cd = A.to(dev), B.to(dev), C0.to(dev).clone()
    st = sadmm.sadmm_gemm_bf16(Ad.data_ptr(), Bd.data_ptr(), Cd.data_ptr(), M, N, K, N, accumulate,
                               int(torch.cuda.current_stream().cuda_stream))
    assert st == 0
    ref = A.double() @ B.double().T + (C0.double() if accumulate else 0)
    err = (Cd.cpu().double() - ref).abs().max().item()
    assert err <= 1e-5 * ref.abs().max().item()


CASES = [
    ("ragged", ConvShape(n=3, c=5, h=11, w=13, f=37, kh=3, kw=3, ph=1, pw=1), 0.7, wl.COL_SHAPE, 0.4),
    ("groups2_5x5", ConvShape(n=2, c=8, h=9, w=9, f=12, kh=5, kw=5, ph=2, pw=2, groups=2), 0.5, wl.COL_SHAPE, 0.5),
    ("stride4_11x11", ConvShape(n=2, c=3, h=35, w=35, f=16, kh=11, kw=11, sh=4, sw=4), 1.0, wl.COL_SHAPE, 0.8),
    ("c3d", ConvShape(n=2, c=4, t=5, h=6, w=7, f=20, kt=3, kh=3, kw=3, pt=1, ph=1, pw=1), 1.0, wl.COL_SHAPE, 0.3),
    # 45 taps: the split tap-mask form (row bits kt*KH + kh, kw bits apart), frames and rows clipped
    ("c3d_45_taps", ConvShape(n=2, c=4, t=6, h=7, w=8, f=16, kt=3, kh=3, kw=5, pt=1, ph=1, pw=2), 0.75, wl.COL_SHAPE,
     0.4),
    ("channel_3x3", ConvShape(n=2, c=24, h=9, w=9, f=40, kh=3, kw=3, ph=1, pw=1), 0.5, wl.COL_CHANNEL, 0.5),
    ("two_filter_tiles", ConvShape(n=2, c=16, h=10, w=10, f=300, kh=3, kw=3, ph=1, pw=1), 1.0, wl.COL_SHAPE, 1.0),
]


def _backward(s, t, kf, ck, kc, relu=True, seed=0, chunk_pixels=0):
    from paper_1807_11091_gb300 import sadmm
    dev = torch.device("cuda", 0)
    rows, cols, _, _ = oracle.project(t["W"], s.taps, kf, ck, kc)
    # oracle forward output: the ReLU decision for both sides
    y = torch.from_numpy(oracle.pruned_conv(t["x"], t["W"], t["bias"], s.desc16(), s.taps, rows, ck, cols,
                                            relu=True)).float()
    g = torch.Generator().manual_seed(seed)
    dy = torch.randn(y.shape, generator=g).to(torch.bfloat16)
    W, x = t["W"].to(dev), t["x"].to(dev)
    fi = torch.as_tensor(rows, dtype=torch.int32, device=dev)
    ci = torch.as_tensor(cols, dtype=torch.int32, device=dev) if ck != wl.COL_NONE else None
    pc = sadmm.PrunedConv(s.desc16(), W, fi if kf < s.f else None, ck, ci, kf, kc if ck != wl.COL_NONE else s.k)
    dW, db, dx = pc.backward(x, dy.to(dev), y=y.to(dev), relu=relu, chunk_pixels=chunk_pixels)
    assert sadmm.device_status() == 0
    rdx, rdW, rdb = oracle.pruned_conv_backward(t["x"], t["W"], t["bias"], s.desc16(), s.taps, rows, ck, cols, dy,
                                                relu=relu, y=y)
    return (dW.cpu().numpy(), db.cpu().numpy(), dx.cpu().numpy()), (rdW.reshape(s.f, -1), rdb, rdx), rows, cols


@pytest.mark.parametrize("case", CASES, ids=lambda c: c[0])
def test_backward_matches_oracle(case):
    name, s, ff, ck, cf = case
    G = s.cg if ck == wl.COL_CHANNEL else s.k
    kf, kc = wl.retained(ff, s.f), (wl.retained(cf, G) if ck != wl.COL_NONE else 0)
    t = wl.gen_tensors(s, seed=13)
    (dW, db, dx), (rdW, rdb, rdx), rows, cols = _backward(s, t, kf, ck, kc)
    assert np.all(np.isfinite(dW)) and np.all(np.isfinite(dx)) and np.all(np.isfinite(db))
    assert_close(dW, rdW, what=f"{name} dW")
    assert_close(db, rdb, what=f"{name} db")
    assert_close(dx, rdx, what=f"{name} dx")
    keep = oracle.masked_weights(np.ones(t["W"].shape), rows, ck, cols, s.taps).reshape(s.f, -1) != 0
    assert np.all(dW[~keep] == 0.0)
    pruned = np.setdiff1d(np.arange(s.f), rows)
    assert np.all(db[pruned] == 0.0)


@pytest.mark.parametrize("li", range(5))
def test_backward_alexnet_layers_batch2(li):
    L = wl.subset_layer(wl.alexnet()[li], 2)
    s = L.shape
    t = wl.gen_tensors(s, seed=L.seed)
    (dW, db, dx), (rdW, rdb, rdx), _, _ = _backward(s, t, L.k_filters, L.colkind, L.k_cols, seed=li)
    assert_close(dW, rdW, what=f"{L.name} dW")
    assert_close(db, rdb, what=f"{L.name} db")
    assert_close(dx, rdx, what=f"{L.name} dx")


def test_backward_without_relu():
    name, s, ff, ck, cf = CASES[0]
    kf, kc = wl.retained(ff, s.f), wl.retained(cf, s.k)
    t = wl.gen_tensors(s, seed=5)
    (dW, db, dx), (rdW, rdb, rdx), _, _ = _backward(s, t, kf, ck, kc, relu=False)
    assert_close(dW, rdW, what="no relu dW")
    assert_close(dx, rdx, what="no relu dx")


@pytest.mark.parametrize("chunk", [32768, 9984, 256])
def test_backward_several_pixel_chunks(chunk):
    """41772 output pixels in chunks as large as a smaller workspace holds:
    32768 + a ragged 9004, five chunks, or 164 chunks of 256, so the weight
    gradient accumulates per pixel split across chunks."""
    s = ConvShape(n=3, c=6, h=120, w=120, f=24, kh=3, kw=3)
    kf, kc = wl.retained(0.75, s.f), wl.retained(0.6, s.k)
    assert s.n * s.oh * s.ow > 32768
    t = wl.gen_tensors(s, seed=21)
    (dW, db, dx), (rdW, rdb, rdx), rows, cols = _backward(s, t, kf, wl.COL_SHAPE, kc, chunk_pixels=chunk)
    assert_close(dW, rdW, what=f"chunks of {chunk}: dW")
    assert_close(db, rdb, what=f"chunks of {chunk}: db")
    assert_close(dx, rdx, what=f"chunks of {chunk}: dx")


def test_backward_workspace_below_one_chunk_is_rejected():
    from paper_1807_11091_gb300 import sadmm
    s = ConvShape(n=1, c=4, h=9, w=9, f=8, kh=3, kw=3)
    t = wl.gen_tensors(s, seed=2)
    dev = torch.device("cuda", 0)
    pc = sadmm.PrunedConv(s.desc16(), t["W"].to(dev), None, wl.COL_NONE, None, s.f, s.k)
    small = sadmm.sadmm_conv_bwd_workspace_size_chunk(pc.plan, 256)
    assert 0 < small <= sadmm.sadmm_conv_bwd_workspace_size(pc.plan)
    ws = torch.empty(small + 2048, dtype=torch.uint8, device=dev)
    wptr = (ws.data_ptr() + 1023) // 1024 * 1024
    x, dy = t["x"].to(dev), torch.zeros((1, 8, 7, 7), dtype=torch.bfloat16, device=dev)
    dx = torch.empty(x.shape, device=dev)
    st = sadmm.sadmm_conv_bwd(pc.plan, x.data_ptr(), dy.data_ptr(), None, sadmm.SADMM_FP32, 0, None, None,
                              dx.data_ptr(), wptr, small - 1024, int(torch.cuda.current_stream().cuda_stream))
    assert st == sadmm.SADMM_EINVAL


def _raw_backward(pc, x, dy, y, want_dw, want_dx):
    from paper_1807_11091_gb300 import sadmm
    dev = x.device
    s_f, K = pc.plan.desc.f, (pc.plan.desc.c // pc.plan.desc.groups) * pc.plan.desc.kt * pc.plan.desc.kh * pc.plan.desc.kw
    dW = torch.full((s_f, K), float("nan"), device=dev) if want_dw else None
    db = torch.full((s_f,), float("nan"), device=dev) if want_dw else None
    dx = torch.full(x.shape, float("nan"), device=dev) if want_dx else None
    ws_bytes = sadmm.sadmm_conv_bwd_workspace_size(pc.plan)
    ws = torch.empty(ws_bytes + 1024, dtype=torch.uint8, device=dev)
    wptr = (ws.data_ptr() + 1023) // 1024 * 1024
    st = sadmm.sadmm_conv_bwd(pc.plan, x.data_ptr(), dy.data_ptr(), y.data_ptr(), sadmm.SADMM_FP32, 1,
                              dW.data_ptr() if dW is not None else None, db.data_ptr() if db is not None else None,
                              dx.data_ptr() if dx is not None else None, wptr, ws_bytes,
                              int(torch.cuda.current_stream().cuda_stream))
    assert st == 0 and sadmm.device_status() == 0
    return dW, db, dx


def test_backward_weight_gradient_deterministic_and_partial_calls():
    """dW and db come out bit-identical on every call (fixed-order sums); a call
    that asks for the weight gradient only, the input gradient only, or the bias
    gradient only gives what the full call gives (dx up to its atomic
    summation order)."""
    from paper_1807_11091_gb300 import sadmm
    name, s, ff, ck, cf = CASES[1]
    kf, kc = wl.retained(ff, s.f), wl.retained(cf, s.k)
    t = wl.gen_tensors(s, seed=31)
    dev = torch.device("cuda", 0)
    rows, cols, _, _ = oracle.project(t["W"], s.taps, kf, ck, kc)
    W, x = t["W"].to(dev), t["x"].to(dev)
    fi = torch.as_tensor(rows, dtype=torch.int32, device=dev)
    ci = torch.as_tensor(cols, dtype=torch.int32, device=dev)
    pc = sadmm.PrunedConv(s.desc16(), W, fi, ck, ci, kf, kc)
    y = pc.forward(x, t["bias"].to(dev))
    g = torch.Generator().manual_seed(7)
    dy = torch.randn(y.shape, generator=g).to(torch.bfloat16).to(dev)
    dW1, db1, dx1 = _raw_backward(pc, x, dy, y, True, True)
    dW2, db2, dx2 = _raw_backward(pc, x, dy, y, True, True)
    assert torch.equal(dW1, dW2) and torch.equal(db1, db2)
    dW3, db3, none = _raw_backward(pc, x, dy, y, True, False)
    assert none is None and torch.equal(dW1, dW3) and torch.equal(db1, db3)
    none, _, dx4 = _raw_backward(pc, x, dy, y, False, True)
    assert torch.isfinite(dx4).all()
    assert_close(dx4.cpu().numpy(), dx1.cpu().double().numpy(), tol=1e-6, what="dx alone")
    # the bias gradient alone (no pixel chunk is gathered)
    db5 = torch.full_like(db1, float("nan"))
    ws_bytes = sadmm.sadmm_conv_bwd_workspace_size(pc.plan)
    ws = torch.empty(ws_bytes + 1024, dtype=torch.uint8, device=dev)
    wptr = (ws.data_ptr() + 1023) // 1024 * 1024
    st = sadmm.sadmm_conv_bwd(pc.plan, x.data_ptr(), dy.data_ptr(), y.data_ptr(), sadmm.SADMM_FP32, 1, None,
                              db5.data_ptr(), None, wptr, ws_bytes, int(torch.cuda.current_stream().cuda_stream))
    assert st == 0 and sadmm.device_status() == 0
    assert torch.equal(db1, db5)


@pytest.mark.parametrize("case", [
    ("slab_stride4_pruned_filters", ConvShape(n=3, c=3, h=51, w=47, f=40, kh=11, kw=11, sh=4, sw=4), 0.6,
     wl.COL_NONE, 1.0),
    ("slab_stem_7x7_s2_p3", ConvShape(n=2, c=3, h=37, w=33, f=24, kh=7, kw=7, sh=2, sw=2, ph=3, pw=3), 1.0,
     wl.COL_SHAPE, 1.0),
    ("slab_channel_5x5_s2", ConvShape(n=2, c=32, h=17, w=16, f=48, kh=5, kw=5, sh=2, sw=2, ph=2, pw=2), 0.5,
     wl.COL_CHANNEL, 0.125),
], ids=lambda c: c[0])
def test_backward_weight_gradient_on_the_slab(case):
    """Input-slab plans take the weight gradient on the space-to-depth slab (dZ
    tiles against shifted slab operands, accumulated per CTA in TMEM, slices
    summed in order): dW, db and dx against the oracle, the pruned entries of dW
    exactly zero, and dW bit-identical across calls."""
    from paper_1807_11091_gb300 import sadmm
    name, s, ff, ck, cf = case
    G = s.cg if ck == wl.COL_CHANNEL else s.k
    kf, kc = wl.retained(ff, s.f), (wl.retained(cf, G) if ck != wl.COL_NONE else 0)
    t = wl.gen_tensors(s, seed=17)
    (dW, db, dx), (rdW, rdb, rdx), rows, cols = _backward(s, t, kf, ck, kc)
    assert_close(dW, rdW, what=f"{name} dW")
    assert_close(db, rdb, what=f"{name} db")
    assert_close(dx, rdx, what=f"{name} dx")
    assert np.all(dW[rdW == 0.0] == 0.0)
    (dW2, _, _), _, _, _ = _backward(s, t, kf, ck, kc)
    assert np.array_equal(dW, dW2)


@pytest.mark.parametrize("li,batch", [(0, 16), (1, 72)], ids=["conv1_b16_slab_many_runs", "conv2_b72_full_chunks"])
def test_backward_alexnet_at_benchmarked_paths(li, batch):
    """The paths the benchmark's batch-128 backward takes, at batches the fp64
    oracle finishes in seconds: CONV1's weight gradient on the slab over 378
    output tiles (2.5 runs per CTA, one fp32 slice each, summed in CTA order);
    CONV2 (two conv groups) in a full 32768-pixel chunk, with the benchmark's
    weight-gradient split for that chunk, then a ragged second chunk."""
    L = wl.subset_layer(wl.alexnet()[li], batch)
    s = L.shape
    t = wl.gen_tensors(s, seed=L.seed)
    if li == 1:
        assert s.n * s.oh * s.ow > 32768
    (dW, db, dx), (rdW, rdb, rdx), rows, cols = _backward(s, t, L.k_filters, L.colkind, L.k_cols, seed=li)
    assert_close(dW, rdW, what=f"{L.name} batch {batch} dW")
    assert_close(db, rdb, what=f"{L.name} batch {batch} db")
    assert_close(dx, rdx, what=f"{L.name} batch {batch} dx")
    assert np.all(dW[rdW == 0.0] == 0.0)
