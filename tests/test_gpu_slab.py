"""GPU parity of the input-slab forward (plan.xs_mode = 1): layers with one conv
group whose kept channels keep every column and whose space-to-depth input has
at most 64 channels -- strided first layers (AlexNet CONV1, a 7x7 stride-2
stem), stride-1 layers with few channels, channel-wise pruned layers.

Every output is pre-filled with NaN; fp32 output within 2e-3 * max|oracle|,
bf16 output within one bf16 ulp of the oracle rounded to bf16.  Each case
asserts that the plan took the slab path."""
import numpy as np
import pytest
import torch

import oracle
import workloads as wl
from workloads import ConvShape

from _helpers import assert_close, gpu_layer, oracle_layer, pruned_filters

pytestmark = pytest.mark.gpu

# (name, shape, filter fraction, column kind, column fraction)
CASES = [
    ("stride4_11x11", ConvShape(n=2, c=3, h=35, w=35, f=16, kh=11, kw=11, sh=4, sw=4), 1.0, wl.COL_NONE, 1.0),
    ("stride4_pruned_filters", ConvShape(n=3, c=3, h=51, w=47, f=40, kh=11, kw=11, sh=4, sw=4), 0.6, wl.COL_NONE,
     1.0),
    ("stem_7x7_s2_p3", ConvShape(n=2, c=3, h=37, w=33, f=24, kh=7, kw=7, sh=2, sw=2, ph=3, pw=3), 1.0, wl.COL_NONE,
     1.0),
    ("stride1_3x3_c16", ConvShape(n=2, c=16, h=21, w=19, f=48, kh=3, kw=3, ph=1, pw=1), 0.75, wl.COL_NONE, 1.0),
    ("channel_3x3", ConvShape(n=2, c=24, h=9, w=9, f=40, kh=3, kw=3, ph=1, pw=1), 0.5, wl.COL_CHANNEL, 0.5),
    ("channel_5x5_stride2", ConvShape(n=2, c=32, h=17, w=16, f=48, kh=5, kw=5, sh=2, sw=2, ph=2, pw=2), 0.5,
     wl.COL_CHANNEL, 0.125),
    ("shape_all_kept", ConvShape(n=2, c=4, h=15, w=16, f=20, kh=5, kw=5, sh=2, sw=2, ph=2, pw=2), 1.0, wl.COL_SHAPE,
     1.0),
    ("rect_stride_kernel", ConvShape(n=2, c=6, h=13, w=10, f=24, kh=3, kw=2, sh=2, sw=1, ph=1, pw=0), 0.75,
     wl.COL_NONE, 1.0),
    ("one_image_many_tiles", ConvShape(n=1, c=3, h=131, w=97, f=64, kh=5, kw=5, sh=2, sw=2, ph=1, pw=2), 1.0,
     wl.COL_NONE, 1.0),
    ("wide_256_filters", ConvShape(n=2, c=3, h=40, w=41, f=256, kh=3, kw=3, sh=2, sw=2, ph=1, pw=1), 1.0,
     wl.COL_NONE, 1.0),
    # stride 4 with padding on both sides and channel pruning
    ("stride4_pads_channels", ConvShape(n=2, c=8, h=37, w=41, f=24, kh=7, kw=7, sh=4, sw=4, ph=2, pw=3), 1.0,
     wl.COL_CHANNEL, 0.5),
    # column stride 3 (does not divide 8): the space-to-depth copy decodes every element
    ("stride3_generic_copy", ConvShape(n=2, c=3, h=25, w=26, f=16, kh=7, kw=7, sh=3, sw=3, ph=1, pw=2), 1.0,
     wl.COL_NONE, 1.0),
    # column stride 8: one input row of 8 columns per chunk
    ("stride8_one_channel", ConvShape(n=2, c=1, h=67, w=70, f=16, kh=12, kw=12, sh=8, sw=8, ph=3, pw=5), 1.0,
     wl.COL_NONE, 1.0),
    # row stride 3, column stride 2: rows (channel, phase) decoded with sh = 3
    ("rows_sh3_sw2", ConvShape(n=2, c=5, h=29, w=22, f=24, kh=6, kw=5, sh=3, sw=2, ph=2, pw=1), 0.75,
     wl.COL_NONE, 1.0),
]


def _k(s, ff, ck, cf):
    G = s.cg if ck == wl.COL_CHANNEL else s.k
    return wl.retained(ff, s.f), (wl.retained(cf, G) if ck != wl.COL_NONE else 0)


def _run(case, seed, **kw):
    name, s, ff, ck, cf = case
    kf, kc = _k(s, ff, ck, cf)
    t = wl.gen_tensors(s, seed=seed)
    fi, ci, y, pc = gpu_layer(s, t, kf, ck, kc, **kw)
    assert pc.plan.xs_mode == 1, f"{name}: the plan did not take the slab path"
    rows, cols, _, _ = oracle.project(t["W"], s.taps, kf, ck, kc)
    assert np.array_equal(fi, rows)
    if ck != wl.COL_NONE:
        assert np.array_equal(ci, cols)
    return s, t, rows, ck, cols, y, pc


@pytest.mark.parametrize("case", CASES, ids=lambda c: c[0])
def test_slab_layers_fp32(case):
    s, t, rows, ck, cols, y, _ = _run(case, seed=301)
    ref = oracle_layer(s, t, rows, ck, cols)
    assert_close(y, ref, what=case[0])
    assert np.all(y[:, pruned_filters(s.f, rows)] == 0.0)


@pytest.mark.parametrize("case", [CASES[1], CASES[2], CASES[4]], ids=lambda c: c[0])
def test_slab_bf16_output_no_relu_no_bias(case):
    s, t, rows, ck, cols, y, _ = _run(case, seed=302, relu=False, use_bias=False, out_dtype=torch.bfloat16)
    ref = oracle_layer(s, t, rows, ck, cols, relu=False, use_bias=False)
    ref_b = torch.from_numpy(ref).to(torch.bfloat16).float().numpy()
    scale = np.abs(ref).max()
    assert np.all(np.abs(y - ref_b) <= np.abs(ref_b) * 2.0 ** -7 + 2e-3 * scale), case[0]
    assert np.all(y[:, pruned_filters(s.f, rows)] == 0.0)


def test_slab_all_filters_pruned_gives_zeros():
    case = ("all_pruned", ConvShape(n=2, c=3, h=23, w=23, f=16, kh=5, kw=5, sh=2, sw=2), 0.0, wl.COL_NONE, 1.0)
    s, t, rows, ck, cols, y, _ = _run(case, seed=303)
    assert len(rows) == 0 and np.all(y == 0.0)


def test_slab_repeated_launches_identical():
    """The plan's space-to-depth buffer is rewritten by every launch: results
    are bit-identical across launches and across a launch on other input."""
    from paper_1807_11091_gb300 import sadmm
    case = CASES[1]
    s, t, rows, ck, cols, y, pc = _run(case, seed=304)
    dev = torch.device("cuda", 0)
    x = t["x"].to(dev)
    bias = t["bias"].to(dev)
    other = torch.randn_like(x.float()).to(torch.bfloat16)
    y2 = torch.full(pc.out_shape(), float("nan"), device=dev)
    pc.forward(other, bias, out=y2)
    pc.forward(x, bias, out=y2)
    assert sadmm.device_status() == 0
    assert np.array_equal(y2.cpu().numpy(), y)


_BY_NAME = {c[0]: c for c in CASES}


@pytest.mark.parametrize("case", [_BY_NAME[n] for n in ("stride4_11x11", "stride4_pads_channels",
                                                       "stride3_generic_copy", "stride8_one_channel")],
                         ids=lambda c: c[0])
def test_slab_input_off_the_16_byte_grid(case):
    """x 2-byte aligned only (a view one element into a buffer, which the ABI
    allows): the output equals the aligned call's bit for bit."""
    s, t, rows, ck, cols, y, pc = _run(case, seed=309)
    dev = torch.device("cuda", 0)
    x = t["x"].to(dev)
    big = torch.empty(x.numel() + 1, dtype=torch.bfloat16, device=dev)
    big[1:].copy_(x.reshape(-1))
    x_off = big[1:].view(x.shape)
    assert x_off.data_ptr() % 16 == 2
    y2 = torch.full(pc.out_shape(), float("nan"), device=dev)
    pc.forward(x_off, t["bias"].to(dev), out=y2)
    from paper_1807_11091_gb300 import sadmm
    assert sadmm.device_status() == 0
    assert np.array_equal(y2.cpu().numpy(), y)


def test_alexnet_conv1_batch128_sampled_images():
    """AlexNet CONV1 at batch 128 (the layer kept whole): indices exact, and
    images 0, 1, 63 and 127 against the oracle element by element."""
    L = wl.alexnet()[0]
    s = L.shape
    t = wl.gen_tensors(s, seed=L.seed)
    fi, ci, y, pc = gpu_layer(s, t, L.k_filters, L.colkind, L.k_cols)
    assert pc.plan.xs_mode == 1 and pc.plan.xs_cs == 48 and pc.plan.xs_r == 3 and pc.plan.xs_wb == 57
    rows, cols, _, _ = oracle.project(t["W"], s.taps, L.k_filters, L.colkind, L.k_cols)
    assert np.array_equal(fi, rows) and np.array_equal(ci, cols)
    for n in (0, 1, 63, 127):
        ref = oracle_layer(s, t, rows, L.colkind, cols, n0=n, n1=n + 1)
        assert_close(y[n:n + 1], ref, what=f"conv1 image {n}")


def test_slab_more_pruned_planes_than_the_shared_table():
    """1060 pruned filters: the first 1024 plane offsets come from shared memory,
    the rest from the plan's list; every pruned plane is zero."""
    case = ("many_pruned", ConvShape(n=2, c=3, h=9, w=11, f=1100, kh=3, kw=3, sh=2, sw=2, pw=1), 40 / 1100,
            wl.COL_NONE, 1.0)
    s, t, rows, ck, cols, y, _ = _run(case, seed=305)
    assert len(rows) == 40
    ref = oracle_layer(s, t, rows, ck, cols)
    assert_close(y, ref, what="many_pruned")
    assert np.all(y[:, pruned_filters(s.f, rows)] == 0.0)


@pytest.mark.parametrize("case", [CASES[1], CASES[4]], ids=lambda c: c[0])
def test_slab_forward_in_two_phases(case):
    """sadmm_conv_fwd_phase: the space-to-depth pass (INPUT) then the conv on
    its copy (REST, x not passed) equals the single call bit for bit; with no
    channel pruning the INPUT pass does not read the packed kept-channel list
    (the list is overwritten here before the pass and the result is the same)."""
    from paper_1807_11091_gb300 import sadmm
    s, t, rows, ck, cols, y, pc = _run(case, seed=306)
    dev = torch.device("cuda", 0)
    x, bias = t["x"].to(dev), t["bias"].to(dev)
    sp = int(torch.cuda.current_stream().cuda_stream)
    y2 = torch.full(pc.out_shape(), float("nan"), device=dev)
    if ck != wl.COL_CHANNEL:
        assert pc.plan.dev == pc.buf.data_ptr()
        off = pc.plan.off_scol + 4 * pc.plan.xs_kpad
        chan = pc.buf[off:off + 4 * pc.plan.xs_cs].view(torch.int32)
        saved = chan.clone()
        chan.fill_(-7)
    assert sadmm.sadmm_conv_fwd_phase(pc.plan, x.data_ptr(), None, 0, None, sadmm.SADMM_FP32,
                                      sadmm.SADMM_FWD_INPUT, sp) == 0
    if ck != wl.COL_CHANNEL:
        chan.copy_(saved)
    assert sadmm.sadmm_conv_fwd_phase(pc.plan, None, bias.data_ptr(), 1, y2.data_ptr(), sadmm.SADMM_FP32,
                                      sadmm.SADMM_FWD_REST, sp) == 0
    assert sadmm.device_status() == 0
    assert np.array_equal(y2.cpu().numpy(), y)


def test_gathered_plan_in_two_phases():
    """For a gathered plan INPUT does nothing and REST runs the whole forward."""
    from paper_1807_11091_gb300 import sadmm
    s = ConvShape(n=2, c=8, h=11, w=12, f=24, kh=3, kw=3, ph=1, pw=1)
    kf, kc = wl.retained(0.75, s.f), wl.retained(0.5, s.k)
    t = wl.gen_tensors(s, seed=307)
    fi, ci, y, pc = gpu_layer(s, t, kf, wl.COL_SHAPE, kc)
    assert pc.plan.xs_mode == 0
    dev = torch.device("cuda", 0)
    x, bias = t["x"].to(dev), t["bias"].to(dev)
    sp = int(torch.cuda.current_stream().cuda_stream)
    y2 = torch.full(pc.out_shape(), float("nan"), device=dev)
    assert sadmm.sadmm_conv_fwd_phase(pc.plan, x.data_ptr(), None, 0, None, sadmm.SADMM_FP32,
                                      sadmm.SADMM_FWD_INPUT, sp) == 0
    assert sadmm.sadmm_conv_fwd_phase(pc.plan, None, bias.data_ptr(), 1, y2.data_ptr(), sadmm.SADMM_FP32,
                                      sadmm.SADMM_FWD_REST, sp) == sadmm.SADMM_EINVAL  # needs x
    assert sadmm.sadmm_conv_fwd_phase(pc.plan, x.data_ptr(), bias.data_ptr(), 1, y2.data_ptr(), sadmm.SADMM_FP32,
                                      sadmm.SADMM_FWD_REST, sp) == 0
    assert sadmm.device_status() == 0
    assert np.array_equal(y2.cpu().numpy(), y)


@pytest.mark.parametrize("case", [
    # 4 channels x 4 x 4 phases: exactly 64 slab channels (eight chunks)
    ("cs_64", ConvShape(n=2, c=4, h=43, w=39, f=32, kh=11, kw=11, sh=4, sw=4), 1.0, wl.COL_NONE, 1.0),
    # a 900-wide input: 450 block pixels per row, a slab of 584 block pixels (73 octets)
    ("wide_rows", ConvShape(n=1, c=3, h=9, w=900, f=16, kh=3, kw=3, sh=2, sw=2, ph=1, pw=1), 1.0, wl.COL_NONE,
     1.0),
], ids=lambda c: c[0])
def test_slab_extreme_geometry(case):
    s, t, rows, ck, cols, y, pc = _run(case, seed=308)
    ref = oracle_layer(s, t, rows, ck, cols)
    assert_close(y, ref, what=case[0])


def test_slab_mma_step_limit():
    """A slab plan issues at most 128 MMAs per tile (their descriptor offsets travel
    in the kernel parameters): 15 x 15 stride 2 over 8 channels is 64 block taps x 32
    slab channels = 128 MMAs and takes the slab path; over 12 channels (192 MMAs) the
    same kernel takes the gathered path.  Both match the oracle."""
    at_cap = ("steps_128", ConvShape(n=2, c=8, h=40, w=40, f=16, kh=15, kw=15, sh=2, sw=2), 1.0, wl.COL_NONE, 1.0)
    s, t, rows, ck, cols, y, pc = _run(at_cap, seed=309)
    assert pc.plan.xs_r * pc.plan.xs_q * pc.plan.xs_cs // 16 == 128
    assert_close(y, oracle_layer(s, t, rows, ck, cols), what="steps_128")
    s = ConvShape(n=2, c=12, h=40, w=40, f=16, kh=15, kw=15, sh=2, sw=2)
    t = wl.gen_tensors(s, seed=310)
    fi, ci, y, pc = gpu_layer(s, t, s.f, wl.COL_NONE, 0)
    assert pc.plan.xs_mode == 0
    rows, cols, _, _ = oracle.project(t["W"], s.taps, s.f, wl.COL_NONE, 0)
    assert np.array_equal(fi, rows)
    assert_close(y, oracle_layer(s, t, rows, wl.COL_NONE, cols), what="steps_192")
