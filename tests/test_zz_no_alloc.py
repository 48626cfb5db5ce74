"""sadmm_project_groups_noalloc: the projection for callers that cannot give the
library device scratch memory (a framework that hands over only its input and
output tensors, or a loop that must not allocate once running).  Its keys live
in a fixed device array inside the library; its results must equal those of
sadmm_project_groups with a caller-provided workspace, call after call.

Kept in a file of its own that pytest collects last."""
import numpy as np
import pytest
import torch

import workloads as wl
from workloads import ConvShape

pytestmark = pytest.mark.gpu

LAYERS = [wl.single2d()[0], wl.alexnet()[1], wl.alexnet()[3], wl.resnet50()[15], wl.c3d()[0],
          wl.sweep(col_fracs=(0.25,), filt_fracs=(0.5,))[0]]


def _run(entry, s, W, kf, ck, kc):
    from paper_1807_11091_gb300 import sadmm
    dev = W.device
    desc = sadmm.make_desc(s.desc16())
    G = 0 if ck == wl.COL_NONE else (s.k if ck == wl.COL_SHAPE else s.cg)
    fi = torch.full((max(kf, 1),), -7, dtype=torch.int32, device=dev)
    ci = torch.full((max(kc, 1),), -7, dtype=torch.int32, device=dev)
    keys = torch.full((s.f + G,), float("nan"), dtype=torch.float64, device=dev)
    stream = torch.cuda.current_stream().cuda_stream
    if entry == "workspace":
        nbytes = sadmm.sadmm_workspace_size(desc, ck)
        ws = torch.empty(nbytes, dtype=torch.uint8, device=dev)
        st = sadmm.sadmm_project_groups(desc, W.data_ptr(), None, sadmm.SADMM_BF16, kf, ck, kc, fi.data_ptr(),
                                        ci.data_ptr(), keys.data_ptr(), ws.data_ptr(), nbytes, stream)
    else:
        st = sadmm.sadmm_project_groups_noalloc(desc, W.data_ptr(), None, sadmm.SADMM_BF16, kf, ck, kc,
                                                fi.data_ptr(), ci.data_ptr(), keys.data_ptr(), stream)
    assert st == 0, st
    assert sadmm.sadmm_last_device_status(stream) == 0
    return fi[:kf].cpu().numpy(), ci[:kc].cpu().numpy(), keys.cpu().numpy()


@pytest.mark.parametrize("layer", LAYERS, ids=lambda l: l.name)
def test_noalloc_projection_equals_workspace_projection(layer):
    s = layer.shape
    W = wl.gen_tensors(s.with_batch(1), seed=layer.seed)["W"].cuda()
    ref = _run("workspace", s, W, layer.k_filters, layer.colkind, layer.k_cols)
    for _ in range(2):  # two calls in a row share (and reuse) the fixed array
        got = _run("noalloc", s, W, layer.k_filters, layer.colkind, layer.k_cols)
        assert np.array_equal(got[0], ref[0]), "filter index list"
        assert np.array_equal(got[1], ref[1]), "column index list"
        np.testing.assert_allclose(got[2], ref[2], rtol=1e-12, atol=0)


def test_noalloc_rejects_layers_beyond_the_fixed_array():
    from paper_1807_11091_gb300 import sadmm
    limit = sadmm.SADMM_NOALLOC_SCRATCH_BYTES
    s = ConvShape(n=1, c=8192, h=3, w=3, f=16, kh=3, kw=3, ph=1, pw=1)  # K = 73728 keys > the array
    desc = sadmm.make_desc(s.desc16())
    assert sadmm.sadmm_workspace_size(desc, wl.COL_SHAPE) > limit
    fake = 1 << 20  # never dereferenced: rejected on the host
    st = sadmm.sadmm_project_groups_noalloc(desc, fake, None, sadmm.SADMM_BF16, 4, wl.COL_SHAPE, 4, fake, fake,
                                            None, None)
    assert st == sadmm.SADMM_EUNSUPPORTED


def test_noalloc_rejects_many_filters_without_column_pruning():
    """The filter keys alone can overflow the array: F = 16384 with no column pruning."""
    from paper_1807_11091_gb300 import sadmm
    s = ConvShape(n=1, c=1, h=3, w=3, f=16384, kh=3, kw=3, ph=1, pw=1)
    desc = sadmm.make_desc(s.desc16())
    assert sadmm.sadmm_workspace_size(desc, wl.COL_NONE) > sadmm.SADMM_NOALLOC_SCRATCH_BYTES
    fake = 1 << 20  # never dereferenced: rejected on the host
    st = sadmm.sadmm_project_groups_noalloc(desc, fake, None, sadmm.SADMM_BF16, 100, wl.COL_NONE, 0, fake, None,
                                            None, None)
    assert st == sadmm.SADMM_EUNSUPPORTED


@pytest.mark.parametrize("f,c,kf,ck,kc", [(192, 16160, 96, wl.COL_SHAPE, 4000),   # exactly at the limit
                                          (192, 16160, 192, wl.COL_CHANNEL, 5000),
                                          (16320, 32, 4000, wl.COL_NONE, 0)])
def test_noalloc_layers_at_the_limit_match_workspace_path(f, c, kf, ck, kc):
    """Layers whose keys fill the array exactly run and equal the workspace path."""
    from paper_1807_11091_gb300 import sadmm
    s = ConvShape(n=1, c=c, h=1, w=1, f=f, kh=1, kw=1)
    desc = sadmm.make_desc(s.desc16())
    assert sadmm.sadmm_workspace_size(desc, ck) == sadmm.SADMM_NOALLOC_SCRATCH_BYTES
    W = wl.gen_tensors(s, seed=77)["W"].cuda()
    ref = _run("workspace", s, W, kf, ck, kc)
    for _ in range(2):
        got = _run("noalloc", s, W, kf, ck, kc)
        assert np.array_equal(got[0], ref[0]) and np.array_equal(got[1], ref[1])
        np.testing.assert_allclose(got[2], ref[2], rtol=1e-12, atol=0)
