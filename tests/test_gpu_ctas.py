"""Forward plans capped to fewer CTAs than SMs (sadmm_plan_init_ctas): the
conv leaves the other SMs free for concurrent work.  The split-K and stream-K
choices follow the cap; the output must match the oracle (indices bit-exact,
output within 2e-3 * max|y|) whatever the cap."""
import numpy as np
import pytest
import torch

import oracle
import workloads as wl

from _helpers import assert_close, pruned_filters

pytestmark = pytest.mark.gpu


def _run(layer, n, max_ctas):
    from paper_1807_11091_gb300 import sadmm
    s = layer.shape.with_batch(n)
    t = wl.gen_tensors(s, seed=layer.seed)
    dev = torch.device("cuda", 0)
    W, x, bias = t["W"].to(dev), t["x"].to(dev), t["bias"].to(dev)
    fi, ci, _ = sadmm.project_groups(s.desc16(), W, layer.k_filters, layer.colkind, layer.k_cols)
    pc = sadmm.PrunedConv(s.desc16(), W, fi if layer.k_filters < s.f else None, layer.colkind, ci,
                          layer.k_filters, layer.k_cols if layer.colkind != wl.COL_NONE else s.k,
                          max_ctas=max_ctas)
    y = torch.full(pc.out_shape(), float("nan"), dtype=torch.float32, device=dev)
    pc.forward(x, bias, relu=True, out=y)
    assert sadmm.device_status() == 0
    rows, cols, _, _ = oracle.project(t["W"], s.taps, layer.k_filters, layer.colkind, layer.k_cols)
    ref = oracle.pruned_conv(t["x"], t["W"], t["bias"], s.desc16(), s.taps, rows, layer.colkind, cols, relu=True)
    assert_close(y.cpu().numpy(), ref, what=f"{layer.name} batch {n} cap {max_ctas}")
    assert np.all(y.cpu().numpy()[:, pruned_filters(s.f, rows)] == 0.0)
    return pc.plan


@pytest.mark.parametrize("cap", [1, 7, -4], ids=["one_cta", "seven", "all_but_4"])
@pytest.mark.parametrize("li", [0, 2, 4], ids=["conv1", "conv3", "conv5"])
def test_capped_plan_parity(li, cap):
    n_sm = torch.cuda.get_device_properties(0).multi_processor_count
    max_ctas = cap if cap > 0 else n_sm + cap
    L = wl.alexnet()[li]
    plan = _run(L, 4, max_ctas)
    assert plan.ctas == max_ctas


def test_cap_resizes_split_and_stream_k():
    """Batch 1 of conv3 has 2 tiles of 9 stages: 8 CTAs split K' 3 ways (3
    stages each), 2 CTAs not at all.  conv3 at batch 16 (22 tiles) on 20 CTAs
    takes the stream-K tail split (runs of 10 stages)."""
    L = wl.alexnet()[2]
    plan = _run(L, 1, 8)
    assert plan.splits == 3 and plan.sk_len == 0
    plan = _run(L, 1, 2)
    assert plan.splits == 1 and plan.sk_len == 0
    plan = _run(L, 16, 20)
    assert plan.splits == 1 and plan.sk_len == 10 and plan.sk_grid == 20
