"""Pins for the pruning-rate bookkeeping against the values Tables 1-2 print,
and for the retained-count rule of the seeded workloads (no GPU)."""
import os

import pytest

import workloads as wl

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "paper_pruning_rates.txt")


def _rows():
    out = []
    with open(GOLDEN) as fh:
        for line in fh:
            if not line.strip() or line.startswith("#"):
                continue
            t, meth, layer, col, row, printed, status = line.split()
            out.append((t, meth, layer, float(col), float(row), float(printed), status))
    return out


@pytest.mark.parametrize("entry", _rows(), ids=lambda e: f"{e[0]}-{e[1]}-{e[2]}")
def test_pruning_rate_reproduces_printed_tables(entry):
    _, _, _, col, row, printed, status = entry
    rate = wl.pruning_rate(col, row)
    if status in ("match", "swapped"):
        assert round(rate, 1) == pytest.approx(printed)
    else:
        assert status == "garbled"
        assert round(rate, 1) != pytest.approx(printed)


def test_retained_count_rule():
    assert wl.retained(0.5, 576) == 288
    assert wl.retained(0.2, 384) == 77
    assert wl.retained(0.2, 1728) == 346
    assert wl.retained(0.3, 3456) == 1037
    assert wl.retained(0.1, 2304) == 230
    assert wl.retained(0.05, 2304) == 115
    assert wl.retained(0.2, 256) == 51


def test_alexnet_shapes_match_the_paper_weight_counts():
    """Sec. 5: conv1 holds about 35K weights and conv2-5 about 2.3M."""
    layers = wl.alexnet()
    counts = [l.shape.f * l.shape.k for l in layers]
    assert counts[0] == 34848
    assert sum(counts[1:]) == 2297856
    assert [l.shape.oh for l in layers] == [55, 27, 13, 13, 13]
