"""Host-side checks of bench.py's arithmetic (no GPU): the retained-MAC count
that the TFLOP/s metric divides, and the parsing of the nvidia-smi clock
samples that decide whether a timed run is kept."""
import types

import numpy as np
import pytest

import oracle
import workloads as wl


def _layers():
    for name in sorted(wl.WORKLOADS):
        for L in wl.get(name):
            yield f"{name}/{L.name}", L


@pytest.mark.parametrize("L", [L for _, L in _layers()], ids=[n for n, _ in _layers()])
def test_flop_count_is_twice_the_kept_weights_times_output_pixels(L):
    """The metric's numerator, 2 * M * F' * K', equals 2 * (output pixels per
    filter) * (weights the projection keeps), counted from the oracle's mask;
    the dense count is the same with nothing pruned."""
    import bench
    L = wl.subset_layer(L, 1)
    s = L.shape
    t = wl.gen_tensors(s, seed=L.seed)
    rows, cols, _, _ = oracle.project(t["W"], s.taps, L.k_filters, L.colkind, L.k_cols)
    kept = int(np.count_nonzero(oracle.masked_weights(np.ones(tuple(t["W"].shape)), rows, L.colkind, cols, s.taps)))
    ref = 2.0 * s.m * kept  # s.m: output pixels of one filter over the batch
    assert L.retained_flops() == ref
    G = s.cg if L.colkind == wl.COL_CHANNEL else s.k
    run = types.SimpleNamespace(s=s, k_filters=L.k_filters, colkind=L.colkind,
                                k_cols=L.k_cols if L.colkind != wl.COL_NONE else 0)
    assert bench.LayerRun.flops(run) == ref
    dense = types.SimpleNamespace(s=s, k_filters=s.f, colkind=L.colkind, k_cols=G if L.colkind != wl.COL_NONE else 0)
    assert bench.LayerRun.flops(dense) == 2.0 * s.m * int(np.prod(t["W"].shape)) == L.dense_flops()


def _line(clk, mx=2070, power=900.0, reasons=("Not Active",) * 4):
    return ", ".join(["2026/01/01 00:00:00.000", "0", str(clk), str(mx), str(power), "0x0"] + list(reasons))


def test_clock_summary_reasons_and_loaded_median():
    import bench
    cs = bench.ClockSampler(0)
    idle = [_line(345, power=120.0)] * 6
    load = [_line(2070, power=1100.0)] * 5 + [_line(1995, power=1250.0)] * 2
    cs.lines = idle + load + ["garbage", _line("[N/A]")]
    s = cs.summary()
    assert s["sm_mhz"] == 2070 and s["sm_max_mhz"] == 2070 and s["reasons"] == [] and s["samples"] == 13
    assert s["power_w_max"] == 1250.0
    cs.lines = load + [_line(1800, power=1300.0, reasons=("Not Active", "Active", "Not Active", "Active"))]
    s = cs.summary()
    assert s["reasons"] == ["hw_thermal_slowdown", "sw_power_cap"]
    cs.lines = [_line(c, power="[N/A]") for c in (1000, 2000, 2070)]
    assert cs.summary()["sm_mhz"] == 2000
    cs.lines = []
    assert cs.summary() == {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}


def test_reference_arm_line_on_rank0(monkeypatch):
    """`bench.py --impl reference` on one process: one JSON line with the GPU
    arm's metric, unit, direction and workload config, the oracle described in
    cpu_baseline, and an e2e entry with no host-device bytes."""
    import contextlib
    import io
    import json

    import bench
    monkeypatch.setenv("RANK", "0")
    monkeypatch.setenv("WORLD_SIZE", "1")
    monkeypatch.setenv("LOCAL_RANK", "0")
    args = types.SimpleNamespace(workload="single2d", steps=2, warmup=3, gpus=1, out_dtype="fp32")
    buf = io.StringIO()
    with contextlib.redirect_stdout(buf):
        assert bench.run_reference(args) == 0
    lines = [ln for ln in buf.getvalue().splitlines() if ln.strip()]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["metric"] == bench.METRIC and d["unit"] == "TFLOP/s"
    assert d["higher_is_better"] is True and d["n_gpus"] == 1 and d["steps"] == 2 and d["warmup"] == 3
    assert d["value"] > 0 and d["ms_per_step"] > 0
    assert d["config"] == bench.workload_config(args, wl.get("single2d"))
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["value"] == d["value"] and cb["sample"]
    assert d["e2e"] == {"value": d["value"], "unit": "TFLOP/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}


def test_traffic_reported_only_for_the_profiled_kernel_sources(monkeypatch, tmp_path):
    """The roofline's `traffic` comes from the committed ncu summary only while
    the forward kernels' sources hash to the sha1 recorded in it, and only for
    the workload it was captured on; otherwise it is null."""
    import bench
    assert bench.conv_traffic("alexnet", "bf16") is None and bench.conv_traffic("resnet50", "fp32") is None
    good = tmp_path / "good.txt"
    good.write_text(f"# comment: 1\nkernel_source_sha1: {bench.conv_source_sha1()}\ndram_bytes_per_call_avg: 123\n")
    monkeypatch.setattr(bench, "TRAFFIC_FILE", str(good))
    assert bench.conv_traffic("alexnet", "fp32") == 123.0
    stale = tmp_path / "stale.txt"
    stale.write_text("kernel_source_sha1: " + "0" * 40 + "\ndram_bytes_per_call_avg: 123\n")
    monkeypatch.setattr(bench, "TRAFFIC_FILE", str(stale))
    assert bench.conv_traffic("alexnet", "fp32") is None
    monkeypatch.setattr(bench, "TRAFFIC_FILE", str(tmp_path / "missing.txt"))
    assert bench.conv_traffic("alexnet", "fp32") is None


def test_gpus_flag_must_match_the_ranks():
    import bench
    assert bench.check_gpus(1, 1) is None and bench.check_gpus(4, 4) is None
    assert "torch.distributed.run" in bench.check_gpus(8, 1)
    assert bench.check_gpus(1, 2) is not None
