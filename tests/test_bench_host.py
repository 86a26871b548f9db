"""Host logic of bench.py that needs no GPU: the clock summary of a timed
region and the rule that rejects it; the stored DRAM-traffic capture of the
tensor-core GEMMs describes the current kernel sources, and its per-launch
figure scales with rows x vocabulary columns as the roofline line assumes."""
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402
from paper_2607_07508_gb300.build import kernel_source_hash  # noqa: E402

CAPTURE = os.path.join(ROOT, "profiles", "dram_traffic_tc_gemm_moe8k.txt")
KERNELS = ("tc_logits_lse_fwd", "tc_dlogits", "tc_dH_gemm", "tc_dW_gemm")


def _rows():
    return [l.split() for l in open(CAPTURE) if l.strip() and not l.startswith("#")]


def test_capture_matches_the_current_gemm_sources():
    """A change to the GEMM sources needs a new capture (the bench then reports
    traffic = null until it exists)."""
    src = kernel_source_hash()
    rows = {f[0]: f for f in _rows() if len(f) == 6}
    assert set(KERNELS) <= set(rows)
    for k in KERNELS:
        assert rows[k][1] == src, f"{k}: capture taken on sources {rows[k][1]}, current {src}"


def test_stored_traffic_scales_with_rows_and_columns():
    for k in KERNELS:
        f = next(r for r in _rows() if r[0] == k)
        rows, cols, rd, wr = int(f[2]), int(f[3]), float(f[4]), float(f[5])
        assert bench.stored_traffic(k, rows, cols) == rd + wr
        assert abs(bench.stored_traffic(k, 2 * rows, cols) - 2 * (rd + wr)) <= 1e-6 * (rd + wr)
        assert abs(bench.stored_traffic(k, rows, cols / 4) - (rd + wr) / 4) <= 1e-6 * (rd + wr)
    assert bench.stored_traffic("no_such_kernel", 1, 1) is None


def _smi(ts, sm, mx, watts, hw="Not Active", hwt="Not Active", swt="Not Active", cap="Not Active"):
    """One line of nvidia-smi --format=csv,noheader,nounits for the sampler's fields."""
    return f"2026/12/02 10:00:{ts:06.3f}, {sm}, {mx}, {watts}, 0x0000000000000000, {hw}, {hwt}, {swt}, {cap}"


def _epoch(ts):
    import datetime
    return datetime.datetime(2026, 12, 2, 10, 0, 0).timestamp() + ts


def test_clock_summary_uses_the_timed_window():
    lines = [_smi(1.0, 900, 2070, 300.0),                      # before the region
             _smi(2.0, 1600, 2070, 1390.0, cap="Active"),
             _smi(2.1, 1650, 2070, 1400.5),
             _smi(2.2, 1700, 2070, 1380.0),
             "garbage line",
             _smi(9.0, 2070, 2070, 200.0, hw="Active")]          # after it
    c = bench.summarise_clocks(lines, _epoch(1.5), _epoch(3.0))
    assert c["sm_mhz"] == 1650 and c["sm_max_mhz"] == 2070
    assert c["samples"] == 3 and c["samples_in_timed_region"] == 3
    assert c["power_w_max"] == 1400.5
    assert c["reasons"] == ["sw_power_cap"]
    # no sample inside the window: every sample is used
    c = bench.summarise_clocks(lines, _epoch(20.0), _epoch(30.0))
    assert c["samples"] == 5 and c["samples_in_timed_region"] == 0
    assert c["reasons"] == ["hw_slowdown", "sw_power_cap"]
    assert bench.summarise_clocks(["x"], 0, 1)["reasons"] == ["no samples"]


def test_clock_rejection_rules():
    ok_cap = {"sm_mhz": 1575, "sm_max_mhz": 2070, "reasons": ["sw_power_cap"]}
    assert bench.clocks_rejection(ok_cap) is None            # the power cap is kept
    assert bench.clocks_rejection({"sm_mhz": 1990, "sm_max_mhz": 2070, "reasons": []}) is None
    for r in ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown"):
        why = bench.clocks_rejection({"sm_mhz": 2000, "sm_max_mhz": 2070, "reasons": [r, "sw_power_cap"]})
        assert why is not None and r in why
    why = bench.clocks_rejection({"sm_mhz": 1200, "sm_max_mhz": 2070, "reasons": []})
    assert why is not None and "lock" in why                 # low clock with no reason
    # no clock record: nothing to reject on
    assert bench.clocks_rejection({"sm_mhz": None, "sm_max_mhz": None,
                                   "reasons": ["nvidia-smi unavailable"]}) is None
