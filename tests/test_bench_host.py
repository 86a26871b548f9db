"""Host logic of bench.py that needs no GPU: the stored DRAM-traffic capture of
the tensor-core GEMMs describes the current kernel sources, and its per-launch
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
