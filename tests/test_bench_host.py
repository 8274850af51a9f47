"""Host logic of the benchmark that needs no GPU: the stored DRAM traffic of
the fused launch is reported only for the kernel source, workload and batch
size it was captured on."""
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402


def _record(tmp_path, h, workload="c1", batch=1, nbytes=107516672):
    (tmp_path / "profiles").mkdir()
    (tmp_path / "profiles" / "k_gemv_c1_dram_traffic.txt").write_text(
        "# comment = ignored\n"
        f"workload = {workload}\nbatch = {batch}\n"
        f"kernel_source_sha256 = {h}\ndram_bytes_per_launch = {nbytes}\n")


def test_traffic_reported_for_the_captured_launch(tmp_path, monkeypatch):
    _record(tmp_path, "abcd" * 4)
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.traffic_per_launch("abcd" * 4, "c1", 1) == 107516672.0


def test_traffic_not_reused_for_other_kernels_workloads_or_batches(tmp_path, monkeypatch):
    _record(tmp_path, "abcd" * 4)
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.traffic_per_launch("0" * 16, "c1", 1) is None
    assert bench.traffic_per_launch("abcd" * 4, "c3", 1) is None
    assert bench.traffic_per_launch("abcd" * 4, "c1", 16) is None


def test_no_record_no_traffic(tmp_path, monkeypatch):
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.traffic_per_launch("abcd" * 4, "c1", 1) is None


def test_kernel_hash_covers_the_fused_kernel_sources():
    assert set(bench.KERNEL_SOURCES) >= {"gemv.cu", "seedq_internal.cuh"}
    h = bench.kernel_source_hash()
    assert len(h) == 16 and int(h, 16) >= 0
    assert h == bench.kernel_source_hash()
