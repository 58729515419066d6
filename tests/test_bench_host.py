"""Host-side accounting of bench.py, on CPU.

The roofline bytes follow the measurement definition of the path: one read
of g plus the (idx, val) codes written by the sparsifier, the codes read
back and the dense sum written by the aggregate.  A DRAM-traffic figure is
reported only while it was taken on the kernel's current source: any edit
of the files that define the kernel turns it into null until it is measured
again.
"""
import os
import shutil

import pytest

import bench

REAL_ROOT = bench.ROOT


def test_algorithmic_bytes_per_step():
    M, d, nnz = 16, 1 << 24, 2682416
    sp, ag = bench.algorithmic_bytes(M, d, 4, nnz)
    assert sp == M * d * 4 + nnz * 8          # one read of fp32 g + the codes written
    assert ag == nnz * 8 + d * 4              # the codes read + the dense fp32 sum written
    sp16, _ = bench.algorithmic_bytes(M, d, 2, nnz)
    assert sp - sp16 == M * d * 2             # bf16 halves only the read of g


def test_job_throughput_counts_every_rank():
    # 1e6 units per rank, 2 ms for the slowest rank, 4 ranks: 2e9 units/s.
    assert bench.job_throughput(1e6, 2.0, 4) == pytest.approx(2e9)


def _tree(tmp_path, traffic_lines):
    """A copy of the files load_traffic reads, under tmp_path."""
    src = os.path.join(REAL_ROOT, "paper_1710_09854_gb300", "csrc")
    dst = tmp_path / "paper_1710_09854_gb300" / "csrc"
    dst.mkdir(parents=True)
    for fn in bench.KERNEL_SOURCES["k_stream_tma"]:
        shutil.copy(os.path.join(src, fn), dst / fn)
    (tmp_path / "profiles").mkdir()
    (tmp_path / "profiles" / "traffic.txt").write_text("\n".join(traffic_lines) + "\n")
    return dst


def test_traffic_is_reported_only_for_the_measured_source(tmp_path, monkeypatch):
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    key = ("k_stream_tma", "c3_d16777216_M16_student_t3", "f32", 0.01)
    dst = _tree(tmp_path, [])
    digest = bench.source_digest("k_stream_tma")
    (tmp_path / "profiles" / "traffic.txt").write_text(
        "# comment\n"
        f"k_stream_tma c3_d16777216_M16_student_t3 f32 0.01 1234567 {digest}\n"
        f"k_stream_tma c5_other f32 0.01 7654321 {'0' * 64}\n")
    assert bench.load_traffic(*key) == 1234567
    assert bench.load_traffic("k_stream_tma", "c5_other", "f32", 0.01) is None   # taken on other source
    assert bench.load_traffic("k_stream_tma", "c3_d16777216_M16_student_t3", "bf16", 0.01) is None
    assert bench.load_traffic("k_sum", "c3_d16777216_M16_student_t3", "f32", 0.01) is None
    # Any edit of the kernel's sources (a comment included) voids the figure.
    with open(dst / "gs_stream_tma.cu", "a") as f:
        f.write("\n// edited\n")
    assert bench.source_digest("k_stream_tma") != digest
    assert bench.load_traffic(*key) is None


def test_missing_traffic_file_reports_null(tmp_path, monkeypatch):
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.load_traffic("k_stream_tma", "c3_d16777216_M16_student_t3", "f32", 0.01) is None


def test_peak_falls_back_without_measured_file(tmp_path, monkeypatch):
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.peaks() == (6800.0, "fallback")
    (tmp_path / "MEASURED_PEAKS.json").write_text('{"hbm_gbs": 6791.4}')
    assert bench.peaks() == (6791.4, "measured")


def _rec(lam, sum_p, capped=0, iters_run=2, flags=0):
    return {"lambda": lam, "sum_p": sum_p, "capped": capped, "iters_run": iters_run, "flags": flags}


def test_algorithm3_summary():
    kappa = 0.01
    recs = [_rec(0.5, 10.0, capped=3), _rec(0.25, 9.0, iters_run=1), _rec(1.0, 10.0, iters_run=3, flags=1)]
    s = bench.alg3_summary(recs, kappa, [1000, 1000, 1000])
    assert s["records"] == 3
    assert (s["lambda_min"], s["lambda_max"]) == (0.25, 1.0)
    assert s["sum_p_over_budget_min"] == pytest.approx(0.9)
    assert s["sum_p_over_budget_max"] == pytest.approx(1.0)
    assert s["iters_run"] == {"1": 1, "2": 1, "3": 1}
    assert s["capped_total"] == 3 and s["exact_fallbacks"] == 1


class _FakeGS:
    """Stands in for the binding: records the calls, returns given records."""
    GS_OK = 0

    def __init__(self, recs, rc=0):
        self.recs, self.rc, self.calls = recs, rc, []

    def info_tensor(self, n):
        return n

    def gs_batched_sparsify(self, g, kappa, iters, seed, step, worker0, idx, val, nnz, info=None, stream=None):
        self.calls.append(("batched", info, iters, seed))

    def gs_segmented_sparsify(self, g, off, kappa, iters, seed, step, worker0, idx, val, nnz, info=None,
                              stream=None):
        self.calls.append(("segmented", info, iters, seed))

    def gs_sync_status(self, stream):
        return self.rc

    def status_string(self, rc):
        return f"status {rc}"

    def decode_info(self, n):
        return self.recs[:n]


def test_algorithm3_state_call(monkeypatch):
    import types
    import numpy as np
    import torch
    monkeypatch.setattr(torch.cuda, "synchronize", lambda *a, **k: None)
    w = types.SimpleNamespace(iters=3, seed=7)
    kappa = 0.1
    # Whole rows: one record per worker, budget kappa * d.
    g = np.zeros((2, 50))
    fake = _FakeGS([_rec(1.0, 5.0), _rec(2.0, 4.0)])
    s = bench.run_alg3_state(fake, g, None, kappa, w, None, None, None, None)
    assert fake.calls == [("batched", 2, 3, 7)]
    assert (s["sum_p_over_budget_min"], s["sum_p_over_budget_max"]) == (pytest.approx(0.8), pytest.approx(1.0))
    # Layer-wise: records ordered worker by worker, segment by segment.
    off = np.array([0, 10, 30])
    fake = _FakeGS([_rec(1.0, 1.0), _rec(1.0, 2.0), _rec(1.0, 1.0), _rec(1.0, 1.0)])
    s = bench.run_alg3_state(fake, np.zeros((2, 30)), off, kappa, w, None, None, None, None)
    assert fake.calls == [("segmented", 4, 3, 7)]
    assert s["records"] == 4
    assert s["sum_p_over_budget_min"] == pytest.approx(0.5)     # worker 1, segment 1: 1 of a budget of 2
    assert s["sum_p_over_budget_max"] == pytest.approx(1.0)
    # A device error is reported, not raised.
    s = bench.run_alg3_state(_FakeGS([], rc=3), g, None, kappa, w, None, None, None, None)
    assert s == {"error": "status 3"}
