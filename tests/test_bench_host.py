"""Host logic of bench.py (no GPU): the committed DRAM-traffic record of a kernel is reported only
while the kernel source it was captured from, and every header that source includes, is unchanged."""
import json
import os

import bench


def test_captured_traffic_follows_the_kernel_source(tmp_path, monkeypatch):
    src = tmp_path / "k.cu"
    src.write_text('#include "a.cuh"\nkernel v1')
    (tmp_path / "a.cuh").write_text('#include "b.h"\nhelpers v1')
    (tmp_path / "b.h").write_text("decls v1")
    prof = tmp_path / "profiles"
    prof.mkdir()
    rec = {"w": {"source": "k.cu", "source_sha256": bench.source_digest(str(src)),
                 "dram_bytes_read": 100, "dram_bytes_write": 20, "summary": "profiles/w.md"}}
    (prof / "traffic.json").write_text(json.dumps(rec))
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.captured_traffic("w") == 120
    assert bench.captured_traffic("other") is None
    (tmp_path / "b.h").write_text("decls v2")   # a header two includes deep changed
    assert bench.captured_traffic("w") is None
    (tmp_path / "b.h").write_text("decls v1")
    assert bench.captured_traffic("w") == 120
    src.write_text('#include "a.cuh"\nkernel v2')   # the kernel itself changed
    assert bench.captured_traffic("w") is None


def test_committed_traffic_record_is_well_formed():
    rec = json.load(open(os.path.join(bench.ROOT, "profiles", "traffic.json")))
    assert rec
    for workload, e in rec.items():
        assert workload in bench.WORKLOADS
        assert os.path.exists(os.path.join(bench.ROOT, e["source"]))
        assert os.path.exists(os.path.join(bench.ROOT, e["summary"]))
        assert e["dram_bytes_read"] > 0 and e["dram_bytes_write"] >= 0
        assert len(e["source_sha256"]) == 64


def test_prefill_scoring_flops_counts_causal_pairs():
    """The setup roofline's FLOPs: 2 products x 2 D per causal (query row, key) pair per query head,
    against a brute-force count of the visible pairs (H2O: every row; SnapKV: a window)."""
    import bench
    for (B, Hq, D, T, rows) in [(1, 1, 64, 7, 7), (2, 4, 128, 50, 50), (1, 2, 64, 40, 8), (3, 8, 128, 33, 1)]:
        pos0 = T - rows
        pairs = sum(1 for i in range(rows) for j in range(T) if j <= pos0 + i)
        assert bench.prefill_scoring_flops(B, Hq, D, T, rows) == 2 * 2 * D * pairs * B * Hq
