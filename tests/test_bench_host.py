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


def test_byte_models_match_per_element_counts():
    """The roofline's algorithmic bytes (one decode launch of one layer) against a count that walks
    the cache token by token, page by page and dim by dim: FP16 and H2O K/V rows, KVQuant codes,
    value ranges, value outliers, CSR offsets and key-outlier entries, RocketKV candidate-page bounds
    of the chosen dims plus the K/V rows of the chosen and the tail pages (incl. a cache shorter
    than one page and one with fewer full pages than k_p)."""
    import bench

    def per_unit_fp16(T, D):
        return sum(2 * D * 2 for _ in range(T))            # K row + V row per token

    def per_unit_kvq(T, D, bits, n_v):
        b = 0
        for _ in range(T):
            b += D * bits // 8                               # key codes
            b += D * bits // 8                               # value codes
            b += 4 + 4                                       # value lo, scale (fp32)
            b += n_v * 4                                     # value outliers (channel << 16 | fp16)
            b += 4                                           # the token's CSR offset
        return b

    def per_unit_rocket(n, D, k_p, r_d, page=16):
        newest_page = (n - 1) // page
        candidates = list(range(newest_page))               # full pages before the newest token's page
        b = 0
        for _ in candidates:
            for _ in range(r_d):
                b += 2 + 2                                   # min and max (fp16) of a chosen dim
        chosen = candidates[:k_p]                            # how many, not which
        for _ in chosen:
            for _ in range(page):
                b += 2 * D * 2
        for _ in range(n - page * newest_page):              # the tail page's tokens
            b += 2 * D * 2
        return b

    for units, T, D in [(64, 8193, 128), (1, 1, 64), (3, 77, 64)]:
        assert bench.alg_bytes_fp16(units, T, D) == units * per_unit_fp16(T, D)
        assert bench.alg_bytes_h2o(units, T, D) == units * per_unit_fp16(T, D)
    for units, T, D, bits, n_v, n_out in [(64, 8198, 128, 4, 2, 81920), (2, 33, 64, 3, 1, 0), (5, 700, 128, 2, 13, 999)]:
        assert bench.alg_bytes_kvquant(units, T, D, bits, n_v, n_out) == units * per_unit_kvq(T, D, bits, n_v) + 4 * n_out
    for units, n, D, k_p, r_d in [(32, 4097, 128, 64, 32), (4, 1, 128, 64, 32), (4, 16, 64, 4, 16),
                                   (4, 17, 64, 4, 16), (2, 100, 64, 64, 16), (2, 4100, 128, 128, 32)]:
        assert bench.alg_bytes_rocket(units, n, D, k_p, r_d) == units * per_unit_rocket(n, D, k_p, r_d), (n, k_p)
    assert bench.overhead_bytes_h2o(128, 3278, 4) == 128 * sum(4 + 4 * 4 for _ in range(3278))


def test_reference_arm_prints_the_contract_line():
    """`bench.py --impl reference` (the fp64 oracle on the host cores, a bounded sample of the headline
    workload) prints one JSON line with the contract's keys, its cpu_baseline and a zero-copy e2e."""
    import json
    import os
    import subprocess
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    out = subprocess.run([sys.executable, "bench.py", "--impl", "reference", "--steps", "1", "--warmup", "0",
                          "--cpu-budget", "1"], cwd=root, capture_output=True, text=True, timeout=600)
    assert out.returncode == 0, out.stderr[-2000:]
    line = json.loads(out.stdout.strip().splitlines()[-1])
    for key in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better",
                "scaling", "vs_baseline", "dtype", "data", "config", "cpu_baseline", "e2e"):
        assert key in line, key
    assert line["impl"] == "reference" and line["value"] > 0 and line["higher_is_better"] is True
    assert line["config"]["workload"] == "kvquant_nuq4_b8_t8192"
    cb = line["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["value"] == line["value"] and cb["sample"]
    assert line["e2e"] == {"value": line["value"], "unit": line["unit"], "h2d_bytes_per_step": 0,
                           "d2h_bytes_per_step": 0}
