"""Host-side arithmetic of bench.py: the per-stage roofline (no GPU)."""
import math
import os
import sys

sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))

import bench  # noqa: E402
import synth  # noqa: E402
from paper_1512_06473_gb300 import costmodel as cm  # noqa: E402

SMEM, HBM = 40273.9, 6781.4  # GB/s


def test_batch1_bounds_and_fractions():
    """AlexNet at batch 1: the conv layers are shared-memory bound, fc6-fc8
    HBM bound by their codes (fc6: 9.44 MB of codes against 37.7 MB of
    look-ups at 6x the bandwidth), max-pools HBM bound; a stage that takes
    exactly its roof time reads 1.0."""
    w = synth.alexnet()
    ms = [1.0] * len(w.layers)
    st = bench.stage_rooflines(w, cm, ms, 1, SMEM, HBM)
    kinds = [(s["kind"], s["bound"]) for s in st]
    assert kinds == [("conv", "smem"), ("maxpool", "hbm"), ("conv", "smem"), ("maxpool", "hbm"),
                     ("conv", "smem"), ("conv", "smem"), ("conv", "smem"), ("maxpool", "hbm"),
                     ("fc", "hbm"), ("fc", "hbm"), ("fc", "hbm")]
    fc6 = w.layers[8]
    M = fc6.Cs // fc6.Csp
    hbm_bytes = 4.0 * (fc6.Cs + fc6.Ct) + fc6.Ct * M + 4.0 * M * fc6.K * fc6.Csp
    roof_ms = hbm_bytes / (HBM * 1e9) * 1e3
    again = bench.stage_rooflines(w, cm, [roof_ms if j == 8 else 1.0 for j in range(len(ms))], 1,
                                  SMEM, HBM)
    assert math.isclose(again[8]["frac"], 1.0, rel_tol=1e-3)


def test_batch128_conv2_matches_the_headline_roofline():
    """At batch 128 conv2 is shared-memory bound with the algorithmic bytes
    bench.py's headline roofline uses (58.48 GB per launch)."""
    w = synth.alexnet()
    st = bench.stage_rooflines(w, cm, [2.0] * len(w.layers), 128, SMEM, HBM)
    assert st[2]["bound"] == "smem"
    alg = 58.477510656e9  # bytes per launch
    assert math.isclose(st[2]["frac"], alg / 2e-3 / (SMEM * 1e9), rel_tol=1e-4)


def test_recorded_traffic_follows_the_kernel_sources(tmp_path, monkeypatch):
    """The DRAM record counts only while the hashed kernel sources are the
    ones it was taken with; another workload, batch or layer has none."""
    import hashlib
    import json
    src = tmp_path / "k.cu"
    src.write_text("kernel v1\n")
    (tmp_path / "profiles").mkdir()
    rec = {"workload": "w", "batch": 4, "layer": 2, "dram_read_bytes": 100,
           "dram_write_bytes": 20, "sources": ["k.cu"],
           "sha256": hashlib.sha256(b"kernel v1\n").hexdigest()}
    (tmp_path / "profiles" / "dram_traffic.txt").write_text("# header\n" + json.dumps(rec) + "\n")
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.recorded_traffic("w", 4, 2) == 120
    assert bench.recorded_traffic("w", 8, 2) is None
    assert bench.recorded_traffic("w", 4, 3) is None
    src.write_text("kernel v2\n")
    assert bench.recorded_traffic("w", 4, 2) is None


def test_job_throughput_counts_every_rank():
    """value = the images all ranks processed / the slowest rank's time."""
    assert bench.job_throughput(128, 1, 20, 0.1331) == 128 * 20 / 0.1331
    assert bench.job_throughput(128, 4, 20, 0.2) == 4 * bench.job_throughput(128, 1, 20, 0.2)
