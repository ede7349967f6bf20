"""Host-side pieces of bench.py (no GPU): argument parsing, workload names,
roofline terms, peaks and the traffic-record lookup, so that the bench's
helpers stay importable and consistent."""
import json
import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402
from paper_2608_08340_gb300 import workloads  # noqa: E402


def test_parse_defaults(monkeypatch):
    monkeypatch.setattr(sys, "argv", ["bench.py"])
    a = bench.parse()
    assert a.gpus == 1 and a.config == 1 and a.impl == "ours" and a.warmup >= 3


def test_roofline_terms_and_names():
    w = workloads.config(1, batch=256)
    nbytes, flops = bench.roofline_terms(w, 1)
    assert nbytes == w.n * w.d * 2 + w.q * w.d * 2
    assert flops == 2.0 * w.q * w.n * w.d
    assert "32768 x 768" in bench.workload_name(1, w)


def test_peaks_and_traffic_records():
    hbm, burst, sustained, src = bench.peaks()
    assert hbm > 0 and burst >= sustained > 0
    with open(os.path.join(ROOT, "profiles", "ncu_traffic.json")) as f:
        table = json.load(f)
    for key, ent in table.items():
        assert ent["dram_bytes_per_launch"] > 0
        # a record is used only while the kernel's code is unchanged
        got = bench.ncu_traffic(key)
        assert got is None or got == ent["dram_bytes_per_launch"]


def test_source_hash_ignores_comments():
    base = bench.source_hash()
    texts = {n: open(os.path.join(ROOT, "paper_2608_08340_gb300", "csrc", n)).read()
             for n in bench.KERNEL_SOURCES}
    commented = bench.source_hash(lambda n: "// note\n" + texts[n] + "\n/* more */\n")
    changed = bench.source_hash(lambda n: texts[n] + ("\nint x;" if n == "search_tc.cu" else ""))
    assert commented == base and changed != base


@pytest.mark.parametrize("cfg", [0, 1, 2, 3, 4])
def test_default_batches(cfg):
    assert bench.default_batch(cfg) > 0
