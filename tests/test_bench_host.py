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
    assert a.gpus == 1 and a.config is None and a.impl == "ours" and a.warmup >= 3
    # no --config: the scale workload is the headline, every other one a sub-entry
    assert bench.HEADLINE == (4, 2048)
    assert sorted(c for c, _ in bench.SUB_WORKLOADS) == [0, 1, 1, 1, 2, 3]


@pytest.mark.parametrize("q", [1, 16, 64, 65, 256, 1000, 2048, 4096])
def test_parity_rows_cover_every_lane_quarter_of_every_tile(q):
    rows = bench.parity_rows(q, seed=3)
    assert len(set(rows.tolist())) == len(rows) and rows.min() >= 0 and rows.max() < q
    if q <= 64:
        assert rows.tolist() == list(range(q))
    else:
        groups = {int(r) // 32 for r in rows}
        assert groups == set(range((q + 31) // 32))      # tile t, quarter g: group 4 t + g


def test_upsert_sequence_replays_the_step_order():
    assert bench.upsert_sequence(5, 3) == [0, 1, 2, 3, 0, 0, 1, 2]


def test_both_arms_print_the_same_config():
    w = workloads.config(0)
    ours = bench.config_dict(0, w, 1)
    assert ours == bench.config_dict(0, w, 1)
    assert {"workload", "n", "d", "q", "k", "l2", "parallelism"} <= set(ours)


def test_sparse_terms_count_postings_by_brute_force():
    w = workloads.config(3, n=50, batch=4)
    got = bench.sparse_terms(w)
    df = {}
    for dd in range(w.n):
        for t in set(w.doc_terms[w.doc_indptr[dd]:w.doc_indptr[dd + 1]].tolist()):
            df[t] = df.get(t, 0) + 1
    assert got["postings_visited"] == sum(df.get(int(t), 0) for t in w.q_terms)
    assert got["postings_distinct_terms"] == sum(df.get(int(t), 0) for t in set(w.q_terms.tolist()))
    nbytes, _ = bench.roofline_terms(w, 3)
    assert nbytes == w.n * w.d * 2 + w.q * w.d * 2 + 8 * got["postings_distinct_terms"]


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
