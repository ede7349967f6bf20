"""GPU parity of the dense search (both kernel families) against the fp64
oracle: hand-worked fixture, the paper-shaped workloads, ragged shapes that
span several tiles, ties and degenerate inputs.  Scores must be within 1e-4 of
the oracle; ids must match except inside near-tie blocks (oracle/check.py)."""
import numpy as np
import pytest
import torch

import oracle
from oracle import check
from paper_2608_08340_gb300 import workloads
from paper_2608_08340_gb300.index import Index

from _golden import load
from _gpu import TOL, check_dense, dev_tensor

pytestmark = pytest.mark.gpu


def _index(data, dtype=None):
    return Index(dev_tensor(data), dtype)


@pytest.mark.parametrize("dtype,path", [("f32", None), ("bf16", "simt"), ("bf16", "tc")])
def test_golden_hand_worked(dtype, path):
    g = load("dense_8chunk.json")
    # the library needs d % 8 == 0: pad the 4-d fixture with zero columns
    E = np.zeros((8, 8), np.float32)
    E[:, :4] = np.asarray(g["E"], np.float32)
    Q = np.zeros((4, 8), np.float32)
    Q[:, :4] = np.asarray(g["Q"], np.float32)
    if dtype == "bf16":
        E, Q = oracle.round_bf16(E), oracle.round_bf16(Q)
    idx = _index(E)
    if path:
        idx.force_path(path)
    ids, sc = idx.search(dev_tensor(Q), g["k"])
    assert ids.cpu().tolist() == g["ids"]
    assert sc.cpu().tolist() == [[float(v) for v in r] for r in g["scores"]]
    if path:
        assert idx.last_path == path


def test_config0_tiny_fp32():
    w = workloads.config(0)
    idx = _index(w.E_data)
    ids, sc = idx.search(dev_tensor(w.Q_data), w.k)
    assert idx.last_path == "simt"
    check_dense(ids, sc, w.E_data, w.Q_data, w.k, "cfg0")


@pytest.fixture(scope="module")
def cfg1():
    w = workloads.config(1, batch=256)
    return w, _index(w.E_data)


@pytest.mark.parametrize("q", [1, 32, 256])
@pytest.mark.parametrize("path", [None, "simt", "tc"])
def test_config1_paper_shaped(cfg1, q, path):
    w, idx = cfg1
    idx.force_path(path)
    try:
        ids, sc = idx.search(dev_tensor(w.Q_data[:q]), w.k)
        torch.cuda.synchronize()
    finally:
        idx.force_path(None)
    check_dense(ids, sc, w.E_data, w.Q_data[:q], w.k, f"cfg1 q={q} path={path}")
    idx.check()


@pytest.mark.parametrize("n,d,q,k", [
    (1000, 64, 3, 5),          # n not a multiple of any tile
    (4097, 136, 17, 10),       # d not a multiple of the 64-wide K block
    (300, 384, 129, 100),      # k close to n, q just past one query tile
    (5000, 128, 257, 1),       # k = 1, three query tiles
    (2000, 256, 2, 256),       # k = K_MAX
    (700, 64, 255, 33),        # list length 128 for k = 33
])
@pytest.mark.parametrize("path", ["simt", "tc"])
def test_ragged_shapes(n, d, q, k, path):
    rng = np.random.default_rng(n + d + q + k)
    E = workloads.to_bf16_bits(workloads._normalise(rng.standard_normal((n, d)).astype(np.float32)))
    Q = workloads.to_bf16_bits(workloads._normalise(rng.standard_normal((q, d)).astype(np.float32)))
    idx = _index(E)
    idx.force_path(path)
    ids, sc = idx.search(dev_tensor(Q), k)
    assert idx.last_path == path
    check_dense(ids, sc, E, Q, k, f"ragged n={n} d={d} q={q} k={k} {path}")


@pytest.mark.parametrize("bn", [128, 256])
def test_tc_tile_widths_agree(bn):
    w = workloads.config(1, n=9000, batch=300)
    idx = _index(w.E_data)
    idx.force_path("tc")
    idx.force_block_n(bn)
    ids, sc = idx.search(dev_tensor(w.Q_data), 10)
    check_dense(ids, sc, w.E_data, w.Q_data, 10, f"bn={bn}")


@pytest.mark.parametrize("path", ["simt", "tc"])
def test_duplicate_rows_tie_to_lower_id(path):
    rng = np.random.default_rng(5)
    base = rng.standard_normal((64, 128)).astype(np.float32)
    E = np.concatenate([base, base, base])          # every row three times
    Eb = oracle.round_bf16(E)
    Qb = Eb[[3, 70, 150]]
    idx = _index(Eb)
    idx.force_path(path)
    ids, sc = idx.search(dev_tensor(Qb), 3)
    ids = ids.cpu().numpy()
    sc = sc.cpu().numpy()
    for i, r in enumerate([3, 70, 150]):
        assert ids[i].tolist() == [r % 64, r % 64 + 64, r % 64 + 128]
        assert sc[i, 0] == sc[i, 1] == sc[i, 2]


@pytest.mark.parametrize("path", ["simt", "tc"])
def test_all_scores_equal_returns_lowest_ids(path):
    E = oracle.round_bf16(np.ones((500, 64), np.float32))
    Q = np.zeros((5, 64), np.uint16)                  # zero queries: every score is 0
    idx = _index(E)
    idx.force_path(path)
    ids, sc = idx.search(dev_tensor(Q), 7)
    assert ids.cpu().tolist() == [list(range(7))] * 5
    assert (sc.cpu().numpy() == 0).all()


def test_k_equal_n_is_full_sort():
    w = workloads.config(0, n=200, batch=4)
    idx = _index(w.E_data)
    ids, sc = idx.search(dev_tensor(w.Q_data), 200)
    check_dense(ids, sc, w.E_data, w.Q_data, 200, "k=n")


def test_argument_errors():
    w = workloads.config(0, n=100, batch=2)
    idx = _index(w.E_data)
    Q = dev_tensor(w.Q_data)
    for k in (0, 101, 257):
        with pytest.raises(Exception):
            idx.search(Q, k)
    ids, sc = idx.search(Q[:0], 5)                    # q = 0 is a no-op
    assert ids.shape == (0, 5)
    with pytest.raises(Exception):
        idx.search(Q.to(torch.bfloat16), 5)           # dtype mismatch


def test_search_host_matches_device_search():
    w = workloads.config(1, n=8192, batch=40)
    idx = _index(w.E_data)
    Qd = dev_tensor(w.Q_data)
    ids_d, sc_d = idx.search(Qd, 5)
    ids_h, sc_h = idx.search_host(Qd.cpu().pin_memory(), 5)
    assert torch.equal(ids_d.cpu(), ids_h)
    assert torch.equal(sc_d.cpu(), sc_h)


def test_fp32_input_into_bf16_index_rounds_to_nearest_even():
    w = workloads.config(0, n=512, batch=4)        # fp32 data
    idx = Index(dev_tensor(w.E_data), torch.bfloat16)
    got = idx.rows().view(torch.int16).numpy().view(np.uint16)
    np.testing.assert_array_equal(got, oracle.round_bf16(w.E_data))
    idx2 = Index(torch.from_numpy(w.E_data), torch.bfloat16)   # from host memory
    got2 = idx2.rows().view(torch.int16).numpy().view(np.uint16)
    np.testing.assert_array_equal(got2, got)


def test_config2_clustered_near_ties_every_query():
    """All 4096 queries of the clustered workload against the oracle."""
    w = workloads.config(2)
    idx = _index(w.E_data)
    ids, sc = idx.search(dev_tensor(w.Q_data), w.k)
    assert idx.last_path == "tc"
    check_dense(ids, sc, w.E_data, w.Q_data, w.k, "cfg2")
    idx.check()


def _lane_quarter_rows(q, seed):
    """Two random rows in every 32-query group (TMEM lane quarter) of every
    128-query tile."""
    rng = np.random.default_rng(seed)
    return np.sort(np.concatenate([rng.choice(np.arange(lo, min(q, lo + 32)),
                                              min(2, q - lo), replace=False)
                                   for lo in range(0, q, 32)]))


@pytest.mark.slow
def test_config4_scale_with_upserts_sampled():
    """1M x 768 bf16, 4 batches of 2048 queries, 4096-row upserts before
    batches 2-4; sampled queries of every batch checked against the oracle
    run on the post-upsert index."""
    w = workloads.config(4, batch=8192)
    E = w.E_data.copy()
    idx = _index(E)
    idx.enable_timing(True)
    for b in range(4):
        if b > 0:
            up_ids, up_rows = workloads.upsert_batch(w.n, w.d, 4096, b, "bf16")
            idx.upsert(up_ids, dev_tensor(up_rows))
            oracle.upsert(E, up_ids, up_rows)
        Qb = w.Q_data[b * 2048:(b + 1) * 2048]
        ids, sc = idx.search(dev_tensor(Qb), w.k)
        # the full-size path: CTA pairs, sampled first pass and counted floors
        assert idx.last_launch["cluster"] == 2
        assert idx.last_timing()["sample_ms"] > 0.0
        # 128 rows: two in every lane quarter of all 16 query tiles
        rows = _lane_quarter_rows(2048, seed=b)
        assert len(rows) == 128
        check_dense(ids, sc, E, Qb, w.k, f"cfg4 batch {b}", rows=rows)
    # the index equals the oracle's post-upsert array
    got = idx.rows().view(torch.int16).numpy().view(np.uint16)
    np.testing.assert_array_equal(got, E)
    idx.check()


@pytest.mark.parametrize("k", [33, 100, 256])
def test_large_k_with_sampled_floor(k):
    """k > 32 over many corpus tiles: the search first scans every 32nd tile
    to get a lower bound of each query's k-th best score, then the full scan
    admits only scores above it.  Results must still be exact."""
    rng = np.random.default_rng(k)
    n, d, q = 160000, 128, 130
    E = workloads.to_bf16_bits(workloads._normalise(rng.standard_normal((n, d)).astype(np.float32)))
    Q = workloads.to_bf16_bits(workloads._normalise(rng.standard_normal((q, d)).astype(np.float32)))
    idx = _index(E)
    ids, sc = idx.search(dev_tensor(Q), k)
    assert idx.last_path == "tc"
    rows = np.sort(rng.choice(q, 12, replace=False))
    check_dense(ids, sc, E, Q, k, f"large k={k}", rows=rows)
    idx.check()


def test_large_k_exact_ties_at_kth():
    """k = 100 over 1500 distinct rows, each stored 30 times (45000 rows, so
    the sampled first pass and the counted floors run): the 100th result
    falls inside a group of 30 equal scores, and the merge, which drops keys
    below the proven floor, must still return the group's lowest ids."""
    rng = np.random.default_rng(0)
    m, reps, d = 1500, 30, 128
    base = oracle.round_bf16(workloads._normalise(rng.standard_normal((m, d)).astype(np.float32)))
    E = np.ascontiguousarray(np.tile(base, (reps, 1)))
    qrows = [3, 777, 1400]
    Q = np.ascontiguousarray(base[qrows])
    Bf = oracle.bf16_to_f32(base).astype(np.float64)
    for r in qrows:       # distinct rows' scores are far apart, so only ties are ambiguous
        s = np.sort(Bf @ Bf[r])[::-1]
        assert (-np.diff(s[:6])).min() > 10 * TOL
    o_ids, _ = oracle.search(E, Q, 100)
    idx = _index(E)
    ids, sc = idx.search(dev_tensor(Q), 100)
    assert idx.last_path == "tc"
    ids, sc = ids.cpu().numpy(), sc.cpu().numpy()
    np.testing.assert_array_equal(ids, o_ids)
    for i in range(len(qrows)):
        grp = ids[i] % m
        for g in np.unique(grp):
            assert len(set(sc[i][grp == g].tolist())) == 1     # copies score alike
    idx.check()


def test_shared_bound_tags_wrap_around():
    """Searches share per-query k-th score bounds tagged with a 32-bit
    generation; when the tag wraps, the bounds array is cleared.  Results
    across the wrap must equal those of a fresh index."""
    from paper_2608_08340_gb300 import _lib
    w = workloads.config(1, n=20000, batch=300)
    ref = _index(w.E_data)
    r_ids, r_sc = ref.search(dev_tensor(w.Q_data), 10)
    idx = _index(w.E_data)
    # Corpus rows as queries: their bounds (self-matches, scores near 1) would
    # wreck the next queries' results if an entry of this search were ever
    # read as current.  This search gets tag 1; the wrap below reuses tag 1.
    idx.search(dev_tensor(w.E_data[:300]), 10)
    idx.set_option(_lib.OPRAG_OPT_BOUND_TAG, -3)         # tag 0xFFFFFFFD
    for _ in range(4):                                   # 0xFFFFFFFE, 0xFFFFFFFF, wrap to 1, 2
        ids, sc = idx.search(dev_tensor(w.Q_data), 10)
        torch.cuda.synchronize()
        assert torch.equal(ids, r_ids)
        assert (sc - r_sc).abs().max().item() == 0.0
    idx.check()


@pytest.mark.parametrize("q,k", [(1024, 5), (1024, 16), (4096, 7), (256, 12),
                                 (1, 5), (37, 16), (200, 9), (600, 16), (600, 3)])
def test_merge_regimes(q, k):
    """The final merge runs as one warp per query over at most 32 partial
    lists (large batches), one, two or four warps per query over more lists
    when k <= 16 (by batch size), or one CTA per query for larger k; all
    must give the exact top-k."""
    rng = np.random.default_rng(q + k)
    n, d = 40000, 256
    E = workloads.to_bf16_bits(workloads._normalise(rng.standard_normal((n, d)).astype(np.float32)))
    Q = workloads.to_bf16_bits(workloads._normalise(rng.standard_normal((q, d)).astype(np.float32)))
    idx = _index(E)
    ids, sc = idx.search(dev_tensor(Q), k)
    assert idx.last_path == "tc"
    rows = np.sort(rng.choice(q, min(q, 40), replace=False))
    check_dense(ids, sc, E, Q, k, f"merge q={q} k={k}", rows=rows)
    idx.check()
