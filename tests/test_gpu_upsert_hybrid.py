"""GPU parity of upsert and of the hybrid (dense + BM25) search against the
fp64 oracle."""
import numpy as np
import pytest
import torch

import oracle
from oracle import check
from paper_2608_08340_gb300 import workloads
from paper_2608_08340_gb300.index import Index

from _golden import load, value
from _gpu import TOL, check_dense, dev_tensor, oracle_topk

pytestmark = pytest.mark.gpu


def _bits(idx):
    return idx.rows().view(torch.int16).numpy().view(np.uint16)


# ------------------------------------------------------------------ upsert

@pytest.mark.parametrize("on_device", [False, True])
def test_upsert_duplicates_last_wins(on_device):
    w = workloads.config(1, n=3000, batch=8)
    idx = Index(dev_tensor(w.E_data))
    ids = np.array([5, 17, 5, 2999, 0, 17, 17], np.int64)
    rows = oracle.round_bf16(np.random.default_rng(3).standard_normal((7, w.d)).astype(np.float32))
    r = dev_tensor(rows) if on_device else dev_tensor(rows).cpu()
    idx.upsert(ids, r)
    E = w.E_data.copy()
    oracle.upsert(E, ids, rows)
    np.testing.assert_array_equal(_bits(idx), E)
    got_ids, got_sc = idx.search(dev_tensor(w.Q_data), 5)
    check_dense(got_ids, got_sc, E, w.Q_data, 5, "after upsert")


def test_upsert_out_of_range_writes_nothing():
    w = workloads.config(1, n=256, batch=2)
    idx = Index(dev_tensor(w.E_data))
    rows = dev_tensor(w.E_data[:2])
    for bad in ([0, 256], [-1, 3]):
        with pytest.raises(Exception) as e:
            idx.upsert(np.array(bad, np.int64), rows)
        assert "RANGE" in str(e.value)
    np.testing.assert_array_equal(_bits(idx), w.E_data)


@pytest.mark.parametrize("on_device", [False, True])
def test_upsert_fp32_rows_into_bf16_index(on_device):
    w = workloads.config(1, n=1024, batch=2)
    idx = Index(dev_tensor(w.E_data))
    rows = np.random.default_rng(9).standard_normal((33, w.d)).astype(np.float32)
    ids = np.arange(100, 133, dtype=np.int64)
    t = torch.from_numpy(rows)
    idx.upsert(ids, t.cuda() if on_device else t)
    E = w.E_data.copy()
    oracle.upsert(E, ids, rows)
    np.testing.assert_array_equal(_bits(idx), E)


def test_upsert_fp32_index():
    w = workloads.config(0, n=512, batch=4)
    idx = Index(dev_tensor(w.E_data))
    ids = np.array([1, 2, 3], np.int64)
    rows = w.Q_data[:3].copy()
    idx.upsert(ids, torch.from_numpy(rows))
    E = w.E_data.copy()
    oracle.upsert(E, ids, rows)
    np.testing.assert_array_equal(idx.rows().numpy(), E)
    got_ids, got_sc = idx.search(dev_tensor(w.Q_data), 5)
    assert got_ids.cpu().numpy()[:3, 0].tolist() == [1, 2, 3]     # self-match
    check_dense(got_ids, got_sc, E, w.Q_data, 5, "fp32 upsert")


def test_upsert_is_stream_ordered_before_search():
    w = workloads.config(1, n=4096, batch=4)
    idx = Index(dev_tensor(w.E_data))
    s = torch.cuda.Stream()
    target = np.array([4000], np.int64)
    with torch.cuda.stream(s):
        idx.upsert(target, dev_tensor(w.Q_data[:1]), stream=s)
        ids, sc = idx.search(dev_tensor(w.Q_data[:1]), 1, stream=s)
    s.synchronize()
    assert ids.item() == 4000


# ------------------------------------------------------------------ hybrid

def _csr(lists):
    indptr = np.zeros(len(lists) + 1, np.int32)
    indptr[1:] = np.cumsum([len(x) for x in lists])
    return indptr, np.array([t for x in lists for t in x], np.int32)


@pytest.mark.parametrize("path,gather", [("simt", False), ("tc", False), ("tc", True)])
def test_hybrid_golden_hand_worked(path, gather):
    g = load("hybrid_4doc.json")
    bm = load("bm25_4doc.json")
    E = np.zeros((4, 8), np.float32)
    E[:, :2] = np.asarray(g["E"], np.float32)
    Q = np.zeros((2, 8), np.float32)
    Q[:, :2] = np.asarray(g["Q"], np.float32)
    idx = Index(dev_tensor(oracle.round_bf16(E)))
    idx.force_path(path)
    dip, dt = _csr(bm["docs"])
    idx.set_sparse(dip, dt, bm["vocab"], bm["k1"], bm["b"])
    idx.gather_lexical(gather)
    qip, qt = _csr(g["query_terms"])
    ids, sc = idx.hybrid_search(dev_tensor(oracle.round_bf16(Q)), torch.from_numpy(qip),
                                torch.from_numpy(qt), g["alpha"], g["k"])
    want = np.array([[value(x) for x in r] for r in g["scores"]])
    # Materialised block: fp32 sums of the exact fp32 weights.  Gathered: a
    # head term's weight enters the tensor cores as a high + low bf16 pair,
    # within 2^-18 of it relatively, so the lexical half (1 - alpha) BM25 / max
    # is within about 2e-6.
    np.testing.assert_allclose(sc.cpu().numpy(), want, atol=1e-5 if gather else 1e-6)
    got = ids.cpu().tolist()
    assert got[0][0] == 0 and sorted(got[0][1:3]) == [1, 2] and got[0][3] == 3
    assert sorted(got[1][:2]) == [1, 2] and sorted(got[1][2:]) == [0, 3]


def _hybrid_check(idx, w, rows, alpha, label, k=None):
    k = k or w.k
    ids, sc = idx.hybrid_search(dev_tensor(w.Q_data), torch.from_numpy(w.q_indptr),
                                torch.from_numpy(w.q_terms), alpha, k)
    ids = ids.cpu().numpy()[rows]
    sc = sc.cpu().numpy()[rows]
    qip = np.zeros(len(rows) + 1, np.int32)
    qts = [w.q_terms[w.q_indptr[r]:w.q_indptr[r + 1]] for r in rows]
    qip[1:] = np.cumsum([len(t) for t in qts])
    qt = np.concatenate(qts).astype(np.int32)
    o_ids, o_sc = oracle_topk(
        lambda kout: oracle.hybrid_search(w.E_data, w.Q_data[rows], w.doc_indptr, w.doc_terms,
                                          w.vocab, qip, qt, alpha, kout, w.k1, w.b),
        k, w.n)
    return check.check_topk(ids, sc, o_ids, o_sc, k, TOL, n=w.n, label=label,
                            query_index=rows)


@pytest.fixture(scope="module")
def cfg3():
    w = workloads.config(3)
    idx = Index(dev_tensor(w.E_data))
    idx.set_sparse(w.doc_indptr, w.doc_terms, w.vocab, w.k1, w.b)
    return w, idx


@pytest.mark.parametrize("gather", [False, True])
def test_config3_hybrid_every_query(cfg3, gather):
    """All 1024 queries of the hybrid workload against the oracle, with the
    BM25 block and with the BM25 gathered in the search epilogue."""
    w, idx = cfg3
    idx.gather_lexical(gather)
    try:
        _hybrid_check(idx, w, np.arange(w.q), w.alpha, f"cfg3 gather={gather}")
    finally:
        idx.gather_lexical(False)
    assert idx.last_path == "tc"
    idx.check()


@pytest.mark.parametrize("alpha", [0.0, 1.0])
def test_config3_alpha_limits(cfg3, alpha):
    w, idx = cfg3
    rows = np.arange(0, w.q, 97)
    _hybrid_check(idx, w, rows, alpha, f"cfg3 alpha={alpha}")


@pytest.mark.parametrize("path", ["simt", "tc"])
def test_hybrid_small_both_paths_with_absent_and_repeated_terms(path):
    w = workloads.config(3, n=3000, batch=9)
    # query 0: a term no chunk holds; query 1: one term repeated; query 2: no terms
    terms = [list(w.q_terms[w.q_indptr[i]:w.q_indptr[i + 1]]) for i in range(w.q)]
    terms[0] = [w.vocab - 1]
    terms[1] = [terms[1][0]] * 4
    terms[2] = []
    w.q_indptr, w.q_terms = _csr(terms)
    idx = Index(dev_tensor(w.E_data))
    idx.force_path(path)
    idx.set_sparse(w.doc_indptr, w.doc_terms, w.vocab, w.k1, w.b)
    _hybrid_check(idx, w, np.arange(w.q), w.alpha, f"hybrid small {path}")


def test_hybrid_without_sparse_side_is_not_ready():
    w = workloads.config(1, n=256, batch=2)
    idx = Index(dev_tensor(w.E_data))
    with pytest.raises(Exception) as e:
        idx.hybrid_search(dev_tensor(w.Q_data), torch.tensor([0, 1, 2]), torch.tensor([1, 2]),
                          0.5, 5)
    assert "NOT_READY" in str(e.value)


# ---------------------------------------------------------------- both forms
# With OPRAG_OPT_LEX_GATHER the lexical part is gathered in the search
# epilogue: the 32 commonest terms through tensor-core MMAs of counts x split
# weights, terms in at least 1/32 of the chunks as fp32 rows (2 per query in
# the landing zone, further ones read directly), the others from their
# postings with per-thread cursors (up to 8 distinct terms), any further
# terms of a long query by a per-chunk search.  Each case runs both forms.


@pytest.mark.parametrize("gather", [False, True])
def test_hybrid_long_queries_with_repeats_and_many_terms(gather):
    """12-40 terms per query: more than 8 distinct postings terms (the
    overflow scan), repeated terms and head terms mixed in."""
    w = workloads.config(3, n=6000, batch=40)
    rng = np.random.default_rng(11)
    lists = []
    for i in range(w.q):
        tail = rng.integers(30, 3000, size=int(rng.integers(12, 41))).tolist()
        head = rng.integers(0, 12, size=3).tolist()
        t = tail + head + tail[:4]                  # the first four tail terms twice
        rng.shuffle(t)
        lists.append(t)
    w.q_indptr, w.q_terms = _csr(lists)
    idx = Index(dev_tensor(w.E_data))
    idx.set_sparse(w.doc_indptr, w.doc_terms, w.vocab, w.k1, w.b)
    idx.gather_lexical(gather)
    _hybrid_check(idx, w, np.arange(w.q), w.alpha, f"long queries gather={gather}")
    assert idx.last_path == "tc"
    idx.check()


@pytest.mark.parametrize("gather", [False, True])
def test_hybrid_more_head_terms_than_tensor_core_slots(gather):
    """60 terms occur in most chunks: the 32 commonest are scored on tensor
    cores, the other 28 through their postings."""
    rng = np.random.default_rng(12)
    n, vocab = 3000, 500
    bags = []
    for _ in range(n):
        common = [t for t in range(60) if rng.random() < 0.85] * int(rng.integers(1, 3))
        bags.append(common + rng.integers(60, vocab, size=int(rng.integers(20, 60))).tolist())
    w = workloads.config(3, n=n, batch=70)
    w.doc_indptr, w.doc_terms = _csr(bags)
    w.vocab = vocab
    lists = [rng.integers(0, 60, size=5).tolist() + rng.integers(60, vocab, size=4).tolist()
             for _ in range(w.q)]
    w.q_indptr, w.q_terms = _csr(lists)
    idx = Index(dev_tensor(w.E_data))
    idx.set_sparse(w.doc_indptr, w.doc_terms, w.vocab, w.k1, w.b)
    idx.gather_lexical(gather)
    for alpha in (w.alpha, 0.0):
        _hybrid_check(idx, w, np.arange(w.q), alpha, f"60 head terms alpha={alpha}")


@pytest.mark.parametrize("gather", [False, True])
@pytest.mark.parametrize("k", [33, 100])
def test_hybrid_large_k_with_sampled_floor(k, gather):
    """k > 32 over 313 corpus tiles: the sampled first pass (every 32nd tile,
    so the postings cursors are placed again at every unit) runs the fused
    epilogue too."""
    w = workloads.config(3, n=40000, batch=130)
    idx = Index(dev_tensor(w.E_data))
    idx.set_sparse(w.doc_indptr, w.doc_terms, w.vocab, w.k1, w.b)
    idx.gather_lexical(gather)
    idx.enable_timing(True)
    rows = np.sort(np.random.default_rng(k).choice(w.q, 24, replace=False))
    _hybrid_check(idx, w, rows, w.alpha, f"hybrid k={k}", k=k)
    assert idx.last_timing()["sample_ms"] > 0.0
    idx.check()


@pytest.mark.parametrize("gather", [False, True])
@pytest.mark.parametrize("n,q,k", [(9000, 300, 16), (129, 5, 7), (4500, 257, 1)])
def test_hybrid_ragged_tiles(n, q, k, gather):
    """Ragged corpus and query tiles, several query tiles per CTA."""
    w = workloads.config(3, n=n, batch=q)
    idx = Index(dev_tensor(w.E_data))
    idx.set_sparse(w.doc_indptr, w.doc_terms, w.vocab, w.k1, w.b)
    idx.gather_lexical(gather)
    _hybrid_check(idx, w, np.arange(w.q), w.alpha, f"ragged n={n} q={q} k={k} gather={gather}", k=k)
    idx.check()
