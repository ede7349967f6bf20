"""Pins the CPU oracle to facts that do not come from the oracle itself:
hand-worked fixtures (tests/golden), a library matmul and a library sort,
closed forms (self-match = squared norm, idf = ln 2 at df = N/2), limits of
BM25 that reduce to textbook tf-idf and to the binary model, invariants
(corpus permutation, alpha = 0 / 1 of the fusion), and IEEE rounding by torch.
Each plausible slip -- a dropped term, a wrong sign, a transposed operand, a
reversed tie-break, a wrong idf variant -- breaks at least one of them."""
import math

import numpy as np
import pytest
import torch

import oracle
from oracle import check
from paper_2608_08340_gb300 import workloads

from _golden import load, value


def _f32(a):
    return np.asarray(a, dtype=np.float32)


# ------------------------------------------------------------------ dense

def test_dense_golden_hand_worked():
    g = load("dense_8chunk.json")
    E, Q = _f32(g["E"]), _f32(g["Q"])
    for data_E, data_Q in ((E, Q), (oracle.round_bf16(E), oracle.round_bf16(Q))):
        ids, sc = oracle.search(data_E, data_Q, g["k"])
        assert ids.tolist() == g["ids"]
        assert sc.tolist() == [[float(v) for v in row] for row in g["scores"]]


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_dense_scores_equal_library_matmul(dtype):
    rng = np.random.default_rng(7)
    E = rng.standard_normal((300, 96)).astype(np.float32)
    Q = rng.standard_normal((5, 96)).astype(np.float32)
    if dtype == "bf16":
        E, Q = oracle.round_bf16(E), oracle.round_bf16(Q)
    S = oracle.dense_scores(E, Q)
    ref = workloads.widen(Q).astype(np.float64) @ workloads.widen(E).astype(np.float64).T
    np.testing.assert_allclose(S, ref, rtol=0, atol=1e-12)


def test_full_sort_equals_library_lexsort_with_ties():
    rng = np.random.default_rng(11)
    # small integers so that many exact ties occur, plus duplicated rows
    E = rng.integers(-2, 3, size=(200, 8)).astype(np.float32)
    E[50] = E[10]
    E[199] = E[10]
    Q = rng.integers(-2, 3, size=(4, 8)).astype(np.float32)
    n = E.shape[0]
    ids, sc = oracle.search(E, Q, n)
    S = Q.astype(np.float64) @ E.astype(np.float64).T
    for i in range(Q.shape[0]):
        order = np.lexsort((np.arange(n), -S[i]))   # score desc, then id asc
        assert ids[i].tolist() == order.tolist()
        np.testing.assert_array_equal(sc[i], S[i][order])


def test_topk_rows_matches_search():
    w = workloads.config(0, n=512, batch=6)
    S = oracle.dense_scores(w.E_data, w.Q_data)
    a_ids, a_sc = oracle.topk_rows(S, 9)
    b_ids, b_sc = oracle.search(w.E_data, w.Q_data, 9)
    np.testing.assert_array_equal(a_ids, b_ids)
    np.testing.assert_array_equal(a_sc, b_sc)


def test_self_match_is_rank_one_with_squared_norm():
    w = workloads.config(1, n=2048, batch=1)
    E = w.E_data
    rows = [0, 17, 1023, 2047]
    Q = E[rows]
    ids, sc = oracle.search(E, Q, 3)
    for j, r in enumerate(rows):
        e = workloads.widen(E[r]).astype(np.float64)
        assert ids[j, 0] == r
        assert sc[j, 0] == pytest.approx(float(np.dot(e, e)), abs=1e-12)
        assert sc[j, 0] == pytest.approx(1.0, abs=1e-2)   # normalised up to bf16 rounding


def test_corpus_permutation_invariance():
    w = workloads.config(1, n=1500, batch=7)
    perm = np.random.default_rng(3).permutation(w.n)
    ids_a, sc_a = oracle.search(w.E_data, w.Q_data, 12)
    ids_b, sc_b = oracle.search(w.E_data[perm], w.Q_data, 12)
    np.testing.assert_array_equal(perm[ids_b], ids_a)
    np.testing.assert_array_equal(sc_b, sc_a)


def test_search_rejects_k_above_n():
    with pytest.raises(RuntimeError):
        oracle.search(np.ones((3, 4), np.float32), np.ones((1, 4), np.float32), 4)


# ------------------------------------------------------------------ BM25

def _csr(lists):
    indptr = np.zeros(len(lists) + 1, np.int32)
    indptr[1:] = np.cumsum([len(x) for x in lists])
    terms = np.array([t for x in lists for t in x], np.int32)
    return indptr, terms


def test_bm25_golden_hand_worked():
    g = load("bm25_4doc.json")
    dip, dt = _csr(g["docs"])
    qip, qt = _csr(g["queries"])
    M, avgdl, df = oracle.bm25(dip, dt, g["vocab"], qip, qt, g["k1"], g["b"])
    assert avgdl == 3.0
    assert df.tolist() == [2, 2, 2, 2, 1, 0]
    want = np.array([[value(x) for x in row] for row in g["expected"]])
    np.testing.assert_allclose(M, want, rtol=1e-14, atol=1e-15)


def _random_corpus(n=60, vocab=40, seed=5):
    rng = np.random.default_rng(seed)
    docs = [rng.integers(0, vocab, size=rng.integers(3, 12)).tolist() for _ in range(n)]
    qs = [rng.integers(0, vocab, size=rng.integers(1, 5)).tolist() for _ in range(9)]
    return docs, qs


def _counts(docs, vocab):
    tf = np.zeros((len(docs), vocab))
    for i, dd in enumerate(docs):
        tf[i] = np.bincount(dd, minlength=vocab)
    return tf


def test_bm25_tfidf_limit():
    """b = 0 and k1 -> infinity: tf (k1+1) / (tf + k1) -> tf, so BM25 becomes
    the textbook sum over query terms of tf * idf."""
    docs, qs = _random_corpus()
    vocab = 40
    dip, dt = _csr(docs)
    qip, qt = _csr(qs)
    M, _, _ = oracle.bm25(dip, dt, vocab, qip, qt, k1=1e12, b=0.0)
    tf = _counts(docs, vocab)
    df = (tf > 0).sum(0)
    N = len(docs)
    idf = np.where(df > 0, np.log1p((N - df + 0.5) / (df + 0.5)), 0.0)
    want = np.stack([sum(tf[:, t] * idf[t] for t in q) for q in qs])
    np.testing.assert_allclose(M, want, rtol=1e-9, atol=1e-12)


def test_bm25_binary_limit():
    """k1 -> 0: every present query term contributes exactly its idf."""
    docs, qs = _random_corpus(seed=9)
    vocab = 40
    dip, dt = _csr(docs)
    qip, qt = _csr(qs)
    M, _, _ = oracle.bm25(dip, dt, vocab, qip, qt, k1=1e-12, b=0.75)
    tf = _counts(docs, vocab)
    df = (tf > 0).sum(0)
    N = len(docs)
    idf = np.where(df > 0, np.log1p((N - df + 0.5) / (df + 0.5)), 0.0)
    want = np.stack([sum((tf[:, t] > 0) * idf[t] for t in q) for q in qs])
    np.testing.assert_allclose(M, want, rtol=1e-9, atol=1e-12)


def test_bm25_idf_is_ln2_for_half_the_corpus():
    """A term held by exactly half of N documents has idf = ln 2; with tf = 1
    in a document of average length the saturation factor is 1 for any k1, b."""
    docs = [[0, 1], [0, 2], [3, 4], [5, 6]]        # term 0 in 2 of 4 docs, all lengths 2
    dip, dt = _csr(docs)
    qip, qt = _csr([[0]])
    for k1, b in ((1.2, 0.75), (2.0, 0.3), (0.5, 1.0)):
        M, _, _ = oracle.bm25(dip, dt, 7, qip, qt, k1, b)
        assert M[0].tolist() == pytest.approx([math.log(2), math.log(2), 0, 0], abs=1e-15)


def test_bm25_monotone_in_term_frequency():
    docs, qs = _random_corpus(seed=13)
    vocab = 40
    dip, dt = _csr(docs)
    qip, qt = _csr([[7]])
    base, _, _ = oracle.bm25(dip, dt, vocab, qip, qt)
    holders = [i for i, dd in enumerate(docs) if 7 in dd]
    assert holders
    bumped = [list(dd) for dd in docs]
    i = holders[0]
    j = next(p for p, t in enumerate(bumped[i]) if t != 7)
    bumped[i][j] = 7                                 # same length, df unchanged
    dip2, dt2 = _csr(bumped)
    after, _, _ = oracle.bm25(dip2, dt2, vocab, qip, qt)
    assert after[0, i] > base[0, i]


def test_bm25_postings_walk_equals_document_scan():
    """Sec. 4.4: the inverted-postings BM25 visits only documents holding a
    query term yet keeps full-corpus BM25 semantics.  An independent postings
    walk (per-term document lists built with numpy) must agree."""
    docs, qs = _random_corpus(n=80, seed=21)
    vocab = 40
    k1, b = 1.2, 0.75
    dip, dt = _csr(docs)
    qip, qt = _csr(qs)
    M, avgdl, df = oracle.bm25(dip, dt, vocab, qip, qt, k1, b)
    tf = _counts(docs, vocab)
    lens = np.array([len(x) for x in docs], np.float64)
    N = len(docs)
    postings = {t: np.nonzero(tf[:, t])[0] for t in range(vocab)}
    out = np.zeros_like(M)
    for qi, q in enumerate(qs):
        for t in q:
            ds = postings[t]
            if ds.size == 0:
                continue
            dft = ds.size
            idf = math.log(1 + (N - dft + 0.5) / (dft + 0.5))
            f = tf[ds, t]
            out[qi, ds] += idf * f * (k1 + 1) / (f + k1 * (1 - b + b * lens[ds] / lens.mean()))
    np.testing.assert_allclose(M, out, rtol=1e-12, atol=1e-14)


# ------------------------------------------------------------------ hybrid

def test_hybrid_golden_hand_worked():
    g = load("hybrid_4doc.json")
    bm = load("bm25_4doc.json")
    dip, dt = _csr(bm["docs"])
    qip, qt = _csr(g["query_terms"])
    ids, sc, mx = oracle.hybrid_search(_f32(g["E"]), _f32(g["Q"]), dip, dt, bm["vocab"], qip,
                                       qt, g["alpha"], g["k"], bm["k1"], bm["b"])
    assert ids.tolist() == g["ids"]
    want = np.array([[value(x) for x in row] for row in g["scores"]])
    np.testing.assert_allclose(sc, want, rtol=0, atol=1e-15)
    assert mx[0] == pytest.approx(value("44/35*ln(2)"), abs=1e-15)
    assert mx[1] == 0.0


def _small_hybrid(seed=4, n=400, q=6):
    w = workloads.config(3, n=n, batch=q)
    return w


def test_hybrid_alpha_one_is_dense_search():
    w = _small_hybrid()
    ids, sc, _ = oracle.hybrid_search(w.E_data, w.Q_data, w.doc_indptr, w.doc_terms, w.vocab,
                                      w.q_indptr, w.q_terms, 1.0, 10)
    d_ids, d_sc = oracle.search(w.E_data, w.Q_data, 10)
    np.testing.assert_array_equal(ids, d_ids)
    np.testing.assert_array_equal(sc, d_sc)


def test_hybrid_alpha_zero_is_normalised_bm25_ranking():
    w = _small_hybrid()
    ids, sc, mx = oracle.hybrid_search(w.E_data, w.Q_data, w.doc_indptr, w.doc_terms, w.vocab,
                                       w.q_indptr, w.q_terms, 0.0, 10)
    M, _, _ = oracle.bm25(w.doc_indptr, w.doc_terms, w.vocab, w.q_indptr, w.q_terms)
    for i in range(w.q):
        order = np.lexsort((np.arange(w.n), -M[i]))[:10]
        assert ids[i].tolist() == order.tolist()
        assert sc[i, 0] == 1.0                         # the best document is the maximum
        assert mx[i] == M[i].max()


# ------------------------------------------------------------------ dense-first rerank

def test_dense_first_golden_hand_worked():
    g = load("dense_first_4doc.json")
    h = load("hybrid_4doc.json")
    bm = load("bm25_4doc.json")
    dip, dt = _csr(bm["docs"])
    qip, qt = _csr(h["query_terms"])
    ids, sc = oracle.hybrid_dense_first(_f32(h["E"]), _f32(h["Q"]), dip, dt, bm["vocab"], qip,
                                        qt, h["alpha"], g["n_cand"], g["k"], bm["k1"], bm["b"])
    assert ids.tolist() == g["ids"]
    want = np.array([[value(x) for x in row] for row in g["scores"]])
    np.testing.assert_allclose(sc, want, rtol=0, atol=1e-15)
    full, _, _ = oracle.hybrid_search(_f32(h["E"]), _f32(h["Q"]), dip, dt, bm["vocab"], qip, qt,
                                      h["alpha"], 2, bm["k1"], bm["b"])
    assert full.tolist() == g["full_hybrid_top2"]


def test_rerank_over_every_chunk_is_the_full_hybrid():
    w = _small_hybrid()
    cand = np.tile(np.arange(w.n, dtype=np.int64), (w.q, 1))
    ids, sc = oracle.rerank(w.E_data, w.Q_data, cand, w.doc_indptr, w.doc_terms, w.vocab,
                            w.q_indptr, w.q_terms, w.alpha, 10, w.k1, w.b)
    h_ids, h_sc, _ = oracle.hybrid_search(w.E_data, w.Q_data, w.doc_indptr, w.doc_terms, w.vocab,
                                          w.q_indptr, w.q_terms, w.alpha, 10, w.k1, w.b)
    np.testing.assert_array_equal(ids, h_ids)
    np.testing.assert_allclose(sc, h_sc, rtol=0, atol=1e-12)


def test_rerank_alpha_one_keeps_the_dense_order():
    w = _small_hybrid()
    ids, sc = oracle.hybrid_dense_first(w.E_data, w.Q_data, w.doc_indptr, w.doc_terms, w.vocab,
                                        w.q_indptr, w.q_terms, 1.0, 32, 10, w.k1, w.b)
    d_ids, d_sc = oracle.search(w.E_data, w.Q_data, 10)
    np.testing.assert_array_equal(ids, d_ids)
    np.testing.assert_array_equal(sc, d_sc)


def test_rerank_ignores_candidate_order_and_empty_slots():
    w = _small_hybrid()
    cand, _ = oracle.search(w.E_data, w.Q_data, 40)
    ids, sc = oracle.rerank(w.E_data, w.Q_data, cand, w.doc_indptr, w.doc_terms, w.vocab,
                            w.q_indptr, w.q_terms, w.alpha, 8, w.k1, w.b)
    rng = np.random.default_rng(3)
    shuffled = np.array([rng.permutation(r) for r in cand])
    padded = np.concatenate([shuffled, -np.ones((w.q, 7), np.int64)], axis=1)
    ids2, sc2 = oracle.rerank(w.E_data, w.Q_data, padded, w.doc_indptr, w.doc_terms, w.vocab,
                              w.q_indptr, w.q_terms, w.alpha, 8, w.k1, w.b)
    np.testing.assert_array_equal(ids, ids2)
    np.testing.assert_array_equal(sc, sc2)


# ------------------------------------------------------------------ embedding tail

def test_embed_pool_golden_hand_worked():
    g = load("embed_pool_2tok.json")
    out = oracle.embed_pool(np.array(g["hidden"], np.float32), np.array(g["mask"], np.uint8))
    want = np.array([[value(x) for x in row] for row in g["normalised_exact"]])
    np.testing.assert_allclose(out, want, rtol=0, atol=1e-15)
    bits = oracle.round_bf16(out.astype(np.float32))
    assert bits.tolist() == g["bf16_bits"]


def test_embed_pool_golden_pooled_rows_are_the_masked_means():
    """The fixture's pooled (pre-normalisation) rows are the exact means of
    the unmasked tokens, and normalising them gives its normalised rows."""
    from fractions import Fraction
    g = load("embed_pool_2tok.json")
    for h, m, pooled, normed in zip(g["hidden"], g["mask"], g["pooled"], g["normalised_exact"]):
        toks = [t for t, keep in zip(h, m) if keep]
        mean = [sum(Fraction(t[j]) for t in toks) / len(toks) for j in range(len(h[0]))]
        assert [Fraction(x) for x in pooled] == mean
        norm = float(sum(x * x for x in mean)) ** 0.5
        want = [float(x) / norm if norm else 0.0 for x in mean]
        np.testing.assert_allclose([value(x) for x in normed], want, rtol=0, atol=1e-15)


def test_embed_pool_single_token_and_identical_tokens_are_the_normalised_token():
    rng = np.random.default_rng(7)
    h = rng.standard_normal((5, 6, 64)).astype(np.float32)
    mask = np.zeros((5, 6), np.uint8)
    mask[:, 2] = 1
    out = oracle.embed_pool(h, mask)
    tok = h[:, 2, :].astype(np.float64)
    np.testing.assert_allclose(out, tok / np.linalg.norm(tok, axis=1, keepdims=True), atol=1e-15)
    same = np.repeat(h[:, :1, :], 6, axis=1)
    np.testing.assert_allclose(oracle.embed_pool(same, np.ones((5, 6), np.uint8)),
                               oracle.embed_pool(same[:, :1, :], np.ones((5, 1), np.uint8)),
                               atol=1e-15)


def test_embed_pool_is_a_unit_vector_invariant_to_scale_and_masked_values():
    rng = np.random.default_rng(8)
    h = rng.standard_normal((4, 9, 48)).astype(np.float32)
    mask = (rng.random((4, 9)) < 0.6).astype(np.uint8)
    mask[:, 0] = 1
    out = oracle.embed_pool(h, mask)
    np.testing.assert_allclose(np.linalg.norm(out, axis=1), 1.0, atol=1e-14)
    np.testing.assert_allclose(oracle.embed_pool(h * np.float32(4.0), mask), out, atol=1e-14)
    h2 = h.copy()
    h2[mask == 0] = 1e3                                   # padding values do not matter
    np.testing.assert_array_equal(oracle.embed_pool(h2, mask), out)
    # the mean of the unmasked tokens, written out with numpy
    m = np.stack([h[b][mask[b] == 1].astype(np.float64).mean(axis=0) for b in range(4)])
    np.testing.assert_allclose(out, m / np.linalg.norm(m, axis=1, keepdims=True), atol=1e-14)


def test_embed_pool_bf16_input_widens_exactly():
    rng = np.random.default_rng(9)
    h = rng.standard_normal((3, 4, 32)).astype(np.float32)
    bits = oracle.round_bf16(h)
    widened = oracle.bf16_to_f32(bits)
    mask = np.ones((3, 4), np.uint8)
    np.testing.assert_array_equal(oracle.embed_pool(bits, mask), oracle.embed_pool(widened, mask))


# ------------------------------------------------------------------ bags, two indices

def test_replace_bags_last_duplicate_wins_appends_and_recomputes_bm25():
    g = load("bm25_4doc.json")
    dip, dt = _csr(g["docs"])
    # doc 1 becomes [4], doc 1 again (wins) becomes [5, 5], doc 5 appended (doc 4 empty)
    ip, tm = oracle.replace_bags(dip, dt, [1, 1, 5], [0, 1, 3, 4], [4, 5, 5, 0])
    assert ip.tolist() == [0, 2, 4, 7, 10, 10, 11]
    assert tm.tolist() == [0, 1, 5, 5, 1, 2, 4, 3, 3, 3, 0]
    # BM25 of term 0 on the new corpus, by hand: N = 6, df(0) = 2 (docs 0 and 5),
    # lengths 2, 2, 3, 3, 0, 1 -> avgdl = 11/6; doc 0: tf 1, L = 1/4 + 3/4 * 2 / (11/6)
    M, avgdl, df = oracle.bm25(ip, tm, g["vocab"], [0, 1], [0], g["k1"], g["b"])
    assert avgdl == pytest.approx(11 / 6, abs=1e-15)
    assert df[0] == 2 and df[5] == 1 and df[2] == 1
    idf = np.log(1 + (6 - 2 + 0.5) / (2 + 0.5))
    L0 = 0.25 + 0.75 * 2 / (11 / 6)
    L5 = 0.25 + 0.75 * 1 / (11 / 6)
    np.testing.assert_allclose(M[0], [idf * 2.2 / (1 + 1.2 * L0), 0, 0, 0, 0,
                                      idf * 2.2 / (1 + 1.2 * L5)], rtol=1e-14)


def test_search_two_is_the_search_of_the_stacked_index():
    w = workloads.config(1, n=500, batch=7)
    Ek, Em = w.E_data[:320], w.E_data[320:]
    ids, src, sc = oracle.search_two(Ek, Em, w.Q_data, 12)
    f_ids, f_sc = oracle.search(w.E_data, w.Q_data, 12)
    np.testing.assert_array_equal(np.where(src == 1, ids + 320, ids), f_ids)
    np.testing.assert_array_equal(sc, f_sc)
    # a memory index equal to the knowledge index: every score appears twice,
    # the knowledge copy first
    ids2, src2, sc2 = oracle.search_two(Ek, Ek, w.Q_data, 6)
    assert (ids2[:, 0::2] == ids2[:, 1::2]).all()
    assert (src2[:, 0::2] == 0).all() and (src2[:, 1::2] == 1).all()


# ------------------------------------------------------------------ upsert

def test_upsert_last_duplicate_wins_and_matches_rebuild():
    w = workloads.config(1, n=300, batch=3)
    E = w.E_data.copy()
    ids = np.array([5, 17, 5, 299, 0], np.int64)
    rows = oracle.round_bf16(np.random.default_rng(1).standard_normal((5, w.d)).astype(np.float32))
    oracle.upsert(E, ids, rows)
    want = w.E_data.copy()
    final = {}
    for i, r in enumerate(ids.tolist()):
        final[r] = i
    for r, i in final.items():
        want[r] = rows[i]
    np.testing.assert_array_equal(E, want)
    # search after upsert == search on the rebuilt array
    a = oracle.search(E, w.Q_data, 7)
    b = oracle.search(want, w.Q_data, 7)
    np.testing.assert_array_equal(a[0], b[0])
    # upserting the same rows again changes nothing
    E2 = E.copy()
    oracle.upsert(E2, ids, rows)
    np.testing.assert_array_equal(E2, E)


def test_upsert_out_of_range_writes_nothing():
    E = np.zeros((4, 8), np.float32)
    with pytest.raises(RuntimeError):
        oracle.upsert(E, np.array([1, 4], np.int64), np.ones((2, 8), np.float32))
    assert not E.any()


def test_upsert_fp32_rows_into_bf16_index_round_to_nearest_even():
    E = np.zeros((2, 4), np.uint16)
    rows = np.array([[1.0 + 2.0 ** -8, 1.0 + 3 * 2.0 ** -8, -0.1, 3.0]], np.float32)
    oracle.upsert(E, np.array([1], np.int64), rows)
    want = torch.from_numpy(rows).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    np.testing.assert_array_equal(E[1], want[0])


def test_round_bf16_matches_torch():
    rng = np.random.default_rng(2)
    x = np.concatenate([rng.standard_normal(100000).astype(np.float32),
                        # exact halfway cases: both parities of the kept bit
                        (np.arange(1, 2000, dtype=np.uint32) << 16 | 0x8000).view(np.float32),
                        np.array([0.0, -0.0, 1e-40, -3.4e38], np.float32)])
    want = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    np.testing.assert_array_equal(oracle.round_bf16(x), want)


# ------------------------------------------------------------------ checker

def test_checker_accepts_exact_and_near_tie_swaps_and_rejects_real_errors():
    or_ids = np.array([4, 9, 2, 7, 1, 3])
    or_sc = np.array([0.9, 0.80003, 0.8, 0.5, 0.49995, 0.1])
    check.check_query(or_ids[:4], or_sc[:4], or_ids, or_sc, 4)
    # ranks 1 and 2 are a near tie (gap 3e-5 < 1e-4): either order passes
    check.check_query([4, 2, 9, 7], [0.9, 0.8, 0.80003, 0.5], or_ids, or_sc, 4)
    # ranks 3 and 4 straddle k = 4 inside one block: id 1 may replace id 7
    check.check_query([4, 9, 2, 1], [0.9, 0.80003, 0.8, 0.49995], or_ids, or_sc, 4)
    with pytest.raises(check.TopkMismatch):          # a swap across a real gap
        check.check_query([9, 4, 2, 7], [0.80003, 0.9, 0.8, 0.5], or_ids, or_sc, 4)
    with pytest.raises(check.TopkMismatch):          # a score off by more than tol
        check.check_query([4, 9, 2, 7], [0.9, 0.80003, 0.8, 0.5003], or_ids, or_sc, 4)
    with pytest.raises(check.TopkMismatch):          # an id outside the top block
        check.check_query([4, 9, 2, 3], [0.9, 0.80003, 0.8, 0.1], or_ids, or_sc, 4)
    with pytest.raises(check.TopkMismatch):          # block at k reaches the list end
        check.check_query([4, 9], [0.9, 0.80003], or_ids[:3], or_sc[:3], 2)
