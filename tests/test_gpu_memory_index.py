"""GPU parity of the index-update rows: append with capacity doubling, the
lexical half of upsert (token bags replaced, BM25 statistics rebuilt) and the
dense search over a knowledge and a memory index together (Sec. 3.2 Op_upsert;
Sec. 4.4 memory-aware retrieval and upsert)."""
import numpy as np
import pytest
import torch

import oracle
from oracle import check
from paper_2608_08340_gb300 import workloads
from paper_2608_08340_gb300.index import Index, search_two

from _gpu import TOL, check_dense, dev_tensor, oracle_topk

pytestmark = pytest.mark.gpu


def _bits(t):
    return t.view(torch.int16).cpu().numpy().view(np.uint16)


def test_append_grows_by_doubling_and_searches_the_whole_index():
    w = workloads.config(1, n=700, batch=40)
    E = w.E_data
    idx = Index(dev_tensor(E[:300]))
    assert idx.append(dev_tensor(E[300:350])) == 300            # device bf16 rows
    for r in range(350, 356):                                    # one row at a time
        assert idx.append(torch.from_numpy(E[r:r + 1].view(np.int16)).view(torch.bfloat16)) == r
    f32 = oracle.bf16_to_f32(E[356:700])                          # host fp32 rows, exact in bf16
    assert idx.append(torch.from_numpy(f32)) == 356
    assert idx.n == 700
    np.testing.assert_array_equal(_bits(idx.rows()), E)
    ids, sc = idx.search(dev_tensor(w.Q_data), 10)
    check_dense(ids, sc, E, w.Q_data, 10, "after appends")
    idx.check()


def _hybrid_check(idx, E, Q, ip, tm, vocab, w, label):
    ids, sc = idx.hybrid_search(dev_tensor(Q), torch.from_numpy(w.q_indptr),
                                torch.from_numpy(w.q_terms), w.alpha, w.k)
    o_ids, o_sc = oracle_topk(
        lambda kout: oracle.hybrid_search(E, Q, ip, tm, vocab, w.q_indptr, w.q_terms, w.alpha,
                                          kout, w.k1, w.b), w.k, E.shape[0])
    check.check_topk(ids.cpu().numpy(), sc.cpu().numpy(), o_ids, o_sc, w.k, TOL,
                     n=E.shape[0], label=label)


def test_update_sparse_keeps_bm25_exact_and_matches_a_fresh_index():
    w = workloads.config(3, n=3000, batch=40)
    idx = Index(dev_tensor(w.E_data))
    idx.set_sparse(w.doc_indptr, w.doc_terms, w.vocab, w.k1, w.b)
    rng = np.random.default_rng(21)
    ids = np.array([5, 17, 5, 2999, 0, 1200], np.int64)         # 5 twice: the second wins
    lens = rng.integers(0, 40, ids.size)
    lens[3] = 0                                                   # an emptied chunk
    bip = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    # draw the new bags from the query terms so that they matter to the queries
    btm = rng.choice(w.q_terms, int(bip[-1])).astype(np.int32)
    idx.update_sparse(ids, bip, btm)
    ip, tm = oracle.replace_bags(w.doc_indptr, w.doc_terms, ids, bip, btm)
    _hybrid_check(idx, w.E_data, w.Q_data, ip, tm, w.vocab, w, "after bag update")
    fresh = Index(dev_tensor(w.E_data))
    fresh.set_sparse(ip, tm, w.vocab, w.k1, w.b)
    qip, qt = torch.from_numpy(w.q_indptr), torch.from_numpy(w.q_terms)
    a = idx.hybrid_search(dev_tensor(w.Q_data), qip, qt, w.alpha, w.k)
    b = fresh.hybrid_search(dev_tensor(w.Q_data), qip, qt, w.alpha, w.k)
    assert torch.equal(a[0], b[0]) and torch.equal(a[1], b[1])
    idx.check()


def test_append_to_a_hybrid_index_gives_empty_bags_then_updates():
    w = workloads.config(3, n=2500, batch=30)
    n0 = 2000
    idx = Index(dev_tensor(w.E_data[:n0]))
    ip0 = w.doc_indptr[:n0 + 1]
    tm0 = w.doc_terms[:ip0[-1]]
    idx.set_sparse(ip0, tm0, w.vocab, w.k1, w.b)
    idx.append(dev_tensor(w.E_data[n0:]))
    new_ids = np.arange(n0, w.n)
    ip, tm = oracle.replace_bags(ip0, tm0, new_ids, np.zeros(new_ids.size + 1, np.int32),
                                 np.zeros(0, np.int32))
    _hybrid_check(idx, w.E_data, w.Q_data, ip, tm, w.vocab, w, "after append (empty bags)")
    # now give the appended chunks their real bags
    sub_ip = w.doc_indptr[n0:] - w.doc_indptr[n0]
    sub_tm = w.doc_terms[w.doc_indptr[n0]:]
    idx.update_sparse(new_ids, sub_ip, sub_tm)
    _hybrid_check(idx, w.E_data, w.Q_data, w.doc_indptr, w.doc_terms, w.vocab, w,
                  "after bags of the appended chunks")
    idx.check()


@pytest.mark.parametrize("nk,nm,k", [(2000, 300, 10), (5000, 40, 64), (100, 3000, 5)])
def test_search_two_matches_the_stacked_oracle(nk, nm, k):
    w = workloads.config(1, n=nk + nm, batch=70)
    E = w.E_data
    kn, mem = Index(dev_tensor(E[:nk])), Index(dev_tensor(E[nk:]))
    ids, src, sc = search_two(kn, mem, dev_tensor(w.Q_data), k)
    torch.cuda.synchronize()
    src = src.cpu().numpy()
    stacked = np.where(src == 1, ids.cpu().numpy() + nk, ids.cpu().numpy())
    assert set(np.unique(src)) <= {0, 1}
    check_dense(stacked, sc.cpu().numpy(), E, w.Q_data, k, f"two indices {nk}+{nm}")
    kn.check()
    mem.check()


@pytest.mark.parametrize("nk,nm,q,k", [(32768, 8192, 256, 5), (9000, 300, 40, 16),
                                       (20000, 45000, 130, 100), (256, 70000, 600, 7),
                                       (1000, 1, 3, 2)])
def test_search_two_is_one_search_over_the_stacked_rows(nk, nm, q, k):
    """The two-index search runs one search pass (and, for k > 32 over many
    tiles, one sampled pass) over the knowledge rows followed by the memory
    rows: its results equal a search of one index holding the stacked rows,
    with memory ids shifted by the knowledge size (scores within 1e-6, ids
    equal outside 1e-6 near-ties: the two runs may tile the rows
    differently); equal scores rank the knowledge index first."""
    w = workloads.config(1, n=nk + nm, batch=q)
    E = w.E_data
    kn, mem = Index(dev_tensor(E[:nk])), Index(dev_tensor(E[nk:]))
    both = Index(dev_tensor(E))
    Q = dev_tensor(w.Q_data)
    ids, src, sc = search_two(kn, mem, Q, k)
    r_ids, r_sc = both.search(Q, k)
    torch.cuda.synchronize()
    src = src.cpu().numpy()
    assert ((src == 0) | (src == 1)).all()
    ids = ids.cpu().numpy()
    assert (ids[src == 0] < nk).all() and (ids[src == 1] < nm).all()
    stacked = np.where(src == 1, ids + nk, ids)
    r_ids, r_sc = r_ids.cpu().numpy(), r_sc.cpu().numpy()
    np.testing.assert_allclose(sc.cpu().numpy(), r_sc, rtol=0, atol=1e-6)
    tie = np.zeros_like(r_sc, dtype=bool)
    tie[:, 1:] |= (r_sc[:, :-1] - r_sc[:, 1:]) <= 1e-6
    tie[:, :-1] |= (r_sc[:, :-1] - r_sc[:, 1:]) <= 1e-6
    np.testing.assert_array_equal(stacked[~tie], r_ids[~tie])
    rows = np.arange(q) if q <= 64 else np.sort(np.random.default_rng(q).choice(q, 48, replace=False))
    check_dense(stacked, sc.cpu().numpy(), E, w.Q_data, k, f"stacked {nk}+{nm}", rows=rows)
    kn.check()
    mem.check()


def test_search_two_ties_rank_knowledge_first():
    """The same row in both indices: the knowledge copy comes first."""
    rng = np.random.default_rng(4)
    E = workloads.to_bf16_bits(workloads._normalise(rng.standard_normal((500, 64)).astype(np.float32)))
    kn, mem = Index(dev_tensor(E)), Index(dev_tensor(E[::-1].copy()))
    ids, src, sc = search_two(kn, mem, dev_tensor(E[:5]), 2)
    torch.cuda.synchronize()
    assert src.cpu().tolist() == [[0, 1]] * 5
    assert ids.cpu().tolist() == [[i, 499 - i] for i in range(5)]
    assert (sc[:, 0] == sc[:, 1]).all()
