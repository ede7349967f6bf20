"""GPU parity of the dense-first hybrid search (Sec. 4.1 Retrieval; Sec. 5.5):
the exact dense top-N, then the fused rerank of only those candidates with
the BM25 maximum taken over the candidates.  The rerank is checked against the
oracle's rerank of the same candidates (the dense top-N itself is checked by
the dense parity tests; near-ties at rank N could otherwise change the set),
and with every chunk a candidate it must equal the full hybrid search: bit
for bit with the materialised BM25 block (the same fp32 sums in query-term
order), and up to the fp32 rounding of the sums with the gathered form (the
head terms' part then comes from tensor-core MMAs)."""
import numpy as np
import pytest
import torch

import oracle
from oracle import check
from paper_2608_08340_gb300 import _lib, workloads
from paper_2608_08340_gb300.index import Index

from _gpu import TOL, dev_tensor

pytestmark = pytest.mark.gpu


def _setup(n, q, seed_cfg=3):
    w = workloads.config(seed_cfg, n=n, batch=q)
    idx = Index(dev_tensor(w.E_data))
    idx.set_sparse(w.doc_indptr, w.doc_terms, w.vocab, w.k1, w.b)
    return w, idx


def _terms(w):
    return torch.from_numpy(w.q_indptr), torch.from_numpy(w.q_terms)


@pytest.mark.parametrize("n,q,n_cand,k", [(6000, 300, 128, 5), (20000, 130, 64, 10),
                                          (3000, 40, 256, 16), (5000, 33, 32, 1)])
def test_dense_first_matches_oracle_rerank(n, q, n_cand, k):
    w, idx = _setup(n, q)
    qip, qt = _terms(w)
    Q = dev_tensor(w.Q_data)
    ids, sc = idx.hybrid_search_dense_first(Q, qip, qt, w.alpha, n_cand, k)
    cand, _ = idx.search(Q, n_cand)                     # the same dense top-N
    torch.cuda.synchronize()
    kout = min(n_cand, k + 48)
    o_ids, o_sc = oracle.rerank(w.E_data, w.Q_data, cand.cpu().numpy(), w.doc_indptr,
                                w.doc_terms, w.vocab, w.q_indptr, w.q_terms, w.alpha, kout,
                                w.k1, w.b)
    check.check_topk(ids.cpu().numpy(), sc.cpu().numpy(), o_ids, o_sc, k, TOL, n=n_cand,
                     label=f"dense-first n={n} q={q} N={n_cand} k={k}")
    idx.check()


@pytest.mark.parametrize("gather", [False, True])
def test_dense_first_over_every_chunk_equals_full_hybrid(gather):
    w, idx = _setup(200, 50)
    idx.gather_lexical(gather)
    qip, qt = _terms(w)
    Q = dev_tensor(w.Q_data)
    d_ids, d_sc = idx.hybrid_search_dense_first(Q, qip, qt, w.alpha, 256, 40)
    h_ids, h_sc = idx.hybrid_search(Q, qip, qt, w.alpha, 10)
    torch.cuda.synchronize()
    if not gather:
        assert torch.equal(d_ids[:, :10], h_ids)
        assert torch.equal(d_sc[:, :10], h_sc)
        return
    # same ranking up to swaps of scores within 1e-5 (different fp32 sum orders)
    check.check_topk(h_ids.cpu().numpy(), h_sc.cpu().numpy(), d_ids.cpu().numpy(),
                     d_sc.cpu().numpy().astype(np.float64), 10, 1e-5, n=200,
                     label="dense-first over every chunk vs gathered hybrid")


def test_dense_first_alpha_one_is_the_dense_search():
    w, idx = _setup(8000, 64)
    qip, qt = _terms(w)
    Q = dev_tensor(w.Q_data)
    ids, sc = idx.hybrid_search_dense_first(Q, qip, qt, 1.0, 128, 8)
    s_ids, s_sc = idx.search(Q, 8)
    torch.cuda.synchronize()
    assert torch.equal(ids, s_ids)
    assert (sc - s_sc).abs().max().item() == 0.0


def test_dense_first_argument_errors():
    w, idx = _setup(500, 4)
    qip, qt = _terms(w)
    Q = dev_tensor(w.Q_data)
    with pytest.raises(RuntimeError):
        idx.hybrid_search_dense_first(Q, qip, qt, w.alpha, 4, 5)          # n_cand < k
    with pytest.raises(RuntimeError):
        idx.hybrid_search_dense_first(Q, qip, qt, w.alpha, 512, 5)        # n_cand > 256
    bare = Index(dev_tensor(w.E_data))
    with pytest.raises(RuntimeError):
        bare.hybrid_search_dense_first(Q, qip, qt, w.alpha, 128, 5)       # no sparse side
