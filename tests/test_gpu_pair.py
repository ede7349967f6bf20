"""GPU parity of the tensor-core search run by CTA pairs (clusters of two CTAs
issuing M = 256 MMAs, each CTA loading half of every 256-row corpus tile),
against the fp64 oracle and against the single-CTA kernel: odd numbers of
query tiles (the last pair's second tile empty or ragged), one query tile
forced onto a pair, buffered lists (k > 32) with the sampled floor, and the
fused hybrid score."""
import numpy as np
import pytest
import torch

from paper_2608_08340_gb300 import workloads
from paper_2608_08340_gb300.index import Index

from _gpu import TOL, check_dense, dev_tensor

pytestmark = pytest.mark.gpu


def _data(n, d, q, seed):
    rng = np.random.default_rng(seed)
    E = workloads.to_bf16_bits(workloads._normalise(rng.standard_normal((n, d)).astype(np.float32)))
    Q = workloads.to_bf16_bits(workloads._normalise(rng.standard_normal((q, d)).astype(np.float32)))
    return E, Q


def _search(idx, Q, k, mode):
    idx.force_path("tc")
    idx.force_block_n(256)
    idx.force_pair(mode)
    out = idx.search(dev_tensor(Q), k)
    torch.cuda.synchronize()
    launch = idx.last_launch
    assert launch["cluster"] == (2 if mode == "pair" else 1), launch
    assert launch["block_n"] == 256 and launch["grid"] % launch["cluster"] == 0
    return out


@pytest.mark.parametrize("n,d,q,k", [
    (9000, 768, 300, 10),      # three query tiles: the second pair has one live tile
    (5000, 128, 257, 1),       # three tiles, the third holds one query
    (4097, 136, 129, 5),       # two tiles, ragged d and n
    (2000, 256, 64, 8),        # one tile forced onto a pair (second CTA idle rows)
    (700, 64, 255, 33),        # buffered lists
    (20000, 1024, 512, 16),    # four tiles, two pairs, several windows of units
])
def test_pair_matches_oracle_and_single(n, d, q, k):
    E, Q = _data(n, d, q, n + d + q + k)
    idx = Index(dev_tensor(E))
    ids_p, sc_p = _search(idx, Q, k, "pair")
    check_dense(ids_p, sc_p, E, Q, k, f"pair n={n} d={d} q={q} k={k}")
    ids_s, sc_s = _search(idx, Q, k, "single")
    assert torch.equal(ids_p, ids_s)
    assert (sc_p - sc_s).abs().max().item() <= TOL
    idx.check()
    idx.close()


@pytest.mark.parametrize("k", [100, 256])
def test_pair_large_k_with_sampled_floor(k):
    n, d, q = 160000, 128, 260
    E, Q = _data(n, d, q, k + 7)
    idx = Index(dev_tensor(E))
    ids, sc = _search(idx, Q, k, "pair")
    rows = np.sort(np.random.default_rng(k).choice(q, 12, replace=False))
    check_dense(ids, sc, E, Q, k, f"pair large k={k}", rows=rows)
    idx.check()
    idx.close()


def test_pair_hybrid_matches_single():
    w = workloads.config(3, n=6000, batch=300)
    idx = Index(dev_tensor(w.E_data))
    idx.set_sparse(w.doc_indptr, w.doc_terms, w.vocab, w.k1, w.b)
    idx.force_path("tc")
    idx.force_block_n(256)
    res = {}
    for mode in ("pair", "single"):
        idx.force_pair(mode)
        res[mode] = idx.hybrid_search(dev_tensor(w.Q_data), torch.from_numpy(w.q_indptr),
                                      torch.from_numpy(w.q_terms), w.alpha, w.k)
        assert idx.last_launch["cluster"] == (2 if mode == "pair" else 1)
    assert torch.equal(res["pair"][0], res["single"][0])
    assert (res["pair"][1] - res["single"][1]).abs().max().item() <= TOL
    idx.check()
    idx.close()


def test_gathered_hybrid_ignores_pair_and_tile_options():
    """The gathered hybrid search (OPRAG_OPT_LEX_GATHER) always runs single
    CTAs on 128-row tiles
    (its two score and two BM25 accumulators fill the TMEM); forcing CTA
    pairs or 256-row tiles changes nothing."""
    w = workloads.config(3, n=6000, batch=300)
    idx = Index(dev_tensor(w.E_data))
    idx.set_sparse(w.doc_indptr, w.doc_terms, w.vocab, w.k1, w.b)
    idx.force_path("tc")
    idx.gather_lexical(True)
    res = {}
    for mode, bn in (("pair", 256), (None, None)):
        idx.force_block_n(bn)
        idx.force_pair(mode)
        res[mode] = idx.hybrid_search(dev_tensor(w.Q_data), torch.from_numpy(w.q_indptr),
                                      torch.from_numpy(w.q_terms), w.alpha, w.k)
        assert idx.last_launch["cluster"] == 1 and idx.last_launch["block_n"] == 128
    assert torch.equal(res["pair"][0], res[None][0])
    assert torch.equal(res["pair"][1], res[None][1])
    idx.check()
    idx.close()
