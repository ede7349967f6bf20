"""GPU parity of the tensor-core search in dual mode (one CTA takes two query
tiles per unit; two MMAs per K-step share the corpus operand, one into each
TMEM accumulator, and each epilogue set filters one tile) against the fp64
oracle and against the single-tile kernel: an odd number of query tiles (the
last unit's second tile ragged or empty), several units per CTA, ragged d and
n, both list lengths dual mode supports, the fused hybrid score, and the
automatic choice for a small batch."""
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
    idx.force_pair(mode)
    out = idx.search(dev_tensor(Q), k)
    torch.cuda.synchronize()
    launch = idx.last_launch
    assert launch["cluster"] == 1, launch
    assert launch["tiles"] == (2 if mode == "dual" else 1), launch
    if mode == "dual":
        assert launch["block_n"] == 128, launch
    return out


@pytest.mark.parametrize("n,d,q,k", [
    (32768, 768, 256, 5),      # the paper-shaped small batch: one or two units per CTA
    (9000, 768, 300, 10),      # three query tiles: the second unit's second tile ragged
    (5000, 128, 257, 1),       # three tiles, the third holds one query
    (4097, 136, 129, 5),       # two tiles, the second holds one query; ragged d and n
    (60000, 256, 512, 16),     # four tiles, several units per CTA, lists of 16
    (3000, 64, 200, 9),        # lists of 16 with k = 9
])
def test_dual_matches_oracle_and_single(n, d, q, k):
    E, Q = _data(n, d, q, n + d + q + k)
    idx = Index(dev_tensor(E))
    ids_d, sc_d = _search(idx, Q, k, "dual")
    rows = None if n * q <= 4_000_000 else np.sort(np.random.default_rng(q).choice(q, 24, replace=False))
    check_dense(ids_d, sc_d, E, Q, k, f"dual n={n} d={d} q={q} k={k}", rows=rows)
    ids_s, sc_s = _search(idx, Q, k, "single")
    assert torch.equal(ids_d, ids_s)
    assert (sc_d - sc_s).abs().max().item() <= TOL
    idx.check()
    idx.close()


def test_dual_is_the_automatic_choice_for_small_batches():
    E, Q = _data(32768, 768, 256, 11)
    idx = Index(dev_tensor(E))
    idx.force_path("tc")
    idx.search(dev_tensor(Q), 5)
    torch.cuda.synchronize()
    assert idx.last_launch["tiles"] == 2, idx.last_launch
    # One query tile, lists of 32 or buffered lists: no dual mode.
    for q, k in ((128, 5), (256, 20), (256, 100)):
        idx.search(dev_tensor(Q[:q]), k)
        torch.cuda.synchronize()
        assert idx.last_launch["tiles"] == 1, (q, k, idx.last_launch)
    idx.check()
    idx.close()


def test_dual_hybrid_matches_single():
    w = workloads.config(3, n=6000, batch=300)
    idx = Index(dev_tensor(w.E_data))
    idx.set_sparse(w.doc_indptr, w.doc_terms, w.vocab, w.k1, w.b)
    idx.force_path("tc")
    res = {}
    for mode in ("dual", "single"):
        idx.force_pair(mode)
        res[mode] = idx.hybrid_search(dev_tensor(w.Q_data), torch.from_numpy(w.q_indptr),
                                      torch.from_numpy(w.q_terms), w.alpha, w.k)
        torch.cuda.synchronize()
        assert idx.last_launch["tiles"] == (2 if mode == "dual" else 1)
    assert torch.equal(res["dual"][0], res["single"][0])
    assert (res["dual"][1] - res["single"][1]).abs().max().item() <= TOL
    idx.check()
    idx.close()


def test_gathered_hybrid_runs_single_ctas_whatever_the_pair_option():
    """The gathered hybrid search (OPRAG_OPT_LEX_GATHER) takes every TMEM
    column for two score and two BM25 accumulators, so it always runs single
    CTAs on 128-row tiles; forcing dual mode changes nothing."""
    w = workloads.config(3, n=6000, batch=300)
    idx = Index(dev_tensor(w.E_data))
    idx.set_sparse(w.doc_indptr, w.doc_terms, w.vocab, w.k1, w.b)
    idx.force_path("tc")
    idx.gather_lexical(True)
    res = {}
    for mode in ("dual", None):
        idx.force_pair(mode)
        res[mode] = idx.hybrid_search(dev_tensor(w.Q_data), torch.from_numpy(w.q_indptr),
                                      torch.from_numpy(w.q_terms), w.alpha, w.k)
        torch.cuda.synchronize()
        assert idx.last_launch["tiles"] == 1 and idx.last_launch["block_n"] == 128
    assert torch.equal(res["dual"][0], res[None][0])
    assert torch.equal(res["dual"][1], res[None][1])
    idx.check()
    idx.close()
