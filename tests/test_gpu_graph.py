"""Graph mode of oprag_search: a search repeated with the same pointers is
captured once and replayed.  The replay must follow the current contents of
the query buffer and of the index, start from cleared shared k-th bounds, and
be rebuilt after the index changes."""
import numpy as np
import pytest
import torch

from paper_2608_08340_gb300 import _lib, workloads
from paper_2608_08340_gb300.index import Index

from _gpu import check_dense, dev_tensor

pytestmark = pytest.mark.gpu


def _bits(t):
    return t.view(torch.int16).cpu().numpy().view(np.uint16)


@pytest.mark.parametrize("k", [10, 100])
def test_graph_replay_follows_new_queries_and_index_changes(k):
    w = workloads.config(1, n=160000 if k > 32 else 20000, batch=130)
    E = w.E_data
    idx = Index(dev_tensor(E))
    idx.set_option(_lib.OPRAG_OPT_GRAPH, 1)
    s = torch.cuda.Stream()
    rng = np.random.default_rng(k)
    Q = dev_tensor(w.Q_data)                      # one buffer, refilled between calls
    ids = torch.empty((w.q, k), dtype=torch.int64, device="cuda")
    sc = torch.empty((w.q, k), dtype=torch.float32, device="cuda")
    with torch.cuda.stream(s):
        for it in range(5):
            # new query contents in the same buffer: self matches of random rows
            rows = rng.choice(w.n, w.q, replace=False)
            Q.copy_(dev_tensor(E[rows]))
            idx.search(Q, k, stream=s, out=(ids, sc))
            s.synchronize()
            assert (ids[:, 0].cpu().numpy() == rows).all(), f"call {it}"
            if it in (2, 4):
                check_dense(ids, sc, E, E[rows], k, f"graph call {it}",
                            rows=np.arange(0, w.q, 13))
    idx.check()


def test_graph_is_rebuilt_after_an_append():
    w = workloads.config(1, n=6000, batch=64)
    idx = Index(dev_tensor(w.E_data[:5000]))
    idx.set_option(_lib.OPRAG_OPT_GRAPH, 1)
    s = torch.cuda.Stream()
    Q = dev_tensor(w.E_data[5000:5064])          # queries equal to rows not yet indexed
    ids = torch.empty((64, 5), dtype=torch.int64, device="cuda")
    sc = torch.empty((64, 5), dtype=torch.float32, device="cuda")
    with torch.cuda.stream(s):
        for _ in range(3):
            idx.search(Q, 5, stream=s, out=(ids, sc))
        s.synchronize()
        assert not (ids[:, 0].cpu().numpy() >= 5000).any()
        idx.append(dev_tensor(w.E_data[5000:]))
        for _ in range(3):
            idx.search(Q, 5, stream=s, out=(ids, sc))
        s.synchronize()
    assert (ids[:, 0].cpu().numpy() == np.arange(5000, 5064)).all()
    idx.check()


def test_graph_mode_on_the_default_stream_runs_directly():
    w = workloads.config(1, n=4000, batch=16)
    idx = Index(dev_tensor(w.E_data))
    idx.set_option(_lib.OPRAG_OPT_GRAPH, 1)
    for _ in range(3):
        ids, sc = idx.search(dev_tensor(w.Q_data), 5)
    check_dense(ids, sc, w.E_data, w.Q_data, 5, "graph mode, default stream")
