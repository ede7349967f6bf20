"""oprag_search_noalloc: the search entry point for callers that must not
allocate device memory while serving (its partial lists live in a static
16 MiB device array instead of the index's growable scratch buffer).

Called through the C ABI and checked against oprag_search on the same inputs,
twice in a row (the static array keeps the previous call's contents, so the
second call checks that nothing leaks between calls).  Kept in a file that
pytest collects last."""
import ctypes

import numpy as np
import pytest
import torch

from paper_2608_08340_gb300 import _lib, workloads
from paper_2608_08340_gb300.index import Index

from _gpu import TOL, dev_tensor

pytestmark = pytest.mark.gpu


def _noalloc(lib, idx, Q, k):
    q = Q.shape[0]
    ids = torch.full((q, k), -7, dtype=torch.int64, device=Q.device)
    sc = torch.full((q, k), 7.0, dtype=torch.float32, device=Q.device)
    rc = lib.oprag_search_noalloc(idx.handle, Q.data_ptr(), q, k, ids.data_ptr(), sc.data_ptr(),
                                  torch.cuda.current_stream().cuda_stream)
    return rc, ids, sc


@pytest.mark.parametrize("cfg,q,k,n", [(1, 256, 5, 20000), (1, 1, 5, 20000), (2, 300, 10, 20000),
                                       (0, 16, 5, None), (1, 64, 100, 2000)])
def test_noalloc_matches_search_twice(cfg, q, k, n):
    lib = _lib.load()
    w = workloads.config(cfg, batch=q, n=n)
    idx = Index(dev_tensor(w.E_data))
    Q = dev_tensor(w.Q_data)
    ref_ids, ref_sc = idx.search(Q, k)
    for _ in range(2):
        rc, ids, sc = _noalloc(lib, idx, Q, k)
        assert rc == 0, lib.oprag_last_error().decode()
        torch.cuda.synchronize()
        assert torch.equal(ids, ref_ids)
        assert (sc - ref_sc).abs().max().item() <= TOL
    idx.check()
    idx.close()


def test_noalloc_refuses_searches_beyond_the_static_array():
    lib = _lib.load()
    w = workloads.config(1, batch=4096, n=20000)
    idx = Index(dev_tensor(w.E_data))
    rc, ids, _ = _noalloc(lib, idx, dev_tensor(w.Q_data), 256)
    assert rc == -1
    msg = lib.oprag_last_error().decode()
    assert "static array" in msg
    assert (ids == -7).all()            # nothing was launched
    idx.close()
