"""oprag_search_noalloc: the search entry point for callers that must not
allocate device memory while serving (a process whose memory pool already
holds the GPU, or one that cannot take the device-wide synchronisation a
cudaMalloc or cudaFree may cause).  Its partial lists, sampled first pass and
shared bounds live in a static 16 MiB device array instead of the index's
growable scratch buffer.

Called through the C ABI on a fresh index, before any oprag_search, and
checked against oprag_search on the same inputs, twice in a row (the static
array keeps the previous call's contents, so the second call checks that
nothing leaks between calls); the index's own buffers must still be empty
after the no-allocation calls.  Kept in a file that pytest collects last."""
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


# (cfg, q, k, n): dual mode (256 queries), one query, single CTAs with lists of
# 16, the fp32 SIMT kernel, and k > 32 (buffered lists) on a small corpus.
@pytest.mark.parametrize("cfg,q,k,n", [(1, 256, 5, 20000), (1, 1, 5, 20000), (2, 300, 10, 20000),
                                       (0, 16, 5, None), (1, 64, 100, 2000)])
def test_noalloc_matches_search_twice(cfg, q, k, n):
    lib = _lib.load()
    w = workloads.config(cfg, batch=q, n=n)
    idx = Index(dev_tensor(w.E_data))
    Q = dev_tensor(w.Q_data)
    got = []
    for _ in range(2):
        rc, ids, sc = _noalloc(lib, idx, Q, k)
        assert rc == 0, lib.oprag_last_error().decode()
        torch.cuda.synchronize()
        got.append((ids, sc))
    # nothing was allocated for the index: its grow-on-demand buffers are empty
    assert idx.buffer_bytes() == {"scratch": 0, "bounds": 0, "lexical": 0}
    idx.check()
    ref_ids, ref_sc = idx.search(Q, k)
    torch.cuda.synchronize()
    for ids, sc in got:
        assert torch.equal(ids, ref_ids)
        assert (sc - ref_sc).abs().max().item() <= TOL
    idx.check()
    idx.close()


@pytest.mark.parametrize("q,k", [(4096, 256), (64, 100)])
def test_noalloc_refuses_searches_beyond_the_static_array(q, k):
    """Thousands of queries with k = 256, and k = 100 over 157 corpus tiles:
    there one 128-row list of 256 keys per CTA (about 38 MB over the grid)
    exceeds the 16 MiB array."""
    lib = _lib.load()
    w = workloads.config(1, batch=q, n=20000)
    idx = Index(dev_tensor(w.E_data))
    rc, ids, _ = _noalloc(lib, idx, dev_tensor(w.Q_data), k)
    assert rc == -1
    msg = lib.oprag_last_error().decode()
    assert "static array" in msg
    torch.cuda.synchronize()
    assert (ids == -7).all()            # nothing was launched
    assert idx.buffer_bytes() == {"scratch": 0, "bounds": 0, "lexical": 0}
    idx.close()
