"""Two guarantees of the index around its kernels.

reserve: after oprag_index_reserve(q_max, k_max) a search of up to q_max
queries and k_max results allocates nothing (its scratch, the sampled first
pass of k > 32 and the shared per-query bounds were sized and cleared there).

bounded waits: every barrier wait of the tensor-core search kernel gives up
after a spin limit, records a device error, drains and returns.  A test hook
shortens the limit so that the waits of a real search run out; the index then
reports OPRAG_ERR_DEVICE once, and the next search with the normal limit is
exact again."""
import numpy as np
import pytest
import torch

from paper_2608_08340_gb300 import workloads
from paper_2608_08340_gb300._lib import OpragError
from paper_2608_08340_gb300.index import Index

from _gpu import check_dense, dev_tensor

pytestmark = pytest.mark.gpu


def test_reserve_covers_later_searches():
    # 40000 rows: 313 corpus tiles of 128, so k = 100 runs the sampled pass
    w = workloads.config(1, n=40000, batch=256)
    idx = Index(dev_tensor(w.E_data))
    idx.reserve(256, 100)
    before = idx.buffer_bytes()
    assert before["scratch"] > 0 and before["bounds"] >= 256 * 8
    Q = dev_tensor(w.Q_data)
    idx.enable_timing(True)
    for k in (5, 16, 32, 100):
        for q in (1, 100, 256):
            ids, sc = idx.search(Q[:q], k)
            t = idx.last_timing()
            if k == 100 and q == 256:
                assert t["sample_ms"] > 0.0          # the first pass ran
                check_dense(ids, sc, w.E_data, w.Q_data[:q], k, "reserved k=100",
                            rows=np.arange(0, 256, 37))
    idx.check()
    assert idx.buffer_bytes() == before


@pytest.mark.parametrize("q,mode", [(64, "single"), (256, "dual")])
def test_bounded_wait_gives_up_and_the_index_recovers(q, mode):
    w = workloads.config(1, n=8192, batch=q)
    idx = Index(dev_tensor(w.E_data))
    idx.force_pair(mode)
    Q = dev_tensor(w.Q_data)
    ref_ids, ref_sc = idx.search(Q, 5)
    idx.check()
    idx.set_wait_limit(1)                 # every wait that is not already complete gives up
    idx.search(Q, 5)
    torch.cuda.synchronize()              # the kernel returned: the context is usable
    with pytest.raises(OpragError) as err:
        idx.check()
    assert err.value.code == -6
    idx.check()                           # reported once, then cleared
    idx.set_wait_limit(0)
    ids, sc = idx.search(Q, 5)
    idx.check()
    assert idx.last_launch["tiles"] == (2 if mode == "dual" else 1)
    assert torch.equal(ids, ref_ids) and torch.equal(sc, ref_sc)
    check_dense(ids, sc, w.E_data, w.Q_data, 5, f"after abort ({mode})")
    idx.close()
