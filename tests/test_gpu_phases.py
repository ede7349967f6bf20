"""The measurement hook of the tensor-core main pass (OPRAG_OPT_PHASES):
per-CTA global-timer stamps come in the order of the CTA's run, and turning
the hook on changes no result."""
import numpy as np
import pytest
import torch

from paper_2608_08340_gb300 import workloads
from paper_2608_08340_gb300.index import Index

from _gpu import dev_tensor

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("q,k", [(256, 5), (64, 32), (300, 100)])
def test_phase_stamps_are_ordered_and_change_nothing(q, k):
    w = workloads.config(1, n=30000, batch=q)
    idx = Index(dev_tensor(w.E_data))
    Q = dev_tensor(w.Q_data)
    ref_ids, ref_sc = idx.search(Q, k)
    idx.enable_phases(True)
    ids, sc = idx.search(Q, k)
    st = idx.last_phases()
    idx.enable_phases(False)
    assert torch.equal(ids, ref_ids) and torch.equal(sc, ref_sc)
    assert st.shape == (idx.last_launch["grid"], 8)
    entry, setup, first, last, commit, e0, e1, exit_ = st.T
    assert (entry > 0).all() and (setup >= entry).all() and (exit_ >= setup).all()
    issuers = first > 0                 # CTAs that issue MMAs (all but pair peers)
    assert issuers.any()
    assert (last[issuers] >= first[issuers]).all() and (commit[issuers] >= last[issuers]).all()
    assert (first[issuers] >= setup[issuers]).all() and (exit_[issuers] >= commit[issuers]).all()
    assert ((e0 > 0) & (e0 <= exit_)).all()
    assert ((e1 == 0) | (e1 <= exit_)).all()
    # a whole pass of this size takes well under a second of global time
    assert (exit_.max() - entry.min()) < 1_000_000_000
    idx.check()
    idx.close()
