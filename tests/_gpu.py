"""Helpers for the GPU parity tests: move workloads to the device, run the
oracle with enough extra ranks for the near-tie rule, and compare."""
import numpy as np
import torch

import oracle
from oracle import check

TOL = 1e-4   # absolute score tolerance of the parity bar


def dev_tensor(a: np.ndarray, device="cuda") -> torch.Tensor:
    """uint16 arrays are bf16 bit patterns; float32 arrays stay float32."""
    if a.dtype == np.uint16:
        return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).view(torch.bfloat16).to(device)
    return torch.from_numpy(np.ascontiguousarray(a)).to(device)


def oracle_topk(fn, k: int, n: int, margin: int = 48):
    """Calls fn(kout) -> (ids, scores, ...) with enough oracle ranks for the
    near-tie rule at rank k (oracle/check.py)."""
    return check.topk_with_margin(fn, k, n, TOL, margin)


def check_dense(ids, scores, E_data, Q_data, k, label="", rows=None):
    """Checks GPU results (torch or numpy) for queries Q_data (or its rows)."""
    ids = ids.cpu().numpy() if isinstance(ids, torch.Tensor) else ids
    scores = scores.cpu().numpy() if isinstance(scores, torch.Tensor) else scores
    Qs = Q_data if rows is None else Q_data[rows]
    gi = ids if rows is None else ids[rows]
    gs = scores if rows is None else scores[rows]
    n = E_data.shape[0]
    o_ids, o_sc = oracle_topk(lambda kout: oracle.search(E_data, Qs, kout), k, n)
    return check.check_topk(gi, gs, o_ids, o_sc, k, TOL, n=n, label=label,
                            query_index=None if rows is None else np.arange(len(Q_data))[rows])
