"""Top-k result checker -- TEST INFRASTRUCTURE (used by tests and smoke()).

Compares a GPU top-k list (fp32 scores) against the oracle's fp64 list for the
same query, following the tie rule of the TopK definition (Sec. 4.4): order
is score descending, then chunk id ascending.

Because the GPU accumulates in fp32 and the oracle in fp64, two oracle
scores closer than ``tol`` may legitimately come out in either order.  The
oracle's ranking is therefore cut into *near-tie blocks*: maximal runs of
consecutive ranks whose adjacent fp64 scores differ by less than ``tol``.
The GPU list passes when
  * every returned (id, score) has |score - s_oracle(id)| <= tol, and
  * for every rank r < k, the id the GPU puts at rank r belongs to the
    oracle's block that contains rank r (inside a block the order is free;
    a block that straddles rank k may contribute any of its members).
The oracle list must extend past the last block that reaches rank k; the
checker reports an error when it does not (ask the oracle for more ranks).
"""
from __future__ import annotations

import numpy as np


class TopkMismatch(AssertionError):
    pass


def near_tie_blocks(scores: np.ndarray, tol: float) -> np.ndarray:
    """Block index per oracle rank: adjacent ranks share a block when their
    scores differ by less than tol."""
    s = np.asarray(scores, dtype=np.float64)
    if s.size == 0:
        return np.zeros(0, np.int64)
    gaps = (s[:-1] - s[1:]) >= tol
    return np.concatenate([[0], np.cumsum(gaps)]).astype(np.int64)


def check_query(gpu_ids, gpu_scores, or_ids, or_scores, k: int, tol: float = 1e-4,
                n: int | None = None, where: str = "") -> None:
    gpu_ids = np.asarray(gpu_ids, dtype=np.int64)[:k]
    gpu_scores = np.asarray(gpu_scores, dtype=np.float64)[:k]
    or_ids = np.asarray(or_ids, dtype=np.int64)
    or_scores = np.asarray(or_scores, dtype=np.float64)
    if gpu_ids.shape[0] != k:
        raise TopkMismatch(f"{where}: GPU returned {gpu_ids.shape[0]} entries, want {k}")
    L = or_ids.shape[0]
    blocks = near_tie_blocks(or_scores, tol)
    if L < k:
        raise TopkMismatch(f"{where}: oracle list shorter than k")
    last_block = blocks[k - 1]
    complete = (n is not None and L >= n)
    if not complete and blocks[L - 1] == last_block:
        raise TopkMismatch(f"{where}: near-tie block at rank k runs to the end of the oracle "
                           f"list ({L} ranks); ask the oracle for more ranks")
    pos = {int(c): i for i, c in enumerate(or_ids)}
    if len(set(gpu_ids.tolist())) != k:
        raise TopkMismatch(f"{where}: duplicate ids in GPU list {gpu_ids.tolist()}")
    for r in range(k):
        cid = int(gpu_ids[r])
        if cid not in pos:
            raise TopkMismatch(f"{where}: rank {r}: id {cid} not among the oracle's top {L}")
        orank = pos[cid]
        if blocks[orank] != blocks[r]:
            raise TopkMismatch(
                f"{where}: rank {r}: id {cid} has oracle rank {orank} (score "
                f"{or_scores[orank]:.9f}); rank {r} belongs to a block with score "
                f"{or_scores[r]:.9f}; GPU ids {gpu_ids.tolist()} oracle ids "
                f"{or_ids[:k + 3].tolist()}")
        err = abs(float(gpu_scores[r]) - float(or_scores[orank]))
        if not err <= tol:
            raise TopkMismatch(f"{where}: rank {r}: id {cid} GPU score {gpu_scores[r]!r} vs "
                               f"oracle {or_scores[orank]!r} (|diff| {err:.3e} > {tol})")


def check_topk(gpu_ids, gpu_scores, or_ids, or_scores, k: int, tol: float = 1e-4,
               n: int | None = None, query_index=None, label: str = "") -> dict:
    """Checks every query row; returns simple statistics on success."""
    gpu_ids = np.asarray(gpu_ids)
    gpu_scores = np.asarray(gpu_scores)
    or_ids = np.asarray(or_ids)
    or_scores = np.asarray(or_scores)
    q = gpu_ids.shape[0]
    exact = 0
    max_err = 0.0
    for i in range(q):
        qi = int(query_index[i]) if query_index is not None else i
        check_query(gpu_ids[i], gpu_scores[i], or_ids[i], or_scores[i], k, tol, n,
                    where=f"{label} query {qi}")
        if np.array_equal(np.asarray(gpu_ids[i][:k], np.int64), np.asarray(or_ids[i][:k], np.int64)):
            exact += 1
        pos = {int(c): j for j, c in enumerate(or_ids[i])}
        for r in range(k):
            e = abs(float(gpu_scores[i][r]) - float(or_scores[i][pos[int(gpu_ids[i][r])]]))
            max_err = max(max_err, e)
    return {"queries": q, "exact_id_lists": exact, "max_abs_score_err": max_err}


def topk_with_margin(fn, k: int, n: int, tol: float = 1e-4, margin: int = 48):
    """Calls fn(kout) -> (ids, scores, ...) with kout = k + margin ranks of the
    oracle, growing the margin until the near-tie block at rank k ends inside
    the returned ranks for every row (or every chunk is returned)."""
    while True:
        kout = min(n, k + margin)
        res = fn(kout)
        ids, sc = res[0], res[1]
        if kout >= n:
            return ids, sc
        if all(near_tie_blocks(sc[i], tol)[-1] != near_tie_blocks(sc[i], tol)[k - 1]
               for i in range(sc.shape[0])):
            return ids, sc
        margin *= 4
