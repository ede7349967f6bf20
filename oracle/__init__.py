"""CPU fp64 oracle for the OpRAG retrieval hot path -- TEST INFRASTRUCTURE.

Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline / reference
arm of ``bench.py`` may import this package.  The product library
(``paper_2608_08340_gb300``) never imports it and shares no code with it.

The arithmetic lives in ``oracle.c`` (plain C, fp64, full sorts); this module
only compiles it with gcc and marshals numpy arrays.  Arrays of dtype
``float32`` are taken as fp32 values, arrays of dtype ``uint16`` as bf16 bit
patterns; both are widened exactly to double inside the C code.

Function -> paper passage:
  dense_scores / search   Sec. 3.2 (Op_retrieve) and the TopK display of Sec. 4.4
  bm25                    Sec. 4.4 (BM25 over the whole corpus with exact
                          statistics; textbook Okapi form)
  hybrid_search           Sec. 4.4 weighted score fusion display
  rerank /                dense-first hybrid policy, Sec. 4.1 Retrieval and
  hybrid_dense_first      Sec. 5.5 (dense top-N, then the fusion over those
                          candidates; BM25 maximum over the candidates)
  embed_pool              Sec. 4.3 (hidden states -> mean pool -> L2 normalise;
                          padded positions masked)
  upsert                  Sec. 3.2 (Op_upsert), Sec. 4.1 (Upsert paragraph)
  replace_bags            the lexical half of Op_upsert (Sec. 3.2, Sec. 4.4)
  search_two              knowledge + memory index, one ranked result (Sec. 4.4)
  round_bf16              storage precision of the index (IEEE RNE)
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "oracle.c")
_OUT_DIR = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_OUT_DIR, "liboracle.so")

F32, BF16 = 0, 1

_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compiles oracle.c into oracle/_build/liboracle.so with gcc (fp64,
    no FMA contraction so results are identical on x86 and Arm hosts)."""
    os.makedirs(_OUT_DIR, exist_ok=True)
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-std=c11", "-D_GNU_SOURCE", "-ffp-contract=off", "-fPIC", "-shared",
           "-pthread", _SRC, "-o", tmp, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        lib = ctypes.CDLL(build())
        P, I64, I32, D = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int, ctypes.c_double
        lib.oracle_dense_scores.argtypes = [P, I32, I64, I32, P, I32, I32, P, I32]
        lib.oracle_topk_rows.argtypes = [P, I32, I64, I64, P, P, I32]
        lib.oracle_search.argtypes = [P, I32, I64, I32, P, I32, I32, I64, P, P, I32]
        lib.oracle_bm25.argtypes = [P, P, I64, I32, D, D, P, P, I32, P, P, P, I32]
        lib.oracle_hybrid_search.argtypes = [P, I32, I64, I32, P, I32, I32, P, P, I32, D, D,
                                             P, P, D, I64, P, P, P, I32]
        lib.oracle_rerank.argtypes = [P, I32, I64, I32, P, I32, I32, P, P, I32, D, D,
                                      P, P, P, I64, D, I64, P, P, I32]
        lib.oracle_embed_pool.argtypes = [P, I32, I32, I32, I32, P, P]
        lib.oracle_upsert.argtypes = [P, I32, I64, I32, P, P, I32, I64]
        lib.oracle_round_bf16.argtypes = [P, I64, P]
        for name in ("oracle_dense_scores", "oracle_topk_rows", "oracle_search", "oracle_bm25",
                     "oracle_hybrid_search", "oracle_rerank", "oracle_embed_pool",
                     "oracle_upsert"):
            getattr(lib, name).restype = ctypes.c_int
        lib.oracle_round_bf16.restype = None
        _lib = lib
        return lib


def _code(a: np.ndarray) -> int:
    if a.dtype == np.float32:
        return F32
    if a.dtype == np.uint16:
        return BF16
    raise TypeError(f"oracle inputs are float32 or uint16 (bf16 bits), got {a.dtype}")


def _ptr(a: np.ndarray):
    return a.ctypes.data_as(ctypes.c_void_p)


def _mat(a, name):
    a = np.ascontiguousarray(a)
    if a.ndim != 2:
        raise ValueError(f"{name} must be 2-D")
    _code(a)
    return a


def _check(rc: int, what: str) -> int:
    if rc < 0:
        raise RuntimeError(f"oracle {what} failed (rc={rc})")
    return rc


def dense_scores(E, Q, nthreads: int = 0) -> np.ndarray:
    """q x n fp64 matrix of inner products <Q[i], E[c]>."""
    E, Q = _mat(E, "E"), _mat(Q, "Q")
    if E.shape[1] != Q.shape[1]:
        raise ValueError("dimension mismatch")
    S = np.empty((Q.shape[0], E.shape[0]), np.float64)
    _check(_load().oracle_dense_scores(_ptr(E), _code(E), E.shape[0], E.shape[1], _ptr(Q),
                                       _code(Q), Q.shape[0], _ptr(S), nthreads), "dense_scores")
    return S


def topk_rows(S, kout: int, nthreads: int = 0):
    """Full-sort top-kout of each row of a fp64 score matrix: (ids int64, scores fp64)."""
    S = np.ascontiguousarray(S, dtype=np.float64)
    q, n = S.shape
    ids = np.empty((q, kout), np.int64)
    sc = np.empty((q, kout), np.float64)
    _check(_load().oracle_topk_rows(_ptr(S), q, n, kout, _ptr(ids), _ptr(sc), nthreads), "topk")
    return ids, sc


def search(E, Q, kout: int, nthreads: int = 0):
    """Exact dense top-kout (score desc, id asc) by full sort: (ids, scores fp64)."""
    E, Q = _mat(E, "E"), _mat(Q, "Q")
    if E.shape[1] != Q.shape[1]:
        raise ValueError("dimension mismatch")
    q = Q.shape[0]
    ids = np.empty((q, kout), np.int64)
    sc = np.empty((q, kout), np.float64)
    used = _check(_load().oracle_search(_ptr(E), _code(E), E.shape[0], E.shape[1], _ptr(Q),
                                        _code(Q), q, kout, _ptr(ids), _ptr(sc), nthreads), "search")
    search.last_threads = used
    return ids, sc


def _csr(indptr, terms):
    return (np.ascontiguousarray(indptr, dtype=np.int32),
            np.ascontiguousarray(terms, dtype=np.int32))


def bm25(doc_indptr, doc_terms, vocab: int, q_indptr, q_terms, k1: float = 1.2,
         b: float = 0.75, nthreads: int = 0):
    """q x n Okapi BM25 matrix by document scan; returns (matrix, avgdl, df)."""
    dip, dt = _csr(doc_indptr, doc_terms)
    qip, qt = _csr(q_indptr, q_terms)
    n, q = dip.shape[0] - 1, qip.shape[0] - 1
    out = np.empty((q, n), np.float64)
    avgdl = ctypes.c_double(0.0)
    df = np.zeros(vocab, np.int64)
    _check(_load().oracle_bm25(_ptr(dip), _ptr(dt), n, vocab, k1, b, _ptr(qip), _ptr(qt), q,
                               _ptr(out), ctypes.byref(avgdl), _ptr(df), nthreads), "bm25")
    return out, avgdl.value, df


def hybrid_search(E, Q, doc_indptr, doc_terms, vocab: int, q_indptr, q_terms, alpha: float,
                  kout: int, k1: float = 1.2, b: float = 0.75, nthreads: int = 0):
    """Fused top-kout of alpha*dense + (1-alpha)*BM25/max BM25: (ids, scores, max_bm25)."""
    E, Q = _mat(E, "E"), _mat(Q, "Q")
    dip, dt = _csr(doc_indptr, doc_terms)
    qip, qt = _csr(q_indptr, q_terms)
    n, q = E.shape[0], Q.shape[0]
    if dip.shape[0] != n + 1 or qip.shape[0] != q + 1:
        raise ValueError("CSR shapes do not match the dense inputs")
    ids = np.empty((q, kout), np.int64)
    sc = np.empty((q, kout), np.float64)
    mx = np.empty(q, np.float64)
    used = _check(_load().oracle_hybrid_search(
        _ptr(E), _code(E), n, E.shape[1], _ptr(Q), _code(Q), q, _ptr(dip), _ptr(dt), vocab,
        k1, b, _ptr(qip), _ptr(qt), alpha, kout, _ptr(ids), _ptr(sc), _ptr(mx), nthreads),
        "hybrid")
    hybrid_search.last_threads = used
    return ids, sc, mx


def rerank(E, Q, cand, doc_indptr, doc_terms, vocab: int, q_indptr, q_terms, alpha: float,
           kout: int, k1: float = 1.2, b: float = 0.75, nthreads: int = 0):
    """Fused top-kout over given candidates (q x N chunk ids, -1 = none), the
    BM25 maximum taken over the candidates: (ids, scores)."""
    E, Q = _mat(E, "E"), _mat(Q, "Q")
    dip, dt = _csr(doc_indptr, doc_terms)
    qip, qt = _csr(q_indptr, q_terms)
    cand = np.ascontiguousarray(cand, dtype=np.int64)
    n, q = E.shape[0], Q.shape[0]
    if dip.shape[0] != n + 1 or qip.shape[0] != q + 1 or cand.shape[0] != q:
        raise ValueError("shapes do not match")
    ids = np.empty((q, kout), np.int64)
    sc = np.empty((q, kout), np.float64)
    _check(_load().oracle_rerank(
        _ptr(E), _code(E), n, E.shape[1], _ptr(Q), _code(Q), q, _ptr(dip), _ptr(dt), vocab,
        k1, b, _ptr(qip), _ptr(qt), _ptr(cand), cand.shape[1], alpha, kout, _ptr(ids), _ptr(sc),
        nthreads), "rerank")
    return ids, sc


def hybrid_dense_first(E, Q, doc_indptr, doc_terms, vocab: int, q_indptr, q_terms,
                       alpha: float, n_cand: int, kout: int, k1: float = 1.2, b: float = 0.75,
                       nthreads: int = 0):
    """Dense-first hybrid: exact dense top-n_cand, then rerank of those: (ids, scores)."""
    cand, _ = search(E, Q, n_cand, nthreads)
    return rerank(E, Q, cand, doc_indptr, doc_terms, vocab, q_indptr, q_terms, alpha, kout,
                  k1, b, nthreads)


def embed_pool(hidden, mask):
    """batch x dim fp64: masked mean over tokens, then L2 normalisation.
    hidden: batch x tokens x dim, float32 or uint16 (bf16 bits); mask:
    batch x tokens, nonzero = a real token."""
    h = np.ascontiguousarray(hidden)
    _code(h)
    if h.ndim != 3:
        raise ValueError("hidden must be 3-D")
    m = np.ascontiguousarray(mask, dtype=np.uint8)
    if m.shape != h.shape[:2]:
        raise ValueError("mask must be batch x tokens")
    out = np.empty((h.shape[0], h.shape[2]), np.float64)
    _check(_load().oracle_embed_pool(_ptr(h), _code(h), h.shape[0], h.shape[1], h.shape[2],
                                     _ptr(m), _ptr(out)), "embed_pool")
    return out


def replace_bags(doc_indptr, doc_terms, ids, bag_indptr, bag_terms):
    """Token bags after replacing those of chunks ids[i] by bag i (a later
    duplicate id wins; ids at n.. append chunks, with empty bags for any chunk
    between n and the largest id): (indptr, terms) of the new CSR.  The
    lexical half of Op_upsert (Sec. 3.2; Sec. 4.4 keeps BM25 exact over the
    corpus, so df and avgdl follow the new bags)."""
    dip, dt = _csr(doc_indptr, doc_terms)
    bip, bt = _csr(bag_indptr, bag_terms)
    ids = np.asarray(ids, dtype=np.int64)
    n = dip.shape[0] - 1
    if ids.size and ids.min() < 0:
        raise ValueError("negative chunk id")
    n_new = max(n, int(ids.max()) + 1 if ids.size else n)
    bags = [list(dt[dip[i]:dip[i + 1]]) for i in range(n)] + [[] for _ in range(n_new - n)]
    for i, c in enumerate(ids.tolist()):
        bags[c] = list(bt[bip[i]:bip[i + 1]])
    ip = np.zeros(n_new + 1, np.int32)
    ip[1:] = np.cumsum([len(b) for b in bags])
    terms = np.array([t for b in bags for t in b], np.int32)
    return ip, terms


def search_two(Ek, Em, Q, kout: int, nthreads: int = 0):
    """Top-kout over two indices (knowledge index Ek, memory index Em, Sec. 4.4:
    both searched the same way, one ranked result): (ids, src, scores) where
    src 0 = Ek, 1 = Em; order score descending, then src, then chunk id."""
    nk = Ek.shape[0]
    both = np.concatenate([np.ascontiguousarray(Ek), np.ascontiguousarray(Em)], axis=0)
    # On the stacked matrix the (score desc, row asc) order is exactly
    # (score desc, src asc, id asc).
    ids, sc = search(both, Q, kout, nthreads)
    src = (ids >= nk).astype(np.int32)
    return np.where(src == 1, ids - nk, ids), src, sc


def upsert(E: np.ndarray, ids, rows) -> None:
    """In-place E[ids[i]] = rows[i] in order; raises on an out-of-range id."""
    if not E.flags.c_contiguous:
        raise ValueError("E must be C-contiguous")
    ids = np.ascontiguousarray(ids, dtype=np.int64)
    rows = _mat(rows, "rows")
    if rows.shape != (ids.shape[0], E.shape[1]):
        raise ValueError("rows shape mismatch")
    _check(_load().oracle_upsert(_ptr(E), _code(E), E.shape[0], E.shape[1], _ptr(ids),
                                 _ptr(rows), _code(rows), ids.shape[0]), "upsert")


def round_bf16(x) -> np.ndarray:
    """fp32 -> bf16 bit patterns, round to nearest even."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    out = np.empty(x.shape, np.uint16)
    _load().oracle_round_bf16(_ptr(x), x.size, _ptr(out))
    return out


def bf16_to_f32(bits) -> np.ndarray:
    """Exact widening of bf16 bit patterns to float32."""
    b = np.ascontiguousarray(bits, dtype=np.uint16)
    return (b.astype(np.uint32) << 16).view(np.float32)
