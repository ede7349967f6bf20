"""Python face of the C ABI: an Index over torch device memory and streams.

Every step of search, hybrid search and upsert runs in the CUDA kernels of
liboprag.so; this module only checks shapes, allocates outputs with torch and
passes pointers.
"""
from __future__ import annotations

import ctypes

_I32 = ctypes.c_int32

import numpy as np
import torch

from . import _lib
from ._lib import OPRAG_BF16, OPRAG_F32, check

_DT = {torch.float32: OPRAG_F32, torch.bfloat16: OPRAG_BF16}


def _stream_ptr(stream) -> int:
    if stream is None:
        stream = torch.cuda.current_stream()
    return int(stream.cuda_stream)


def _ptr(t) -> int:
    return int(t.data_ptr())


class Index:
    """Chunk-embedding index on the current CUDA device.

    emb: (n, d) float32 or bfloat16 tensor on the host or a CUDA device.
    dtype: storage type (torch.float32 or torch.bfloat16); defaults to emb's.
    """

    def __init__(self, emb: torch.Tensor, dtype: torch.dtype | None = None):
        if emb.dim() != 2 or emb.dtype not in _DT:
            raise ValueError("emb must be a 2-D float32 or bfloat16 tensor")
        emb = emb.contiguous()
        dtype = dtype or emb.dtype
        if dtype not in _DT:
            raise ValueError("dtype must be float32 or bfloat16")
        self._lib = _lib.load()
        h = ctypes.c_void_p()
        check(self._lib.oprag_index_create(ctypes.byref(h), _ptr(emb), emb.shape[0], emb.shape[1],
                                           _DT[dtype], _DT[emb.dtype], int(emb.is_cuda)))
        self._h = h
        self.n, self.d = int(emb.shape[0]), int(emb.shape[1])
        self.dtype = dtype
        self.device = torch.device("cuda", torch.cuda.current_device())

    # -- lifetime
    def close(self) -> None:
        if getattr(self, "_h", None) is not None and self._h.value:
            self._lib.oprag_index_destroy(self._h)
            self._h = ctypes.c_void_p()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    @property
    def handle(self) -> int:
        return int(self._h.value or 0)

    # -- searches
    def _queries(self, queries: torch.Tensor) -> torch.Tensor:
        if queries.dim() != 2 or queries.shape[1] != self.d:
            raise ValueError(f"queries must be (q, {self.d})")
        if queries.dtype != self.dtype:
            raise ValueError(f"queries must be {self.dtype}")
        if not queries.is_cuda:
            raise ValueError("queries must be on the GPU (use search_host for host buffers)")
        return queries.contiguous()

    def search(self, queries: torch.Tensor, k: int, stream=None, out=None):
        """Exact top-k: (ids int64 (q, k), scores float32 (q, k)), best first."""
        queries = self._queries(queries)
        q = int(queries.shape[0])
        if out is None:
            ids = torch.empty((q, k), dtype=torch.int64, device=queries.device)
            scores = torch.empty((q, k), dtype=torch.float32, device=queries.device)
        else:
            ids, scores = out
        check(self._lib.oprag_search(self._h, _ptr(queries), q, k, _ptr(ids), _ptr(scores),
                                     _stream_ptr(stream)))
        return ids, scores

    def search_host(self, queries: torch.Tensor, k: int, stream=None, out=None):
        """Search with host (ideally pinned) buffers; synchronous."""
        if queries.is_cuda or queries.dtype != self.dtype or queries.shape[-1] != self.d:
            raise ValueError("queries must be a host tensor of the index dtype")
        queries = queries.contiguous()
        q = int(queries.shape[0])
        if out is None:
            ids = torch.empty((q, k), dtype=torch.int64)
            scores = torch.empty((q, k), dtype=torch.float32)
        else:
            ids, scores = out
        check(self._lib.oprag_search_host(self._h, _ptr(queries), q, k, _ptr(ids), _ptr(scores),
                                          _stream_ptr(stream)))
        return ids, scores

    def set_sparse(self, doc_indptr, doc_terms, vocab: int, k1: float = 1.2, b: float = 0.75):
        """Attaches per-chunk term-id bags (host CSR) for BM25."""
        ip = np.ascontiguousarray(doc_indptr, dtype=np.int32)
        tm = np.ascontiguousarray(doc_terms, dtype=np.int32)
        if ip.shape[0] != self.n + 1:
            raise ValueError("doc_indptr must have n + 1 entries")
        check(self._lib.oprag_index_set_sparse(self._h, ip.ctypes.data, tm.ctypes.data, vocab,
                                               k1, b))

    def hybrid_search(self, queries: torch.Tensor, q_indptr: torch.Tensor, q_terms: torch.Tensor,
                      alpha: float, k: int, stream=None):
        """Fused alpha * dense + (1 - alpha) * BM25 / max BM25 top-k."""
        queries = self._queries(queries)
        q = int(queries.shape[0])
        qip = q_indptr.to(device=queries.device, dtype=torch.int32).contiguous()
        qt = q_terms.to(device=queries.device, dtype=torch.int32).contiguous()
        if qt.numel() == 0:
            qt = torch.zeros(1, dtype=torch.int32, device=queries.device)
        if qip.numel() != q + 1:
            raise ValueError("q_indptr must have q + 1 entries")
        ids = torch.empty((q, k), dtype=torch.int64, device=queries.device)
        scores = torch.empty((q, k), dtype=torch.float32, device=queries.device)
        check(self._lib.oprag_hybrid_search(self._h, _ptr(queries), q, _ptr(qip), _ptr(qt),
                                            float(alpha), k, _ptr(ids), _ptr(scores),
                                            _stream_ptr(stream)))
        return ids, scores

    def hybrid_search_dense_first(self, queries: torch.Tensor, q_indptr: torch.Tensor,
                                  q_terms: torch.Tensor, alpha: float, n_cand: int, k: int,
                                  stream=None):
        """Dense top-n_cand, then the fused rerank of those candidates (BM25
        maximum over the candidates); top-k (ids, scores)."""
        queries = self._queries(queries)
        q = int(queries.shape[0])
        qip = q_indptr.to(device=queries.device, dtype=torch.int32).contiguous()
        qt = q_terms.to(device=queries.device, dtype=torch.int32).contiguous()
        if qt.numel() == 0:
            qt = torch.zeros(1, dtype=torch.int32, device=queries.device)
        if qip.numel() != q + 1:
            raise ValueError("q_indptr must have q + 1 entries")
        ids = torch.empty((q, k), dtype=torch.int64, device=queries.device)
        scores = torch.empty((q, k), dtype=torch.float32, device=queries.device)
        check(self._lib.oprag_hybrid_search_dense_first(
            self._h, _ptr(queries), q, _ptr(qip), _ptr(qt), float(alpha), n_cand, k, _ptr(ids),
            _ptr(scores), _stream_ptr(stream)))
        return ids, scores

    # -- upsert
    def upsert(self, ids, rows: torch.Tensor, stream=None) -> None:
        """rows[i] overwrites chunk ids[i] (host int64 ids; later duplicates win)."""
        ids_np = np.ascontiguousarray(ids.cpu().numpy() if isinstance(ids, torch.Tensor) else ids,
                                      dtype=np.int64)
        if rows.dim() != 2 or rows.shape[1] != self.d or rows.shape[0] != ids_np.shape[0]:
            raise ValueError("rows must be (len(ids), d)")
        if rows.dtype not in _DT:
            raise ValueError("rows must be float32 or bfloat16")
        rows = rows.contiguous()
        check(self._lib.oprag_upsert(self._h, ids_np.ctypes.data, _ptr(rows), ids_np.shape[0],
                                     _DT[rows.dtype], int(rows.is_cuda), _stream_ptr(stream)))

    def append(self, rows: torch.Tensor, stream=None) -> int:
        """Appends rows as chunks n, n + 1, ...; returns the first new id."""
        if rows.dim() != 2 or rows.shape[1] != self.d or rows.dtype not in _DT:
            raise ValueError(f"rows must be (m, {self.d}) float32 or bfloat16")
        rows = rows.contiguous()
        first = ctypes.c_int64()
        check(self._lib.oprag_append(self._h, _ptr(rows), int(rows.shape[0]), _DT[rows.dtype],
                                     int(rows.is_cuda), ctypes.byref(first), _stream_ptr(stream)))
        self.n += int(rows.shape[0])
        return int(first.value)

    def update_sparse(self, ids, bag_indptr, bag_terms) -> None:
        """Replaces the token bags of chunks ids (host CSR bags, later duplicates win)."""
        ids_np = np.ascontiguousarray(ids, dtype=np.int64)
        ip = np.ascontiguousarray(bag_indptr, dtype=np.int32)
        tm = np.ascontiguousarray(bag_terms, dtype=np.int32)
        if ip.shape[0] != ids_np.shape[0] + 1:
            raise ValueError("bag_indptr must have len(ids) + 1 entries")
        if tm.size == 0:
            tm = np.zeros(1, np.int32)
        check(self._lib.oprag_index_update_sparse(self._h, ids_np.ctypes.data, ids_np.shape[0],
                                                  ip.ctypes.data, tm.ctypes.data))

    # -- misc
    def rows(self, first: int = 0, count: int | None = None) -> torch.Tensor:
        count = self.n - first if count is None else count
        out = torch.empty((count, self.d), dtype=self.dtype)
        check(self._lib.oprag_index_get_rows(self._h, first, count, _ptr(out)))
        return out

    def reserve(self, q_max: int, k_max: int) -> None:
        check(self._lib.oprag_index_reserve(self._h, q_max, k_max))

    def check(self) -> None:
        check(self._lib.oprag_index_check(self._h))

    def set_option(self, option: int, value: int) -> None:
        check(self._lib.oprag_index_set_option(self._h, option, value))

    def force_path(self, path: str | None) -> None:
        self.set_option(_lib.OPRAG_OPT_PATH, {None: 0, "simt": 1, "tc": 2}[path])

    def force_pair(self, mode: str | None) -> None:
        """None: automatic; "single": one CTA per MMA, one query tile per unit;
        "pair": CTA pairs; "dual": one CTA, two query tiles per unit."""
        self.set_option(_lib.OPRAG_OPT_PAIR, {None: 0, "single": 1, "pair": 2, "dual": 3}[mode])

    def force_block_n(self, bn: int | None) -> None:
        self.set_option(_lib.OPRAG_OPT_BLOCK_N, bn or 0)

    def enable_timing(self, on: bool = True) -> None:
        self.set_option(_lib.OPRAG_OPT_TIMING, int(on))

    def last_timing(self) -> dict:
        """Device milliseconds of the last timed search's kernels: lexical pass,
        sampled first pass (k > 32 over many tiles), main search pass, merge."""
        a, b, c, m = ctypes.c_float(), ctypes.c_float(), ctypes.c_float(), ctypes.c_float()
        check(self._lib.oprag_index_last_timing(self._h, ctypes.byref(a), ctypes.byref(b),
                                                ctypes.byref(c), ctypes.byref(m)))
        return {"lexical_ms": a.value, "sample_ms": b.value, "search_ms": c.value,
                "merge_ms": m.value}

    def buffer_bytes(self) -> dict:
        """Bytes held by the index's grow-on-demand device buffers."""
        a, b, c = ctypes.c_int64(), ctypes.c_int64(), ctypes.c_int64()
        check(self._lib.oprag_index_buffer_bytes(self._h, ctypes.byref(a), ctypes.byref(b),
                                                 ctypes.byref(c)))
        return {"scratch": a.value, "bounds": b.value, "lexical": c.value}

    def gather_lexical(self, on: bool = True) -> None:
        """Hybrid search: gather BM25 in the search epilogue (True) instead of
        reading a materialised q x n BM25 block (False, the default)."""
        self.set_option(_lib.OPRAG_OPT_LEX_GATHER, int(on))

    PHASES = ("entry", "setup", "first_stage", "last_stage", "last_commit", "epi0_done",
              "epi1_done", "exit")

    def enable_phases(self, on: bool = True) -> None:
        """Measurement hook: per-CTA global-timer stamps of the main pass."""
        self.set_option(_lib.OPRAG_OPT_PHASES, int(on))

    def last_phases(self) -> np.ndarray:
        """(ctas, 8) int64 global-timer stamps (ns) of the last main pass, in
        the order of PHASES (0 where a CTA records none)."""
        n = ctypes.c_int32()
        check(self._lib.oprag_index_last_phases(self._h, None, 0, ctypes.byref(n)))
        out = np.zeros((n.value, 8), np.int64)
        check(self._lib.oprag_index_last_phases(
            self._h, out.ctypes.data_as(ctypes.POINTER(ctypes.c_int64)), out.size,
            ctypes.byref(n)))
        return out

    def set_wait_limit(self, cycles: int) -> None:
        """Test hook: spin limit of the search kernels' barrier waits (0 = default)."""
        self.set_option(_lib.OPRAG_OPT_WAIT_LIMIT, int(cycles))

    @property
    def last_launch(self) -> dict:
        """Main kernel launch of the last search: grid (CTAs), cluster (2 = CTA
        pairs), block_n, query tiles per CTA and unit (2 = dual mode); zeros
        for the SIMT kernel."""
        g, c, b, t = _I32(), _I32(), _I32(), _I32()
        check(self._lib.oprag_index_last_launch(self._h, ctypes.byref(g), ctypes.byref(c),
                                                ctypes.byref(b)))
        check(self._lib.oprag_index_last_tiles_per_cta(self._h, ctypes.byref(t)))
        return {"grid": g.value, "cluster": c.value, "block_n": b.value, "tiles": t.value}

    @property
    def last_path(self) -> str:
        return {0: "none", 1: "simt", 2: "tc"}[self._lib.oprag_index_last_path(self._h)]


def embed_pool(hidden: torch.Tensor, mask: torch.Tensor, out_dtype: torch.dtype = torch.bfloat16,
               stream=None) -> torch.Tensor:
    """Tail of Op_embed: masked mean pool over tokens, then L2 normalisation.

    hidden: (batch, tokens, dim) bfloat16 or float32 CUDA tensor; mask:
    (batch, tokens) bool or uint8 (nonzero = a real token).  Returns
    (batch, dim) in out_dtype (bfloat16 or float32), usable as queries."""
    lib = _lib.load()
    if hidden.dim() != 3 or hidden.dtype not in _DT or not hidden.is_cuda:
        raise ValueError("hidden must be a 3-D bfloat16 or float32 CUDA tensor")
    if out_dtype not in _DT:
        raise ValueError("out_dtype must be bfloat16 or float32")
    b, t, d = (int(x) for x in hidden.shape)
    hidden = hidden.contiguous()
    m = mask.to(device=hidden.device, dtype=torch.uint8).contiguous()
    if tuple(m.shape) != (b, t):
        raise ValueError("mask must be (batch, tokens)")
    out = torch.empty((b, d), dtype=out_dtype, device=hidden.device)
    check(lib.oprag_embed_pool(_ptr(hidden), _DT[hidden.dtype], b, t, d, _ptr(m), _ptr(out),
                               _DT[out_dtype], _stream_ptr(stream)))
    return out


def search_two(knowledge: Index, memory: Index, queries: torch.Tensor, k: int, stream=None):
    """Dense top-k over a knowledge and a memory index: (ids, src, scores);
    src 0 = knowledge, 1 = memory; ids are chunk ids within their index."""
    queries = knowledge._queries(queries)
    q = int(queries.shape[0])
    ids = torch.empty((q, k), dtype=torch.int64, device=queries.device)
    src = torch.empty((q, k), dtype=torch.int32, device=queries.device)
    scores = torch.empty((q, k), dtype=torch.float32, device=queries.device)
    check(knowledge._lib.oprag_search_two(knowledge._h, memory._h, _ptr(queries), q, k, _ptr(ids),
                                          _ptr(src), _ptr(scores), _stream_ptr(stream)))
    return ids, src, scores



_PLAN_FIELDS = ("grid", "block_n", "cluster", "dual", "qt", "uqt", "nt", "win", "pmax",
                "stages", "smem", "scratch", "sets")


def plan_search(n: int, d: int, q: int, k: int, num_sms: int = 148, force_block_n: int = 0,
                force_pair: int = 0, pair_capacity: int = 74) -> dict:
    """Host-side plan of a tensor-core search (no device work, no GPU needed):
    launch shape, schedule, shared memory and list scratch."""
    out = (ctypes.c_int64 * len(_PLAN_FIELDS))()
    check(_lib.load().oprag_plan_search(n, d, q, k, num_sms, force_block_n, force_pair,
                                        pair_capacity, out))
    return dict(zip(_PLAN_FIELDS, (int(v) for v in out)))
