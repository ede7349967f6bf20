"""Seeded synthetic inputs for the retrieval hot path.

This module draws random inputs only; it holds none of the retrieval
arithmetic (no scoring, no BM25 statistics, no ranking).  It serves both the
CUDA path (tests, bench, smoke) and the CPU oracle, which is why it lives on
its own.

The shapes follow the paper's serving experiments: 32K chunks (Sec. 5.1),
768-dimensional embeddings (Sec. 4.4 memory estimate), 1024 queries per
scenario (Sec. 5.1), L2-normalised vectors (Sec. 4.3 embedding chain: mean
pool then L2 normalise).  The paper's corpus (WikiText-103) and LLM weights are
not available, so i.i.d. Gaussian directions (and a clustered mixture to stress
near ties) stand in for the embeddings, and Zipf-distributed token bags stand
in for the chunk text that BM25 indexes.

Recipe (all numpy PCG64 ``default_rng``):
  * dense rows: float32 standard normals drawn in chunks of 65536 rows
    (chunk c from its own generator seeded (seed, c)), normalised in float64,
    cast to float32; bf16 inputs are the
    round-to-nearest-even bf16 of that float32 (torch ``.to(bfloat16)``).
  * clustered rows: centres ~ N(0, I); each row picks a centre uniformly;
    x = c + sigma * z; then normalised as above.
  * token bags: chunk length uniform on [len_lo, len_hi]; tokens i.i.d. from a
    Zipf(s) law truncated to ranks 1..vocab; term id = rank - 1.
  * seeds: corpus rows 1000 + cfg, query rows 2000 + cfg, cluster centres and
    chunk token bags 3000 + cfg, query terms 3500 + cfg, upsert round r ids
    4000 + r and rows 4500 + r.
"""
from __future__ import annotations

import dataclasses

import numpy as np

_CHUNK = 65536


def _normalise(x: np.ndarray) -> np.ndarray:
    x64 = x.astype(np.float64)
    norms = np.sqrt(np.einsum("ij,ij->i", x64, x64))
    norms[norms == 0.0] = 1.0
    return (x64 / norms[:, None]).astype(np.float32)


def to_bf16_bits(x32: np.ndarray) -> np.ndarray:
    """float32 -> bf16 bit patterns (uint16), round to nearest even."""
    import torch
    t = torch.from_numpy(np.ascontiguousarray(x32, dtype=np.float32))
    return t.to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16).copy()


def gaussian_rows(n: int, d: int, seed: int) -> np.ndarray:
    """n x d float32 L2-normalised Gaussian directions.  Rows come in chunks of
    65536; chunk c draws from its own generator seeded (seed, c), so the
    chunks can be drawn on several threads and the result does not depend on
    how many."""
    out = np.empty((n, d), np.float32)

    def fill(c: int) -> None:
        lo, hi = c * _CHUNK, min(n, (c + 1) * _CHUNK)
        rng = np.random.default_rng([seed, c])
        out[lo:hi] = _normalise(rng.standard_normal((hi - lo, d), dtype=np.float32))

    chunks = range((n + _CHUNK - 1) // _CHUNK)
    if len(chunks) <= 1:
        for c in chunks:
            fill(c)
    else:
        import concurrent.futures as cf
        import os
        with cf.ThreadPoolExecutor(max_workers=min(len(chunks), os.cpu_count() or 1)) as ex:
            list(ex.map(fill, chunks))
    return out


def cluster_centres(n_clusters: int, d: int, seed: int) -> np.ndarray:
    rng = np.random.default_rng(seed)
    return rng.standard_normal((n_clusters, d), dtype=np.float32)


def clustered_rows(n: int, centres: np.ndarray, sigma: float, seed: int) -> np.ndarray:
    """n x d float32 rows near uniformly chosen centres, then normalised."""
    rng = np.random.default_rng(seed)
    k, d = centres.shape
    out = np.empty((n, d), np.float32)
    for lo in range(0, n, _CHUNK):
        hi = min(n, lo + _CHUNK)
        pick = rng.integers(0, k, size=hi - lo)
        z = rng.standard_normal((hi - lo, d), dtype=np.float32)
        out[lo:hi] = _normalise(centres[pick] + np.float32(sigma) * z)
    return out


def zipf_sampler(vocab: int, s: float):
    ranks = np.arange(1, vocab + 1, dtype=np.float64)
    w = ranks ** (-s)
    cdf = np.cumsum(w)
    cdf /= cdf[-1]

    def draw(rng: np.random.Generator, size: int) -> np.ndarray:
        u = rng.random(size)
        return np.minimum(np.searchsorted(cdf, u, side="right"), vocab - 1).astype(np.int32)
    return draw


def token_bags(n: int, vocab: int, s: float, len_lo: int, len_hi: int, seed: int):
    """Per-chunk token lists in CSR form: (indptr int32 [n+1], terms int32)."""
    rng = np.random.default_rng(seed)
    lens = rng.integers(len_lo, len_hi + 1, size=n).astype(np.int64)
    indptr = np.zeros(n + 1, np.int64)
    np.cumsum(lens, out=indptr[1:])
    terms = zipf_sampler(vocab, s)(rng, int(indptr[-1]))
    return indptr.astype(np.int32), terms


def query_terms(q: int, per_query: int, vocab: int, s: float, seed: int):
    """Each query gets per_query Zipf-drawn term ids (repeats allowed), CSR form."""
    rng = np.random.default_rng(seed)
    terms = zipf_sampler(vocab, s)(rng, q * per_query)
    indptr = (np.arange(q + 1, dtype=np.int64) * per_query).astype(np.int32)
    return indptr, terms


@dataclasses.dataclass
class Workload:
    """One synthetic search workload.  ``E_data``/``Q_data`` are what the index
    and the search receive: float32 values for "f32" workloads, bf16 bit
    patterns (uint16) for "bf16" workloads.  ``E``/``Q`` give the exact float32
    values of those inputs."""
    name: str
    dtype: str                      # "f32" or "bf16"
    k: int
    E_data: np.ndarray
    Q_data: np.ndarray
    doc_indptr: np.ndarray | None = None
    doc_terms: np.ndarray | None = None
    q_indptr: np.ndarray | None = None
    q_terms: np.ndarray | None = None
    vocab: int = 0
    k1: float = 1.2
    b: float = 0.75
    alpha: float = 0.5

    @property
    def n(self) -> int:
        return int(self.E_data.shape[0])

    @property
    def d(self) -> int:
        return int(self.E_data.shape[1])

    @property
    def q(self) -> int:
        return int(self.Q_data.shape[0])

    @property
    def E(self) -> np.ndarray:
        return widen(self.E_data)

    @property
    def Q(self) -> np.ndarray:
        return widen(self.Q_data)


def widen(a: np.ndarray) -> np.ndarray:
    """float32 values of an input array (bf16 bit patterns are widened exactly)."""
    if a.dtype == np.uint16:
        return (a.astype(np.uint32) << 16).view(np.float32)
    return a


def make_dense(name: str, n: int, d: int, q: int, k: int, dtype: str, cfg: int,
               clusters: int = 0, sigma: float = 0.05) -> Workload:
    if clusters:
        centres = cluster_centres(clusters, d, 3000 + cfg)
        E = clustered_rows(n, centres, sigma, 1000 + cfg)
        Q = clustered_rows(q, centres, sigma, 2000 + cfg)
    else:
        E = gaussian_rows(n, d, 1000 + cfg)
        Q = gaussian_rows(q, d, 2000 + cfg)
    if dtype == "f32":
        return Workload(name, dtype, k, E, Q)
    return Workload(name, dtype, k, to_bf16_bits(E), to_bf16_bits(Q))


def add_sparse(w: Workload, cfg: int, vocab: int = 30522, s: float = 1.1, len_lo: int = 150,
               len_hi: int = 250, terms_per_query: int = 8) -> Workload:
    w.doc_indptr, w.doc_terms = token_bags(w.n, vocab, s, len_lo, len_hi, 3000 + cfg)
    w.q_indptr, w.q_terms = query_terms(w.q, terms_per_query, vocab, s, 3500 + cfg)
    w.vocab = vocab
    return w


def upsert_batch(n: int, d: int, m: int, round_index: int, dtype: str):
    """m distinct random row ids (without replacement) and fresh normalised rows
    (float32 for "f32", bf16 bit patterns for "bf16")."""
    rng = np.random.default_rng(4000 + round_index)
    ids = rng.choice(n, size=m, replace=False).astype(np.int64)
    rows = gaussian_rows(m, d, 4500 + round_index)
    return ids, (rows if dtype == "f32" else to_bf16_bits(rows))


CONFIG_NAMES = {
    0: "tiny dense top-5: 1024 x 384 fp32, 16 queries",
    1: "paper-shaped dense top-5: 32768 x 768 bf16, query batches 1/32/256",
    2: "clustered dense top-10: 32768 x 1024 bf16, 256 clusters sigma 0.05, 4096 queries",
    3: "hybrid top-5: 32768 x 768 bf16 + Zipf(1.1) BM25 (k1 1.2, b 0.75), 1024 queries, alpha 0.5",
    4: "scale dense top-100: 1048576 x 768 bf16, 4 x 2048 queries, 4096-row upserts between batches",
}


def config(i: int, batch: int | None = None, n: int | None = None) -> Workload:
    """The five workload shapes.  ``batch`` overrides the query count (config 1
    uses 1, 32 or 256; config 4 uses 2048 per batch); ``n`` overrides the corpus
    size for scaled-down test runs."""
    if i == 0:
        return make_dense("cfg0", n or 1024, 384, batch or 16, 5, "f32", 0)
    if i == 1:
        return make_dense("cfg1", n or 32768, 768, batch or 256, 5, "bf16", 1)
    if i == 2:
        return make_dense("cfg2", n or 32768, 1024, batch or 4096, 10, "bf16", 2, clusters=256)
    if i == 3:
        w = make_dense("cfg3", n or 32768, 768, batch or 1024, 5, "bf16", 3)
        return add_sparse(w, 3)
    if i == 4:
        return make_dense("cfg4", n or 1048576, 768, batch or 2048, 100, "bf16", 4)
    raise ValueError(f"unknown config {i}")
