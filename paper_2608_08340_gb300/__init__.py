"""GB300-native retrieval hot path of OpRAG (arxiv 2608.08340).

Exact top-k inner-product search, hybrid dense + BM25 fusion and index upsert
on one GPU, implemented as hand-written sm_103a CUDA kernels behind the C ABI
of include/oprag.h (library: paper_2608_08340_gb300/_build/liboprag.so).
"""
from ._lib import OPRAG_BF16, OPRAG_F32, OPRAG_K_MAX, OpragError  # noqa: F401


def __getattr__(name):
    if name == "Index":
        from .index import Index
        return Index
    raise AttributeError(name)
