// Lexical rerank of a dense top-N: the dense-first hybrid policy (Sec. 4.1
// Retrieval; Sec. 5.5).  Per query: BM25 of each candidate chunk through the
// sparse index, the BM25 maximum over the candidates, the weighted fusion of
// Sec. 4.4 and the ranked top-k of the fused scores.
//
// One warp per query; lane l holds candidates l * E .. l * E + E - 1.  A
// candidate's BM25 is the sum of its query terms' weights in the query's term
// order: a dense term's weight is read from its row, a sparse term's is found
// by a binary search of the term's postings (the E searches of a lane are
// interleaved so that their loads overlap).  The sums and the fused score are
// formed exactly as in the BM25 pass and the fused search epilogue, so with
// every chunk a candidate the result equals the full hybrid search bit for
// bit.  The N fused keys are sorted by one warp bitonic sort.
#include "common.cuh"
#include "internal.h"

namespace oprag {

namespace {

constexpr int kRerankWarps = 4;

template <int E>
__global__ void __launch_bounds__(kRerankWarps * 32)
rerank_kernel(SparseIndex sp, int q, int ncand, const int64_t* __restrict__ cand_ids,
              const float* __restrict__ cand_scores, const int32_t* __restrict__ q_indptr,
              const int32_t* __restrict__ q_terms, float alpha, int k,
              int64_t* __restrict__ out_ids, float* __restrict__ out_scores) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int qi = blockIdx.x * kRerankWarps + warp;
  if (qi >= q) return;
  int32_t doc[E];
  float dense[E], lex[E];
#pragma unroll
  for (int e = 0; e < E; ++e) {
    const int c = lane * E + e;
    const int64_t id = c < ncand ? cand_ids[static_cast<int64_t>(qi) * ncand + c] : -1;
    doc[e] = static_cast<int32_t>(id);
    dense[e] = c < ncand ? cand_scores[static_cast<int64_t>(qi) * ncand + c] : 0.f;
    lex[e] = 0.f;
  }
  const int t0 = q_indptr[qi], t1 = q_indptr[qi + 1];
  for (int ti = t0; ti < t1; ++ti) {
    const int32_t term = q_terms[ti];
    if (term < 0 || term >= sp.vocab) continue;
    const int slot = sp.dense_slot[term];
    float w[E];
    if (slot >= 0) {
      const float* row = sp.dense_w + slot * sp.dense_ld;
#pragma unroll
      for (int e = 0; e < E; ++e) w[e] = doc[e] >= 0 ? row[doc[e]] : 0.f;
    } else {
      const int64_t p0 = sp.post_ptr[term], p1 = sp.post_ptr[term + 1];
      int64_t lo[E], hi[E];
#pragma unroll
      for (int e = 0; e < E; ++e) {
        lo[e] = p0;
        hi[e] = doc[e] >= 0 ? p1 : p0;
      }
      // Lower bound of each candidate in the term's (ascending) postings.
      bool more = p0 < p1;
      while (more) {
        more = false;
#pragma unroll
        for (int e = 0; e < E; ++e) {
          if (lo[e] < hi[e]) {
            const int64_t mid = (lo[e] + hi[e]) >> 1;
            if (sp.post[mid].x < doc[e]) lo[e] = mid + 1;
            else hi[e] = mid;
            more |= lo[e] < hi[e];
          }
        }
      }
#pragma unroll
      for (int e = 0; e < E; ++e) {
        w[e] = 0.f;
        if (doc[e] >= 0 && lo[e] < p1) {
          const int2 pe = sp.post[lo[e]];
          if (pe.x == doc[e]) w[e] = __int_as_float(pe.y);
        }
      }
    }
#pragma unroll
    for (int e = 0; e < E; ++e) lex[e] += w[e];
  }
  // BM25 maximum over the candidates (BM25 is never negative).
  float m = 0.f;
#pragma unroll
  for (int e = 0; e < E; ++e)
    if (doc[e] >= 0) m = fmaxf(m, lex[e]);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
  const float inv_max = m > 0.f ? 1.f / m : 0.f;
  const float a = alpha, b1 = 1.f - alpha;
  uint64_t key[E];
#pragma unroll
  for (int e = 0; e < E; ++e)
    key[e] = doc[e] >= 0 ? make_key(fmaf(a, dense[e], b1 * (lex[e] * inv_max)),
                                    static_cast<uint32_t>(doc[e]))
                         : kEmptyKey;
  warp_sort_desc<E>(key);
#pragma unroll
  for (int e = 0; e < E; ++e) {
    const int r = lane * E + e;
    if (r < k) {
      const int64_t o = static_cast<int64_t>(qi) * k + r;
      out_ids[o] = key[e] == kEmptyKey ? -1 : static_cast<int64_t>(key_id(key[e]));
      out_scores[o] = key[e] == kEmptyKey ? -INFINITY : key_score(key[e]);
    }
  }
}

}  // namespace

cudaError_t launch_rerank(const SparseIndex& sp, int q, int ncand, const int64_t* cand_ids,
                          const float* cand_scores, const int32_t* q_indptr,
                          const int32_t* q_terms, float alpha, int k, int64_t* out_ids,
                          float* out_scores, cudaStream_t st) {
  if (q <= 0) return cudaSuccess;
  if (ncand < 1 || ncand > kRerankMaxCand || k > ncand) return cudaErrorInvalidValue;
  const dim3 grid((q + kRerankWarps - 1) / kRerankWarps), block(kRerankWarps * 32);
  const int e = (ncand + 31) / 32;
  if (e <= 1)
    rerank_kernel<1><<<grid, block, 0, st>>>(sp, q, ncand, cand_ids, cand_scores, q_indptr,
                                             q_terms, alpha, k, out_ids, out_scores);
  else if (e <= 2)
    rerank_kernel<2><<<grid, block, 0, st>>>(sp, q, ncand, cand_ids, cand_scores, q_indptr,
                                             q_terms, alpha, k, out_ids, out_scores);
  else if (e <= 4)
    rerank_kernel<4><<<grid, block, 0, st>>>(sp, q, ncand, cand_ids, cand_scores, q_indptr,
                                             q_terms, alpha, k, out_ids, out_scores);
  else
    rerank_kernel<8><<<grid, block, 0, st>>>(sp, q, ncand, cand_ids, cand_scores, q_indptr,
                                             q_terms, alpha, k, out_ids, out_scores);
  return cudaGetLastError();
}

}  // namespace oprag
