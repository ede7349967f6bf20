// Lexical half of the hybrid search (Sec. 4.4): BM25 of every (query, chunk)
// pair through inverted postings, which "visits only documents that contain
// query terms while preserving exact full-corpus BM25 semantics".
//
// The per-posting weight idf(t) * tf (k1 + 1) / (tf + k1 (1 - b + b |d| / avgdl))
// does not depend on the query, so it is computed once on the host when the
// sparse side is attached; a query's BM25 for chunk d is then the sum of the
// weights of its terms' postings at d, taken in the order of the query's term
// list (a repeated term counts again).
//
// One CTA per (query, tile of 8192 chunks) accumulates those sums in shared
// memory, one term at a time (the postings of one term hold each chunk at
// most once, so the adds of a term never collide and the summation order is
// fixed).  It writes the tile's row of the q x n BM25 matrix and folds the
// tile maximum into the per-query maximum that normalises the lexical score.
#include "common.cuh"
#include "internal.h"

namespace oprag {

namespace {

constexpr int kDocTile = 8192;
constexpr int kBm25Threads = 256;
constexpr int kTermsPerPass = kBm25Threads / 32;

// First position in [lo, hi) whose value is >= key (hi if none); the array is
// ascending.  Warp-collective: 32 probes per round.
__device__ int64_t warp_lower_bound(const int32_t* a, int64_t lo, int64_t hi, int32_t key) {
  const int lane = threadIdx.x & 31;
  while (hi - lo > 32) {
    const int64_t step = (hi - lo + 31) / 32;
    const int64_t pos = lo + lane * step;
    const bool less = pos < hi && a[pos] < key;
    const int c = __popc(__ballot_sync(0xffffffffu, less));
    if (c == 0) return lo;
    const int64_t next = lo + static_cast<int64_t>(c) * step;
    lo = lo + static_cast<int64_t>(c - 1) * step + 1;
    if (c < 32 && next < hi) hi = next;
  }
  const int64_t pos = lo + lane;
  const bool less = pos < hi && a[pos] < key;
  return lo + __popc(__ballot_sync(0xffffffffu, less));
}

__global__ void __launch_bounds__(kBm25Threads)
bm25_matrix_kernel(SparseIndex sp, int64_t n, const int32_t* __restrict__ q_indptr,
                   const int32_t* __restrict__ q_terms, float* __restrict__ out, int64_t ld,
                   float* __restrict__ out_max) {
  __shared__ float acc[kDocTile];
  __shared__ int64_t rng_lo[kTermsPerPass], rng_hi[kTermsPerPass];
  __shared__ float red[kBm25Threads / 32];
  const int qi = blockIdx.x;
  const int64_t d0 = static_cast<int64_t>(blockIdx.y) * kDocTile;
  const int64_t d1 = min(n, d0 + kDocTile);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  for (int i = threadIdx.x; i < kDocTile; i += blockDim.x) acc[i] = 0.f;

  const int t0 = q_indptr[qi], t1 = q_indptr[qi + 1];
  for (int base = t0; base < t1; base += kTermsPerPass) {
    // Locate each term's postings inside [d0, d1): one warp per term.
    const int ti = base + warp;
    if (ti < t1) {
      const int32_t term = q_terms[ti];
      int64_t lo = 0, hi = 0;
      if (term >= 0 && term < sp.vocab) {
        const int64_t p0 = sp.post_ptr[term], p1 = sp.post_ptr[term + 1];
        lo = warp_lower_bound(sp.post_doc, p0, p1, static_cast<int32_t>(d0));
        hi = warp_lower_bound(sp.post_doc, lo, p1, static_cast<int32_t>(d1));
      }
      if (lane == 0) {
        rng_lo[warp] = lo;
        rng_hi[warp] = hi;
      }
    }
    __syncthreads();
    const int nt = min(kTermsPerPass, t1 - base);
    for (int w = 0; w < nt; ++w) {
      for (int64_t p = rng_lo[w] + threadIdx.x; p < rng_hi[w]; p += blockDim.x)
        acc[sp.post_doc[p] - d0] += sp.post_w[p];
      __syncthreads();
    }
  }

  float m = 0.f;
  float* orow = out + static_cast<int64_t>(qi) * ld;
  for (int64_t dd = d0 + threadIdx.x; dd < d1; dd += blockDim.x) {
    const float v = acc[dd - d0];
    orow[dd] = v;
    m = fmaxf(m, v);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
  if (lane == 0) red[warp] = m;
  __syncthreads();
  if (threadIdx.x == 0) {
    float bm = red[0];
    for (int w = 1; w < kBm25Threads / 32; ++w) bm = fmaxf(bm, red[w]);
    // BM25 is never negative, so the float order equals the int order.
    atomicMax(reinterpret_cast<int*>(out_max + qi), __float_as_int(bm));
  }
}

}  // namespace

cudaError_t launch_bm25_matrix(const SparseIndex& sp, int64_t n, const int32_t* q_indptr,
                               const int32_t* q_terms, int q, float* out, int64_t ld,
                               float* out_max, cudaStream_t st) {
  if (q <= 0) return cudaSuccess;
  cudaError_t e = cudaMemsetAsync(out_max, 0, sizeof(float) * q, st);
  if (e != cudaSuccess) return e;
  const dim3 grid(q, static_cast<unsigned>((n + kDocTile - 1) / kDocTile));
  bm25_matrix_kernel<<<grid, kBm25Threads, 0, st>>>(sp, n, q_indptr, q_terms, out, ld, out_max);
  return cudaGetLastError();
}

}  // namespace oprag
