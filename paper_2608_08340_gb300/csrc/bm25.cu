// Lexical half of the hybrid search (Sec. 4.4): BM25 of every (query, chunk)
// pair through inverted postings, touching only the chunks that hold a query
// term and giving the same scores as a scan of the whole corpus.
//
// The per-posting weight idf(t) * tf (k1 + 1) / (tf + k1 (1 - b + b |d| / avgdl))
// does not depend on the query, so it is computed once on the host when the
// sparse side is attached; a query's BM25 for chunk d is then the sum of the
// weights of its terms' postings at d, taken in the order of the query's term
// list (a repeated term counts again).
//
// One CTA per (query, tile of 8192 chunks) accumulates those sums in shared
// memory, one term at a time in the query's order; a table built with the
// postings gives where each sparse term's postings enter the tile.  A dense term (held by
// more than half of the chunks, stored as a row of weights with zeros where
// absent) is added element-wise with 16-byte loads, each thread keeping the
// same elements, so consecutive dense terms need no barrier; a sparse term
// scatters its postings (each chunk at most once per term, so its adds never
// collide).  Adding a zero weight leaves an fp32 sum unchanged, so both forms
// give the same sums in the same order.  The CTA writes the tile's row of the
// q x n BM25 matrix and folds the tile maximum into the per-query maximum
// that normalises the lexical score.
#include "common.cuh"
#include "internal.h"

namespace oprag {

namespace {

constexpr int kDocTile = kBm25DocTile;
constexpr int kBm25Threads = 256;
constexpr int kTermsPerPass = kBm25Threads / 32;
constexpr int kScatterUnroll = 4;      // postings loaded per thread before the adds
constexpr int kDenseBatch = 8;         // dense-row float4 groups loaded per thread before the adds
constexpr int kSkipTerm = -2;          // term id outside the vocabulary

__global__ void __launch_bounds__(kBm25Threads)
bm25_matrix_kernel(SparseIndex sp, int64_t n, const int32_t* __restrict__ q_indptr,
                   const int32_t* __restrict__ q_terms, float* __restrict__ out, int64_t ld,
                   float* __restrict__ out_max) {
  __shared__ __align__(16) float acc[kDocTile];
  __shared__ int64_t rng_lo[kTermsPerPass], rng_hi[kTermsPerPass];
  __shared__ int slot_of[kTermsPerPass];
  __shared__ float red[kBm25Threads / 32];
  const int qi = blockIdx.x;
  const int64_t d0 = static_cast<int64_t>(blockIdx.y) * kDocTile;
  const int64_t d1 = min(n, d0 + kDocTile);
  const int nv = static_cast<int>((d1 - d0 + 3) / 4);     // float4 groups of this tile
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  float4* acc4 = reinterpret_cast<float4*>(acc);

  for (int i = threadIdx.x; i < kDocTile / 4; i += blockDim.x) acc4[i] = make_float4(0.f, 0.f, 0.f, 0.f);

  const int t0 = q_indptr[qi], t1 = q_indptr[qi + 1];
  bool pending = true;      // element-wise work since the last barrier came from a scatter
  for (int base = t0; base < t1; base += kTermsPerPass) {
    // Classify each term of the pass and locate a sparse term's postings
    // inside [d0, d1) in the per-tile table: one thread per term, its three
    // loads issued together.
    const int ti = base + warp;
    if (ti < t1 && lane == 0) {
      const int32_t term = q_terms[ti];
      int slot = kSkipTerm;
      int64_t lo = 0, hi = 0;
      if (term >= 0 && term < sp.vocab) {
        const int64_t* tp = sp.tile_ptr + static_cast<int64_t>(term) * (sp.ntiles + 1) + blockIdx.y;
        const int64_t a = tp[0], z = tp[1];
        slot = sp.dense_slot[term];
        if (slot < 0) {
          lo = a;
          hi = z;
        }
      }
      slot_of[warp] = slot;
      rng_lo[warp] = lo;
      rng_hi[warp] = hi;
    }
    __syncthreads();
    pending = false;
    bool dirty = false;     // unsynchronised adds since the last barrier
    const int nt = min(kTermsPerPass, t1 - base);
    for (int w = 0; w < nt; ++w) {
      const int slot = slot_of[w];
      if (slot == kSkipTerm) continue;
      if (slot >= 0) {
        // Dense term: thread i owns float4 groups i, i + 256, ...; after
        // another dense term nothing needs ordering.
        if (pending) __syncthreads();
        // The row's groups are loaded kDenseBatch at a time, all before the
        // adds, so a dense term costs one L2 round trip per batch.
        const float4* row = reinterpret_cast<const float4*>(sp.dense_w + slot * sp.dense_ld + d0);
        for (int i0 = threadIdx.x; i0 < nv; i0 += kDenseBatch * kBm25Threads) {
          float4 x[kDenseBatch];
#pragma unroll
          for (int u = 0; u < kDenseBatch; ++u) {
            const int i = i0 + u * kBm25Threads;
            x[u] = i < nv ? __ldg(row + i) : make_float4(0.f, 0.f, 0.f, 0.f);
          }
#pragma unroll
          for (int u = 0; u < kDenseBatch; ++u) {
            const int i = i0 + u * kBm25Threads;
            if (i < nv) {
              float4 a = acc4[i];
              a.x += x[u].x;
              a.y += x[u].y;
              a.z += x[u].z;
              a.w += x[u].w;
              acc4[i] = a;
            }
          }
        }
        pending = false;
        dirty = true;
      } else {
        if (dirty) __syncthreads();
        const int64_t lo = rng_lo[w], hi = rng_hi[w];
        for (int64_t p = lo + threadIdx.x; p < hi; p += kScatterUnroll * blockDim.x) {
          int2 e[kScatterUnroll];
#pragma unroll
          for (int u = 0; u < kScatterUnroll; ++u) {
            const int64_t pp = p + static_cast<int64_t>(u) * blockDim.x;
            e[u] = pp < hi ? __ldg(sp.post + pp) : make_int2(-1, 0);
          }
#pragma unroll
          for (int u = 0; u < kScatterUnroll; ++u)
            if (e[u].x >= 0) acc[e[u].x - d0] += __int_as_float(e[u].y);
        }
        pending = true;
        dirty = true;
      }
    }
    __syncthreads();        // the next pass rewrites the term table; the output reads acc
  }

  float m = 0.f;
  float4* orow =
      out != nullptr ? reinterpret_cast<float4*>(out + static_cast<int64_t>(qi) * ld + d0) : nullptr;
  for (int i = threadIdx.x; i < nv; i += blockDim.x) {
    const float4 v = acc4[i];
    if (orow != nullptr) orow[i] = v;
    m = fmaxf(fmaxf(m, fmaxf(v.x, v.y)), fmaxf(v.z, v.w));
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

// One thread per query, by the classes of its terms: the head terms' counts
// (as bf16, twice: against the high and the low half of the split weights),
// its first kLexMidReg distinct mid rows and first kLexRegTerms distinct tail
// terms that have postings, each with its multiplicity, in first-occurrence
// order, and the raw term index where a further distinct one first occurs
// (the end of the query's terms if none does).
__global__ void lex_prep_kernel(const int32_t* __restrict__ lex_class,
                                const int64_t* __restrict__ post_ptr, int vocab,
                                const int32_t* __restrict__ q_indptr,
                                const int32_t* __restrict__ q_terms, int q, LexPrep out) {
  const int qi = blockIdx.x * blockDim.x + threadIdx.x;
  if (qi >= q) return;
  float cnt[kLexHeadTerms];
#pragma unroll
  for (int i = 0; i < kLexHeadTerms; ++i) cnt[i] = 0.f;
  const int t0 = q_indptr[qi], t1 = q_indptr[qi + 1];
  int4* tails = out.terms + static_cast<int64_t>(qi) * kLexRegTerms;
  int2* mids = out.mid + static_cast<int64_t>(qi) * kLexMidReg;
  int nt = 0, nm = 0, first_ovf = t1;
  for (int i = t0; i < t1; ++i) {
    const int32_t term = q_terms[i];
    if (term < 0 || term >= vocab) continue;
    const int c = lex_class[term];
    if (c >= 0) {
#pragma unroll
      for (int s = 0; s < kLexHeadTerms; ++s) cnt[s] += s == c ? 1.f : 0.f;
    } else if (c <= -2) {
      const int row = -2 - c;
      int j = 0;
      while (j < nm && mids[j].x != row) ++j;
      if (j < nm) mids[j].y = __float_as_int(__int_as_float(mids[j].y) + 1.f);
      else if (nm < kLexMidReg) mids[nm++] = make_int2(row, __float_as_int(1.f));
      else if (first_ovf == t1) first_ovf = i;
    } else {
      const int64_t a = post_ptr[term], b = post_ptr[term + 1];
      if (a >= b) continue;
      int j = 0;
      while (j < nt && tails[j].w != term) ++j;
      if (j < nt)
        tails[j].z = __float_as_int(__int_as_float(tails[j].z) + 1.f);
      else if (nt < kLexRegTerms)
        tails[nt++] = make_int4(static_cast<int>(a), static_cast<int>(b), __float_as_int(1.f), term);
      else if (first_ovf == t1)
        first_ovf = i;
    }
  }
  out.term_cnt[qi] = nt;
  out.mid_cnt[qi] = nm;
  out.ovf[qi] = first_ovf;
  __nv_bfloat16* row = static_cast<__nv_bfloat16*>(out.qcount) + static_cast<int64_t>(qi) * kLexK;
#pragma unroll
  for (int s = 0; s < kLexHeadTerms; ++s) {
    row[s] = __float2bfloat16_rn(cnt[s]);
    row[kLexHeadTerms + s] = __float2bfloat16_rn(cnt[s]);
  }
}

}  // namespace

cudaError_t launch_lex_prep(const int32_t* lex_class, const int64_t* post_ptr, int vocab,
                            const int32_t* q_indptr, const int32_t* q_terms, int q,
                            const LexPrep& out, cudaStream_t st) {
  if (q <= 0) return cudaSuccess;
  lex_prep_kernel<<<(q + 127) / 128, 128, 0, st>>>(lex_class, post_ptr, vocab, q_indptr, q_terms,
                                                   q, out);
  return cudaGetLastError();
}

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
