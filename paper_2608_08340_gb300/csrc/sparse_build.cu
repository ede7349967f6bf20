// Device side of building the lexical index (Sec. 3.2 Op_upsert applied to
// the token bags; Sec. 4.4 BM25 over inverted postings).  The host hands over
// the integer structure -- a term-major inverted index of (chunk, tf) pairs,
// chunks ascending inside a term, the chunks' token counts and each term's
// idf -- and these kernels compute every per-posting Okapi weight
//   w(t, d) = idf(t) * tf (k1 + 1) / (tf + k1 (1 - b + b |d| / avgdl))
// in fp64 (IEEE operations without contraction, so a rebuild gives the same
// bits as a fresh build) and write it where the searches read it: the
// postings of the sparse terms, the dense rows of the common terms, the
// split bf16 operand of the tensor-core head terms and the mid-frequency
// rows of the gathered hybrid search; then the per-tile entry points of the
// postings.
#include "common.cuh"
#include "internal.h"

namespace oprag {

namespace {

// One warp per term (grid-stride over terms).
__global__ void lex_weights_kernel(LexBuild lb) {
  const int lane = threadIdx.x & 31;
  const int64_t warp0 = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = (static_cast<int64_t>(gridDim.x) * blockDim.x) >> 5;
  const double kp1 = __dadd_rn(lb.k1, 1.0);
  for (int64_t t = warp0; t < lb.vocab; t += nwarps) {
    const int64_t a = lb.term_start[t], z = lb.term_start[t + 1];
    if (a == z) continue;
    const double idf = lb.idf[t];
    const int slot = lb.slot[t];
    const int cls = lb.lex_class[t];
    const int64_t pbase = lb.post_ptr[t];
    for (int64_t i = a + lane; i < z; i += 32) {
      const int2 e = lb.inv[i];                   // (chunk, tf)
      const double tf = static_cast<double>(e.y);
      const double len = static_cast<double>(lb.doc_len[e.x]);
      const double ratio = lb.avgdl > 0.0 ? __ddiv_rn(len, lb.avgdl) : 0.0;
      const double norm = __dadd_rn(__dsub_rn(1.0, lb.b), __dmul_rn(lb.b, ratio));
      const double num = __dmul_rn(__dmul_rn(idf, tf), kp1);
      const double den = __dadd_rn(tf, __dmul_rn(lb.k1, norm));
      const float w = static_cast<float>(__ddiv_rn(num, den));
      if (slot >= 0) {
        lb.dense_w[static_cast<int64_t>(slot) * lb.dense_ld + e.x] = w;
      } else {
        lb.post[pbase + (i - a)] = make_int2(e.x, __float_as_int(w));
      }
      if (cls >= 0) {
        const __nv_bfloat16 hi = __float2bfloat16_rn(w);
        lb.wsplit[static_cast<int64_t>(e.x) * kLexK + cls] = hi;
        lb.wsplit[static_cast<int64_t>(e.x) * kLexK + kLexHeadTerms + cls] =
            __float2bfloat16_rn(w - __bfloat162float(hi));
      } else if (cls <= -2) {
        lb.mid_w[static_cast<int64_t>(-2 - cls) * lb.mid_ld + e.x] = w;
      }
    }
  }
}

// One thread per (term, tile boundary b): the first posting of the term whose
// chunk is >= b * kBm25DocTile.
__global__ void tile_ptr_kernel(const int64_t* __restrict__ post_ptr, const int2* __restrict__ post,
                                int vocab, int ntiles, int64_t* __restrict__ tile_ptr) {
  const int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  const int64_t per = ntiles + 1;
  if (i >= static_cast<int64_t>(vocab) * per) return;
  const int64_t t = i / per, b = i % per;
  const int64_t doc0 = b * kBm25DocTile;
  int64_t lo = post_ptr[t], hi = post_ptr[t + 1];
  while (lo < hi) {
    const int64_t mid = (lo + hi) >> 1;
    if (post[mid].x < doc0) lo = mid + 1; else hi = mid;
  }
  tile_ptr[i] = lo;
}

}  // namespace

cudaError_t launch_lex_build(const LexBuild& lb, int ntiles, int64_t* tile_ptr, cudaStream_t st) {
  if (lb.vocab <= 0) return cudaSuccess;
  const int64_t warps = lb.vocab;
  const int blocks = static_cast<int>(std::min<int64_t>((warps + 7) / 8, 8192));
  lex_weights_kernel<<<blocks, 256, 0, st>>>(lb);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  const int64_t cells = static_cast<int64_t>(lb.vocab) * (ntiles + 1);
  tile_ptr_kernel<<<static_cast<unsigned>((cells + 255) / 256), 256, 0, st>>>(
      lb.post_ptr, lb.post, lb.vocab, ntiles, tile_ptr);
  return cudaGetLastError();
}

}  // namespace oprag
