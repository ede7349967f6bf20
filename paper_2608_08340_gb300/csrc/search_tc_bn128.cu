// Tensor-core search kernels with 128-row corpus tiles (one query tile per
// unit): dense scores, and the hybrid search reading the BM25 block.
#include "search_tc.cuh"

namespace oprag {
namespace tc {

cudaError_t launch_bn128(const TcMaps& m, const TcParams& prm, int grid, int lex, cudaStream_t st) {
  return lex == kLexBlock ? launch_bn<128, kLexBlock>(m, prm, grid, st)
                          : launch_bn<128, kLexNone>(m, prm, grid, st);
}

}  // namespace tc
}  // namespace oprag
