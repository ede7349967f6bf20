// Tensor-core search kernels in dual mode (two query tiles per unit,
// 128-row corpus tiles, double-buffered accumulators; lists of 8 or 16 keys),
// dense or hybrid from the BM25 block.
#include "search_tc.cuh"

namespace oprag {
namespace tc {

cudaError_t launch_dual128(const TcMaps& m, const TcParams& prm, int grid, int lex,
                           cudaStream_t st) {
  return lex == kLexBlock ? launch_dual<kLexBlock>(m, prm, grid, st)
                          : launch_dual<kLexNone>(m, prm, grid, st);
}

}  // namespace tc
}  // namespace oprag
