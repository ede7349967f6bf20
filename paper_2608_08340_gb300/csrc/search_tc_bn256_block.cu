// Tensor-core search kernels with 256-row corpus tiles, hybrid scores read
// from the BM25 block.
#include "search_tc.cuh"

namespace oprag {
namespace tc {

cudaError_t launch_bn256_block(const TcMaps& m, const TcParams& prm, int grid, cudaStream_t st) {
  return launch_bn<256, kLexBlock>(m, prm, grid, st);
}

}  // namespace tc
}  // namespace oprag
