// Tensor-core search kernels, CTA pairs (M = 256), 256-row corpus tiles,
// hybrid scores read from the BM25 block.
#include "search_tc.cuh"

namespace oprag {
namespace tc {

cudaError_t launch_pair256_block(const TcMaps& m, const TcParams& prm, int grid, cudaStream_t st) {
  return launch_pair<kLexBlock>(m, prm, grid, st);
}

}  // namespace tc
}  // namespace oprag
