// Tensor-core search kernels with 256-row corpus tiles, dense scores.
#include "search_tc.cuh"

namespace oprag {
namespace tc {

cudaError_t launch_bn256_dense(const TcMaps& m, const TcParams& prm, int grid, cudaStream_t st) {
  return launch_bn<256, kLexNone>(m, prm, grid, st);
}

}  // namespace tc
}  // namespace oprag
