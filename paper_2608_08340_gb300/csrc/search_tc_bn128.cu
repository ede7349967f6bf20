// Tensor-core search kernels with 128-row corpus tiles (small query batches).
#include "search_tc.cuh"

namespace oprag {
namespace tc {

cudaError_t launch_bn128(const CUtensorMap& mq, const CUtensorMap& me, const TcParams& prm, int grid,
                        bool hybrid, cudaStream_t st) {
  return launch_bn<128>(mq, me, prm, grid, hybrid, st);
}

}  // namespace tc
}  // namespace oprag
