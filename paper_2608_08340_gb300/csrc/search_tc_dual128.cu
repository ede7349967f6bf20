// Tensor-core search kernels in dual mode (two query tiles per unit,
// 128-row corpus tiles, double-buffered accumulators; lists of 8 or 16 keys).
#include "search_tc.cuh"

namespace oprag {
namespace tc {

cudaError_t launch_dual128(const CUtensorMap& mq, const CUtensorMap& me, const TcParams& prm,
                           int grid, bool hybrid, cudaStream_t st) {
  switch (list_len_for(prm.k)) {
    case 8:
      return hybrid ? launch_dual_variant<8, true>(mq, me, prm, grid, st)
                    : launch_dual_variant<8, false>(mq, me, prm, grid, st);
    case 16:
      return hybrid ? launch_dual_variant<16, true>(mq, me, prm, grid, st)
                    : launch_dual_variant<16, false>(mq, me, prm, grid, st);
    default:
      return cudaErrorInvalidValue;
  }
}

}  // namespace tc
}  // namespace oprag
