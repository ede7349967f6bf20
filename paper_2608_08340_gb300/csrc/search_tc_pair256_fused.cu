// Tensor-core search kernels, CTA pairs (M = 256), 256-row corpus tiles,
// fused dense + lexical scores.
#include "search_tc.cuh"

namespace oprag {
namespace tc {

cudaError_t launch_pair256_fused(const CUtensorMap& mq, const CUtensorMap& me, const TcParams& prm,
                                 int grid, cudaStream_t st) {
  switch (list_len_for(prm.k)) {
    case 8: return launch_pair_variant<256, 8, true>(mq, me, prm, grid, st);
    case 16: return launch_pair_variant<256, 16, true>(mq, me, prm, grid, st);
    case 32: return launch_pair_variant<256, 32, true>(mq, me, prm, grid, st);
    case 128: return launch_pair_variant<256, 128, true>(mq, me, prm, grid, st);
    default: return launch_pair_variant<256, 256, true>(mq, me, prm, grid, st);
  }
}

}  // namespace tc
}  // namespace oprag
