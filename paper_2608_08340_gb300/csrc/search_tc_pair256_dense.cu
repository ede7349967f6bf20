// Tensor-core search kernels, CTA pairs (M = 256), 256-row corpus tiles,
// dense scores.
#include "search_tc.cuh"

namespace oprag {
namespace tc {

cudaError_t launch_pair256_dense(const CUtensorMap& mq, const CUtensorMap& me, const TcParams& prm,
                                 int grid, cudaStream_t st) {
  switch (list_len_for(prm.k)) {
    case 8: return launch_pair_variant<256, 8, false>(mq, me, prm, grid, st);
    case 16: return launch_pair_variant<256, 16, false>(mq, me, prm, grid, st);
    case 32: return launch_pair_variant<256, 32, false>(mq, me, prm, grid, st);
    case 128: return launch_pair_variant<256, 128, false>(mq, me, prm, grid, st);
    default: return launch_pair_variant<256, 256, false>(mq, me, prm, grid, st);
  }
}

int pair_capacity_query() {
  constexpr size_t smem = smem_for<256, 16, true>();
  if (cudaFuncSetAttribute(tc_search_kernel<256, 16, false, true>,
                           cudaFuncAttributeMaxDynamicSharedMemorySize,
                           static_cast<int>(smem)) != cudaSuccess)
    return 0;
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(2);
  cfg.blockDim = dim3(threads_for(16));
  cfg.dynamicSmemBytes = smem;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, tc_search_kernel<256, 16, false, true>, &cfg) !=
      cudaSuccess)
    return 0;
  return n;
}

}  // namespace tc
}  // namespace oprag
