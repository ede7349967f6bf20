// Tensor-core search kernels, CTA pairs (M = 256), 256-row corpus tiles,
// dense scores.
#include "search_tc.cuh"

namespace oprag {
namespace tc {

cudaError_t launch_pair256_dense(const TcMaps& m, const TcParams& prm, int grid, cudaStream_t st) {
  return launch_pair<kLexNone>(m, prm, grid, st);
}

int pair_capacity_query() {
  constexpr size_t smem = smem_for<256, 16, true>();
  if (cudaFuncSetAttribute(tc_search_kernel<256, 16, kLexNone, true>,
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
  if (cudaOccupancyMaxActiveClusters(&n, tc_search_kernel<256, 16, kLexNone, true>, &cfg) !=
      cudaSuccess)
    return 0;
  return n;
}

}  // namespace tc
}  // namespace oprag
