// Tensor-core search kernels of the gathered hybrid search: 128-row corpus
// tiles, the head terms' BM25 as one more K block into a second
// accumulator, mid rows and tail postings read in the epilogue.
#include "search_tc.cuh"

namespace oprag {
namespace tc {

cudaError_t launch_bn128_gather(const TcMaps& m, const TcParams& prm, int grid, cudaStream_t st) {
  return launch_bn<128, kLexGather>(m, prm, grid, st);
}

}  // namespace tc
}  // namespace oprag
