// SIMT streaming search kernels for fp32 indices.
#include "search_simt.cuh"

namespace oprag {
namespace simt {

cudaError_t launch_f32(int qc, const void* E, const void* Q, const SearchShape& s,
                       const Fusion& fu, void* scratch, int grid, ListSet* lists, cudaStream_t st) {
  switch (qc) {
    case 1: return launch_qc<float, 1>(E, Q, s, fu, scratch, grid, lists, st);
    case 2: return launch_qc<float, 2>(E, Q, s, fu, scratch, grid, lists, st);
    case 4: return launch_qc<float, 4>(E, Q, s, fu, scratch, grid, lists, st);
    default: return launch_qc<float, 8>(E, Q, s, fu, scratch, grid, lists, st);
  }
}

}  // namespace simt
}  // namespace oprag
