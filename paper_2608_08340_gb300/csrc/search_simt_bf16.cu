// SIMT streaming search kernels for bf16 indices.
#include "search_simt.cuh"

namespace oprag {
namespace simt {

cudaError_t launch_bf16(int qc, const void* E, const void* Q, const SearchShape& s,
                        const Fusion& fu, void* scratch, int grid, ListSet* lists, cudaStream_t st) {
  switch (qc) {
    case 1: return launch_qc<__nv_bfloat16, 1>(E, Q, s, fu, scratch, grid, lists, st);
    case 2: return launch_qc<__nv_bfloat16, 2>(E, Q, s, fu, scratch, grid, lists, st);
    case 4: return launch_qc<__nv_bfloat16, 4>(E, Q, s, fu, scratch, grid, lists, st);
    default: return launch_qc<__nv_bfloat16, 8>(E, Q, s, fu, scratch, grid, lists, st);
  }
}

}  // namespace simt
}  // namespace oprag
