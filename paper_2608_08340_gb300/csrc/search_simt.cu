// Host side of the SIMT streaming search of search_simt.cuh: grid size,
// scratch size and the choice of the query-chunk width.
#include "search_simt.cuh"

namespace oprag {

using namespace simt;

namespace {

size_t smem_bytes(int qc, int d, int K) {
  return sizeof(float) * qc * d + sizeof(uint64_t) * kSimtWarps * qc * K +
         sizeof(uint64_t) * qc * 2 * (K < 32 ? 32 : K);
}

// Queries per CTA chunk: up to 8, fewer when the shared-memory copy of the
// queries and the lists would not fit.
int qc_for(const SearchShape& s) {
  const int K = list_len_for(s.k);
  int qc = s.q <= 1 ? 1 : s.q <= 2 ? 2 : s.q <= 4 ? 4 : 8;
  while (qc > 1 && smem_bytes(qc, s.d, K) > 200 * 1024) qc >>= 1;
  return qc;
}

}  // namespace

int simt_grid(const SearchShape& s, int num_sms) {
  // Enough warps to keep ~48 KB of loads in flight per SM; at least one row
  // per warp.
  int64_t grid = static_cast<int64_t>(num_sms) * 2;
  const int64_t max_grid = (s.n + kSimtWarps - 1) / kSimtWarps;
  if (grid > max_grid) grid = max_grid;
  if (grid < 1) grid = 1;
  return static_cast<int>(grid);
}

size_t simt_scratch_bytes(int dtype, const SearchShape& s, int grid) {
  (void)dtype;
  const int QC = qc_for(s);
  const int K = list_len_for(s.k);
  const int64_t chunks = (s.q + QC - 1) / QC;
  size_t bytes = sizeof(uint64_t) * static_cast<size_t>(chunks) * grid * QC * K;
  if (K > 32) bytes += sizeof(uint64_t) * static_cast<size_t>(chunks) * grid * kSimtWarps * QC * 2 * K;
  return bytes;
}

cudaError_t launch_simt_search(int dtype, const void* E, const void* Q, const SearchShape& s,
                               const Fusion& fu, void* scratch, int grid, ListSet* lists,
                               cudaStream_t st) {
  const int QC = qc_for(s);
  return dtype == kF32 ? launch_f32(QC, E, Q, s, fu, scratch, grid, lists, st)
                       : launch_bf16(QC, E, Q, s, fu, scratch, grid, lists, st);
}

}  // namespace oprag
