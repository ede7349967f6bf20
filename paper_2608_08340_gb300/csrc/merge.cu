// Global top-k reduction: merges the partial lists that the search kernels
// leave per (query tile, producer) into the final ranked top-k of each query.
// This is the "local candidates, then global top-k reduction" step of
// Op_retrieve (Sec. 3.2; Sec. 4.1 Retrieval), done inside one GPU: the
// producers are corpus slices instead of index shards.
#include "common.cuh"
#include "internal.h"

namespace oprag {

namespace {

constexpr int kMergeWarps = 8;

// One CTA per query.  Warp w merges producers w, w+8, ... into its own buffer;
// warp 0 then merges the eight warp results and writes the answer.
template <int KP>
__global__ void __launch_bounds__(kMergeWarps * 32)
merge_kernel(ListSet ls, int q, int k, int64_t* __restrict__ out_ids,
             float* __restrict__ out_scores) {
  constexpr int kCap = 2 * KP;
  extern __shared__ __align__(16) uint64_t smem_keys[];
  const int qi = blockIdx.x;
  if (qi >= q) return;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int tile = qi / ls.TH, row = qi % ls.TH;

  WarpMerger<KP> m;
  m.init(smem_keys + warp * kCap, k);
  for (int p = warp; p < ls.P; p += kMergeWarps) {
    const uint64_t* list =
        ls.keys + (static_cast<int64_t>(tile) * ls.P + p) * ls.TH * ls.stride +
        static_cast<int64_t>(row) * ls.stride;
    m.offer_list(list, k);
  }
  m.finish();
  __syncthreads();
  if (warp != 0) return;

  WarpMerger<KP> f;
  f.init(smem_keys + kMergeWarps * kCap, k);
  for (int w = 0; w < kMergeWarps; ++w) f.offer_list(smem_keys + w * kCap, k);
  f.finish();
  for (int i = lane; i < k; i += 32) {
    const uint64_t key = f.sbuf[i];
    const int64_t o = static_cast<int64_t>(qi) * k + i;
    out_ids[o] = key == kEmptyKey ? -1 : static_cast<int64_t>(key_id(key));
    out_scores[o] = key == kEmptyKey ? -INFINITY : key_score(key);
  }
}

template <int KP>
cudaError_t launch_merge_kp(const ListSet& ls, int q, int k, int64_t* ids, float* scores,
                            cudaStream_t st) {
  const size_t smem = static_cast<size_t>(kMergeWarps + 1) * 2 * KP * sizeof(uint64_t);
  merge_kernel<KP><<<q, kMergeWarps * 32, smem, st>>>(ls, q, k, ids, scores);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_merge(const ListSet& ls, int q, int k, int64_t* out_ids, float* out_scores,
                         cudaStream_t st) {
  if (q <= 0) return cudaSuccess;
  if (k <= 32) return launch_merge_kp<32>(ls, q, k, out_ids, out_scores, st);
  if (k <= 64) return launch_merge_kp<64>(ls, q, k, out_ids, out_scores, st);
  if (k <= 128) return launch_merge_kp<128>(ls, q, k, out_ids, out_scores, st);
  return launch_merge_kp<256>(ls, q, k, out_ids, out_scores, st);
}

}  // namespace oprag
