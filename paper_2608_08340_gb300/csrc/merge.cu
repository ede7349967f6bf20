// Global top-k reduction: merges the partial lists that the search kernels
// leave per (query tile, producer) into the final ranked top-k of each query.
// This is the step of Op_retrieve (Sec. 3.2; Sec. 4.1 Retrieval) that reduces
// local candidates to the global top-k, done inside one GPU: the producers
// are corpus slices instead of index shards.
//
// Three merges by list count and k: one warp per query over at most 32
// sorted lists (head by head), one warp per query over more lists when
// k <= 16, and the block merge of merge.cuh (one CTA per query) otherwise.
#include "merge.cuh"

namespace oprag {

namespace {

constexpr int kMergeWarps = 8;

template <int KP>
__global__ void __launch_bounds__(kMergeWarps * 32)
merge_kernel(ListSet ls, int q, int k, int64_t* __restrict__ out_ids,
             float* __restrict__ out_scores, float* __restrict__ kth_out,
             float* __restrict__ levels_out) {
  extern __shared__ __align__(16) uint64_t smem_keys[];
  // Launched as a programmatic dependent of the search kernel: wait until
  // that grid has finished and its lists are visible.
  asm volatile("griddepcontrol.wait;" ::: "memory");
  const int qi = blockIdx.x;
  if (qi >= q) return;
  merge_one_query<KP>(ls, qi, k, kMergeWarps, out_ids, out_scores, kth_out, levels_out, smem_keys);
}

template <int KP>
cudaError_t launch_merge_kp(const ListSet& ls, int q, int k, int64_t* ids, float* scores,
                            cudaStream_t st, float* kth_out, float* levels_out) {
  const size_t smem = static_cast<size_t>(kMergeWarps + 1) * 2 * KP * sizeof(uint64_t);
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(q);
  cfg.blockDim = dim3(kMergeWarps * 32);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, merge_kernel<KP>, ls, q, k, ids, scores, kth_out, levels_out);
}

// Few lists per query (at most 32): one warp per query merges the sorted
// lists directly.  Lane l holds the head of list l (with the next keys
// prefetched in registers); each round the warp takes the largest head
// (keys are unique, so exactly one lane wins) and that lane advances.
// CTAs of two warps under 64 registers a thread fit beside a running search
// CTA, so the early-launched merge waits in place.
constexpr int kHeads = 8;           // keys prefetched per list
constexpr int kWayWarps = 2;        // queries per CTA

__global__ void __launch_bounds__(kWayWarps * 32, 16)
merge_kway_kernel(ListSet ls, int q, int k, int64_t* __restrict__ out_ids,
                  float* __restrict__ out_scores, float* __restrict__ kth_out,
                  float* __restrict__ levels_out) {
  asm volatile("griddepcontrol.wait;" ::: "memory");
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int qi = blockIdx.x * kWayWarps + warp;
  if (qi >= q) return;
  const int tile = qi / ls.TH, row = qi % ls.TH;
  const int np = merge_list_count(ls, tile);
  const int kl = min(k, ls.klen);
  const uint64_t* list = ls.keys + ((static_cast<int64_t>(tile) * ls.P + lane) * ls.TH + row) *
                                       static_cast<int64_t>(ls.stride);
  const bool has_list = lane < np;
  uint64_t h[kHeads];
  int next = 0;       // keys of this list fetched so far
  auto refill = [&]() {
#pragma unroll
    for (int i = 0; i < kHeads; ++i) h[i] = next + i < kl ? list[next + i] : kEmptyKey;
    next += kHeads;
  };
  if (has_list) refill();
  else {
#pragma unroll
    for (int i = 0; i < kHeads; ++i) h[i] = kEmptyKey;
  }
  int avail = kHeads;
  uint64_t mine = kEmptyKey;      // the answer of rank (lane + 32 * m) for the current m
  for (int r = 0; r < k; ++r) {
    uint64_t best = h[0];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) best = umax64(best, __shfl_xor_sync(0xffffffffu, best, o));
    if (best != kEmptyKey && h[0] == best) {
#pragma unroll
      for (int i = 0; i + 1 < kHeads; ++i) h[i] = h[i + 1];
      h[kHeads - 1] = kEmptyKey;
      if (--avail == 0 && next < kl) {
        refill();
        avail = kHeads;
      }
    }
    if ((r & 31) == lane) mine = best;
    if ((r & 31) == 31 || r == k - 1) {
      const int i = (r & ~31) + lane;
      if (i <= r) {
        const int64_t o = static_cast<int64_t>(qi) * k + i;
        out_ids[o] = mine == kEmptyKey ? -1 : static_cast<int64_t>(key_id(mine));
        out_scores[o] = mine == kEmptyKey ? -INFINITY : key_score(mine);
      }
    }
    if (r == k - 1 && kth_out != nullptr && lane == 0)
      kth_out[qi] = best == kEmptyKey ? -INFINITY : key_score(best);
    if (levels_out != nullptr && lane < kLevels && r == level_rank(k, lane) - 1)
      levels_out[static_cast<int64_t>(qi) * kLevels + lane] =
          best == kEmptyKey ? -INFINITY : key_score(best);
  }
}

// More than 32 lists and k <= 16: one warp per query, two queries per CTA of
// 64 threads with at most 64 registers a thread, so that a CTA fits on an SM
// beside a running search CTA: launched early (programmatic dependent launch),
// it waits in place and starts as soon as the search grid ends.  Lane l reads
// the keys l, l + 32, ... of the query's np * kl candidates (64 / KL
// independent loads at a time, within the register budget) and keeps the
// best KL sorted in registers;
// then the lanes' sorted lists are merged head by head as above.
constexpr int kSmallWarps = 2;

template <int KL>
__global__ void __launch_bounds__(kSmallWarps * 32, 16)
merge_small_kernel(ListSet ls, int q, int k, int64_t* __restrict__ out_ids,
                   float* __restrict__ out_scores, float* __restrict__ kth_out,
                   float* __restrict__ levels_out) {
  asm volatile("griddepcontrol.wait;" ::: "memory");
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int qi = blockIdx.x * kSmallWarps + warp;
  if (qi >= q) return;
  const int tile = qi / ls.TH, row = qi % ls.TH;
  const int np = merge_list_count(ls, tile);
  const int kl = min(k, ls.klen);
  const int total = np * kl;
  const uint64_t* base = ls.keys + (static_cast<int64_t>(tile) * ls.P * ls.TH + row) * ls.stride;
  const int64_t list_step = static_cast<int64_t>(ls.TH) * ls.stride;
  constexpr int kLoadBatch = 64 / KL;
  uint64_t top[KL];
#pragma unroll
  for (int i = 0; i < KL; ++i) top[i] = kEmptyKey;
  for (int g = lane; g < total; g += 32 * kLoadBatch) {
    uint64_t key[kLoadBatch];
#pragma unroll
    for (int u = 0; u < kLoadBatch; ++u) {
      const int i = g + 32 * u;
      key[u] = kEmptyKey;
      if (i < total) {
        const int pl = i / kl;
        key[u] = base[pl * list_step + (i - pl * kl)];
      }
    }
#pragma unroll
    for (int u = 0; u < kLoadBatch; ++u) {
      const uint64_t x = key[u];
      if (x > top[KL - 1]) {
#pragma unroll
        for (int i = KL - 1; i > 0; --i)
          top[i] = x > top[i - 1] ? top[i - 1] : (x > top[i] ? x : top[i]);
        top[0] = x > top[0] ? x : top[0];
      }
    }
  }
  uint64_t mine = kEmptyKey;
  for (int r = 0; r < k; ++r) {
    uint64_t best = top[0];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) best = umax64(best, __shfl_xor_sync(0xffffffffu, best, o));
    if (best != kEmptyKey && top[0] == best) {
#pragma unroll
      for (int i = 0; i + 1 < KL; ++i) top[i] = top[i + 1];
      top[KL - 1] = kEmptyKey;
    }
    if ((r & 31) == lane) mine = best;
    if ((r & 31) == 31 || r == k - 1) {
      const int i = (r & ~31) + lane;
      if (i <= r) {
        const int64_t o = static_cast<int64_t>(qi) * k + i;
        out_ids[o] = mine == kEmptyKey ? -1 : static_cast<int64_t>(key_id(mine));
        out_scores[o] = mine == kEmptyKey ? -INFINITY : key_score(mine);
      }
    }
    if (r == k - 1 && kth_out != nullptr && lane == 0)
      kth_out[qi] = best == kEmptyKey ? -INFINITY : key_score(best);
    if (levels_out != nullptr && lane < kLevels && r == level_rank(k, lane) - 1)
      levels_out[static_cast<int64_t>(qi) * kLevels + lane] =
          best == kEmptyKey ? -INFINITY : key_score(best);
  }
}

template <typename Kern>
cudaError_t launch_warp_per_query(Kern kern, int warps, const ListSet& ls, int q, int k,
                                  int64_t* out_ids, float* out_scores, cudaStream_t st,
                                  float* kth_out, float* levels_out) {
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3((q + warps - 1) / warps);
  cfg.blockDim = dim3(warps * 32);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, ls, q, k, out_ids, out_scores, kth_out, levels_out);
}

}  // namespace

namespace {

// One thread per query: a two-way merge of the queries' ranked lists.
__global__ void merge_two_kernel(int q, const int64_t* __restrict__ a_ids,
                                 const float* __restrict__ a_sc, int ka,
                                 const int64_t* __restrict__ b_ids,
                                 const float* __restrict__ b_sc, int kb, int k,
                                 int64_t* __restrict__ out_ids, int32_t* __restrict__ out_src,
                                 float* __restrict__ out_scores) {
  const int qi = blockIdx.x * blockDim.x + threadIdx.x;
  if (qi >= q) return;
  const int64_t* ai = a_ids + static_cast<int64_t>(qi) * ka;
  const float* as = a_sc + static_cast<int64_t>(qi) * ka;
  const int64_t* bi = b_ids + static_cast<int64_t>(qi) * kb;
  const float* bs = b_sc + static_cast<int64_t>(qi) * kb;
  int i = 0, j = 0;
  for (int r = 0; r < k; ++r) {
    const bool a_ok = i < ka && ai[i] >= 0;
    const bool b_ok = j < kb && bi[j] >= 0;
    // At equal scores list a (the knowledge index) comes first.
    const bool take_a = a_ok && (!b_ok || !(bs[j] > as[i]));
    const int64_t o = static_cast<int64_t>(qi) * k + r;
    if (take_a) {
      out_ids[o] = ai[i];
      out_scores[o] = as[i];
      out_src[o] = 0;
      ++i;
    } else if (b_ok) {
      out_ids[o] = bi[j];
      out_scores[o] = bs[j];
      out_src[o] = 1;
      ++j;
    } else {
      out_ids[o] = -1;
      out_scores[o] = -INFINITY;
      out_src[o] = -1;
    }
  }
}

}  // namespace

cudaError_t launch_merge_two(int q, const int64_t* a_ids, const float* a_sc, int ka,
                             const int64_t* b_ids, const float* b_sc, int kb, int k,
                             int64_t* out_ids, int32_t* out_src, float* out_scores,
                             cudaStream_t st) {
  if (q <= 0) return cudaSuccess;
  merge_two_kernel<<<(q + 127) / 128, 128, 0, st>>>(q, a_ids, a_sc, ka, b_ids, b_sc, kb, k,
                                                    out_ids, out_src, out_scores);
  return cudaGetLastError();
}

cudaError_t launch_merge(const ListSet& ls, int q, int k, int64_t* out_ids, float* out_scores,
                         cudaStream_t st, float* kth_out, float* levels_out) {
  if (q <= 0) return cudaSuccess;
  if (ls.P <= 32)
    return launch_warp_per_query(merge_kway_kernel, kWayWarps, ls, q, k, out_ids, out_scores, st,
                                 kth_out, levels_out);
  if (k <= 8)
    return launch_warp_per_query(merge_small_kernel<8>, kSmallWarps, ls, q, k, out_ids,
                                 out_scores, st, kth_out, levels_out);
  if (k <= 16)
    return launch_warp_per_query(merge_small_kernel<16>, kSmallWarps, ls, q, k, out_ids,
                                 out_scores, st, kth_out, levels_out);
  if (k <= 32) return launch_merge_kp<32>(ls, q, k, out_ids, out_scores, st, kth_out, levels_out);
  if (k <= 64) return launch_merge_kp<64>(ls, q, k, out_ids, out_scores, st, kth_out, levels_out);
  if (k <= 128) return launch_merge_kp<128>(ls, q, k, out_ids, out_scores, st, kth_out, levels_out);
  return launch_merge_kp<256>(ls, q, k, out_ids, out_scores, st, kth_out, levels_out);
}

}  // namespace oprag
