// Global top-k reduction: merges the partial lists that the search kernels
// leave per (query tile, producer) into the final ranked top-k of each query.
// This is the step of Op_retrieve (Sec. 3.2; Sec. 4.1 Retrieval) that reduces
// local candidates to the global top-k, done inside one GPU: the producers
// are corpus slices instead of index shards.
//
// Four merges: for unsorted lists (buffered tensor-core lists, k > 32) and
// for sorted lists of at most 32 keys merged into k > 32, one warp per query
// over all their keys; otherwise for sorted lists, by list count and k, one
// warp per query over at most 32 lists (head by head), one to four warps per
// query over up to 512 lists when k <= 16 (also head by head), and the block
// merge of merge.cuh (one CTA per query).
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
    const uint64_t best = warp_max_key(h[0]);
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
        store_result(ls, out_ids, out_scores, o, mine);
      }
    }
    if (r == k - 1 && kth_out != nullptr && lane == 0)
      kth_out[qi] = best == kEmptyKey ? -INFINITY : key_score(best);
    if (levels_out != nullptr && lane < kLevels && r == level_rank(k, lane) - 1)
      levels_out[static_cast<int64_t>(qi) * kLevels + lane] =
          best == kEmptyKey ? -INFINITY : key_score(best);
  }
}

// More than 32 lists and k <= 16, at most kSmallLists lists per lane: W
// warps per query (W = 1, 2 or 4 by list count; CTAs of four warps, 4 / W
// queries each).
// Launched early (programmatic dependent
// launch), a CTA waits in place and starts as soon as the search grid ends.
// Lane l of warp w holds lists p = 32 w + l + 32 W u (u < kSmallLists): the
// first kSmallKeys keys of each, fetched with 16-byte loads all issued
// together.  Then the query's 32 W lanes take the k best head by head:
// each round the lanes' best heads go through a warp maximum (and, when
// W > 1, a maximum over the query's warps in shared memory); keys are
// unique, so one lane owns the winner and advances that list (fetching its
// next keys once the held ones are used up, which only k > kSmallKeys can
// need).
constexpr int kSmallThreads = 128;
constexpr int kSmallLists = 4;
constexpr int kSmallKeys = 6;

template <int W>
__global__ void __launch_bounds__(kSmallThreads, 4)
merge_small_kernel(ListSet ls, int q, int k, int64_t* __restrict__ out_ids,
                   float* __restrict__ out_scores, float* __restrict__ kth_out,
                   float* __restrict__ levels_out) {
  constexpr int kQPerCta = kSmallThreads / 32 / W;
  __shared__ uint64_t heads[2][kSmallThreads / 32];
  asm volatile("griddepcontrol.wait;" ::: "memory");
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int qs = warp / W, wq = warp % W;      // query slot in the CTA, warp of the query
  const int qi = blockIdx.x * kQPerCta + qs;
  if (qi >= q) return;                         // all W warps of the slot leave together
  const int tile = qi / ls.TH, row = qi % ls.TH;
  const int np = merge_list_count(ls, tile);
  const int kl = min(k, ls.klen);
  const uint64_t* base = ls.keys + (static_cast<int64_t>(tile) * ls.P * ls.TH + row) * ls.stride;
  const int64_t list_step = static_cast<int64_t>(ls.TH) * ls.stride;
  // Keys at or past kl of a list are not candidates; a missing list is empty.
  auto fetch = [&](int u, int from, uint64_t (&dst)[kSmallKeys]) {
    const int p = wq * 32 + lane + u * 32 * W;
    const uint64_t* l = base + p * list_step + from;
#pragma unroll
    for (int j = 0; j < kSmallKeys; j += 2) {
      ulonglong2 v = make_ulonglong2(kEmptyKey, kEmptyKey);
      if (p < np && from + j < kl) v = *reinterpret_cast<const ulonglong2*>(l + j);
      dst[j] = v.x;
      dst[j + 1] = from + j + 1 < kl ? v.y : kEmptyKey;
    }
  };
  uint64_t key[kSmallLists][kSmallKeys];
  int used[kSmallLists];
#pragma unroll
  for (int u = 0; u < kSmallLists; ++u) {
    fetch(u, 0, key[u]);
    used[u] = 0;
  }
  uint64_t mine = kEmptyKey;
  for (int r = 0; r < k; ++r) {
    uint64_t own = key[0][0];
#pragma unroll
    for (int u = 1; u < kSmallLists; ++u) own = umax64(own, key[u][0]);
    uint64_t best = warp_max_key(own);
    if constexpr (W > 1) {
      if (lane == 0) heads[r & 1][warp] = best;
      // The query's W warps (named barrier 1 + slot; constant ids, so
      // that the kernel reserves only the barriers it uses).
      if (qs == 0) asm volatile("bar.sync 1, %0;" ::"n"(32 * W) : "memory");
      else asm volatile("bar.sync 2, %0;" ::"n"(32 * W) : "memory");
#pragma unroll
      for (int j = 0; j < W; ++j) best = umax64(best, heads[r & 1][qs * W + j]);
    }
    if (best != kEmptyKey && own == best) {
      bool done = false;
#pragma unroll
      for (int u = 0; u < kSmallLists; ++u) {
        if (!done && key[u][0] == best) {
          done = true;
#pragma unroll
          for (int j = 0; j + 1 < kSmallKeys; ++j) key[u][j] = key[u][j + 1];
          key[u][kSmallKeys - 1] = kEmptyKey;
          if (++used[u] % kSmallKeys == 0 && used[u] < kl) fetch(u, used[u], key[u]);
        }
      }
    }
    if (wq != 0) continue;
    if ((r & 31) == lane) mine = best;
    if ((r & 31) == 31 || r == k - 1) {
      const int i = (r & ~31) + lane;
      if (i <= r) {
        const int64_t o = static_cast<int64_t>(qi) * k + i;
        store_result(ls, out_ids, out_scores, o, mine);
      }
    }
    if (r == k - 1 && kth_out != nullptr && lane == 0)
      kth_out[qi] = best == kEmptyKey ? -INFINITY : key_score(best);
    if (levels_out != nullptr && lane < kLevels && r == level_rank(k, lane) - 1)
      levels_out[static_cast<int64_t>(qi) * kLevels + lane] =
          best == kEmptyKey ? -INFINITY : key_score(best);
  }
}

// Unsorted lists (ListSet::counts), k > 32, and short sorted lists merged
// into k > 32 (read whole, as if unsorted): one warp per query.  The warp
// scans the query's list counts into offsets in shared memory, reads the
// concatenated keys 32 x kUnsortedLoads at a time (a lane's keys come in
// increasing order, so it finds each key's list by moving a cursor forward
// over the offsets, rarely more than one step), drops keys below the counted floor and
// keeps the rest in a WarpMerger, whose buffer is sorted only when it fills
// up and once at the end.  A good floor leaves a few hundred keys of the
// several thousand read, so a query usually costs one sort; the warps of
// different queries share nothing and need no barrier.
constexpr int kUnsortedWarps = 4;
constexpr int kUnsortedLoads = 8;

// Shared memory of merge_unsorted_kernel: a merger buffer and P + 1
// offsets per warp.
template <int KP>
size_t unsorted_smem_bytes(int P) {
  return kUnsortedWarps * (2 * KP * sizeof(uint64_t) + (static_cast<size_t>(P) + 4) / 4 * 16);
}

template <int KP>
__global__ void __launch_bounds__(kUnsortedWarps * 32)
merge_unsorted_kernel(ListSet ls, int q, int k, int64_t* __restrict__ out_ids,
                      float* __restrict__ out_scores, float* __restrict__ kth_out,
                      float* __restrict__ levels_out) {
  extern __shared__ __align__(16) uint64_t smem_u[];
  asm volatile("griddepcontrol.wait;" ::: "memory");
  constexpr int kCap = 2 * KP;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int qi = blockIdx.x * kUnsortedWarps + warp;
  if (qi >= q) return;
  const int tile = qi / ls.TH, row = qi % ls.TH;
  const int np = merge_list_count(ls, tile);
  const int offs_len = (ls.P + 4) / 4 * 4;
  int* offs = reinterpret_cast<int*>(smem_u + kUnsortedWarps * kCap) + warp * offs_len;
  const int* cnt = ls.counts != nullptr
                       ? ls.counts + static_cast<int64_t>(tile) * ls.P * ls.TH + row
                       : nullptr;
  const int fixed = min(ls.klen, ls.stride);     // keys of a sorted list
  const uint64_t* base = ls.keys + (static_cast<int64_t>(tile) * ls.P * ls.TH + row) * ls.stride;
  const int64_t list_step = static_cast<int64_t>(ls.TH) * ls.stride;

  // offs[p]: keys of the lists before p (exclusive scan, 32 lists a round)
  int total = 0;
  for (int p0 = 0; p0 < np; p0 += 32) {
    const int p = p0 + lane;
    const int c = p >= np          ? 0
                  : cnt == nullptr ? fixed
                                   : max(0, min(cnt[static_cast<int64_t>(p) * ls.TH], ls.stride));
    int incl = c;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int t = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += t;
    }
    if (p < np) offs[p] = total + incl - c;
    total += __shfl_sync(0xffffffffu, incl, 31);
  }
  if (lane == 0) offs[np] = total;
  __syncwarp();

  WarpMerger<KP> m;
  m.init(smem_u + warp * kCap, k);
  m.worst = merge_floor_key(ls, qi, k);
  int cur = 0;      // this lane's list: offs[cur] <= its next key's index
  for (int g = 0; g < total; g += 32 * kUnsortedLoads) {
    uint64_t key[kUnsortedLoads];
#pragma unroll
    for (int u = 0; u < kUnsortedLoads; ++u) {
      const int i = g + u * 32 + lane;
      key[u] = kEmptyKey;
      if (i < total) {
        // the list holding key i: the last p with offs[p] <= i (offs[np] =
        // total > i ends the walk)
        while (offs[cur + 1] <= i) ++cur;
        key[u] = base[cur * list_step + (i - offs[cur])];
      }
    }
#pragma unroll
    for (int u = 0; u < kUnsortedLoads; ++u)
      if (g + u * 32 < total) merge_offer32(m, key[u]);
  }
  m.finish();
  if (kth_out != nullptr && lane == 0) {
    const uint64_t kk = m.sbuf[k - 1];
    kth_out[qi] = kk == kEmptyKey ? -INFINITY : key_score(kk);
  }
  if (levels_out != nullptr && lane < kLevels) {
    const uint64_t kk = m.sbuf[level_rank(k, lane) - 1];
    levels_out[static_cast<int64_t>(qi) * kLevels + lane] =
        kk == kEmptyKey ? -INFINITY : key_score(kk);
  }
  for (int i = lane; i < k; i += 32)
    store_result(ls, out_ids, out_scores, static_cast<int64_t>(qi) * k + i, m.sbuf[i]);
}

template <int KP>
cudaError_t launch_unsorted_kp(const ListSet& ls, int q, int k, int64_t* ids, float* scores,
                               cudaStream_t st, float* kth_out, float* levels_out) {
  const size_t smem = unsorted_smem_bytes<KP>(ls.P);
  if (smem > 48 * 1024) {
    const cudaError_t e =
        cudaFuncSetAttribute(merge_unsorted_kernel<KP>,
                             cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
    if (e != cudaSuccess) return e;
  }
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3((q + kUnsortedWarps - 1) / kUnsortedWarps);
  cfg.blockDim = dim3(kUnsortedWarps * 32);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, merge_unsorted_kernel<KP>, ls, q, k, ids, scores, kth_out,
                            levels_out);
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

template <int W>
cudaError_t launch_small_w(const ListSet& ls, int q, int k, int64_t* out_ids, float* out_scores,
                           cudaStream_t st, float* kth_out, float* levels_out) {
  constexpr int kQPerCta = kSmallThreads / 32 / W;
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3((q + kQPerCta - 1) / kQPerCta);
  cfg.blockDim = dim3(kSmallThreads);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, merge_small_kernel<W>, ls, q, k, out_ids, out_scores, kth_out,
                            levels_out);
}

// Warps per query of merge_small_kernel: the fewest whose lanes hold all of
// a query's lists (kSmallLists each).  The lists' loads are issued together
// whatever W is, and with one warp per query the head-by-head rounds need no
// barrier.  Returns cudaErrorNotSupported when four warps do not suffice (the
// caller then takes the block merge).
cudaError_t launch_small(const ListSet& ls, int q, int k, int64_t* out_ids, float* out_scores,
                         cudaStream_t st, float* kth_out, float* levels_out) {
  constexpr int kPerWarp = kSmallLists * 32;
  const int W = ls.P <= kPerWarp ? 1 : ls.P <= 2 * kPerWarp ? 2 : 4;
  if (ls.P > W * kPerWarp) return cudaErrorNotSupported;
  if (W == 4) return launch_small_w<4>(ls, q, k, out_ids, out_scores, st, kth_out, levels_out);
  if (W == 2) return launch_small_w<2>(ls, q, k, out_ids, out_scores, st, kth_out, levels_out);
  return launch_small_w<1>(ls, q, k, out_ids, out_scores, st, kth_out, levels_out);
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
  // Unsorted lists, or sorted lists of at most 32 keys merged into more
  // (the sampled first pass of a search with k > 32): one sort per query
  // instead of k head-by-head rounds.
  if (ls.counts != nullptr || (k > 32 && ls.klen <= 32 && ls.stride <= 32)) {
    if (k <= 64) return launch_unsorted_kp<64>(ls, q, k, out_ids, out_scores, st, kth_out, levels_out);
    if (k <= 128)
      return launch_unsorted_kp<128>(ls, q, k, out_ids, out_scores, st, kth_out, levels_out);
    return launch_unsorted_kp<256>(ls, q, k, out_ids, out_scores, st, kth_out, levels_out);
  }
  if (ls.P <= 32)
    return launch_warp_per_query(merge_kway_kernel, kWayWarps, ls, q, k, out_ids, out_scores, st,
                                 kth_out, levels_out);
  if (k <= 16) {
    const cudaError_t e = launch_small(ls, q, k, out_ids, out_scores, st, kth_out, levels_out);
    if (e != cudaErrorNotSupported) return e;
  }
  if (k <= 32) return launch_merge_kp<32>(ls, q, k, out_ids, out_scores, st, kth_out, levels_out);
  if (k <= 64) return launch_merge_kp<64>(ls, q, k, out_ids, out_scores, st, kth_out, levels_out);
  if (k <= 128) return launch_merge_kp<128>(ls, q, k, out_ids, out_scores, st, kth_out, levels_out);
  return launch_merge_kp<256>(ls, q, k, out_ids, out_scores, st, kth_out, levels_out);
}

}  // namespace oprag
