// Block merge of one query's partial lists (the global top-k reduction of
// Op_retrieve, Sec. 3.2 / Sec. 4.1 Retrieval), run by the merge kernel with
// one CTA per query.
//
// The P * kl candidate keys of the query (the first kl of each producer's
// sorted list) are split evenly over the CTA's warps; a warp fetches four
// 32-key groups at once (independent loads, so L2 latency is paid once per
// group of four) and filters them against its running k-th best.  Warp 0 then
// merges the warps' results and writes the query's ranked top-k.
#pragma once
#include "common.cuh"
#include "internal.h"

namespace oprag {

template <int KP>
__device__ __forceinline__ void merge_offer32(WarpMerger<KP>& m, uint64_t key) {
  const int lane = threadIdx.x & 31;
  const bool pass = key > m.worst;
  const uint32_t bits = __ballot_sync(0xffffffffu, pass);
  if (bits == 0) return;
  if (m.count > WarpMerger<KP>::kCap - 32) m.compact();
  if (pass) m.sbuf[m.count + __popc(bits & ((1u << lane) - 1u))] = key;
  m.count += __popc(bits);
}

// Writes result o of the merge: a key's id (split into the corpus and the id
// within it for a search over two stacked corpora) and score, or the empty
// result (-1, -inf).
__device__ __forceinline__ void store_result(const ListSet& ls, int64_t* out_ids, float* out_scores,
                                             int64_t o, uint64_t key) {
  if (key == kEmptyKey) {
    out_ids[o] = -1;
    out_scores[o] = -INFINITY;
    if (ls.out_src != nullptr) ls.out_src[o] = -1;
    return;
  }
  int64_t id = static_cast<int64_t>(key_id(key));
  if (ls.out_src != nullptr) {
    const bool second = id >= ls.split;
    ls.out_src[o] = second ? 1 : 0;
    if (second) id -= ls.split;
  }
  out_ids[o] = id;
  out_scores[o] = key_score(key);
}

// Lists that exist for the query tile `tile` (see ListSet).
__device__ __forceinline__ int merge_list_count(const ListSet& ls, int tile) {
  int np = ls.P;
  if (ls.C > 0) {
    int c0 = static_cast<int>(static_cast<int64_t>(tile / ls.pair) * ls.C / ls.qt) - 1;
    c0 = c0 < 0 ? 0 : c0;
    np = min(ls.P, (ls.C - c0) * ls.sets);
  }
  return np;
}

// The smallest key that can still be among the query's k best: a counted
// floor f whose band counts up to it sum to k or more proves k real scores
// >= f, so every key of the top k has a score >= f (the key of score f with
// the largest id ranks below all of them).  kEmptyKey (admit all) without
// counted floors.
__device__ __forceinline__ uint64_t merge_floor_key(const ListSet& ls, int qi, int k) {
  if (ls.levels == nullptr || ls.level_cnt == nullptr) return kEmptyKey;
  int sum = 0;
#pragma unroll
  for (int i = 0; i < kLevels; ++i) {
    const int64_t o = static_cast<int64_t>(qi) * kLevels + i;
    sum += ls.level_cnt[o];
    if (sum >= k) {
      const float f = ls.levels[o];
      return f > -INFINITY ? make_key(f, kNoId) : kEmptyKey;
    }
  }
  return kEmptyKey;
}

// Shared memory: (nw + 1) * 2 * KP keys.  All threads of the CTA call this;
// it ends with a barrier, so the buffer can be reused.
template <int KP>
__device__ __forceinline__ void merge_one_query(const ListSet& ls, int qi, int k, int nw,
                                int64_t* __restrict__ out_ids, float* __restrict__ out_scores,
                                float* __restrict__ kth_out, float* __restrict__ levels_out,
                                uint64_t* smem_keys) {
  constexpr int kCap = 2 * KP;
  constexpr int kUnroll = 4;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int tile = qi / ls.TH, row = qi % ls.TH;
  const uint64_t* base = ls.keys + (static_cast<int64_t>(tile) * ls.P * ls.TH + row) * ls.stride;
  const int64_t list_step = static_cast<int64_t>(ls.TH) * ls.stride;
  const int np = merge_list_count(ls, tile);
  const int kl = min(k, ls.klen);         // keys read from each list
  const int total = np * kl;
  const int lo = static_cast<int>(static_cast<int64_t>(total) * warp / nw);
  const int hi = static_cast<int>(static_cast<int64_t>(total) * (warp + 1) / nw);

  WarpMerger<KP> m;
  m.init(smem_keys + warp * kCap, k);
  for (int g = lo; g < hi; g += 32 * kUnroll) {
    uint64_t key[kUnroll];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const int i = g + u * 32 + lane;
      key[u] = kEmptyKey;
      if (i < hi) {
        const int p = i / kl;
        key[u] = base[p * list_step + (i - p * kl)];
      }
    }
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) merge_offer32(m, key[u]);
  }
  m.finish();
  __syncthreads();
  if (warp == 0) {
    WarpMerger<KP> f;
    f.init(smem_keys + nw * kCap, k);
    const int all = nw * k;
    for (int g = 0; g < all; g += 32 * kUnroll) {
      uint64_t key[kUnroll];
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) {
        const int i = g + u * 32 + lane;
        key[u] = kEmptyKey;
        if (i < all) {
          const int w = i / k;
          key[u] = smem_keys[w * kCap + (i - w * k)];
        }
      }
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) merge_offer32(f, key[u]);
    }
    f.finish();
    if (kth_out != nullptr && lane == 0) {
      const uint64_t kk = f.sbuf[k - 1];
      kth_out[qi] = kk == kEmptyKey ? -INFINITY : key_score(kk);
    }
    if (levels_out != nullptr && lane < kLevels) {
      const uint64_t kk = f.sbuf[level_rank(k, lane) - 1];
      levels_out[static_cast<int64_t>(qi) * kLevels + lane] =
          kk == kEmptyKey ? -INFINITY : key_score(kk);
    }
    for (int i = lane; i < k; i += 32) {
      const uint64_t key = f.sbuf[i];
      const int64_t o = static_cast<int64_t>(qi) * k + i;
      store_result(ls, out_ids, out_scores, o, key);
    }
  }
  __syncthreads();
}

}  // namespace oprag
