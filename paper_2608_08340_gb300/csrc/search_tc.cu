// Host planning for the tensor-core search kernel of search_tc.cuh: tile
// size, persistent grid, window size and list bound, scratch size and TMA
// descriptors.
#include <algorithm>
#include <vector>

#include "search_tc.cuh"

namespace oprag {

using namespace tc;

namespace {

// ----------------------------------------------------------------- host

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  if (fn == nullptr) {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult qres;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault,
                                         &qres) == cudaSuccess &&
        qres == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(ptr);
  }
  return fn;
}

// Row-major rows x d bf16 matrix, boxes of 64 columns x box_rows rows, 128-byte swizzle;
// rows past the end read as zero.
bool make_map(CUtensorMap* m, const void* base, int64_t rows, int d, int box_rows) {
  EncodeTiledFn enc = encode_fn();
  if (enc == nullptr) return false;
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(d), static_cast<cuuint64_t>(rows)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(d) * 2};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(kBlockK), static_cast<cuuint32_t>(box_rows)};
  cuuint32_t estr[2] = {1, 1};
  return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box,
             estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) ==
         CUDA_SUCCESS;
}

}  // namespace

int tc_pair_capacity() { return pair_capacity_query(); }

TcPlan tc_plan(const SearchShape& s, int num_sms, int force_block_n, int tile_stride,
               int force_pair, int pair_capacity) {
  TcPlan pl{};
  pl.qt = (s.q + kBlockM - 1) / kBlockM;
  int bn = 256;
  if (s.fused_lex) {
    // The gathered hybrid search: single CTAs, 128-row tiles, one epilogue
    // set (its accumulators take all 512 TMEM columns).
    bn = 128;
  } else if (force_block_n == 128 || force_block_n == 256) {
    bn = force_block_n;
  } else {
    // Few units (small query batches): 128-row tiles give every SM more of
    // them; the MMA rate per row is the same for N = 128 and N = 256.
    const int64_t units256 =
      static_cast<int64_t>(pl.qt) * ((s.n + 255) / 256 + (s.n_second + 255) / 256);
    if (units256 < 4LL * num_sms) bn = 128;
  }
  // Dual mode: every unit takes two query tiles and one 128-row corpus tile,
  // so a CTA reads each corpus tile once for 256 queries, and its four
  // accumulators let one unit's epilogue overlap the next unit.  Automatic
  // when there are at least two query tiles and at most four dual units per
  // CTA (small batches, where the copies into the SMs, not the MMAs, bound
  // the kernel; measured on 32768 x 768: faster up to 512 queries, slower at
  // 1024); it needs the two epilogue sets of lists of 8 or 16.
  const bool dual_ok = !s.fused_lex && pl.qt >= 2 && list_len_for(s.k) <= 16 &&
                       force_pair != 2 && (force_block_n == 0 || force_block_n == 128);
  const int64_t dual_units =
      static_cast<int64_t>((pl.qt + 1) / 2) * ((s.n + 127) / 128 + (s.n_second + 127) / 128);
  pl.dual = dual_ok && (force_pair == 3 || (force_pair == 0 && dual_units <= 4LL * num_sms));
  if (pl.dual) bn = 128;
  pl.block_n = bn;
  // CTA pairs cut the operand bytes each SM loads per MMA by a third; they
  // need 256-row corpus tiles and a device that fits clusters of two.  They
  // run on request, and by default for large batches with buffered lists
  // (k > 32, at least 8 query tiles): measured on GB300, 1M x 768 with 2048
  // queries and k = 100 takes 2524 instead of 2591 us; with lists of 16
  // (32768 x 1024, 4096 queries, k = 10) pairs are no faster.
  const bool pair = !s.fused_lex && bn == 256 && pair_capacity > 0 &&
                    (force_pair == 2 ||
                     (force_pair == 0 && list_len_for(s.k) > 32 && pl.qt >= 8));
  pl.pair = pair ? 2 : 1;
  pl.uqt = pair || pl.dual ? (pl.qt + 1) / 2 : pl.qt;
  pl.tile_stride = tile_stride < 1 ? 1 : tile_stride;
  // two stacked corpora: the second's tiles follow the first's
  pl.nt_first = static_cast<int>((s.n + bn - 1) / bn);
  const int64_t all_tiles = pl.nt_first + (s.n_second + bn - 1) / bn;
  pl.nt = static_cast<int>((all_tiles + pl.tile_stride - 1) / pl.tile_stride);
  const int64_t units = static_cast<int64_t>(pl.nt) * pl.uqt;
  const int slots = pair ? pair_capacity : num_sms;     // schedule units in flight
  int C = static_cast<int>(units < slots ? units : slots);
  if (C < 1) C = 1;
  pl.grid = C * pl.pair;
  // Windows of about 32 MB of corpus.  Inside a window every CTA works on
  // a contiguous share of (query tile, corpus tile) units, so at any moment
  // the CTAs read tiles spread over the whole window: a window that stays in
  // L2 is read from HBM about once.  With few query tiles the CTAs of
  // one query tile already read the corpus in step, and one window over a
  // small corpus (<= 80 MB) keeps the list count per query tile low (up to 8
  // query tiles: measured, windows then cost more in lists than they save).
  const int64_t tile_bytes = static_cast<int64_t>(bn) * s.d * 2;
  const int64_t corpus = tile_bytes * pl.nt;
  const int win32 = static_cast<int>(std::max<int64_t>(1, (int64_t(32) << 20) / tile_bytes));
  pl.win = corpus <= (int64_t(80) << 20) && pl.uqt <= 8 ? pl.nt : std::min(win32, pl.nt);
  // Exact per-tile range of schedule slots (CTAs or pairs), by replaying
  // the schedule of UnitSeq.
  int per_tile = 1;
  std::vector<int> hi(pl.uqt, -1);
  bool ok = true;
  for (int w = 0; static_cast<int64_t>(w) * pl.win < pl.nt; ++w) {
    const int tw = std::min(pl.win, pl.nt - w * pl.win);
    const int64_t uw = static_cast<int64_t>(pl.uqt) * tw;
    for (int c = 0; c < C; ++c) {
      const int64_t l0 = uw * c / C, l1 = uw * (c + 1) / C;
      if (l0 >= l1) continue;
      for (int64_t j = l0 / tw; j <= (l1 - 1) / tw; ++j) {
        if (c < first_cta(static_cast<int>(j), pl.uqt, C)) ok = false;
        hi[j] = std::max(hi[j], c);
      }
    }
  }
  for (int j = 0; j < pl.uqt; ++j)
    per_tile = std::max(per_tile, hi[j] - first_cta(j, pl.uqt, C) + 1);
  if (!ok) per_tile = C;  // not expected; every slot then gets a list per tile
  pl.sets = pl.dual ? 1 : epi_sets(list_len_for(s.k), s.fused_lex);
  pl.pmax = per_tile * pl.sets;
  const int K = list_len_for(s.k);
  // Shared memory of the launch (the same sum as smem_for<BN, K, pair, dual>).
  const size_t b_stage = static_cast<size_t>(pair ? bn / 2 : bn) * 128;
  const size_t a_stage = kAStageBytes * (pl.dual ? 2 : 1);
  pl.stages = pair        ? stages_for<256, true>()
              : pl.dual     ? stages_for<128, false, true>()
              : s.fused_lex ? stages_for<128, false, false, true>()
                            : (bn == 128 ? stages_for<128>() : stages_for<256>());
  pl.smem = static_cast<size_t>(pl.stages) * (a_stage + b_stage) +
            static_cast<size_t>(epi_sets(K, s.fused_lex)) * 128 * kStageRowBytes +
            lex_land_bytes(s.fused_lex) + 1024 + 256;
  return pl;
}

// List rows: one per (query tile, producer, query row); pair and dual modes
// cover 2 * uqt tiles (an odd qt leaves the last pair's second tile empty).
static size_t list_rows(const TcPlan& pl) {
  return static_cast<size_t>(pl.uqt) * (pl.pair == 2 || pl.dual ? 2 : 1) * pl.pmax * kBlockM;
}

size_t tc_scratch_bytes(const SearchShape& s, const TcPlan& pl) {
  const int K = list_len_for(s.k);
  const int stride = K > 32 ? 2 * K : K;
  const size_t rows = list_rows(pl);
  size_t bytes = rows * stride * sizeof(uint64_t);
  if (K > 32) bytes += rows * (sizeof(uint64_t) + sizeof(int));
  return bytes;
}

cudaError_t launch_tc_search(const void* E, const void* Q, const SearchShape& s, const Fusion& fu,
                             const TcPlan& pl, void* scratch, int* dev_err, ListSet* lists,
                             cudaStream_t st, const float* init_floor, uint64_t* qfloor,
                             uint32_t gen, const float* levels, int* level_cnt,
                             long long wait_limit, unsigned long long* phases,
                             const void* E2) {
  TcMaps maps;
  // With a single query tile only its real rows are loaded (the remaining
  // rows of the A tile hold stale data whose TMEM lanes the epilogue never
  // reads); rows are loaded in multiples of 8, the swizzle atom height.
  // Pair mode: each CTA loads all 128 rows of its tile and half of the
  // corpus tile.
  const int a_rows =
      pl.qt == 1 && pl.pair == 1 && !pl.dual ? std::min(kBlockM, (s.q + 7) / 8 * 8) : kBlockM;
  if (!make_map(&maps.q, Q, s.q, s.d, a_rows) ||
      !make_map(&maps.e, E, s.n, s.d, pl.block_n / pl.pair))
    return cudaErrorInvalidValue;
  const bool hybrid = fu.gathered();
  const int lex = hybrid ? kLexGather : fu.bm25 != nullptr ? kLexBlock : kLexNone;
  if (hybrid != s.fused_lex) return cudaErrorInvalidValue;
  if (hybrid) {
    // head-term counts (q x kLexK) and split weights (n x kLexK): one K block
    if (pl.block_n != 128 || pl.pair != 1 || pl.dual ||
        !make_map(&maps.qb, fu.lex_qcount, s.q, kLexK, a_rows) ||
        !make_map(&maps.eb, fu.lex_wsplit, s.n, kLexK, pl.block_n))
      return cudaErrorInvalidValue;
  } else if (s.n_second > 0) {
    // the second stacked corpus (dense search over two indices)
    if (E2 == nullptr || fu.bm25 != nullptr ||
        !make_map(&maps.eb, E2, s.n_second, s.d, pl.block_n / pl.pair))
      return cudaErrorInvalidValue;
    maps.qb = maps.q;
  } else {
    maps.qb = maps.q;
    maps.eb = maps.e;
  }
  const int K = list_len_for(s.k);
  const int stride = K > 32 ? 2 * K : K;
  const size_t rows = list_rows(pl);
  TcParams prm{};
  prm.n = s.n + s.n_second;
  prm.n_first = s.n;
  prm.nt_first = pl.nt_first;
  prm.d = s.d;
  prm.q = s.q;
  prm.k = s.k;
  prm.qt = pl.uqt;
  prm.nt = pl.nt;
  prm.win = pl.win;
  prm.pmax = pl.pmax;
  prm.kblocks = (s.d + kBlockK - 1) / kBlockK;
  prm.a_bytes = static_cast<uint32_t>(a_rows) * kBlockK * 2;
  prm.tile_stride = pl.tile_stride;
  prm.init_floor = init_floor;
  prm.fu = fu;
  prm.lists = static_cast<uint64_t*>(scratch);
  prm.meta_worst = prm.lists + rows * stride;
  prm.meta_count = reinterpret_cast<int*>(prm.meta_worst + (K > 32 ? rows : 0));
  prm.dev_err = dev_err;
  prm.wait_limit = wait_limit > 0 ? wait_limit : kWaitLimitCycles;
  prm.phases = phases;
  // Register lists publish their k-th scores; buffered lists use counted floors.
  prm.qfloor = K <= 32 ? qfloor : nullptr;
  prm.gen = gen;
  prm.levels = K > 32 ? levels : nullptr;
  prm.level_cnt = K > 32 ? level_cnt : nullptr;
  lists->keys = prm.lists;
  lists->P = pl.pmax;
  lists->TH = kBlockM;
  lists->stride = stride;
  lists->C = pl.grid / pl.pair;
  lists->qt = pl.uqt;
  lists->sets = pl.dual ? 1 : epi_sets(K, hybrid);
  lists->klen = K;
  lists->pair = pl.dual ? 2 : pl.pair;
  if (K > 32) {
    lists->counts = prm.meta_count;
    lists->levels = prm.levels;
    lists->level_cnt = prm.level_cnt;
  }
  if (hybrid) return launch_bn128_gather(maps, prm, pl.grid, st);
  if (pl.dual) {
    if (pl.block_n != 128) return cudaErrorInvalidValue;
    return launch_dual128(maps, prm, pl.grid, lex, st);
  }
  if (pl.pair == 2) {
    if (pl.block_n != 256) return cudaErrorInvalidValue;
    return lex == kLexBlock ? launch_pair256_block(maps, prm, pl.grid, st)
                            : launch_pair256_dense(maps, prm, pl.grid, st);
  }
  if (pl.block_n == 128) return launch_bn128(maps, prm, pl.grid, lex, st);
  return lex == kLexBlock ? launch_bn256_block(maps, prm, pl.grid, st)
                          : launch_bn256_dense(maps, prm, pl.grid, st);
}

}  // namespace oprag
