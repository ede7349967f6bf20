// Tensor-core search for bf16 indices on sm_103a: the query x chunk score
// contraction of Sec. 4.4 (dense scores of a query against the whole
// embedding matrix in one matrix operation) as a tcgen05 GEMM, with the partial top-k
// selection (Sec. 4.4, Sec. 7) fused into the epilogue so that the q x n
// score matrix never reaches HBM.
//
// Work decomposition.  Queries are cut into tiles of 128 (the MMA M side, one
// query per TMEM lane) and the corpus into tiles of BN rows (the MMA N side).
// A unit is (query tile j, corpus tile t).  The corpus tiles are grouped into
// windows that stay in L2; inside a window the units are ordered j-major and
// cut into one contiguous share per CTA of the persistent grid (UnitSeq), so
// all CTAs read inside the same window at the same time while each CTA meets
// only one or two query tiles.  A CTA keeps one running top-K list per query
// of each tile it meets and leaves it as one partial list of that tile for
// the merge kernel (list slot = CTA offset from the first CTA of the tile).
//
// Roles (320 threads with two epilogue sets, 192 with one):
//   warp 0, lane 0: TMA producer.  Per K block of 64 bf16 (one 128-byte
//                   swizzle row) it loads the 128 x 64 query tile and the
//                   BN x 64 corpus tile into a pipeline stage.
//   warp 1        : allocates 2 x BN TMEM columns (two fp32 accumulators);
//                   lane 0 issues tcgen05.mma (M = 128, N = BN, K = 16).
//   warps 2..     : epilogue, one or two sets of four warps; with two sets,
//                   set s drains accumulator s.  Each thread owns one query
//                   (one TMEM lane), reads its BN scores with tcgen05.ld and
//                   filters them against a lower bound of that query's k-th
//                   best score (its own list, the unit, and the bounds that
//                   the other lists publish).
// The two accumulators let the MMAs of one unit overlap the filtering of the
// previous one(s).  Every mbarrier wait is bounded (see common.cuh).
#pragma once
#include <cuda.h>

#include "common.cuh"
#include "internal.h"

namespace oprag {
namespace tc {

constexpr int kBlockM = 128;
constexpr int kBlockK = 64;                 // bf16 per 128-byte row
constexpr int kUmmaK = 16;
// Epilogue warp sets: two (one per accumulator, 320 threads) for register
// lists up to 16 keys and for buffered lists; one set (192 threads) for lists
// of 32.  Ten warps put three on two of the SM's four schedulers, which caps
// a thread at 168 registers; with six warps it may use 255.  Buffered lists
// fit the cap because their epilogue waits for each TMEM load before
// filtering (no registers in flight across the filter); with two sets each
// set has two units' time per unit.  Measured on GB300, 1M x 768 with 2048
// queries and k = 100: main pass 2026 instead of 2060 us.
// The gathered hybrid search keeps one set (its postings cursors advance
// through consecutive units).
__host__ __device__ constexpr int epi_sets(int K, bool lex = false) {
  return (K <= 16 || K > 32) && !lex ? 2 : 1;
}
__host__ __device__ constexpr int threads_for(int K, bool lex = false) {
  return 64 + 128 * epi_sets(K, lex);
}
constexpr uint32_t kAStageBytes = kBlockM * kBlockK * 2;
constexpr int kSmemBudget = 200 * 1024;

struct TcParams {
  int64_t n;            // corpus rows (of both corpora when two are stacked)
  int64_t n_first;      // rows of the first corpus (n for one corpus)
  int nt_first;         // corpus tiles of the first corpus (nt-unstrided; all for one)
  int d;
  int q;
  int k;
  int qt;               // query tiles of 128
  int nt;               // corpus tiles of BN rows
  int win;              // corpus tiles per L2 window
  int pmax;             // lists per query tile (CTAs that may touch it x kEpiSets)
  int kblocks;
  uint32_t a_bytes;     // bytes of one query K block actually loaded (rows x 128)
  int tile_stride;      // scanned corpus tile i is tile i * tile_stride
  const float* init_floor;  // optional per-query lower bound of the k-th best score
  Fusion fu;
  uint64_t* lists;      // [(j * pmax + producer) * 128 + row] * stride
  int* meta_count;      // buffered lists: kept keys per (list, row)
  uint64_t* meta_worst; // buffered lists: K-th key per (list, row)
  int* dev_err;
  // Cycles a wait on an mbarrier may spin before the kernel gives up
  // (kWaitLimitCycles unless a test shortens it).
  long long wait_limit;
  // Optional (register lists only): per query, a lower bound of its k-th best
  // score shared by every list of the search, tagged with `gen` (entries of
  // other searches read as -inf); see shared_floor_read.
  uint64_t* qfloor;
  uint32_t gen;
  // Optional (buffered lists): per query, kLevels candidate floors (best
  // first, non-increasing) and one counter per band: counter i counts pushed
  // keys whose best reached floor is floor i.  Counters 0..i summed count the
  // pushed keys >= floor i; once that sum reaches k, floor i bounds the
  // query's k-th best score for every list.
  const float* levels;
  int* level_cnt;
  // Optional (measurement): kPhases global-timer stamps per CTA (PhaseMark).
  unsigned long long* phases;
};

// Points of a CTA's run whose global-timer values a measurement run records
// (TcParams::phases, slot blockIdx.x * kPhases + mark).
enum PhaseMark : int {
  kPhEntry = 0,        // first instruction
  kPhSetup = 1,        // barriers initialised, TMEM allocated (after the setup barrier)
  kPhFirstStage = 2,   // MMA issuer: first pipeline stage landed
  kPhLastStage = 3,    // MMA issuer: last pipeline stage landed
  kPhLastCommit = 4,   // MMA issuer: last unit's MMAs issued and committed
  kPhEpi0Done = 5,     // epilogue set 0: last unit filtered
  kPhEpi1Done = 6,     // epilogue set 1 (two sets): last unit filtered
  kPhExit = 7,         // after the final barrier, before TMEM is freed
  kPhases = 8
};

__device__ __forceinline__ unsigned long long global_timer() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ void note_phase(const TcParams& p, int mark) {
  if (p.phases != nullptr) p.phases[static_cast<size_t>(blockIdx.x) * kPhases + mark] = global_timer();
}

// Units of one CTA in processing order.  The corpus tiles are cut into
// windows of `win` tiles (sized to stay in L2); inside a window the units
// (query tile j, corpus tile t) are ordered j-major and split into C equal
// contiguous shares, share c going to CTA c.  So all CTAs sweep the windows
// together (each window is read from HBM once and re-read from L2), while a
// CTA meets only the one or two query tiles its share covers and scans their
// corpus tiles in increasing order.
struct UnitSeq {
  int nt, win, qt, C, cta;
  int w, tw;
  int64_t l, l_end;

  __device__ __forceinline__ void start(const TcParams& p, int cta_, int C_) {
    nt = p.nt;
    win = p.win;
    qt = p.qt;
    stride = p.tile_stride;
    C = C_;
    cta = cta_;
    w = -1;
    next_window();
  }
  __device__ __forceinline__ void next_window() {
    while (true) {
      ++w;
      if (static_cast<int64_t>(w) * win >= nt) {
        l = l_end = 0;
        return;
      }
      tw = min(win, nt - w * win);
      const int64_t uw = static_cast<int64_t>(qt) * tw;
      l = uw * cta / C;
      l_end = uw * (cta + 1) / C;
      if (l < l_end) return;
    }
  }
  __device__ __forceinline__ bool valid() const { return static_cast<int64_t>(w) * win < nt; }
  __device__ __forceinline__ void next() {
    if (++l >= l_end) next_window();
  }
  __device__ __forceinline__ int j() const { return static_cast<int>(l / tw); }
  __device__ __forceinline__ int t() const { return (w * win + static_cast<int>(l % tw)) * stride; }
  int stride;
};

// First CTA whose shares can reach query tile j (the host checks the bound).
__host__ __device__ __forceinline__ int first_cta(int j, int qt, int C) {
  const int c = static_cast<int>(static_cast<int64_t>(j) * C / qt) - 1;
  return c < 0 ? 0 : c;
}

// Corpus rows one CTA loads per stage: BN, or BN / 2 when a CTA pair shares
// the tile (each CTA of the pair loads half of its rows).
template <int BN, bool kPair>
constexpr uint32_t b_stage_bytes() {
  return static_cast<uint32_t>(kPair ? BN / 2 : BN) * 128;
}

// Query rows per stage: one 128-row tile, or two in dual mode.
template <bool kDual>
constexpr uint32_t a_stage_bytes() {
  return kAStageBytes * (kDual ? 2u : 1u);
}

// Per-thread landing zone of the gathered hybrid search's copies: kLexMidReg
// rows of 32 floats, then 2 postings per tail term; the 400-byte stride (100
// words) spreads the lanes over the banks.  One set of 128 threads.
constexpr int kLexLandStride = 400;
__host__ __device__ constexpr int lex_land_bytes(bool lex) {
  return lex ? 128 * kLexLandStride : 0;
}

// kExtra: further shared memory of the launch (the BM25 block form's second
// staging tile per epilogue warp, block_land_bytes).
template <int BN, bool kPair = false, bool kDual = false, bool kLex = false, int kExtra = 0>
constexpr int stages_for() {
  return (kSmemBudget - lex_land_bytes(kLex) - kExtra) /
                     (a_stage_bytes<kDual>() + b_stage_bytes<BN, kPair>()) > 8
             ? 8
             : (kSmemBudget - lex_land_bytes(kLex) - kExtra) /
                   (a_stage_bytes<kDual>() + b_stage_bytes<BN, kPair>());
}

// Per epilogue thread: one 32-float row where a chunk's scores are staged so
// that candidate columns can be read back by index.
constexpr int kStageRowBytes = 32 * 4;

template <int BN, int K, bool kPair = false, bool kDual = false, bool kLex = false, int kExtra = 0>
constexpr size_t smem_for() {
  return static_cast<size_t>(stages_for<BN, kPair, kDual, kLex, kExtra>()) *
             (a_stage_bytes<kDual>() + b_stage_bytes<BN, kPair>()) +
         static_cast<size_t>(epi_sets(K, kLex)) * 128 * kStageRowBytes + lex_land_bytes(kLex) +
         kExtra + 1024 + 256;
}

// ----------------------------------------------------------------- PTX

__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, uint64_t* bar, int x,
                                            int y) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%3, %4}], [%2];" ::"r"(smem_addr(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(smem_addr(bar)), "r"(x), "r"(y)
      : "memory");
}

__device__ __forceinline__ void prefetch_map(const CUtensorMap* map) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(map)) : "memory");
}

__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}

__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

__device__ __forceinline__ void tmem_alloc(uint32_t* slot, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                   smem_addr(slot)),
               "r"(ncols)
               : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
               : "memory");
}

// Shared-memory matrix descriptor: K-major operand in the 128-byte swizzle
// layout written by TMA (8-row groups 1024 bytes apart).
__device__ __forceinline__ uint64_t sw128_desc(uint32_t saddr) {
  uint64_t desc = 0;
  desc |= static_cast<uint64_t>((saddr & 0x3FFFFu) >> 4);   // start address
  desc |= static_cast<uint64_t>(1) << 16;                    // leading byte offset (unused)
  desc |= static_cast<uint64_t>(1024 >> 4) << 32;            // stride byte offset
  desc |= static_cast<uint64_t>(1) << 46;                    // descriptor version
  desc |= static_cast<uint64_t>(2) << 61;                    // 128-byte swizzle
  return desc;
}

// Instruction descriptor, kind::f16: bf16 A and B (both K-major), fp32 D.
__host__ __device__ constexpr uint32_t idesc_bf16(int m, int n) {
  return (1u << 4) | (1u << 7) | (1u << 10) | (static_cast<uint32_t>(n >> 3) << 17) |
         (static_cast<uint32_t>(m >> 4) << 24);
}

__device__ __forceinline__ void mma_bf16(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t idesc,
                                         uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(a), "l"(b), "r"(idesc), "r"(accumulate)
      : "memory");
}

__device__ __forceinline__ void mma_commit(uint64_t* bar) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
          smem_addr(bar))
      : "memory");
}

// ----------------------------------------------------------- CTA pairs
// A cluster of two CTAs can issue one MMA with M = 256 (cta_group::2): each
// CTA holds 128 rows of A and half of the N rows of B in its own shared
// memory at the same offsets, and each CTA's TMEM receives the 128 x N
// accumulator of its own A rows.  Rank 0 of the pair issues the MMAs.  A
// kernel uses one cta_group for all of its tcgen05 instructions.

__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}

__device__ __forceinline__ uint32_t cluster_index() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%clusterid.x;" : "=r"(r));
  return r;
}

// Every thread of both CTAs; orders shared-memory writes before the barrier
// with reads after it across the cluster.
__device__ __forceinline__ void cluster_sync() {
  asm volatile("barrier.cluster.arrive.release;\n\tbarrier.cluster.wait.acquire;" ::: "memory");
}

// Address of the same shared-memory variable in the CTA of cluster rank `rank`.
__device__ __forceinline__ uint32_t cluster_addr(const void* p, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(smem_addr(p)), "r"(rank));
  return r;
}

__device__ __forceinline__ void mbar_arrive_cluster(uint32_t caddr) {
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(caddr)
               : "memory");
}

// TMA load into this CTA's shared memory whose completion is counted on an
// mbarrier of either CTA of the pair (cluster address).
__device__ __forceinline__ void tma_load_2d_pair(void* dst, const CUtensorMap* map, uint32_t bar_caddr,
                                                 int x, int y) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes.cta_group::2"
      " [%0], [%1, {%3, %4}], [%2];" ::"r"(smem_addr(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(bar_caddr), "r"(x), "r"(y)
      : "memory");
}

__device__ __forceinline__ void tmem_alloc_pair(uint32_t* slot, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                   smem_addr(slot)),
               "r"(ncols)
               : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void tmem_dealloc_pair(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
               : "memory");
}

__device__ __forceinline__ void mma_bf16_pair(uint32_t d_tmem, uint64_t a, uint64_t b,
                                              uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(a), "l"(b), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Arrives once on the mbarrier at this offset in every CTA of `mask` when the
// pair's MMAs issued so far have completed.
__device__ __forceinline__ void mma_commit_pair_mc(uint64_t* bar, uint16_t mask) {
  asm volatile(
      "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64"
      " [%0], %1;" ::"r"(smem_addr(bar)),
      "h"(mask)
      : "memory");
}

__device__ __forceinline__ void mma_commit_pair(uint64_t* bar) {
  asm volatile(
      "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
          smem_addr(bar))
      : "memory");
}

// Issues a 32-column TMEM load (32 lanes x 32 columns of 32 bits); the
// registers are valid only after tmem_wait_ld() on the same array.
__device__ __forceinline__ void tmem_ld32_async(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
      "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]),
        "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]),
        "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
}

// Waits for the outstanding TMEM loads.  The registers are passed through the
// asm so that no use of them can be scheduled before the wait.
__device__ __forceinline__ void tmem_wait_ld(uint32_t (&r)[32]) {
  asm volatile("tcgen05.wait::ld.sync.aligned;"
               : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]), "+r"(r[4]), "+r"(r[5]),
                 "+r"(r[6]), "+r"(r[7]), "+r"(r[8]), "+r"(r[9]), "+r"(r[10]), "+r"(r[11]),
                 "+r"(r[12]), "+r"(r[13]), "+r"(r[14]), "+r"(r[15]), "+r"(r[16]), "+r"(r[17]),
                 "+r"(r[18]), "+r"(r[19]), "+r"(r[20]), "+r"(r[21]), "+r"(r[22]), "+r"(r[23]),
                 "+r"(r[24]), "+r"(r[25]), "+r"(r[26]), "+r"(r[27]), "+r"(r[28]), "+r"(r[29]),
                 "+r"(r[30]), "+r"(r[31])
               :
               : "memory");
}

// ------------------------------------------------------- shared k-th floors
// Every list that holds k scores >= f proves that the query's k-th best score
// is >= f, so any list may drop scores below f.  Lists publish such bounds per
// query with a 64-bit atomic max of (gen << 32 | order-preserving bits of f)
// and read the current value before each unit; an entry of another search
// (other gen) reads as -inf, so the array never needs clearing.
__device__ __forceinline__ uint32_t ordered_bits(float f) {
  const uint32_t b = __float_as_uint(f);
  return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}

__device__ __forceinline__ float from_ordered_bits(uint32_t o) {
  return __uint_as_float((o & 0x80000000u) ? (o & 0x7FFFFFFFu) : ~o);
}

__device__ __forceinline__ float shared_floor_read(const uint64_t* qf, int64_t qi, uint32_t gen) {
  const unsigned long long v = __ldcg(reinterpret_cast<const unsigned long long*>(qf + qi));
  return static_cast<uint32_t>(v >> 32) == gen ? from_ordered_bits(static_cast<uint32_t>(v))
                                               : -INFINITY;
}

__device__ __forceinline__ void shared_floor_raise(uint64_t* qf, int64_t qi, uint32_t gen, float f) {
  atomicMax(reinterpret_cast<unsigned long long*>(qf + qi),
            (static_cast<unsigned long long>(gen) << 32) | ordered_bits(f));
}

// Sorts N (a power of two) values descending in registers (bitonic network;
// 240 exchanges for N = 32); the stages are template instances so that every
// index is a constant.
template <int N, int KS, int JS>
__device__ __forceinline__ void bitonic_stage(float (&a)[N]) {
#pragma unroll
  for (int i = 0; i < N; ++i) {
    const int l = i ^ JS;
    if (l > i) {
      const float hi = fmaxf(a[i], a[l]), lo = fminf(a[i], a[l]);
      const bool desc = (i & KS) == 0;
      a[i] = desc ? hi : lo;
      a[l] = desc ? lo : hi;
    }
  }
  if constexpr (JS > 1) bitonic_stage<N, KS, JS / 2>(a);
}

template <int N, int KS = 2>
__device__ __forceinline__ void bitonic_desc(float (&a)[N]) {
  static_assert(N >= 2 && (N & (N - 1)) == 0, "power of two");
  bitonic_stage<N, KS, KS / 2>(a);
  if constexpr (KS < N) bitonic_desc<N, KS * 2>(a);
}

// Three-input maximum (one instruction on sm_100 and later).
__device__ __forceinline__ float fmax3(float a, float b, float c) {
  float r;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
  return r;
}

// max of 32 values: 16 three- and two-input maxima (the epilogue's filter runs
// this once per 32 scores, so its instruction count bounds the epilogue).
__device__ __forceinline__ float max32(const float (&v)[32]) {
  float a[12];
#pragma unroll
  for (int i = 0; i < 10; ++i) a[i] = fmax3(v[3 * i], v[3 * i + 1], v[3 * i + 2]);
  a[10] = v[30];
  a[11] = v[31];
  const float b0 = fmax3(a[0], a[1], a[2]), b1 = fmax3(a[3], a[4], a[5]);
  const float b2 = fmax3(a[6], a[7], a[8]), b3 = fmax3(a[9], a[10], a[11]);
  return fmaxf(fmax3(b0, b1, b2), b3);
}

// Waits without looking at the abort word (used to drain in-flight copies and
// MMAs before the CTA exits); still bounded.
__device__ __forceinline__ bool mbar_drain(uint64_t* bar, uint32_t parity, int* dev_err) {
  const long long t0 = clock64();
  while (!mbar_test(bar, parity)) {
    if (clock64() - t0 > kWaitLimitCycles) {
      atomicExch(dev_err, static_cast<int>(kDevErrWaitTimeout));
      return false;
    }
  }
  return true;
}

// ----------------------------------------------------------------- lists

template <int K, bool kBuf = (K > 32)>
struct EpiList;

template <int K>
struct EpiList<K, false> {
  static constexpr int kStride = K;
  // Only the best kk = min(k, K) keys of a list can reach the query's top-k
  // (the merges read no more).  The list keeps them in its last kk slots,
  // under pad = K - kk sentinel slots of +inf that no score passes, so the
  // insertion network is unchanged and the floor (the last slot) is the
  // kk-th best score.  Stored lists hold their kk keys first.
  RegTopK<K> t;
  int pad = 0;
  __device__ __forceinline__ void set_k(int k) { pad = k < K ? K - k : 0; }
  __device__ __forceinline__ void init_mem(const TcParams& p, int64_t sr, int) {
#pragma unroll
    for (int i = 0; i < K; i += 2)
      *reinterpret_cast<ulonglong2*>(p.lists + sr * K + i) = make_ulonglong2(0ull, 0ull);
  }
  __device__ __forceinline__ void pad_top() {
#pragma unroll
    for (int i = 0; i + 1 < K; ++i)
      if (i < pad) t.s[i] = INFINITY;
  }
  // Stored order -> slots: shift right by pad (a barrel shifter, so that
  // every register index is a constant).
  __device__ __forceinline__ void load(const TcParams& p, int64_t sr) {
    t.load(p.lists + sr * K);
#pragma unroll
    for (int w = K / 2; w >= 1; w /= 2) {
      const bool on = (pad & w) != 0;
#pragma unroll
      for (int j = K - 1; j >= 0; --j) {
        t.s[j] = on ? (j >= w ? t.s[j - w] : INFINITY) : t.s[j];
        t.id[j] = on ? (j >= w ? t.id[j - w] : kNoId) : t.id[j];
      }
    }
    t.floor = t.s[K - 1];
  }
  // Slots -> stored order: shift left by pad, empty keys behind.
  __device__ __forceinline__ void save(const TcParams& p, int64_t sr) {
    RegTopK<K> o = t;
#pragma unroll
    for (int w = 1; w <= K / 2; w *= 2) {
      const bool on = (pad & w) != 0;
#pragma unroll
      for (int j = 0; j < K; ++j) {
        o.s[j] = on ? (j + w < K ? o.s[j + w] : -INFINITY) : o.s[j];
        o.id[j] = on ? (j + w < K ? o.id[j + w] : kNoId) : o.id[j];
      }
    }
    o.store(p.lists + sr * K);
  }
  __device__ __forceinline__ void clear() {
    t.init();
    pad_top();
  }
  __device__ __forceinline__ bool full() const { return t.full(); }
  __device__ __forceinline__ float floor() const { return t.floor; }
  __device__ __forceinline__ void push(float s, uint32_t id) { t.push(s, id); }
  __device__ __forceinline__ void insert(float s, uint32_t id) { t.insert(s, id); }
  // The k-th best score held, for the k the list was set up with.
  __device__ __forceinline__ float kth(int) const { return t.floor; }
  __device__ __forceinline__ void sync(bool, bool) {}
  __device__ __forceinline__ void read_ahead() {}
};

template <int K>
struct EpiList<K, true> {
  static constexpr int kStride = 2 * K;
  BufTopK<K> t;
  // Counted floors of the current query (see TcParams::levels).
  float lvl[kLevels];
  int* cnt;
  // Their counts as read one unit earlier.  Counts only grow, so an older
  // reading still proves its floors, and reading ahead keeps the L2 latency
  // off the epilogue's path (it runs once per unit).
  int4 seen;
  __device__ __forceinline__ void set_query(const TcParams& p, int64_t q_index, bool valid) {
    cnt = valid && p.levels != nullptr ? p.level_cnt + q_index * kLevels : nullptr;
#pragma unroll
    for (int i = 0; i < kLevels; ++i) lvl[i] = cnt != nullptr ? p.levels[q_index * kLevels + i] : INFINITY;
    seen = cnt != nullptr ? __ldcg(reinterpret_cast<const int4*>(cnt)) : make_int4(0, 0, 0, 0);
    proven = kLevels;
  }
  // Reads the counts for the next unit of the same query.
  __device__ __forceinline__ void read_ahead() {
    if (cnt != nullptr) seen = __ldcg(reinterpret_cast<const int4*>(cnt));
  }
  // Index of the best floor proven by the last reading (kLevels: none).
  int proven;
  // The best counted floor that k pushed keys reached by the last reading
  // (-inf if none); also sets `proven`.
  __device__ __forceinline__ float proven_floor(int k) {
    proven = kLevels;
    if (cnt == nullptr) return -INFINITY;
    const int4 c = seen;
    const int cs[kLevels] = {c.x, c.y, c.z, c.w};
    float f = -INFINITY;
    int sum = 0;
#pragma unroll
    for (int i = 0; i < kLevels; ++i) {
      sum += cs[i];
      if (sum >= k && proven == kLevels) {
        proven = i;
        f = lvl[i];
      }
    }
    return f;
  }
  __device__ __forceinline__ void init_mem(const TcParams& p, int64_t sr, int qidx) {
    p.meta_count[sr] = 0;
    // A known lower bound f of the k-th best score admits only scores >= f
    // (the key with the largest possible id ranks below every such score).
    const float f = p.init_floor != nullptr ? p.init_floor[qidx] : -INFINITY;
    p.meta_worst[sr] = f > -INFINITY ? make_key(f, kNoId) : kEmptyKey;
  }
  __device__ __forceinline__ void load(const TcParams& p, int64_t sr) {
    t.buf = p.lists + sr * kStride;
    t.count = p.meta_count[sr];
    t.worst = p.meta_worst[sr];
    t.floor = key_floor(t.worst);
  }
  __device__ __forceinline__ void save(const TcParams& p, int64_t sr) {
    p.meta_count[sr] = t.count;
    p.meta_worst[sr] = t.worst;
  }
  __device__ __forceinline__ void set_k(int) {}
  __device__ __forceinline__ void clear() {
    t.buf = nullptr;
    t.count = 0;
    t.worst = kEmptyKey;
    t.floor = -INFINITY;
    cnt = nullptr;
    proven = kLevels;
  }
  __device__ __forceinline__ bool full() const { return t.worst != kEmptyKey; }
  __device__ __forceinline__ float floor() const { return t.floor; }
  __device__ __forceinline__ void push(float s, uint32_t id) { t.push(s, id); }
  // Pushes a candidate; a pushed key counts once, in the band of the best
  // floor it reaches (a fire-and-forget add).  Sums of k counts prove k real
  // keys >= a floor, which then bounds the query's k-th best for every list;
  // a pushed key leaves its list only when the list holds K >= k better
  // keys, so the proof stays valid.  A key whose band is at or below the
  // best proven floor (`proven`) can prove nothing new and is not counted
  // (counts stay lower bounds).
  __device__ __forceinline__ void insert(float s, uint32_t id) {
    if (!(s > -INFINITY)) return;
    const uint64_t key = make_key(s, id);
    if (key <= t.worst) return;
    t.buf[t.count++] = key;
    if (cnt != nullptr) {
      int band = kLevels;
#pragma unroll
      for (int i = kLevels - 1; i >= 0; --i)
        if (s >= lvl[i]) band = i;
      if (band < proven) atomicAdd(cnt + band, 1);
    }
  }
  __device__ __forceinline__ void sync(bool final, bool active) { t.sync(final, active); }
  // No final sort: a list ends as its count and that many keys in no order
  // (they include its best K), and the merge reads it so.  Sorting 32 lanes'
  // buffers one after another at the end of the kernel, where nothing
  // overlaps it, cost more than the merge's extra reads.
};

// ----------------------------------------------------------- lexical gather
// The mid and tail terms of one thread's query in the gathered hybrid search
// (Sec. 4.4, inverted-postings BM25; see Fusion).  Per chunk of 32 corpus
// rows the thread copies, with cp.async into its landing zone in shared
// memory (no registers held while the copies fly), the chunk's 32 weights of
// each listed mid row and the next two postings of each listed tail term.
// A tail term's cursor (chunk ids ascending) is kept across the chunks and
// units that the thread filters in increasing chunk order, so each posting
// is read once; it is re-placed by binary search when the thread's query
// changes or its units are not consecutive.  Tail terms have under one
// posting per 32 chunks on average; a longer run falls back to dependent
// loads.  Terms past the listed ones (long queries) are searched per chunk.

static_assert(kLexMidReg * 128 + kLexRegTerms * 16 <= kLexLandStride, "landing zone");

__device__ __forceinline__ void cp_async16(void* dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_addr(dst)), "l"(src)
               : "memory");
}

__device__ __forceinline__ void cp_async8(void* dst, const void* src) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 8;" ::"r"(smem_addr(dst)), "l"(src)
               : "memory");
}

// 16 bytes, or 16 zero bytes when !in (nothing is read from src then).
__device__ __forceinline__ void cp_async16_zfill(void* dst, const void* src, bool in) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(smem_addr(dst)), "l"(src),
               "r"(in ? 16 : 0)
               : "memory");
}

__device__ __forceinline__ void cp_async_commit() {
  asm volatile("cp.async.commit_group;" ::: "memory");
}

__device__ __forceinline__ void cp_async_wait_all() {
  asm volatile("cp.async.wait_group 0;" ::: "memory");
}

__device__ __forceinline__ void cp_async_commit_wait_all() {
  asm volatile("cp.async.commit_group;\n\tcp.async.wait_group 0;" ::: "memory");
}

struct LexCursor {
  int base[kLexRegTerms], cur[kLexRegTerms], end[kLexRegTerms], term[kLexRegTerms];
  float mul[kLexRegTerms];
  int mrow[kLexMidReg];
  float mmul[kLexMidReg];
  int nreg = 0, nmid = 0;      // listed tail terms and mid rows
  int ovf = 0, ovf_end = 0;    // raw term range scanned for further terms
  int64_t next_doc = -1;       // first chunk that continues the cursors (-1: none)

  __device__ __forceinline__ void set_query(const TcParams& p, int64_t qi) {
    nreg = p.fu.lex_term_cnt[qi];
    nmid = p.fu.lex_mid_cnt[qi];
    ovf = p.fu.lex_ovf[qi];
    ovf_end = p.fu.q_indptr[qi + 1];
#pragma unroll
    for (int i = 0; i < kLexRegTerms; ++i) {
      const int4 e = i < nreg ? p.fu.lex_terms[qi * kLexRegTerms + i] : make_int4(0, 0, 0, -1);
      base[i] = cur[i] = e.x;
      end[i] = e.y;
      mul[i] = __int_as_float(e.z);
      term[i] = e.w;
    }
#pragma unroll
    for (int m = 0; m < kLexMidReg; ++m) {
      const int2 e = m < nmid ? p.fu.lex_mid[qi * kLexMidReg + m] : make_int2(-1, 0);
      mrow[m] = e.x;
      mmul[m] = __int_as_float(e.y);
    }
    next_doc = -1;
  }

  // Places every tail cursor on the term's first posting with chunk >= d
  // (interleaved binary searches: one load per term and step in flight).
  __device__ __forceinline__ void seek(const int2* post, int64_t d) {
    int lo[kLexRegTerms], hi[kLexRegTerms];
#pragma unroll
    for (int i = 0; i < kLexRegTerms; ++i) {
      lo[i] = i < nreg ? base[i] : 0;
      hi[i] = i < nreg ? end[i] : 0;
    }
    bool more = true;
    while (more) {
      int x[kLexRegTerms];
#pragma unroll
      for (int i = 0; i < kLexRegTerms; ++i)
        x[i] = lo[i] < hi[i] ? __ldg(&post[(lo[i] + hi[i]) >> 1].x) : 0;
      more = false;
#pragma unroll
      for (int i = 0; i < kLexRegTerms; ++i) {
        if (lo[i] < hi[i]) {
          const int mid = (lo[i] + hi[i]) >> 1;
          if (x[i] < d) lo[i] = mid + 1; else hi[i] = mid;
          more |= lo[i] < hi[i];
        }
      }
    }
#pragma unroll
    for (int i = 0; i < kLexRegTerms; ++i) cur[i] = lo[i];
  }

  // Copies the chunk's mid-row weights and the tail terms' next postings
  // (chunks id0 .. id0 + 31) into the landing zone and waits for them.
  __device__ __forceinline__ void fetch(const TcParams& p, int64_t id0, unsigned char* land) {
    float* lm = reinterpret_cast<float*>(land);
    int2* lt = reinterpret_cast<int2*>(land + kLexMidReg * 128);
#pragma unroll
    for (int m = 0; m < kLexMidReg; ++m) {
      if (m < nmid) {
        const float* src = p.fu.mid_w + static_cast<int64_t>(mrow[m]) * p.fu.mid_ld + id0;
#pragma unroll
        for (int g = 0; g < 8; ++g) cp_async16(lm + m * 32 + 4 * g, src + 4 * g);
      }
    }
    const int2* post = p.fu.lex_post;
#pragma unroll
    for (int i = 0; i < kLexRegTerms; ++i) {
#pragma unroll
      for (int u = 0; u < 2; ++u) {
        if (i < nreg && cur[i] + u < end[i]) cp_async8(lt + 2 * i + u, post + cur[i] + u);
        else lt[2 * i + u] = make_int2(0x7FFFFFFF, 0);
      }
    }
    cp_async_commit_wait_all();
  }

  // The chunk's mid-row part of element i (landing zone filled by fetch).
  __device__ __forceinline__ float4 mid4(const unsigned char* land, int g) const {
    const float* lm = reinterpret_cast<const float*>(land);
    float4 r = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
    for (int m = 0; m < kLexMidReg; ++m) {
      if (m < nmid) {
        const float4 x = *reinterpret_cast<const float4*>(lm + m * 32 + 4 * g);
        r.x = fmaf(mmul[m], x.x, r.x);
        r.y = fmaf(mmul[m], x.y, r.y);
        r.z = fmaf(mmul[m], x.z, r.z);
        r.w = fmaf(mmul[m], x.w, r.w);
      }
    }
    return r;
  }

  // Adds the chunk's tail-term (and long-query) BM25 into the thread's
  // staging row (float4 groups XOR-swizzled by swz), which holds zeros on
  // entry, and advances the tail cursors past the chunk.
  __device__ __forceinline__ void tail(const TcParams& p, int64_t id0, const unsigned char* land,
                                       float* srow, int swz) {
    const int2* post = p.fu.lex_post;
    const int2* lt = reinterpret_cast<const int2*>(land + kLexMidReg * 128);
    const int64_t lim = id0 + 32;
    auto add = [&](int2 e, float m) {
      const int i = static_cast<int>(e.x - id0);
      srow[((((i & 31) >> 2) ^ swz) << 2) | (i & 3)] += m * __int_as_float(e.y);
    };
#pragma unroll
    for (int i = 0; i < kLexRegTerms; ++i) {
      const int2 e0 = lt[2 * i], e1 = lt[2 * i + 1];
      if (e0.x < lim) {
        add(e0, mul[i]);
        int c = cur[i] + 1;
        if (e1.x < lim) {
          add(e1, mul[i]);
          ++c;
          while (c < end[i]) {
            const int2 e = __ldg(post + c);
            if (e.x >= lim) break;
            add(e, mul[i]);
            ++c;
          }
        }
        cur[i] = c;
      }
    }
    // Further terms of a long query (each occurrence once): mid rows read
    // directly, tail terms by a binary search per chunk.
    for (int j = ovf; j < ovf_end; ++j) {
      const int32_t tm = p.fu.q_terms[j];
      if (tm < 0 || tm >= p.fu.vocab) continue;
      const int cls = p.fu.lex_class[tm];
      if (cls >= 0) continue;
      if (cls <= -2) {
        bool listed = false;
#pragma unroll
        for (int m = 0; m < kLexMidReg; ++m) listed |= m < nmid && mrow[m] == -2 - cls;
        if (listed) continue;
        const float* row = p.fu.mid_w + static_cast<int64_t>(-2 - cls) * p.fu.mid_ld + id0;
        for (int i = 0; i < 32; ++i) srow[(((i >> 2) ^ swz) << 2) | (i & 3)] += __ldg(row + i);
        continue;
      }
      bool listed = false;
#pragma unroll
      for (int i = 0; i < kLexRegTerms; ++i) listed |= term[i] == tm;
      if (listed) continue;
      int lo = static_cast<int>(p.fu.post_ptr[tm]);
      const int stop = static_cast<int>(p.fu.post_ptr[tm + 1]);
      int hi = stop;
      while (lo < hi) {
        const int mid = (lo + hi) >> 1;
        if (__ldg(&post[mid].x) < id0) lo = mid + 1; else hi = mid;
      }
      for (; lo < stop; ++lo) {
        const int2 e = __ldg(post + lo);
        if (e.x >= lim) break;
        add(e, 1.f);
      }
    }
  }
};

// ----------------------------------------------------------------- kernel

// kPair: the grid is made of clusters of two CTAs that share every unit: a
// unit covers query tiles 2J and 2J + 1 (one per CTA) and corpus tile t of BN
// rows (BN / 2 loaded by each CTA); rank 0 issues M = 256 MMAs for both.  Per
// MMA each CTA then reads 128 x 16 + BN / 2 x 16 operand elements instead of
// 128 x 16 + BN x 16.  The unit sequence (UnitSeq) runs over pairs: p.qt
// counts pairs of query tiles and the pair index plays the CTA index.
//
// kDual (BN = 128): every unit covers query tiles 2J and 2J + 1 and corpus
// tile t; a stage holds both query tiles' K-block and the corpus tile's, and
// the MMA warp issues two MMAs per K-step that share the corpus operand, one
// into each accumulator of the unit's buffer (four accumulators of BN
// columns: buffer u & 1, query tile s at column (2 (u & 1) + s) BN).
// Epilogue set s filters query tile 2J + s, so one unit's epilogue overlaps
// the next unit's copies and MMAs.  Per unit the CTA reads the corpus tile
// once for 256 queries.
//
// kLex: the lexical part of the hybrid search (Sec. 4.4 fusion).
// kLexNone: dense scores.  kLexBlock: the epilogue reads BM25(q, d) from the
// q x ld block that the BM25 pass materialised.  kLexGather (single CTAs,
// BN = 128, one epilogue set): the gathered hybrid
// search.  After the unit's score K blocks the producer loads one more stage,
// the query tile's head-term counts (map_qb) and the corpus tile's split
// head-term weights (map_eb), and the MMA issuer accumulates their product
// into a second accumulator (the head terms' BM25, columns 2 BN + acc BN);
// the epilogue adds the other terms from the postings (LexCursor) and fuses.
constexpr int kLexNone = 0, kLexBlock = 1, kLexGather = 2;

// The BM25 block form's second staging tile: 32 x 32 floats per epilogue
// warp, so that the next chunk's copy of the block flies while one chunk is
// filtered.
template <int K, int L>
constexpr int block_land_bytes() {
  return L == kLexBlock ? epi_sets(K) * 128 * kStageRowBytes : 0;
}

template <int BN, int K, int kLex, bool kPair = false, bool kDual = false>
__global__ void __launch_bounds__(threads_for(K, kLex == kLexGather), 1)
tc_search_kernel(const __grid_constant__ CUtensorMap map_q, const __grid_constant__ CUtensorMap map_e,
                 const __grid_constant__ CUtensorMap map_qb,
                 const __grid_constant__ CUtensorMap map_eb, const TcParams p) {
  static_assert(!(kPair && kDual), "pair and dual modes are exclusive");
  static_assert(!kDual || epi_sets(K) == 2, "dual mode needs one epilogue set per query tile");
  static_assert(!kDual || BN == 128, "dual mode double-buffers four accumulators of 128 columns");
  constexpr bool kHybrid = kLex == kLexGather;   // the gathered form
  static_assert(!kHybrid || (!kPair && !kDual && BN == 128),
                "the gathered hybrid search runs single CTAs on 128-row tiles");
  constexpr int kLand = block_land_bytes<K, kLex>();
  constexpr int S = stages_for<BN, kPair, kDual, kHybrid, kLand>();
  constexpr uint32_t kAStage = a_stage_bytes<kDual>();
  constexpr uint32_t kBStageBytes = b_stage_bytes<BN, kPair>();
  constexpr uint32_t kTmemCols = (kDual ? 4 : 2) * BN * (kHybrid ? 2 : 1);
  constexpr int kEpiSets = epi_sets(K, kHybrid);
  // Stages per unit: the score K blocks, plus the head-term block (hybrid).
  const int unit_kb = p.kblocks + (kHybrid ? 1 : 0);
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  if (threadIdx.x == 0) note_phase(p, kPhEntry);
  unsigned char* base = reinterpret_cast<unsigned char*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  unsigned char* sA = base;
  unsigned char* sB = sA + S * kAStage;
  float* stage_rows = reinterpret_cast<float*>(sB + S * kBStageBytes);   // epilogue staging
  // hybrid: each epilogue thread's landing zone of the lexical copies
  unsigned char* lex_land = reinterpret_cast<unsigned char*>(stage_rows + kEpiSets * 128 * 32);
  float* block_land = reinterpret_cast<float*>(lex_land + lex_land_bytes(kHybrid));
  uint64_t* full = reinterpret_cast<uint64_t*>(reinterpret_cast<unsigned char*>(block_land) + kLand);
  uint64_t* empty = full + S;
  uint64_t* tfull = empty + S;
  uint64_t* tempty = tfull + 4;
  uint64_t* mma_done = tempty + 4;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(mma_done + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // Pair mode: rank 0 of each cluster is the leader (issues the MMAs, owns
  // the full / tempty / mma_done barriers that count both CTAs).
  const uint32_t rank = kPair ? cluster_rank() : 0u;
  const bool leader = rank == 0;
  const int cta = kPair ? static_cast<int>(cluster_index()) : static_cast<int>(blockIdx.x);
  const int C = kPair ? static_cast<int>(gridDim.x) / 2 : static_cast<int>(gridDim.x);
  // Bytes one stage brings into the leader's full barrier (both CTAs in pair mode).
  const uint32_t stage_tx = (p.a_bytes * (kDual ? 2u : 1u) + kBStageBytes) * (kPair ? 2u : 1u);
  // Row coordinates of this CTA's part of unit (J, t).
  auto a_row = [&](int J) {
    return (kPair ? 2 * J + static_cast<int>(rank) : kDual ? 2 * J : J) * kBlockM;
  };
  // Corpus tile t: tiles [0, nt_first) of the first corpus (map_e), then
  // those of the second (map_eb) when two are stacked (dense searches only).
  auto b_row = [&](int t) {
    const int tl = t < p.nt_first ? t : t - p.nt_first;
    return tl * BN + (kPair ? static_cast<int>(rank) * (BN / 2) : 0);
  };
  auto b_map = [&](int t) -> const CUtensorMap* {
    return kLex == kLexNone && t >= p.nt_first ? &map_eb : &map_e;
  };

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 4; ++b) {     // accumulators 2 and 3: dual mode only
      mbar_init(&tfull[b], 1);
      mbar_init(&tempty[b], kPair ? 8 : 4);   // four epilogue warps per CTA
    }
    mbar_init(mma_done, 1);
    *abort_flag = 0;
    fence_mbar_init();
    prefetch_map(&map_q);
    prefetch_map(&map_e);
    if (kHybrid || p.n_first < p.n) {
      prefetch_map(&map_qb);
      prefetch_map(&map_eb);
    }
  }
  // The peer's copies and arrivals target the leader's barriers: both CTAs'
  // barriers are initialised before either CTA issues anything.
  if constexpr (kPair) cluster_sync();
  auto load_stage = [&](int s, int kb, int J, int t) {
    if (kPair) {
      if (leader) mbar_arrive_expect_tx(&full[s], stage_tx);
      const uint32_t bar = cluster_addr(&full[s], 0);                  // the leader's full[s]
      tma_load_2d_pair(sA + s * kAStage, &map_q, bar, kb * kBlockK, a_row(J));
      tma_load_2d_pair(sB + s * kBStageBytes, b_map(t), bar, kb * kBlockK, b_row(t));
    } else if (kHybrid && kb == p.kblocks) {
      // the head-term stage: counts x split weights (one 64-element K block)
      mbar_arrive_expect_tx(&full[s], stage_tx);
      tma_load_2d(sA + s * kAStage, &map_qb, &full[s], 0, a_row(J));
      tma_load_2d(sB + s * kBStageBytes, &map_eb, &full[s], 0, b_row(t));
    } else {
      mbar_arrive_expect_tx(&full[s], stage_tx);
      tma_load_2d(sA + s * kAStage, &map_q, &full[s], kb * kBlockK, a_row(J));
      if constexpr (kDual)
        tma_load_2d(sA + s * kAStage + kAStageBytes, &map_q, &full[s], kb * kBlockK,
                    a_row(J) + kBlockM);
      tma_load_2d(sB + s * kBStageBytes, b_map(t), &full[s], kb * kBlockK, b_row(t));
    }
  };
  int pre_issued = 0;           // stages the producer issued before the setup barrier
  if (threadIdx.x == 0) {
    // The ring is empty: start the first loads while TMEM is being allocated.
    UnitSeq us;
    us.start(p, cta, C);
    for (; us.valid() && pre_issued < S; us.next()) {
      for (int kb = 0; kb < unit_kb && pre_issued < S; ++kb, ++pre_issued)
        load_stage(pre_issued, kb, us.j(), us.t());
      if (pre_issued >= S) break;
    }
  }
  if (warp == 1) {
    if constexpr (kPair) tmem_alloc_pair(tmem_slot, kTmemCols);
    else tmem_alloc(tmem_slot, kTmemCols);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (threadIdx.x == 0) note_phase(p, kPhSetup);
  const uint32_t tmem_base = *tmem_slot;
  // Let the merge kernel that follows on the stream get scheduled; it waits
  // for this grid to finish before reading the lists.
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

  if (warp == 0) {
    if (lane == 0) {
      // ------------------------------------------------ TMA producer
      int s = 0;
      uint32_t ph = 0;
      uint32_t issued = 0, parity = 0;    // per stage: ever issued, parity of last issue
      bool ok = true;
      int skip = pre_issued;              // already issued before the setup barrier
      UnitSeq us;
      for (us.start(p, cta, C); ok && us.valid(); us.next()) {
        const int j = us.j();
        const int t = us.t();
        for (int kb = 0; kb < unit_kb; ++kb) {
          if (skip > 0) {
            --skip;
            issued |= 1u << s;
            parity &= ~(1u << s);
            if (++s == S) { s = 0; ph ^= 1u; }
            continue;
          }
          if (!mbar_wait(&empty[s], ph ^ 1u, abort_flag, p.dev_err, p.wait_limit)) { ok = false; break; }
          load_stage(s, kb, j, t);
          issued |= 1u << s;
          parity = (parity & ~(1u << s)) | (ph << s);
          if (++s == S) { s = 0; ph ^= 1u; }
        }
      }
      // The leader's full barriers also count the peer's copies.
      if (leader)
        for (int i = 0; i < S; ++i)
          if (issued & (1u << i)) mbar_drain(&full[i], (parity >> i) & 1u, p.dev_err);
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0 && leader) {
      // ------------------------------------------------ MMA issuer
      constexpr uint32_t idesc = idesc_bf16(kPair ? 2 * kBlockM : kBlockM, BN);
      int s = 0;
      uint32_t ph = 0;
      int acc = 0;
      uint32_t acc_ph = 0;
      bool ok = true;
      bool landed = false;
      UnitSeq us;
      for (us.start(p, cta, C); ok && us.valid(); us.next()) {
        if constexpr (kDual) {
          // Both accumulators of buffer acc take this unit.
          const int a0i = 2 * acc, a1i = 2 * acc + 1;
          if (!mbar_wait(&tempty[a0i], acc_ph ^ 1u, abort_flag, p.dev_err, p.wait_limit)) break;
          if (!mbar_wait(&tempty[a1i], acc_ph ^ 1u, abort_flag, p.dev_err, p.wait_limit)) break;
          tc_fence_after();
          const uint32_t d0 = tmem_base + static_cast<uint32_t>(a0i * BN);
          const uint32_t d1 = tmem_base + static_cast<uint32_t>(a1i * BN);
          for (int kb = 0; kb < p.kblocks; ++kb) {
            if (!mbar_wait(&full[s], ph, abort_flag, p.dev_err, p.wait_limit)) { ok = false; break; }
            tc_fence_after();
            if (p.phases != nullptr) {
              if (!landed) note_phase(p, kPhFirstStage);
              landed = true;
              note_phase(p, kPhLastStage);
            }
            const uint64_t a0 = sw128_desc(smem_addr(sA + s * kAStage));
            const uint64_t a1 = sw128_desc(smem_addr(sA + s * kAStage + kAStageBytes));
            const uint64_t b = sw128_desc(smem_addr(sB + s * kBStageBytes));
#pragma unroll
            for (int kk = 0; kk < kBlockK / kUmmaK; ++kk) {
              const uint32_t accum = (kb | kk) != 0 ? 1u : 0u;
              mma_bf16(d0, a0 + 2 * kk, b + 2 * kk, idesc, accum);
              mma_bf16(d1, a1 + 2 * kk, b + 2 * kk, idesc, accum);
            }
            mma_commit(&empty[s]);
            if (++s == S) { s = 0; ph ^= 1u; }
          }
          if (!ok) break;
          mma_commit(&tfull[a0i]);
          mma_commit(&tfull[a1i]);
          if (++acc == 2) { acc = 0; acc_ph ^= 1u; }
          continue;
        }
        if (!mbar_wait<kPair>(&tempty[acc], acc_ph ^ 1u, abort_flag, p.dev_err, p.wait_limit)) break;
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(acc * BN);
        for (int kb = 0; kb < unit_kb; ++kb) {
          if (!mbar_wait(&full[s], ph, abort_flag, p.dev_err, p.wait_limit)) { ok = false; break; }
          tc_fence_after();
          if (p.phases != nullptr) {
            if (!landed) note_phase(p, kPhFirstStage);
            landed = true;
            note_phase(p, kPhLastStage);
          }
          const uint64_t a = sw128_desc(smem_addr(sA + s * kAStage));
          const uint64_t b = sw128_desc(smem_addr(sB + s * kBStageBytes));
          if (kHybrid && kb == p.kblocks) {
            // head-term BM25 of the unit into the second accumulator
            const uint32_t d_lex = tmem_base + static_cast<uint32_t>((2 + acc) * BN);
#pragma unroll
            for (int kk = 0; kk < kBlockK / kUmmaK; ++kk)
              mma_bf16(d_lex, a + 2 * kk, b + 2 * kk, idesc, kk != 0 ? 1u : 0u);
            mma_commit(&empty[s]);
          } else if constexpr (kPair) {
#pragma unroll
            for (int kk = 0; kk < kBlockK / kUmmaK; ++kk)
              mma_bf16_pair(d_tmem, a + 2 * kk, b + 2 * kk, idesc, (kb | kk) != 0 ? 1u : 0u);
            mma_commit_pair_mc(&empty[s], 0x3);
          } else {
#pragma unroll
            for (int kk = 0; kk < kBlockK / kUmmaK; ++kk)
              mma_bf16(d_tmem, a + 2 * kk, b + 2 * kk, idesc, (kb | kk) != 0 ? 1u : 0u);
            mma_commit(&empty[s]);
          }
          if (++s == S) { s = 0; ph ^= 1u; }
        }
        if (!ok) break;
        if constexpr (kPair) mma_commit_pair_mc(&tfull[acc], 0x3);
        else mma_commit(&tfull[acc]);
        if (++acc == 2) { acc = 0; acc_ph ^= 1u; }
      }
      note_phase(p, kPhLastCommit);
      if constexpr (kPair) mma_commit_pair(mma_done);
      else mma_commit(mma_done);
      mbar_drain(mma_done, 0, p.dev_err);
    }
    __syncwarp();
  } else {
    // ------------------------------------------------ epilogue
    // kEpiSets sets of four warps; set s filters the units whose sequence
    // number is s modulo kEpiSets (with two sets, two units are filtered at
    // the same time).  Each set keeps its own lists.  Dual mode: set s
    // filters query tile 2J + s of every unit, from accumulator s.
    const int set = (warp - 2) >> 2;
    const int eg = warp & 3;                 // TMEM lane group of this warp
    const int row = eg * 32 + lane;          // query row within a tile
    constexpr int kRowSets = kDual ? 1 : kEpiSets;   // list slots per producer and tile
    const int per_tile = p.pmax / kRowSets;  // CTAs (pairs) per unit query tile with a list slot
    // Unit query tile J covers this CTA's query tile qtile(J) (one of a pair's two).
    auto qtile = [&](int J) {
      return kPair ? 2 * J + static_cast<int>(rank) : kDual ? 2 * J + set : J;
    };
    auto list_row = [&](int J) -> int64_t {
      const int pc = cta - first_cta(J, p.qt, C);
      return (static_cast<int64_t>(qtile(J)) * p.pmax + pc * kRowSets + (kDual ? 0 : set)) *
                 kBlockM + row;
    };
    auto owns = [&](int J) {
      const int pc = cta - first_cta(J, p.qt, C);
      return pc >= 0 && pc < per_tile;
    };
    EpiList<K> list;
    list.set_k(p.k);
    list.clear();
    LexCursor lex;             // hybrid: the query's postings cursors

    // This CTA owns the list slots (J, cta - first_cta(J)); empty them first.
    for (int J = 0; J < p.qt; ++J) {
      const int qi = qtile(J) * kBlockM + row;
      if (owns(J) && qi < p.q) list.init_mem(p, list_row(J), qi);
    }

    int cur_j = -1;
    int64_t cur_sr = 0;
    bool cur_valid = false;
    uint32_t acc_ph = 0;                     // phase bit per accumulator (bit acc)
    UnitSeq us;
    int seq = 0;
    for (us.start(p, cta, C); us.valid(); us.next(), ++seq) {
      if (!kDual && seq % kEpiSets != set) continue;
      // Accumulator (TMEM columns acc * BN, barriers tfull / tempty [acc]).
      const int acc = kDual ? 2 * (seq & 1) + set : (seq & 1);
      const int J = us.j();
      const int j = qtile(J);                // this CTA's query tile
      const int64_t t = us.t();
      // Chunk ids of this corpus tile: its rows, after the first corpus's
      // n_first ids when it belongs to a stacked second corpus.
      const bool second = t >= p.nt_first;
      const int64_t id_base = second ? p.n_first + (t - p.nt_first) * BN : t * BN;
      const int64_t id_end = second ? p.n : p.n_first;
      const bool valid = j * kBlockM + row < p.q;
      const bool warp_live = j * kBlockM + eg * 32 < p.q;
      if (J != cur_j) {
        if (cur_j >= 0 && cur_valid) list.save(p, cur_sr);
        if (!owns(J)) {              // cannot happen when the host plan holds
          atomicExch(p.dev_err, 2);
          *abort_flag = 1;
        }
        cur_j = J;
        cur_sr = list_row(J);
        cur_valid = valid && owns(J);
        if (cur_valid) list.load(p, cur_sr); else list.clear();
        if constexpr (K > 32) list.set_query(p, static_cast<int64_t>(j) * kBlockM + row, cur_valid);
        if constexpr (kHybrid) {
          if (cur_valid) lex.set_query(p, static_cast<int64_t>(j) * kBlockM + row);
        }
      }
      const bool act = cur_valid;
      if constexpr (kHybrid) {
        // Place the postings cursors at this unit's first chunk (while its
        // MMAs run) unless they continue from the previous unit.
        if (act && lex.next_doc != t * BN) lex.seek(p.fu.lex_post, t * BN);
        lex.next_doc = (t + 1) * BN;
      }
      // Shared bound of this query's k-th best score, read while the MMAs run.
      float gfl = -INFINITY;
      if constexpr (K <= 32) {
        if (p.qfloor != nullptr && act)
          gfl = shared_floor_read(p.qfloor, static_cast<int64_t>(j) * kBlockM + row, p.gen);
      } else {
        if (act) gfl = list.proven_floor(p.k);
      }
      // The warp leaves together when a wait gives up: the TMEM loads below
      // are warp-collective.
      const bool got = mbar_wait(&tfull[acc], (acc_ph >> acc) & 1u, abort_flag, p.dev_err,
                                 p.wait_limit);
      if (!__all_sync(0xffffffffu, got)) break;
      // Hands the accumulator back once this warp's TMEM loads of the unit
      // are done.  Pair mode: the epilogue warps of both CTAs release it at
      // the leader.
      bool released = false;
      auto release_acc = [&]() {
        tc_fence_before();
        __syncwarp();
        if (lane == 0) {
          if constexpr (kPair) mbar_arrive_cluster(cluster_addr(&tempty[acc], 0));
          else mbar_arrive(&tempty[acc]);
        }
        released = true;
      };
      tc_fence_after();
      if constexpr (K > 32) list.read_ahead();
      if (warp_live) {
        float inv_max = 0.f;
        if (kLex != kLexNone && act) {
          const float m = p.fu.bm25_max[j * kBlockM + row];
          inv_max = m > 0.f ? 1.f / m : 0.f;
        }
        const uint32_t taddr = tmem_base + (static_cast<uint32_t>(eg * 32) << 16) +
                               static_cast<uint32_t>(acc * BN);
        // This thread's staging row; float4 groups are XOR-swizzled by lane so
        // that the 32 lanes' 16-byte stores spread over all banks.
        float* srow = stage_rows + ((warp - 2) * 32 + lane) * 32;
        const int swz = lane & 7;
        unsigned char* land = lex_land + ((warp - 2) * 32 + lane) * kLexLandStride;
        // BM25 block form: the warp's 32 x 32 tile of the block for chunk c
        // sits in the staging rows (c even) or in the second tile (c odd);
        // the filter stages the chunk's candidates in the same tile, and the
        // next chunk's copy goes to the other one while this one is filtered.
        constexpr int NC = BN / 32;              // 32-column chunks of a unit
        float* wtile[2] = {stage_rows + (warp - 2) * 32 * 32, block_land + (warp - 2) * 32 * 32};
        auto row_of = [&](int c) -> float* {
          return kLex == kLexBlock && (c & 1) ? wtile[1] + lane * 32 : srow;
        };
        int block_next = -1;     // chunk whose block tile is in flight (-1: none)
        // Copies chunk c's tile row by row with cp.async (eight lanes per
        // 128-byte row, four rows per round: a lane reading its own row would
        // touch 32 lines per load) straight into the rows of the lanes that
        // own the query rows.  Rows past the batch and columns past the
        // block's width read as 0; columns past the corpus become -inf later.
        auto copy_block = [&](int c) {
          float* tile = wtile[c & 1];
          const int sub = lane >> 3, part = lane & 7;
          const int64_t col = id_base + c * 32 + part * 4;
          int64_t qrow = static_cast<int64_t>(j) * kBlockM + eg * 32 + sub;
          const float* src = p.fu.bm25 + qrow * p.fu.ld + col;
#pragma unroll 1
          for (int rr = sub; rr < 32; rr += 4) {
            const bool in = qrow < p.q && col < p.fu.ld;
            cp_async16_zfill(tile + rr * 32 + ((part ^ (rr & 7)) << 2), in ? src : p.fu.bm25, in);
            src += 4 * p.fu.ld;
            qrow += 4;
          }
          cp_async_commit();
        };
        // Scores of one chunk (corpus rows id0 .. id0 + 31), fused with the
        // lexical part when hybrid, -inf past the end of the corpus.  Called
        // by every lane of a live warp (the TMEM load is warp-collective).
        auto scores = [&](const uint32_t (&r)[32], int c, float (&v)[32]) {
#pragma unroll
          for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
          const int64_t id0 = id_base + c * 32;
          if constexpr (kLex == kLexBlock) {
            if (block_next != c) {
              __syncwarp();                      // the tile's last readers are done
              copy_block(c);
            }
            cp_async_wait_all();
            __syncwarp();
            if (act) {
              const float a = p.fu.alpha, b1 = 1.f - p.fu.alpha;
              const float* row = row_of(c);
#pragma unroll
              for (int g = 0; g < 8; ++g) {
                const float4 x = *reinterpret_cast<const float4*>(row + ((g ^ swz) << 2));
                v[4 * g] = fmaf(a, v[4 * g], b1 * (x.x * inv_max));
                v[4 * g + 1] = fmaf(a, v[4 * g + 1], b1 * (x.y * inv_max));
                v[4 * g + 2] = fmaf(a, v[4 * g + 2], b1 * (x.z * inv_max));
                v[4 * g + 3] = fmaf(a, v[4 * g + 3], b1 * (x.w * inv_max));
              }
            }
            // The other tile's last users (the previous chunk's filter, which
            // ends with a warp barrier) are done: start the next chunk's copy.
            block_next = c + 1 < NC ? c + 1 : -1;
            if (block_next >= 0) copy_block(block_next);
          }
          if constexpr (kHybrid) {
            // head terms from the second accumulator, the other terms from
            // the postings (gathered into the staging row while the TMEM
            // load is in flight), then the Sec. 4.4 weighted fusion
            uint32_t rl[32];
            tmem_ld32_async(taddr + 2 * BN + c * 32, rl);
            if (act) {
              lex.fetch(p, id0, land);
#pragma unroll
              for (int g = 0; g < 8; ++g)
                *reinterpret_cast<float4*>(srow + (g << 2)) = make_float4(0.f, 0.f, 0.f, 0.f);
              lex.tail(p, id0, land, srow, swz);
            }
            tmem_wait_ld(rl);
            if (act) {
              const float a = p.fu.alpha, b1 = 1.f - p.fu.alpha;
#pragma unroll
              for (int g = 0; g < 8; ++g) {
                const float4 x = *reinterpret_cast<const float4*>(srow + ((g ^ swz) << 2));
                const float4 y = lex.mid4(land, g);
                v[4 * g] = fmaf(
                    a, v[4 * g], b1 * ((__uint_as_float(rl[4 * g]) + x.x + y.x) * inv_max));
                v[4 * g + 1] = fmaf(
                    a, v[4 * g + 1], b1 * ((__uint_as_float(rl[4 * g + 1]) + x.y + y.y) * inv_max));
                v[4 * g + 2] = fmaf(
                    a, v[4 * g + 2], b1 * ((__uint_as_float(rl[4 * g + 2]) + x.z + y.z) * inv_max));
                v[4 * g + 3] = fmaf(
                    a, v[4 * g + 3], b1 * ((__uint_as_float(rl[4 * g + 3]) + x.w + y.w) * inv_max));
              }
            }
          }
          if (id0 + 32 > id_end) {
#pragma unroll
            for (int i = 0; i < 32; ++i)
              if (id0 + i >= id_end) v[i] = -INFINITY;
          }
        };
        // Filters one chunk against max(list floor, unit bound).
        auto process = [&](const uint32_t (&r)[32], int c, float bound) {
          float v[32];
          scores(r, c, v);
          const int64_t id0 = id_base + c * 32;
          if (__any_sync(0xffffffffu, act && max32(v) >= fmaxf(list.floor(), bound))) {
            // Room for this chunk's keys in a buffered list (a compaction
            // raises the list's floor, so the floor is read after it).
            list.sync(false, act);
            const float fl = fmaxf(list.floor(), bound);
            // Lanes insert their candidates together, one column per round,
            // so the warp runs max-per-lane rounds instead of the sum.
            uint32_t mask = 0;
            if (act) {
              // Four independent 8-bit parts (short dependency chains).
              uint32_t part[4] = {0u, 0u, 0u, 0u};
#pragma unroll
              for (int i = 0; i < 32; ++i) part[i >> 3] |= (v[i] >= fl ? 1u : 0u) << i;
              mask = (part[0] | part[1]) | (part[2] | part[3]);
              float* crow = row_of(c);
#pragma unroll
              for (int g = 0; g < 8; ++g)
                *reinterpret_cast<float4*>(crow + ((g ^ swz) << 2)) =
                    make_float4(v[4 * g], v[4 * g + 1], v[4 * g + 2], v[4 * g + 3]);
            }
            const float* crow = row_of(c);
            // Warp-uniform number of rounds; each round takes the lowest
            // remaining candidate column of every lane (ids stay increasing)
            // and inserts it with the branch-free network, so rounds are
            // straight-line code and the next extraction overlaps the insert.
            const int rounds = __reduce_max_sync(0xffffffffu, __popc(mask));
#pragma unroll 2
            for (int r = 0; r < rounds; ++r) {
              const int i = __ffs(mask) - 1;
              const bool has = mask != 0;
              mask &= mask - 1;
              const float s = has ? crow[((((i & 31) >> 2) ^ swz) << 2) | (i & 3)] : -INFINITY;
              list.insert(s, static_cast<uint32_t>(id0 + i));
            }
          }
          __syncwarp();
        };
        static_assert(NC % 2 == 0, "chunks are processed in pairs");
        uint32_t ra[32], rb[32];
        float bound = -INFINITY;
        // (Hybrid: no group bound for a fresh list, whose scores would need
        // a second walk of the postings.)
        if constexpr (K <= 32 && !kHybrid) {
          if (__any_sync(0xffffffffu, act && !list.full())) {
            // A list that is not full yet would take almost every score of
            // this unit as a candidate.  Cut the unit's columns into groups:
            // the k-th largest group maximum is reached by k distinct scores
            // of the unit, so it is <= the unit's k-th best score, and no
            // score below it can be among the query's k best.  Lists of 16
            // or 32 use 32 groups and sort their maxima (a tight bound pays
            // for the sort when each insertion costs 16-32 steps); lists of
            // 8 use 8 groups (a sort of 8 values).
            if constexpr (K <= 8) {
              constexpr int G = K / NC;         // groups per 32-column chunk
              static_assert(G >= 1 && 32 % G == 0, "group layout");
              // Group maxima enter gm through a shift (constant indices in a
              // loop that is not unrolled).
              float gm[K];
#pragma unroll 1
              for (int c = 0; c < NC; ++c) {
                __syncwarp();
                tmem_ld32_async(taddr + c * 32, ra);
                tmem_wait_ld(ra);
                float v[32];
                scores(ra, c, v);
#pragma unroll
                for (int i = K - 1; i >= G; --i) gm[i] = gm[i - G];
#pragma unroll
                for (int g = 0; g < G; ++g) {
                  constexpr int L = 32 / G;
                  float m = v[g * L];
#pragma unroll
                  for (int i = 1; i + 1 < L; i += 2) m = fmax3(m, v[g * L + i], v[g * L + i + 1]);
                  if constexpr (L % 2 == 0) m = fmaxf(m, v[g * L + L - 1]);
                  gm[g] = m;
                }
              }
              // The k-th largest group maximum (K groups, k <= K).
              bitonic_desc<K>(gm);
              bound = reg_select(gm, (p.k < K ? p.k : K) - 1);
            } else {
            constexpr int GPC = 32 / NC;        // groups per 32-column chunk
            constexpr int L = 32 / GPC;         // columns per group
            static_assert(GPC * NC == 32 && L >= 2, "group layout");
            float gm[32];
#pragma unroll
            for (int c = 0; c < NC; ++c) {
              __syncwarp();
              tmem_ld32_async(taddr + c * 32, ra);
              tmem_wait_ld(ra);
              float v[32];
              scores(ra, c, v);
#pragma unroll
              for (int g = 0; g < GPC; ++g) {
                float m = v[g * L];
#pragma unroll
                for (int i = 1; i + 1 < L; i += 2) m = fmax3(m, v[g * L + i], v[g * L + i + 1]);
                if constexpr (L % 2 == 0) m = fmaxf(m, v[g * L + L - 1]);
                gm[c * GPC + g] = m;
              }
            }
            bitonic_desc<32>(gm);
            const int kk = p.k < 32 ? p.k : 32;
            bound = reg_select(gm, kk - 1);
            }
          }
        }
        const float lb = fmaxf(bound, gfl);     // admission bound of this unit
        __syncwarp();
        if constexpr (K > 32) {
          // Buffered lists: one chunk at a time, each load waited for before
          // the filter (see epi_sets).
#pragma unroll 1
          for (int c = 0; c < NC; ++c) {
            tmem_ld32_async(taddr + c * 32, ra);
            tmem_wait_ld(ra);
            if (!kHybrid && c + 1 == NC) release_acc();   // see below
            process(ra, c, lb);
          }
        } else {
        // Register lists: the next chunk's load flies while one is filtered.
        tmem_ld32_async(taddr, ra);
#pragma unroll 1
        for (int c = 0; c < NC; c += 2) {
          tmem_wait_ld(ra);
          tmem_ld32_async(taddr + (c + 1) * 32, rb);
          process(ra, c, lb);
          tmem_wait_ld(rb);
          if (c + 2 < NC) tmem_ld32_async(taddr + (c + 2) * 32, ra);
          // The unit's last TMEM load has landed: hand the accumulator back
          // to the MMA before filtering the last chunk (the gathered hybrid
          // form still reads its second accumulator while filtering).
          // Measured on GB300: 32768 x 1024 with 4096 queries and k = 10,
          // 217.6 instead of 218.9 us a step; 1M x 768 with 2048 queries and
          // k = 100, main pass 1835 instead of 1868 us.
          if (!kHybrid && c + 2 >= NC) release_acc();
          process(rb, c + 1, lb);
        }
        }
        if constexpr (K <= 32) {
          // Publish what this list now proves about the query's k-th best.
          if (p.qfloor != nullptr && act) {
            const float pub = fmaxf(list.kth(p.k), bound);
            if (pub > gfl)
              shared_floor_raise(p.qfloor, static_cast<int64_t>(j) * kBlockM + row, p.gen, pub);
          }
        }
      }
      if (!released) release_acc();
      acc_ph ^= 1u << acc;
    }
    if (cur_j >= 0 && cur_valid) list.save(p, cur_sr);
    // The set's last warp to finish (the slots start at zero).
    if (p.phases != nullptr && lane == 0)
      atomicMax(p.phases + static_cast<size_t>(blockIdx.x) * kPhases + kPhEpi0Done + set,
                global_timer());
  }

  tc_fence_before();
  // Pair mode: neither CTA leaves (or frees TMEM) while the other may still
  // signal its barriers; the leader's MMAs have drained (mma_done) by now.
  if constexpr (kPair) cluster_sync();
  else __syncthreads();
  tc_fence_after();
  if (threadIdx.x == 0) note_phase(p, kPhExit);
  if (warp == 1) {
    if constexpr (kPair) tmem_dealloc_pair(tmem_base, kTmemCols);
    else tmem_dealloc(tmem_base, kTmemCols);
  }
}

// ----------------------------------------------------------------- launch

// Tensor maps of one launch: queries and corpus (score K blocks), and for the
// gathered hybrid search the head-term counts and split weights (otherwise
// copies of the first two, unused).
struct TcMaps {
  CUtensorMap q, e, qb, eb;
};

// Pair mode: clusters of two CTAs; `grid` counts CTAs (even).
template <int BN, int K, int L>
cudaError_t launch_pair_variant(const TcMaps& m, const TcParams& prm, int grid, cudaStream_t st) {
  constexpr size_t smem = smem_for<BN, K, true, false, false, block_land_bytes<K, L>()>();
  static bool configured = false;
  if (!configured) {
    cudaError_t e = cudaFuncSetAttribute(tc_search_kernel<BN, K, L, true>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    configured = true;
  }
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(threads_for(K));
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, tc_search_kernel<BN, K, L, true>, m.q, m.e, m.qb, m.eb, prm);
}

// Clusters of two CTAs of a pair-mode search kernel that fit on the device at
// once (the kernels' shared-memory use keeps one CTA per SM).
int pair_capacity_query();

template <int BN, int K, int L>
cudaError_t launch_variant(const TcMaps& m, const TcParams& prm, int grid, cudaStream_t st) {
  constexpr bool g = L == kLexGather;
  constexpr size_t smem = smem_for<BN, K, false, false, g, block_land_bytes<K, L>()>();
  static bool configured = false;
  if (!configured) {
    cudaError_t e = cudaFuncSetAttribute(tc_search_kernel<BN, K, L>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    configured = true;
  }
  tc_search_kernel<BN, K, L><<<grid, threads_for(K, g), smem, st>>>(m.q, m.e, m.qb, m.eb, prm);
  return cudaGetLastError();
}

// Dual mode (two query tiles per unit); 128-row corpus tiles, lists of 8 or 16.
template <int K, int L>
cudaError_t launch_dual_variant(const TcMaps& m, const TcParams& prm, int grid, cudaStream_t st) {
  constexpr size_t smem = smem_for<128, K, false, true, false, block_land_bytes<K, L>()>();
  static bool configured = false;
  if (!configured) {
    cudaError_t e = cudaFuncSetAttribute(tc_search_kernel<128, K, L, false, true>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    configured = true;
  }
  tc_search_kernel<128, K, L, false, true><<<grid, threads_for(K), smem, st>>>(m.q, m.e, m.qb,
                                                                               m.eb, prm);
  return cudaGetLastError();
}

template <int BN, int L>
cudaError_t launch_bn(const TcMaps& m, const TcParams& prm, int grid, cudaStream_t st) {
  switch (list_len_for(prm.k)) {
    case 8: return launch_variant<BN, 8, L>(m, prm, grid, st);
    case 16: return launch_variant<BN, 16, L>(m, prm, grid, st);
    case 32: return launch_variant<BN, 32, L>(m, prm, grid, st);
    case 128: return launch_variant<BN, 128, L>(m, prm, grid, st);
    default: return launch_variant<BN, 256, L>(m, prm, grid, st);
  }
}

template <int L>
cudaError_t launch_pair(const TcMaps& m, const TcParams& prm, int grid, cudaStream_t st) {
  switch (list_len_for(prm.k)) {
    case 8: return launch_pair_variant<256, 8, L>(m, prm, grid, st);
    case 16: return launch_pair_variant<256, 16, L>(m, prm, grid, st);
    case 32: return launch_pair_variant<256, 32, L>(m, prm, grid, st);
    case 128: return launch_pair_variant<256, 128, L>(m, prm, grid, st);
    default: return launch_pair_variant<256, 256, L>(m, prm, grid, st);
  }
}

template <int L>
cudaError_t launch_dual(const TcMaps& m, const TcParams& prm, int grid, cudaStream_t st) {
  switch (list_len_for(prm.k)) {
    case 8: return launch_dual_variant<8, L>(m, prm, grid, st);
    case 16: return launch_dual_variant<16, L>(m, prm, grid, st);
    default: return cudaErrorInvalidValue;
  }
}

// Instantiations live in their own translation units (parallel builds).
cudaError_t launch_bn128(const TcMaps& m, const TcParams& prm, int grid, int lex, cudaStream_t st);
cudaError_t launch_bn128_gather(const TcMaps& m, const TcParams& prm, int grid, cudaStream_t st);
cudaError_t launch_bn256_dense(const TcMaps& m, const TcParams& prm, int grid, cudaStream_t st);
cudaError_t launch_bn256_block(const TcMaps& m, const TcParams& prm, int grid, cudaStream_t st);
cudaError_t launch_pair256_dense(const TcMaps& m, const TcParams& prm, int grid, cudaStream_t st);
cudaError_t launch_pair256_block(const TcMaps& m, const TcParams& prm, int grid, cudaStream_t st);
cudaError_t launch_dual128(const TcMaps& m, const TcParams& prm, int grid, int lex,
                           cudaStream_t st);

}  // namespace tc
}  // namespace oprag
