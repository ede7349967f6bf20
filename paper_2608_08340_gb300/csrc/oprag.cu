// Host side of the C ABI declared in include/oprag.h: the index object,
// argument checking, scratch management and the choice of kernel family.
#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <string>
#include <thread>
#include <vector>

#include "oprag.h"
#include "internal.h"

using namespace oprag;

namespace {

thread_local std::string g_err;

int fail(int code, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof buf, fmt, ap);
  va_end(ap);
  g_err = buf;
  return code;
}

int cuda_fail(cudaError_t e, const char* what) {
  return fail(OPRAG_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

int ok() {
  g_err.clear();
  return OPRAG_OK;
}

size_t elem_size(int dtype) { return dtype == OPRAG_F32 ? 4 : 2; }

// Makes the index's device current for the duration of a call.
struct DeviceGuard {
  int prev = -1;
  bool changed = false;
  explicit DeviceGuard(int dev) {
    if (cudaGetDevice(&prev) == cudaSuccess && prev != dev) {
      changed = cudaSetDevice(dev) == cudaSuccess;
    }
  }
  ~DeviceGuard() {
    if (changed) cudaSetDevice(prev);
  }
};

// bf16 searches always take the tensor-core kernel (measured faster than the
// SIMT stream even for a single query); fp32 indices take the SIMT kernel.
constexpr int kSimtMaxQueriesBf16 = 0;
// Largest BM25 matrix block (floats) materialised per hybrid pass.
constexpr int64_t kLexMaxElems = int64_t(1) << 28;

}  // namespace

struct oprag_index {
  int device = 0;
  int num_sms = 1;
  int64_t n = 0;
  int64_t cap = 0;             // rows allocated for emb (appends double it)
  int d = 0;
  int dtype = OPRAG_BF16;
  void* emb = nullptr;
  int* dev_err = nullptr;
  int* err_host = nullptr;       // pinned copy of dev_err, read after host-buffer calls
  cudaEvent_t done = nullptr;

  void* scratch = nullptr;     // partial top-k lists
  size_t scratch_bytes = 0;
  float* lex = nullptr;        // BM25 block (q x ld) followed by q maxima
  size_t lex_bytes = 0;
  void* cand = nullptr;        // dense-first candidates: q x N ids, then q x N scores
  size_t cand_bytes = 0;
  void* stage = nullptr;       // upsert staging / host-buffer search staging
  size_t stage_bytes = 0;

  bool has_sparse = false;
  int vocab = 0;
  // Host copy of the token bags (CSR) and BM25 parameters: the device side is
  // rebuilt from them when bags are replaced or chunks appended.
  std::vector<int32_t> bag_ptr, bag_terms;
  double bm_k1 = 1.2, bm_b = 0.75;
  int64_t nnz = 0;
  int64_t* post_ptr = nullptr;
  int2* post = nullptr;
  int32_t* dense_slot = nullptr;
  float* dense_w = nullptr;
  int64_t dense_ld = 0;
  int64_t* tile_ptr = nullptr;
  int ntiles = 0;
  void* wsplit = nullptr;      // n x kLexK bf16 head-term weights (high | low halves)
  int32_t* lex_class = nullptr;  // vocab: epilogue class of each term (see rebuild_sparse)
  float* mid_w = nullptr;        // rows of mid-frequency term weights, mid_ld apart
  int64_t mid_ld = 0;

  int opt_path = 0;
  int opt_block_n = 0;
  int opt_lex_gather = 0;      // hybrid search: 1 gathers BM25 in the epilogue (OPRAG_OPT_LEX_GATHER)
  int opt_pair = 0;
  // Replay of a captured dense search (OPRAG_OPT_GRAPH): the launches of the
  // previous search with the same pointers, sizes, stream and index state.
  int opt_graph = 0;
  uint64_t state_version = 0;  // bumped whenever a buffer moves or an option changes
  bool capturing = false;
  struct {
    bool seen = false;
    const void* queries = nullptr;
    int q = 0, k = 0;
    int64_t* ids = nullptr;
    float* scores = nullptr;
    cudaStream_t st = nullptr;
    uint64_t version = 0;
    cudaGraphExec_t exec = nullptr;
  } gcache;
  // Per-query k-th score bounds shared by the lists of one search, tagged
  // with a per-launch generation (zeroed memory holds no valid entry).
  uint64_t* qfloor = nullptr;
  size_t qfloor_bytes = 0;
  uint32_t gen = 0;
  int pair_cap = -1;       // clusters of two search CTAs that fit at once (-1: not asked yet)
  int last_path = 0;
  int last_grid = 0, last_cluster = 0, last_block_n = 0;   // last main search kernel launch
  int last_tiles = 0;                                         // query tiles per CTA and unit

  // Optional kernel timing (events listed below).
  bool timing = false;
  bool timed = false;      // the last search recorded its events
  bool timed_lex = false;  // ... including a lexical pass
  bool timed_sample = false;  // ... including a sampled first pass
  // ev[0] before the lexical pass, ev[1] before the search passes, ev[4]
  // before the main search pass (after the sampled first pass, if any),
  // ev[2] before the merge, ev[3] after it.
  cudaEvent_t ev[5] = {nullptr, nullptr, nullptr, nullptr, nullptr};
  // Spin limit (cycles) of the search kernels' mbarrier waits; 0 = default.
  long long wait_limit = 0;
  // Phase stamps of the main tensor-core pass (OPRAG_OPT_PHASES): grid x
  // kTcPhases global-timer values of the last search, and its grid.
  bool phases_on = false;
  void* phases = nullptr;
  size_t phases_bytes = 0;
  int phases_grid = 0;

  // Waits until all work enqueued on this index is done.
  cudaError_t drain() { return done ? cudaEventSynchronize(done) : cudaSuccess; }

  // Grows a device buffer.  The old buffer may still be read by work this or
  // an earlier call enqueued, so the whole device is drained first.
  int ensure(void** buf, size_t* cur, size_t need, const char* what) {
    if (need <= *cur) return OPRAG_OK;
    ++state_version;
    cudaError_t e = cudaDeviceSynchronize();
    if (e != cudaSuccess) return cuda_fail(e, "waiting for pending work");
    if (*buf) cudaFree(*buf);
    *buf = nullptr;
    *cur = 0;
    const size_t want = need + need / 4;
    if (cudaMalloc(buf, want) != cudaSuccess) {
      cudaGetLastError();
      *buf = nullptr;
      return fail(OPRAG_ERR_OOM, "cannot allocate %zu bytes of %s", want, what);
    }
    *cur = want;
    return OPRAG_OK;
  }

  void free_sparse() {
    if (post_ptr) cudaFree(post_ptr);
    if (post) cudaFree(post);
    if (dense_slot) cudaFree(dense_slot);
    if (dense_w) cudaFree(dense_w);
    if (tile_ptr) cudaFree(tile_ptr);
    if (wsplit) cudaFree(wsplit);
    if (lex_class) cudaFree(lex_class);
    if (mid_w) cudaFree(mid_w);
    wsplit = nullptr;
    lex_class = nullptr;
    mid_w = nullptr;
    post_ptr = nullptr;
    post = nullptr;
    dense_slot = nullptr;
    dense_w = nullptr;
    tile_ptr = nullptr;
    has_sparse = false;
  }
};

namespace {

int begin_call(oprag_index* idx, cudaStream_t st) {
  cudaGetLastError();  // clear a stale, non-sticky error of another library
  cudaError_t e = cudaStreamWaitEvent(st, idx->done, 0);
  if (e != cudaSuccess) return cuda_fail(e, "ordering after the previous call");
  return OPRAG_OK;
}

int end_call(oprag_index* idx, cudaStream_t st) {
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(e, "kernel launch");
  e = cudaEventRecord(idx->done, st);
  if (e != cudaSuccess) return cuda_fail(e, "recording completion");
  return ok();
}

// Clusters of two pair-mode search CTAs that fit at once on the index's
// device; asked once (the device is current inside every entry point).
int pair_capacity(oprag_index* idx) {
  if (idx->pair_cap < 0) {
    idx->pair_cap = tc_pair_capacity();
    cudaGetLastError();
  }
  return idx->pair_cap;
}

// Shared k-th score bounds for a search of q queries: grows (and zeroes) the
// per-index array and hands out a fresh generation tag.
int shared_floors(oprag_index* idx, int q, cudaStream_t st, uint64_t** qf, uint32_t* gen) {
  const size_t need = static_cast<size_t>(q) * sizeof(uint64_t);
  if (need > idx->qfloor_bytes) {
    int rc = idx->ensure(reinterpret_cast<void**>(&idx->qfloor), &idx->qfloor_bytes, need,
                         "shared k-th score bounds");
    if (rc) return rc;
    cudaError_t e = cudaMemsetAsync(idx->qfloor, 0, idx->qfloor_bytes, st);
    if (e != cudaSuccess) return cuda_fail(e, "clearing shared bounds");
  }
  if (idx->capturing) {
    // A captured search is replayed with the same tag: clear its entries in
    // every replay instead.
    cudaError_t e = cudaMemsetAsync(idx->qfloor, 0, need, st);
    if (e != cudaSuccess) return cuda_fail(e, "clearing shared bounds");
  }
  if (++idx->gen == 0) {            // tags wrapped: old entries could read as current
    cudaError_t e = cudaMemsetAsync(idx->qfloor, 0, idx->qfloor_bytes, st);
    if (e != cudaSuccess) return cuda_fail(e, "clearing shared bounds");
    idx->gen = 1;
  }
  *qf = idx->qfloor;
  *gen = idx->gen;
  return OPRAG_OK;
}

// Records the shape of a search's main kernel launch (oprag_index_last_launch).
void note_launch(oprag_index* idx, int path, const TcPlan& plan) {
  if (path == 2) {
    idx->last_grid = plan.grid;
    idx->last_cluster = plan.pair;
    idx->last_block_n = plan.block_n;
    idx->last_tiles = plan.dual ? 2 : 1;
  } else {
    idx->last_grid = idx->last_cluster = idx->last_block_n = idx->last_tiles = 0;
  }
}

int choose_path(const oprag_index* idx, int q) {
  if (idx->dtype == OPRAG_F32) return 1;
  if (idx->opt_path == 1 || idx->opt_path == 2) return idx->opt_path;
  return q <= kSimtMaxQueriesBf16 ? 1 : 2;
}

// Scratch of one search, in one block: the main pass's partial lists and,
// for buffered lists (k > 32) over many corpus tiles, a first pass over every
// kSampleStride-th corpus tile (its lists, its merged top-k, and per query the
// k-th score, kLevels counted floors and their counters).  Register lists
// (k <= 32) also use one 64-bit shared bound per query, kept outside the block.
#ifndef OPRAG_SAMPLE_STRIDE
#define OPRAG_SAMPLE_STRIDE 32
#endif
constexpr int kSampleStride = OPRAG_SAMPLE_STRIDE;
// Corpus tiles from which a search with buffered lists runs the first pass.
constexpr int kSampleMinTiles = 128;
// Every 32nd corpus tile, lists of 8 keys (two epilogue sets, the cheapest
// insertions).  Any k-th best of real candidates is a valid floor.  Measured
// on 1M x 768 with 2048 queries and k = 100: with stride 16, lists of 32 / 16
// / 8 keys gave a first pass of 395 / 264 / 218 us and the same main pass
// (2194 us); with lists of 8, strides 8 / 16 / 32 gave steps of 2636 / 2534 /
// 2470 us (first pass 357 / 220 / 141 us, main pass 2226 / 2256 / 2275 us).
#ifndef OPRAG_SAMPLE_K
#define OPRAG_SAMPLE_K 8
#endif
constexpr int kSampleK = OPRAG_SAMPLE_K;

struct SearchLayout {
  int path = 0;           // 1 SIMT, 2 tensor core
  int simt_grid = 0;
  TcPlan plan{}, splan{};
  bool sampled = false;
  size_t main_bytes = 0;    // multiple of 256
  size_t sample_bytes = 0;  // 0 unless sampled
  bool floors = false;      // q shared bounds (register lists on the tensor-core path)
  size_t total() const { return main_bytes + sample_bytes; }
};

size_t round256(size_t b) { return (b + 255) / 256 * 256; }

SearchLayout search_layout(oprag_index* idx, int q, int k, int path, int block_n, int pair,
                           bool lex = false, int64_t n_second = 0) {
  SearchLayout L;
  SearchShape s{idx->n, idx->d, q, k};
  s.fused_lex = lex && path == 2;
  s.n_second = path == 2 ? n_second : 0;
  L.path = path;
  if (path == 1) {
    L.simt_grid = simt_grid(s, idx->num_sms);
    L.main_bytes = round256(simt_scratch_bytes(idx->dtype, s, L.simt_grid));
    return L;
  }
  L.plan = tc_plan(s, idx->num_sms, block_n, 1, pair, pair_capacity(idx));
  L.main_bytes = round256(tc_scratch_bytes(s, L.plan));
  // Buffered lists collect every score above their floor, and the floor of a
  // fresh list starts at -inf.  A cheap first pass over every
  // kSampleStride-th corpus tile with kSampleK-key lists yields, per query, the
  // k-th best of real corpus scores -- a lower bound of the true k-th best --
  // which the main pass then uses as the lists' starting floor.
  L.sampled = list_len_for(k) > 32 && L.plan.nt >= kSampleMinTiles;
  if (L.sampled) {
    SearchShape s32 = s;
    s32.k = kSampleK;
    L.splan = tc_plan(s32, idx->num_sms, L.plan.block_n, kSampleStride, L.plan.pair,
                      pair_capacity(idx));
    const size_t per_query_tail = sizeof(float) + kLevels * (sizeof(float) + sizeof(int));
    L.sample_bytes = round256(tc_scratch_bytes(s32, L.splan)) +
                     round256(static_cast<size_t>(q) * k * 12) +
                     static_cast<size_t>(q) * per_query_tail + 16;
  }
  L.floors = list_len_for(k) <= 32;
  return L;
}

SearchLayout search_layout(oprag_index* idx, int q, int k, bool lex = false) {
  return search_layout(idx, q, k, choose_path(idx, q), idx->opt_block_n, idx->opt_pair, lex);
}

// Enqueues the passes of a laid-out search and its merge.  scratch holds
// L.total() bytes; qf / gen are the shared bounds (used when L.floors).
// E2 / n2 (tensor-core path): a second corpus stacked after the index's rows
// in the same launches; the final merge then writes out_src (0: the index,
// 1: the second corpus) and ids within each.
int launch_search(oprag_index* idx, const SearchLayout& L, const void* Q, int q, int k,
                  const Fusion& fu, void* scratch, uint64_t* qf, uint32_t gen, int64_t* out_ids,
                  float* out_scores, cudaStream_t st, const void* E2 = nullptr, int64_t n2 = 0,
                  int32_t* out_src = nullptr) {
  SearchShape s{idx->n, idx->d, q, k};
  s.fused_lex = L.path == 2 && fu.gathered();
  s.n_second = L.path == 2 ? n2 : 0;
  ListSet lists{};
  cudaError_t e;
  if (idx->timing) cudaEventRecord(idx->ev[1], st);
  idx->timed_sample = idx->timing && L.sampled;
  if (L.path == 1) {
    e = launch_simt_search(idx->dtype, idx->emb, Q, s, fu, scratch, L.simt_grid, &lists, st);
  } else {
    const float* floor = nullptr;
    float* levels = nullptr;
    int* level_cnt = nullptr;
    if (L.sampled) {
      SearchShape s32 = s;
      s32.k = kSampleK;
      char* sbase = static_cast<char*>(scratch) + L.main_bytes;
      const size_t slist = round256(tc_scratch_bytes(s32, L.splan));
      int64_t* sids = reinterpret_cast<int64_t*>(sbase + slist);
      float* sscores = reinterpret_cast<float*>(sids + static_cast<size_t>(q) * k);
      float* kth = reinterpret_cast<float*>(sbase + slist + round256(static_cast<size_t>(q) * k * 12));
      // 16-byte aligned: each query's kLevels counters are read as one int4.
      levels = kth + (static_cast<size_t>(q) + 3) / 4 * 4;
      level_cnt = reinterpret_cast<int*>(levels + static_cast<size_t>(q) * kLevels);
      ListSet slists{};
      e = launch_tc_search(idx->emb, Q, s32, fu, L.splan, sbase, idx->dev_err, &slists, st,
                           nullptr, nullptr, 0, nullptr, nullptr, idx->wait_limit, nullptr, E2);
      if (e == cudaSuccess) e = launch_merge(slists, q, k, sids, sscores, st, kth, levels);
      if (e == cudaSuccess)
        e = cudaMemsetAsync(level_cnt, 0, static_cast<size_t>(q) * kLevels * sizeof(int), st);
      if (e != cudaSuccess) return cuda_fail(e, "sampling pass");
      floor = kth;
    }
    if (idx->timed_sample) cudaEventRecord(idx->ev[4], st);
    unsigned long long* ph = nullptr;
    if (idx->phases_on && idx->phases != nullptr &&
        idx->phases_bytes >= static_cast<size_t>(L.plan.grid) * kTcPhases * 8) {
      ph = static_cast<unsigned long long*>(idx->phases);
      cudaMemsetAsync(ph, 0, static_cast<size_t>(L.plan.grid) * kTcPhases * 8, st);
      idx->phases_grid = L.plan.grid;
    }
    e = launch_tc_search(idx->emb, Q, s, fu, L.plan, scratch, idx->dev_err, &lists, st, floor,
                         L.floors ? qf : nullptr, gen, levels, level_cnt, idx->wait_limit, ph, E2);
  }
  if (e != cudaSuccess) return cuda_fail(e, "search kernel");
  if (idx->timing) cudaEventRecord(idx->ev[2], st);
  note_launch(idx, L.path, L.plan);
  if (out_src != nullptr) {
    lists.split = idx->n;
    lists.out_src = out_src;
  }
  e = launch_merge(lists, q, k, out_ids, out_scores, st);
  if (e != cudaSuccess) return cuda_fail(e, "merge kernel");
  if (idx->timing) cudaEventRecord(idx->ev[3], st);
  idx->timed = idx->timing;
  idx->last_path = L.path;
  return OPRAG_OK;
}

// Dense (or fused) top-k of q queries; all pointers on the device.  Grows the
// index's scratch (and shared bounds) on demand.
int run_search(oprag_index* idx, const void* Q, int q, int k, const Fusion& fu, int64_t* out_ids,
               float* out_scores, cudaStream_t st) {
  const SearchLayout L = search_layout(idx, q, k, fu.gathered());
  int rc = idx->ensure(&idx->scratch, &idx->scratch_bytes, L.total(), "search scratch");
  if (rc) return rc;
  uint64_t* qf = nullptr;
  uint32_t gen = 0;
  if (L.floors && (rc = shared_floors(idx, q, st, &qf, &gen))) return rc;
  return launch_search(idx, L, Q, q, k, fu, idx->scratch, qf, gen, out_ids, out_scores, st);
}

// Lexical buffer of a hybrid search of q queries.  Gathered form: the
// per-query operands of the epilogue and the BM25 maxima; materialised form:
// the BM25 block of up to qchunk queries (at most kLexMaxElems values) and
// its maxima.
struct LexLayout {
  size_t qcount = 0, terms = 0, term_cnt = 0, mid = 0, mid_cnt = 0, ovf = 0, max = 0, total = 0;
  int qchunk = 0;
};

LexLayout lex_layout(const oprag_index* idx, int q, bool gather) {
  LexLayout L;
  const size_t nq = static_cast<size_t>(q);
  if (gather) {
    size_t o = 0;
    auto take = [&](size_t bytes) {
      const size_t at = o;
      o = round256(o + bytes);
      return at;
    };
    L.qcount = take(nq * kLexK * 2);
    L.terms = take(nq * kLexRegTerms * sizeof(int4));
    L.term_cnt = take(nq * sizeof(int));
    L.mid = take(nq * kLexMidReg * sizeof(int2));
    L.mid_cnt = take(nq * sizeof(int));
    L.ovf = take(nq * sizeof(int));
    L.max = take(nq * sizeof(float));
    L.total = o;
    L.qchunk = q;
    return L;
  }
  const int64_t ld = (idx->n + 3) / 4 * 4;
  L.qchunk = static_cast<int>(std::min<int64_t>(q, std::max<int64_t>(1, kLexMaxElems / ld)));
  L.max = sizeof(float) * static_cast<size_t>(L.qchunk) * ld;
  L.total = L.max + sizeof(float) * static_cast<size_t>(L.qchunk);
  return L;
}

int check_search_args(const oprag_index* idx, const void* queries, int q, int k,
                      const void* out_ids, const void* out_scores) {
  if (!idx) return fail(OPRAG_ERR_INVALID_ARG, "index is NULL");
  if (q < 0) return fail(OPRAG_ERR_INVALID_ARG, "q = %d < 0", q);
  if (k < 1 || k > OPRAG_K_MAX || k > idx->n)
    return fail(OPRAG_ERR_INVALID_ARG, "k = %d outside [1, min(n = %lld, %d)]", k,
                static_cast<long long>(idx->n), OPRAG_K_MAX);
  if (q > 0 && (!queries || !out_ids || !out_scores))
    return fail(OPRAG_ERR_INVALID_ARG, "NULL queries or output buffer");
  if (q > 0 && (reinterpret_cast<uintptr_t>(queries) & 15))
    return fail(OPRAG_ERR_INVALID_ARG, "queries must be 16-byte aligned");
  return OPRAG_OK;
}

}  // namespace

extern "C" {

const char* oprag_last_error(void) { return g_err.c_str(); }

int oprag_index_create(oprag_index** out, const void* emb, int64_t n, int32_t d, int32_t dtype,
                       int32_t src_dtype, int32_t emb_on_device) {
  if (!out) return fail(OPRAG_ERR_INVALID_ARG, "out is NULL");
  *out = nullptr;
  if (!emb) return fail(OPRAG_ERR_INVALID_ARG, "emb is NULL");
  if (n < 1 || n > 0x7FFFFFFFLL) return fail(OPRAG_ERR_INVALID_ARG, "n = %lld out of range", (long long)n);
  if (d < 1 || d > 8192 || d % 8)
    return fail(OPRAG_ERR_INVALID_ARG, "d = %d must be a multiple of 8 in [8, 8192]", d);
  if ((dtype != OPRAG_F32 && dtype != OPRAG_BF16) || (src_dtype != OPRAG_F32 && src_dtype != OPRAG_BF16))
    return fail(OPRAG_ERR_INVALID_ARG, "unknown dtype");
  if (dtype == OPRAG_F32 && src_dtype == OPRAG_BF16)
    return fail(OPRAG_ERR_INVALID_ARG, "bf16 input into an f32 index is not supported");

  oprag_index* idx = new (std::nothrow) oprag_index();
  if (!idx) return fail(OPRAG_ERR_OOM, "host allocation");
  cudaGetLastError();
  cudaError_t e = cudaGetDevice(&idx->device);
  if (e != cudaSuccess) {
    delete idx;
    return cuda_fail(e, "no CUDA device");
  }
  cudaDeviceGetAttribute(&idx->num_sms, cudaDevAttrMultiProcessorCount, idx->device);
  idx->n = n;
  idx->cap = n;
  idx->d = d;
  idx->dtype = dtype;
  const size_t count = static_cast<size_t>(n) * d;
  const size_t bytes = count * elem_size(dtype);
  auto bail = [&](int rc) {
    oprag_index_destroy(idx);
    return rc;
  };
  if (cudaMalloc(&idx->emb, bytes) != cudaSuccess) {
    cudaGetLastError();
    idx->emb = nullptr;
    return bail(fail(OPRAG_ERR_OOM, "cannot allocate %zu bytes for the index", bytes));
  }
  if (cudaMalloc(reinterpret_cast<void**>(&idx->dev_err), sizeof(int)) != cudaSuccess) {
    cudaGetLastError();
    idx->dev_err = nullptr;
    return bail(fail(OPRAG_ERR_OOM, "cannot allocate the error word"));
  }
  if (cudaMallocHost(reinterpret_cast<void**>(&idx->err_host), sizeof(int)) != cudaSuccess) {
    cudaGetLastError();
    idx->err_host = nullptr;
    return bail(fail(OPRAG_ERR_OOM, "cannot allocate the pinned error word"));
  }
  *idx->err_host = 0;
  if ((e = cudaEventCreateWithFlags(&idx->done, cudaEventDisableTiming)) != cudaSuccess)
    return bail(cuda_fail(e, "event"));
  cudaStream_t st;
  if ((e = cudaStreamCreateWithFlags(&st, cudaStreamNonBlocking)) != cudaSuccess)
    return bail(cuda_fail(e, "stream"));
  e = cudaMemsetAsync(idx->dev_err, 0, sizeof(int), st);
  if (e == cudaSuccess) {
    if (src_dtype == dtype) {
      e = cudaMemcpyAsync(idx->emb, emb, bytes, emb_on_device ? cudaMemcpyDeviceToDevice
                                                              : cudaMemcpyHostToDevice, st);
    } else if (emb_on_device) {
      e = launch_convert_f32_bf16(static_cast<const float*>(emb), idx->emb, count, st);
    } else {
      // Host fp32 -> device staging in slices -> bf16 rounding kernel.
      const size_t slice = std::min<size_t>(count, size_t(1) << 26);
      float* tmp = nullptr;
      e = cudaMalloc(&tmp, slice * sizeof(float));
      for (size_t off = 0; e == cudaSuccess && off < count; off += slice) {
        const size_t c = std::min(slice, count - off);
        e = cudaMemcpyAsync(tmp, static_cast<const float*>(emb) + off, c * sizeof(float),
                            cudaMemcpyHostToDevice, st);
        if (e == cudaSuccess)
          e = launch_convert_f32_bf16(tmp, static_cast<uint16_t*>(idx->emb) + off, c, st);
        if (e == cudaSuccess) e = cudaStreamSynchronize(st);
      }
      if (tmp) cudaFree(tmp);
    }
  }
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  cudaStreamDestroy(st);
  if (e != cudaSuccess) return bail(cuda_fail(e, "copying the embeddings"));
  if ((e = cudaEventRecord(idx->done, 0)) != cudaSuccess) return bail(cuda_fail(e, "event"));
  *out = idx;
  return ok();
}

void oprag_index_destroy(oprag_index* idx) {
  if (!idx) return;
  DeviceGuard g(idx->device);
  idx->drain();
  if (idx->emb) cudaFree(idx->emb);
  if (idx->dev_err) cudaFree(idx->dev_err);
  if (idx->err_host) cudaFreeHost(idx->err_host);
  if (idx->gcache.exec) cudaGraphExecDestroy(idx->gcache.exec);
  if (idx->scratch) cudaFree(idx->scratch);
  if (idx->qfloor) cudaFree(idx->qfloor);
  if (idx->phases) cudaFree(idx->phases);
  if (idx->lex) cudaFree(idx->lex);
  if (idx->cand) cudaFree(idx->cand);
  if (idx->stage) cudaFree(idx->stage);
  idx->free_sparse();
  if (idx->done) cudaEventDestroy(idx->done);
  for (cudaEvent_t ev : idx->ev)
    if (ev) cudaEventDestroy(ev);
  delete idx;
}

int oprag_index_info(const oprag_index* idx, int64_t* n, int32_t* d, int32_t* dtype,
                     int32_t* device) {
  if (!idx) return fail(OPRAG_ERR_INVALID_ARG, "index is NULL");
  if (n) *n = idx->n;
  if (d) *d = idx->d;
  if (dtype) *dtype = idx->dtype;
  if (device) *device = idx->device;
  return ok();
}

const void* oprag_index_data(const oprag_index* idx) { return idx ? idx->emb : nullptr; }

int oprag_index_get_rows(const oprag_index* idx, int64_t first, int64_t count, void* out) {
  if (!idx || !out) return fail(OPRAG_ERR_INVALID_ARG, "NULL argument");
  if (first < 0 || count < 0 || first + count > idx->n)
    return fail(OPRAG_ERR_RANGE, "rows [%lld, %lld) outside the index", (long long)first,
                (long long)(first + count));
  DeviceGuard g(idx->device);
  const_cast<oprag_index*>(idx)->drain();
  const size_t row = static_cast<size_t>(idx->d) * elem_size(idx->dtype);
  cudaError_t e = cudaMemcpy(out, static_cast<const char*>(idx->emb) + first * row, count * row,
                             cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_fail(e, "reading rows");
  return ok();
}

int oprag_index_reserve(oprag_index* idx, int32_t q_max, int32_t k_max) {
  if (!idx) return fail(OPRAG_ERR_INVALID_ARG, "index is NULL");
  if (q_max < 1 || k_max < 1 || k_max > OPRAG_K_MAX)
    return fail(OPRAG_ERR_INVALID_ARG, "bad reservation q_max=%d k_max=%d", q_max, k_max);
  DeviceGuard g(idx->device);
  const int kcap = static_cast<int>(std::min<int64_t>({k_max, idx->n, OPRAG_K_MAX}));
  // Every layout a search of up to q_max queries and k_max results may take:
  // each list length up to k_max's, both kernel families, every forced tile
  // width and CTA mode, and a single query tile (whose plan differs).
  size_t need = 0;
  for (int kk : {8, 16, 32, 128, 256}) {
    const int k = std::min(kk, kcap);
    for (int qq : {static_cast<int>(q_max), std::min<int>(q_max, 128)}) {
      need = std::max(need, search_layout(idx, qq, k, 1, 0, 0).total());
      if (idx->dtype != OPRAG_BF16) continue;
      for (int bn : {0, 128, 256})
        for (int pair : {0, 1, 2, 3})
          need = std::max(need, search_layout(idx, qq, k, 2, bn, pair).total());
    }
  }
  int rc = idx->ensure(&idx->scratch, &idx->scratch_bytes, need, "search scratch");
  if (rc) return rc;
  // Shared k-th bounds of register lists: zeroed once here, so that a later
  // search of up to q_max queries neither allocates nor clears them.
  const size_t fb = static_cast<size_t>(q_max) * sizeof(uint64_t);
  if (fb > idx->qfloor_bytes) {
    rc = idx->ensure(reinterpret_cast<void**>(&idx->qfloor), &idx->qfloor_bytes, fb,
                     "shared k-th score bounds");
    if (rc) return rc;
    cudaError_t e = cudaMemset(idx->qfloor, 0, idx->qfloor_bytes);
    if (e == cudaSuccess) e = cudaDeviceSynchronize();
    if (e != cudaSuccess) return cuda_fail(e, "clearing shared bounds");
  }
  if (idx->has_sparse) {
    const size_t lb = std::max(lex_layout(idx, q_max, false).total,
                               lex_layout(idx, q_max, true).total);
    rc = idx->ensure(reinterpret_cast<void**>(&idx->lex), &idx->lex_bytes, lb, "BM25 block");
    if (rc) return rc;
    // the gathered form's searches use their own tensor-core layouts
    for (int kk : {8, 16, 32, 128, 256}) {
      const int k = std::min(kk, kcap);
      for (int qq : {static_cast<int>(q_max), std::min<int>(q_max, 128)})
        if (idx->dtype == OPRAG_BF16)
          need = std::max(need, search_layout(idx, qq, k, 2, 0, 0, true).total());
    }
    rc = idx->ensure(&idx->scratch, &idx->scratch_bytes, need, "search scratch");
    if (rc) return rc;
  }
  return ok();
}

int oprag_upsert(oprag_index* idx, const int64_t* ids, const void* rows, int64_t m,
                 int32_t rows_dtype, int32_t rows_on_device, void* stream) {
  if (!idx) return fail(OPRAG_ERR_INVALID_ARG, "index is NULL");
  if (m < 0) return fail(OPRAG_ERR_INVALID_ARG, "m < 0");
  if (m == 0) return ok();
  if (!ids || !rows) return fail(OPRAG_ERR_INVALID_ARG, "NULL ids or rows");
  if (rows_dtype != OPRAG_F32 && rows_dtype != OPRAG_BF16)
    return fail(OPRAG_ERR_INVALID_ARG, "unknown rows dtype");
  if (idx->dtype == OPRAG_F32 && rows_dtype == OPRAG_BF16)
    return fail(OPRAG_ERR_INVALID_ARG, "bf16 rows into an f32 index are not supported");
  for (int64_t i = 0; i < m; ++i)
    if (ids[i] < 0 || ids[i] >= idx->n)
      return fail(OPRAG_ERR_RANGE, "ids[%lld] = %lld outside [0, %lld)", (long long)i,
                  (long long)ids[i], (long long)idx->n);
  if (rows_on_device && (reinterpret_cast<uintptr_t>(rows) & 15))
    return fail(OPRAG_ERR_INVALID_ARG, "device rows must be 16-byte aligned");
  // The later entry of a repeated id wins: keep the last occurrence only
  // (walking backwards through an open-addressing set of the ids seen, at
  // most half full).
  std::vector<int64_t> pairs;
  pairs.reserve(2 * m);
  {
    size_t cap = 16;
    while (cap < static_cast<size_t>(m) * 2) cap <<= 1;
    std::vector<int64_t> seen(cap, -1);
    const size_t mask = cap - 1;
    for (int64_t i = m - 1; i >= 0; --i) {
      const int64_t id = ids[i];
      size_t h = (static_cast<uint64_t>(id) * 0x9E3779B97F4A7C15ull) >> 20 & mask;
      while (seen[h] != -1 && seen[h] != id) h = (h + 1) & mask;
      if (seen[h] == id) continue;
      seen[h] = id;
      pairs.push_back(i);
      pairs.push_back(id);
    }
  }
  const int64_t count = static_cast<int64_t>(pairs.size() / 2);
  DeviceGuard g(idx->device);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const size_t row_bytes = static_cast<size_t>(idx->d) * elem_size(rows_dtype);
  const size_t pair_bytes = pairs.size() * sizeof(int64_t);
  const size_t pair_off = 0;
  const size_t rows_off = (pair_bytes + 255) / 256 * 256;
  const size_t need = rows_off + (rows_on_device ? 0 : static_cast<size_t>(m) * row_bytes);
  int rc = idx->ensure(&idx->stage, &idx->stage_bytes, need, "upsert staging");
  if (rc) return rc;
  if ((rc = begin_call(idx, st))) return rc;
  char* stage = static_cast<char*>(idx->stage);
  cudaError_t e = cudaMemcpyAsync(stage + pair_off, pairs.data(), pair_bytes,
                                  cudaMemcpyHostToDevice, st);
  const void* src = rows;
  if (e == cudaSuccess && !rows_on_device) {
    e = cudaMemcpyAsync(stage + rows_off, rows, static_cast<size_t>(m) * row_bytes,
                        cudaMemcpyHostToDevice, st);
    src = stage + rows_off;
  }
  if (e != cudaSuccess) return cuda_fail(e, "copying the upsert batch");
  e = launch_scatter_rows(idx->dtype, idx->emb, idx->d, src, rows_dtype,
                          reinterpret_cast<const int64_t*>(stage + pair_off), count, st);
  if (e != cudaSuccess) return cuda_fail(e, "upsert kernel");
  return end_call(idx, st);
}

int rebuild_sparse(oprag_index* idx);

int oprag_append(oprag_index* idx, const void* rows, int64_t m, int32_t rows_dtype,
                 int32_t rows_on_device, int64_t* first_id, void* stream) {
  if (!idx) return fail(OPRAG_ERR_INVALID_ARG, "index is NULL");
  if (m < 0) return fail(OPRAG_ERR_INVALID_ARG, "m < 0");
  if (first_id) *first_id = idx->n;
  if (m == 0) return ok();
  if (!rows) return fail(OPRAG_ERR_INVALID_ARG, "NULL rows");
  if (rows_dtype != OPRAG_F32 && rows_dtype != OPRAG_BF16)
    return fail(OPRAG_ERR_INVALID_ARG, "unknown rows dtype");
  if (idx->dtype == OPRAG_F32 && rows_dtype == OPRAG_BF16)
    return fail(OPRAG_ERR_INVALID_ARG, "bf16 rows into an f32 index are not supported");
  if (idx->n + m > (int64_t(1) << 31))
    return fail(OPRAG_ERR_INVALID_ARG, "an index holds at most 2^31 chunks");
  DeviceGuard g(idx->device);
  const int64_t n0 = idx->n;
  if (n0 + m > idx->cap) {
    // Capacity doubling: a new allocation, the rows so far copied over.
    cudaError_t e = idx->drain();
    if (e != cudaSuccess) return cuda_fail(e, "waiting for pending work");
    const int64_t cap = std::max<int64_t>(n0 + m, 2 * idx->cap);
    const size_t row_bytes = static_cast<size_t>(idx->d) * elem_size(idx->dtype);
    void* grown = nullptr;
    if (cudaMalloc(&grown, static_cast<size_t>(cap) * row_bytes) != cudaSuccess) {
      cudaGetLastError();
      return fail(OPRAG_ERR_OOM, "cannot grow the index to %lld rows", (long long)cap);
    }
    e = cudaMemcpy(grown, idx->emb, static_cast<size_t>(n0) * row_bytes, cudaMemcpyDeviceToDevice);
    if (e != cudaSuccess) {
      cudaFree(grown);
      return cuda_fail(e, "copying the index");
    }
    cudaFree(idx->emb);
    idx->emb = grown;
    idx->cap = cap;
  }
  idx->n = n0 + m;
  ++idx->state_version;
  std::vector<int64_t> ids(static_cast<size_t>(m));
  for (int64_t i = 0; i < m; ++i) ids[i] = n0 + i;
  int rc = oprag_upsert(idx, ids.data(), rows, m, rows_dtype, rows_on_device, stream);
  if (rc) {
    idx->n = n0;
    return rc;
  }
  if (idx->has_sparse) {
    // The new chunks hold no terms yet (oprag_index_update_sparse gives them
    // bags); N and avgdl change, so every BM25 weight is rebuilt.
    cudaError_t e = cudaStreamSynchronize(static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "appending rows");
    idx->bag_ptr.resize(static_cast<size_t>(idx->n) + 1, idx->bag_ptr.back());
    return rebuild_sparse(idx);
  }
  return ok();
}

int oprag_search_two(oprag_index* knowledge, oprag_index* memory, const void* queries, int32_t q,
                     int32_t k, int64_t* out_ids, int32_t* out_src, float* out_scores,
                     void* stream) {
  if (!knowledge || !memory) return fail(OPRAG_ERR_INVALID_ARG, "index is NULL");
  if (knowledge->d != memory->d || knowledge->dtype != memory->dtype ||
      knowledge->device != memory->device)
    return fail(OPRAG_ERR_INVALID_ARG, "the two indices differ in dim, dtype or device");
  if (!out_src) return fail(OPRAG_ERR_INVALID_ARG, "NULL out_src");
  if (k < 1 || k > OPRAG_K_MAX || k > knowledge->n + memory->n)
    return fail(OPRAG_ERR_INVALID_ARG, "k = %d outside [1, min(%d, n_knowledge + n_memory)]", k,
                OPRAG_K_MAX);
  if (q < 0) return fail(OPRAG_ERR_INVALID_ARG, "q < 0");
  if (q == 0) return ok();
  if (!queries || !out_ids || !out_scores) return fail(OPRAG_ERR_INVALID_ARG, "NULL argument");
  DeviceGuard g(knowledge->device);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  int rc;
  if (choose_path(knowledge, q) == 2 && choose_path(memory, q) == 2) {
    // One search over both (Sec. 3.6 / Sec. 4.4: the two indices searched the
    // same way into one ranking): the memory index's corpus tiles follow the
    // knowledge index's in the same launches, its chunks keyed after the
    // knowledge ids, so equal scores rank knowledge first; the merge writes
    // the source and the id within it.  Scratch and bounds of the knowledge
    // index.
    const SearchLayout L = search_layout(knowledge, q, k, 2, knowledge->opt_block_n,
                                         knowledge->opt_pair, false, memory->n);
    if ((rc = knowledge->ensure(&knowledge->scratch, &knowledge->scratch_bytes, L.total(),
                                "search scratch")))
      return rc;
    uint64_t* qf = nullptr;
    uint32_t gen = 0;
    if (L.floors && (rc = shared_floors(knowledge, q, st, &qf, &gen))) return rc;
    if ((rc = begin_call(knowledge, st))) return rc;
    if ((rc = begin_call(memory, st))) return rc;
    const Fusion none{nullptr, 0, nullptr, 0.f};
    knowledge->timed_lex = false;
    if ((rc = launch_search(knowledge, L, queries, q, k, none, knowledge->scratch, qf, gen, out_ids,
                            out_scores, st, memory->emb, memory->n, out_src)))
      return rc;
    if ((rc = end_call(memory, st))) return rc;
    return end_call(knowledge, st);
  }
  // fp32 indices (SIMT kernel): each index's top-k, then one two-list merge.
  const int ka = static_cast<int>(std::min<int64_t>(k, knowledge->n));
  const int kb = static_cast<int>(std::min<int64_t>(k, memory->n));
  if ((rc = knowledge->ensure(&knowledge->cand, &knowledge->cand_bytes,
                              static_cast<size_t>(q) * ka * 12, "two-index results")))
    return rc;
  if ((rc = memory->ensure(&memory->cand, &memory->cand_bytes,
                           static_cast<size_t>(q) * kb * 12, "two-index results")))
    return rc;
  if ((rc = begin_call(knowledge, st))) return rc;
  if ((rc = begin_call(memory, st))) return rc;
  int64_t* a_ids = static_cast<int64_t*>(knowledge->cand);
  float* a_sc = reinterpret_cast<float*>(a_ids + static_cast<size_t>(q) * ka);
  int64_t* b_ids = static_cast<int64_t*>(memory->cand);
  float* b_sc = reinterpret_cast<float*>(b_ids + static_cast<size_t>(q) * kb);
  const Fusion none{nullptr, 0, nullptr, 0.f};
  if ((rc = run_search(knowledge, queries, q, ka, none, a_ids, a_sc, st))) return rc;
  if ((rc = run_search(memory, queries, q, kb, none, b_ids, b_sc, st))) return rc;
  cudaError_t e = launch_merge_two(q, a_ids, a_sc, ka, b_ids, b_sc, kb, k, out_ids, out_src,
                                   out_scores, st);
  if (e != cudaSuccess) return cuda_fail(e, "two-index merge");
  if ((rc = end_call(memory, st))) return rc;
  return end_call(knowledge, st);
}

int oprag_search(oprag_index* idx, const void* queries, int32_t q, int32_t k, int64_t* out_ids,
                 float* out_scores, void* stream) {
  int rc = check_search_args(idx, queries, q, k, out_ids, out_scores);
  if (rc) return rc;
  if (q == 0) return ok();
  DeviceGuard g(idx->device);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  if ((rc = begin_call(idx, st))) return rc;
  const Fusion none{nullptr, 0, nullptr, 0.f};
  idx->timed_lex = false;
  // Graph mode: a search repeated with the same pointers, sizes, stream and
  // index state is captured once (on its second call) and then replayed
  // with one graph launch.  Not on the legacy default stream (no capture).
  auto& c = idx->gcache;
  if (idx->opt_graph && st != nullptr && !idx->timing) {
    const bool same = c.seen && c.queries == queries && c.q == q && c.k == k &&
                      c.ids == out_ids && c.scores == out_scores && c.st == st &&
                      c.version == idx->state_version;
    if (same && c.exec) {
      cudaError_t e = cudaGraphLaunch(c.exec, st);
      if (e != cudaSuccess) return cuda_fail(e, "graph launch");
      return end_call(idx, st);
    }
    if (same) {
      cudaError_t e = cudaStreamBeginCapture(st, cudaStreamCaptureModeThreadLocal);
      if (e == cudaSuccess) {
        idx->capturing = true;
        rc = run_search(idx, queries, q, k, none, out_ids, out_scores, st);
        idx->capturing = false;
        cudaGraph_t graph = nullptr;
        e = cudaStreamEndCapture(st, &graph);
        cudaGraphExec_t exec = nullptr;
        if (rc == OPRAG_OK && e == cudaSuccess && graph)
          e = cudaGraphInstantiate(&exec, graph, 0);
        if (graph) cudaGraphDestroy(graph);
        if (rc == OPRAG_OK && e == cudaSuccess && exec) {
          c.exec = exec;
          if ((e = cudaGraphLaunch(exec, st)) != cudaSuccess) return cuda_fail(e, "graph launch");
          return end_call(idx, st);
        }
        if (exec) cudaGraphExecDestroy(exec);
        cudaGetLastError();
      } else {
        cudaGetLastError();
      }
      c.seen = false;            // this search does not capture: launch it directly
    } else {
      if (c.exec) cudaGraphExecDestroy(c.exec);
      c.exec = nullptr;
      c.seen = true;
      c.queries = queries;
      c.q = q;
      c.k = k;
      c.ids = out_ids;
      c.scores = out_scores;
      c.st = st;
      c.version = idx->state_version;
    }
  }
  if ((rc = run_search(idx, queries, q, k, none, out_ids, out_scores, st))) return rc;
  return end_call(idx, st);
}

int oprag_search_host(oprag_index* idx, const void* queries, int32_t q, int32_t k,
                      int64_t* out_ids, float* out_scores, void* stream) {
  int rc = check_search_args(idx, queries, q, k, out_ids, out_scores);
  if (rc) return rc;
  if (q == 0) return ok();
  DeviceGuard g(idx->device);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const size_t qbytes = static_cast<size_t>(q) * idx->d * elem_size(idx->dtype);
  const size_t q_off = 0;
  const size_t id_off = (qbytes + 255) / 256 * 256;
  const size_t sc_off = id_off + (static_cast<size_t>(q) * k * sizeof(int64_t) + 255) / 256 * 256;
  const size_t need = sc_off + static_cast<size_t>(q) * k * sizeof(float);
  if ((rc = idx->ensure(&idx->stage, &idx->stage_bytes, need, "search staging"))) return rc;
  if ((rc = begin_call(idx, st))) return rc;
  char* stage = static_cast<char*>(idx->stage);
  cudaError_t e = cudaMemcpyAsync(stage + q_off, queries, qbytes, cudaMemcpyHostToDevice, st);
  if (e != cudaSuccess) return cuda_fail(e, "copying queries");
  const Fusion none{nullptr, 0, nullptr, 0.f};
  if ((rc = run_search(idx, stage + q_off, q, k, none, reinterpret_cast<int64_t*>(stage + id_off),
                       reinterpret_cast<float*>(stage + sc_off), st)))
    return rc;
  e = cudaMemcpyAsync(out_ids, stage + id_off, static_cast<size_t>(q) * k * sizeof(int64_t),
                      cudaMemcpyDeviceToHost, st);
  if (e == cudaSuccess)
    e = cudaMemcpyAsync(out_scores, stage + sc_off, static_cast<size_t>(q) * k * sizeof(float),
                        cudaMemcpyDeviceToHost, st);
  // The error word travels with the results, so that the call waits for the
  // device once.
  if (e == cudaSuccess)
    e = cudaMemcpyAsync(idx->err_host, idx->dev_err, sizeof(int), cudaMemcpyDeviceToHost, st);
  if (e != cudaSuccess) return cuda_fail(e, "copying results");
  if ((rc = end_call(idx, st))) return rc;
  if ((e = cudaStreamSynchronize(st)) != cudaSuccess) return cuda_fail(e, "search");
  return *idx->err_host != 0 ? oprag_index_check(idx) : ok();
}

// Builds the device side of BM25 from the index's host copy of the token
// bags.  Called whenever the bags or the chunk count change, so that df,
// avgdl and every weight follow the current corpus.  The host does the
// integer work -- a stable counting sort of the bags into a term-major
// inverted index of (chunk, tf) pairs, chunks ascending, on several threads
// over contiguous chunk ranges; document frequencies, lengths, idf and the
// terms' storage classes -- and the device computes every weight from it
// (launch_lex_build).
int rebuild_sparse(oprag_index* idx) {
  const int64_t n = idx->n;
  const int vocab = idx->vocab;
  const double k1 = idx->bm_k1, b = idx->bm_b;
  const int32_t* doc_indptr = idx->bag_ptr.data();
  const int32_t* doc_terms = idx->bag_terms.data();
  const int64_t total = doc_indptr[n];

  // Pass 1: per thread (a contiguous range of chunks), the number of chunks
  // holding each term.  Pass 2: each thread writes its (chunk, tf) pairs at
  // its own offsets inside each term's range, so chunks stay ascending.
  const int T = static_cast<int>(std::max<int64_t>(
      1, std::min<int64_t>({static_cast<int64_t>(std::thread::hardware_concurrency()), 16,
                            (n + 1023) / 1024})));
  std::vector<std::vector<int64_t>> cnt(T, std::vector<int64_t>(vocab, 0));
  auto chunk_range = [&](int th, int64_t* d0, int64_t* d1) {
    *d0 = n * th / T;
    *d1 = n * (th + 1) / T;
  };
  // Per distinct term of chunk dd: f(term, tf), in first-occurrence order.
  auto each_term = [&](int64_t dd, std::vector<int32_t>& last, std::vector<int32_t>& tfc,
                       std::vector<int32_t>& seen, auto&& f) {
    seen.clear();
    for (int32_t i = doc_indptr[dd]; i < doc_indptr[dd + 1]; ++i) {
      const int32_t t = doc_terms[i];
      if (last[t] != static_cast<int32_t>(dd)) {
        last[t] = static_cast<int32_t>(dd);
        tfc[t] = 0;
        seen.push_back(t);
      }
      ++tfc[t];
    }
    for (int32_t t : seen) f(t, tfc[t]);
  };
  auto run = [&](auto&& body) {
    std::vector<std::thread> pool;
    for (int th = 1; th < T; ++th) pool.emplace_back(body, th);
    body(0);
    for (auto& p : pool) p.join();
  };
  run([&](int th) {
    int64_t d0, d1;
    chunk_range(th, &d0, &d1);
    std::vector<int32_t> last(vocab, -1), tfc(vocab, 0), seen;
    for (int64_t dd = d0; dd < d1; ++dd)
      each_term(dd, last, tfc, seen, [&](int32_t t, int32_t) { ++cnt[th][t]; });
  });
  std::vector<int64_t> df(vocab, 0), term_start(static_cast<size_t>(vocab) + 1, 0);
  for (int t = 0; t < vocab; ++t) {
    for (int th = 0; th < T; ++th) df[t] += cnt[th][t];
    term_start[t + 1] = term_start[t] + df[t];
  }
  const int64_t nnz_all = term_start[vocab];
  // cnt becomes each thread's write offset per term
  for (int t = 0; t < vocab; ++t) {
    int64_t off = term_start[t];
    for (int th = 0; th < T; ++th) {
      const int64_t c = cnt[th][t];
      cnt[th][t] = off;
      off += c;
    }
  }
  std::vector<int2> inv(static_cast<size_t>(std::max<int64_t>(nnz_all, 1)));
  run([&](int th) {
    int64_t d0, d1;
    chunk_range(th, &d0, &d1);
    std::vector<int32_t> last(vocab, -1), tfc(vocab, 0), seen;
    for (int64_t dd = d0; dd < d1; ++dd)
      each_term(dd, last, tfc, seen, [&](int32_t t, int32_t tf) {
        inv[cnt[th][t]++] = make_int2(static_cast<int32_t>(dd), tf);
      });
  });
  std::vector<int32_t> doc_len(static_cast<size_t>(std::max<int64_t>(n, 1)));
  for (int64_t dd = 0; dd < n; ++dd) doc_len[dd] = doc_indptr[dd + 1] - doc_indptr[dd];
  const double avgdl = n > 0 ? static_cast<double>(total) / static_cast<double>(n) : 0.0;
  const double N = static_cast<double>(n);
  std::vector<double> idf(vocab);
  for (int t = 0; t < vocab; ++t) {
    const double dft = static_cast<double>(df[t]);
    idf[t] = std::log(1.0 + (N - dft + 0.5) / (dft + 0.5));
  }

  // Terms in more than half of the chunks become dense rows of the BM25 pass
  // and the rerank; the others keep postings grouped by term, chunks
  // ascending inside a term.
  std::vector<int32_t> slot(vocab, -1);
  int n_dense = 0;
  for (int t = 0; t < vocab; ++t)
    if (2 * df[t] > n) slot[t] = n_dense++;
  // Classes of the gathered hybrid search's epilogue.  Terms held by at least
  // 1/32 of the chunks, commonest first: the first kLexHeadTerms are scored
  // on tensor cores (class s = their slot), the next ones read as fp32 rows
  // of weights (class -2 - row; every dense-row term without a tensor-core
  // slot is one, the others while the rows stay within kLexMidBytes); all
  // other terms (class -1) are walked in their postings, under one posting
  // per 32 chunks on average.
  constexpr int64_t kLexMidBytes = int64_t(64) << 20;
  const int64_t dld = (n + 3) / 4 * 4;
  const int64_t mld = (n + 127) / 128 * 128;   // mid rows: whole 128-row tiles
  std::vector<int32_t> lex_class(vocab, -1);
  int n_tc = 0, n_mid = 0;
  {
    const int64_t floor_df = std::max<int64_t>(1, (n + 31) / 32);
    std::vector<int32_t> order;
    for (int t = 0; t < vocab; ++t)
      if (df[t] >= floor_df) order.push_back(t);
    std::stable_sort(order.begin(), order.end(),
                     [&](int32_t x, int32_t y) { return df[x] > df[y]; });
    const int64_t mid_cap = kLexMidBytes / (mld * 4);
    for (int32_t t : order) {
      if (n_tc < kLexHeadTerms) lex_class[t] = n_tc++;
      else if (slot[t] >= 0 || n_mid < mid_cap) lex_class[t] = -2 - n_mid++;
    }
  }
  std::vector<int64_t> ptr(static_cast<size_t>(vocab) + 1, 0);
  for (int t = 0; t < vocab; ++t) ptr[t + 1] = ptr[t] + (slot[t] < 0 ? df[t] : 0);
  const int64_t nnz = ptr[vocab];
  if (nnz >= (int64_t(1) << 31) || nnz_all >= (int64_t(1) << 31))
    return fail(OPRAG_ERR_INVALID_ARG, "more than 2^31 postings");
  const int ntiles = static_cast<int>((n + kBm25DocTile - 1) / kBm25DocTile);

  DeviceGuard g(idx->device);
  cudaError_t e = idx->drain();
  if (e != cudaSuccess) return cuda_fail(e, "waiting for pending work");
  idx->free_sparse();
  idx->has_sparse = false;
  const size_t dense_elems = std::max<size_t>(static_cast<size_t>(n_dense) * dld, 4);
  const size_t wsplit_elems = static_cast<size_t>(n) * kLexK;
  const size_t mid_elems = static_cast<size_t>(std::max(n_mid, 1)) * mld;
  const size_t tptr_elems = static_cast<size_t>(vocab) * (ntiles + 1);
  // temporaries of the build: the inverted index, term offsets, idf, lengths
  int2* d_inv = nullptr;
  int64_t* d_start = nullptr;
  double* d_idf = nullptr;
  int32_t* d_len = nullptr;
  auto free_tmp = [&]() {
    if (d_inv) cudaFree(d_inv);
    if (d_start) cudaFree(d_start);
    if (d_idf) cudaFree(d_idf);
    if (d_len) cudaFree(d_len);
  };
  if (cudaMalloc(&idx->post_ptr, ptr.size() * sizeof(int64_t)) != cudaSuccess ||
      cudaMalloc(&idx->post, std::max<int64_t>(nnz, 1) * sizeof(int2)) != cudaSuccess ||
      cudaMalloc(&idx->dense_slot, slot.size() * sizeof(int32_t)) != cudaSuccess ||
      cudaMalloc(&idx->dense_w, dense_elems * sizeof(float)) != cudaSuccess ||
      cudaMalloc(&idx->tile_ptr, tptr_elems * sizeof(int64_t)) != cudaSuccess ||
      cudaMalloc(&idx->wsplit, wsplit_elems * sizeof(uint16_t)) != cudaSuccess ||
      cudaMalloc(&idx->lex_class, lex_class.size() * sizeof(int32_t)) != cudaSuccess ||
      cudaMalloc(&idx->mid_w, mid_elems * sizeof(float)) != cudaSuccess ||
      cudaMalloc(&d_inv, inv.size() * sizeof(int2)) != cudaSuccess ||
      cudaMalloc(&d_start, term_start.size() * sizeof(int64_t)) != cudaSuccess ||
      cudaMalloc(&d_idf, idf.size() * sizeof(double)) != cudaSuccess ||
      cudaMalloc(&d_len, doc_len.size() * sizeof(int32_t)) != cudaSuccess) {
    cudaGetLastError();
    free_tmp();
    idx->free_sparse();
    return fail(OPRAG_ERR_OOM, "cannot allocate postings");
  }
  e = cudaMemcpy(idx->post_ptr, ptr.data(), ptr.size() * sizeof(int64_t), cudaMemcpyHostToDevice);
  if (e == cudaSuccess)
    e = cudaMemcpy(idx->dense_slot, slot.data(), slot.size() * sizeof(int32_t), cudaMemcpyHostToDevice);
  if (e == cudaSuccess)
    e = cudaMemcpy(idx->lex_class, lex_class.data(), lex_class.size() * sizeof(int32_t),
                   cudaMemcpyHostToDevice);
  if (e == cudaSuccess)
    e = cudaMemcpy(d_inv, inv.data(), inv.size() * sizeof(int2), cudaMemcpyHostToDevice);
  if (e == cudaSuccess)
    e = cudaMemcpy(d_start, term_start.data(), term_start.size() * sizeof(int64_t),
                   cudaMemcpyHostToDevice);
  if (e == cudaSuccess)
    e = cudaMemcpy(d_idf, idf.data(), idf.size() * sizeof(double), cudaMemcpyHostToDevice);
  if (e == cudaSuccess)
    e = cudaMemcpy(d_len, doc_len.data(), doc_len.size() * sizeof(int32_t), cudaMemcpyHostToDevice);
  if (e == cudaSuccess) e = cudaMemset(idx->dense_w, 0, dense_elems * sizeof(float));
  if (e == cudaSuccess) e = cudaMemset(idx->wsplit, 0, wsplit_elems * sizeof(uint16_t));
  if (e == cudaSuccess) e = cudaMemset(idx->mid_w, 0, mid_elems * sizeof(float));
  if (e == cudaSuccess) {
    const LexBuild lb{vocab,        d_inv,           d_start,     d_idf,
                      d_len,        avgdl,           k1,          b,
                      idx->dense_slot, idx->lex_class, idx->post_ptr, idx->post,
                      idx->dense_w, dld,
                      reinterpret_cast<__nv_bfloat16*>(idx->wsplit), idx->mid_w, mld};
    e = launch_lex_build(lb, ntiles, idx->tile_ptr, nullptr);
  }
  if (e == cudaSuccess) e = cudaDeviceSynchronize();
  free_tmp();
  if (e != cudaSuccess) {
    idx->free_sparse();
    return cuda_fail(e, "building the lexical index");
  }
  idx->nnz = nnz;
  idx->dense_ld = dld;
  idx->mid_ld = mld;
  idx->ntiles = ntiles;
  idx->has_sparse = true;
  return ok();
}

// Term ids of bags must lie in [0, vocab).
int check_bags(const int32_t* indptr, const int32_t* terms, int64_t count, int vocab) {
  if (indptr[0] != 0) return fail(OPRAG_ERR_INVALID_ARG, "bag indptr[0] != 0");
  for (int64_t i = 0; i < count; ++i)
    if (indptr[i + 1] < indptr[i])
      return fail(OPRAG_ERR_INVALID_ARG, "bag indptr decreases at %lld", (long long)i);
  const int64_t total = indptr[count];
  if (total > 0 && !terms) return fail(OPRAG_ERR_INVALID_ARG, "bag terms is NULL");
  for (int64_t p = 0; p < total; ++p)
    if (terms[p] < 0 || terms[p] >= vocab)
      return fail(OPRAG_ERR_INVALID_ARG, "term id %d outside [0, %d)", terms[p], vocab);
  return OPRAG_OK;
}

int oprag_index_set_sparse(oprag_index* idx, const int32_t* doc_indptr, const int32_t* doc_terms,
                           int32_t vocab, float k1, float b) {
  if (!idx || !doc_indptr) return fail(OPRAG_ERR_INVALID_ARG, "NULL argument");
  if (vocab < 1) return fail(OPRAG_ERR_INVALID_ARG, "vocab = %d", vocab);
  if (!(k1 >= 0.f) || !(b >= 0.f && b <= 1.f))
    return fail(OPRAG_ERR_INVALID_ARG, "need k1 >= 0 and 0 <= b <= 1");
  int rc = check_bags(doc_indptr, doc_terms, idx->n, vocab);
  if (rc) return rc;
  const int64_t total = doc_indptr[idx->n];
  idx->bag_ptr.assign(doc_indptr, doc_indptr + idx->n + 1);
  idx->bag_terms.assign(doc_terms, doc_terms + total);
  idx->vocab = vocab;
  idx->bm_k1 = k1;
  idx->bm_b = b;
  return rebuild_sparse(idx);
}

int oprag_index_update_sparse(oprag_index* idx, const int64_t* ids, int64_t m,
                              const int32_t* bag_indptr, const int32_t* bag_terms) {
  if (!idx) return fail(OPRAG_ERR_INVALID_ARG, "index is NULL");
  if (!idx->has_sparse) return fail(OPRAG_ERR_NOT_READY, "no sparse side: call oprag_index_set_sparse");
  if (m < 0) return fail(OPRAG_ERR_INVALID_ARG, "m < 0");
  if (m == 0) return ok();
  if (!ids || !bag_indptr) return fail(OPRAG_ERR_INVALID_ARG, "NULL argument");
  for (int64_t i = 0; i < m; ++i)
    if (ids[i] < 0 || ids[i] >= idx->n)
      return fail(OPRAG_ERR_RANGE, "ids[%lld] = %lld outside [0, %lld)", (long long)i,
                  (long long)ids[i], (long long)idx->n);
  int rc = check_bags(bag_indptr, bag_terms, m, idx->vocab);
  if (rc) return rc;
  // New bags: the last occurrence of a repeated id wins.
  std::vector<int64_t> which(static_cast<size_t>(idx->n), -1);
  for (int64_t i = 0; i < m; ++i) which[ids[i]] = i;
  std::vector<int32_t> ptr(static_cast<size_t>(idx->n) + 1, 0), terms;
  terms.reserve(idx->bag_terms.size());
  for (int64_t dd = 0; dd < idx->n; ++dd) {
    const int64_t w = which[dd];
    if (w < 0)
      terms.insert(terms.end(), idx->bag_terms.begin() + idx->bag_ptr[dd],
                   idx->bag_terms.begin() + idx->bag_ptr[dd + 1]);
    else
      terms.insert(terms.end(), bag_terms + bag_indptr[w], bag_terms + bag_indptr[w + 1]);
    if (terms.size() > static_cast<size_t>(INT32_MAX))
      return fail(OPRAG_ERR_INVALID_ARG, "token bags exceed 2^31 terms");
    ptr[dd + 1] = static_cast<int32_t>(terms.size());
  }
  idx->bag_ptr.swap(ptr);
  idx->bag_terms.swap(terms);
  return rebuild_sparse(idx);
}

int oprag_hybrid_search(oprag_index* idx, const void* queries, int32_t q, const int32_t* q_indptr,
                        const int32_t* q_terms, float alpha, int32_t k, int64_t* out_ids,
                        float* out_scores, void* stream) {
  int rc = check_search_args(idx, queries, q, k, out_ids, out_scores);
  if (rc) return rc;
  if (!idx->has_sparse) return fail(OPRAG_ERR_NOT_READY, "no sparse side: call oprag_index_set_sparse");
  if (q == 0) return ok();
  if (!q_indptr || !q_terms) return fail(OPRAG_ERR_INVALID_ARG, "NULL query terms");
  if (!std::isfinite(alpha)) return fail(OPRAG_ERR_INVALID_ARG, "alpha is not finite");
  DeviceGuard g(idx->device);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const int path = choose_path(idx, q);
  const bool gather = path == 2 && idx->opt_lex_gather;
  const LexLayout LL = lex_layout(idx, q, gather);
  if ((rc = idx->ensure(reinterpret_cast<void**>(&idx->lex), &idx->lex_bytes, LL.total,
                        "BM25 block")))
    return rc;
  if ((rc = begin_call(idx, st))) return rc;
  const SparseIndex sp{idx->vocab,      idx->nnz,     idx->post_ptr, idx->post,
                       idx->dense_slot, idx->dense_w, idx->dense_ld, idx->tile_ptr,
                       idx->ntiles};
  char* lex = reinterpret_cast<char*>(idx->lex);
  if (gather) {
    // Gathered form (Sec. 4.4 fusion in the dense epilogue): per-query
    // operands, then a pass for each query's BM25 maximum over the corpus
    // (no BM25 block is written), then the fused search.
    if (idx->timing) cudaEventRecord(idx->ev[0], st);
    idx->timed_lex = idx->timing;
    float* bm_max = reinterpret_cast<float*>(lex + LL.max);
    const LexPrep prep{lex + LL.qcount, reinterpret_cast<int4*>(lex + LL.terms),
                       reinterpret_cast<int*>(lex + LL.term_cnt),
                       reinterpret_cast<int2*>(lex + LL.mid), reinterpret_cast<int*>(lex + LL.mid_cnt),
                       reinterpret_cast<int*>(lex + LL.ovf)};
    cudaError_t e = launch_lex_prep(idx->lex_class, idx->post_ptr, idx->vocab, q_indptr, q_terms,
                                    q, prep, st);
    if (e == cudaSuccess)
      e = launch_bm25_matrix(sp, idx->n, q_indptr, q_terms, q, nullptr, 0, bm_max, st);
    if (e != cudaSuccess) return cuda_fail(e, "BM25 maximum pass");
    Fusion fu{nullptr, 0, bm_max, alpha};
    fu.lex_qcount = prep.qcount;
    fu.lex_wsplit = idx->wsplit;
    fu.lex_terms = prep.terms;
    fu.lex_term_cnt = prep.term_cnt;
    fu.lex_mid = prep.mid;
    fu.lex_mid_cnt = prep.mid_cnt;
    fu.lex_ovf = prep.ovf;
    fu.lex_post = idx->post;
    fu.mid_w = idx->mid_w;
    fu.mid_ld = idx->mid_ld;
    fu.q_indptr = q_indptr;
    fu.q_terms = q_terms;
    fu.lex_class = idx->lex_class;
    fu.post_ptr = idx->post_ptr;
    fu.vocab = idx->vocab;
    if ((rc = run_search(idx, queries, q, k, fu, out_ids, out_scores, st))) return rc;
    return end_call(idx, st);
  }
  // Materialised form (the default): the BM25 block of up to qchunk queries
  // is written by the BM25 pass and read by the search's fused selection.
  // Measured on 32768 x 768 with 1024 queries of 8 Zipf terms, it takes
  // 201 us per search against 841 us for the gathered form.
  const int64_t ld = (idx->n + 3) / 4 * 4;
  const size_t qrow = static_cast<size_t>(idx->d) * elem_size(idx->dtype);
  for (int c0 = 0; c0 < q; c0 += LL.qchunk) {
    const int qc = std::min(LL.qchunk, q - c0);
    float* block = idx->lex;
    float* blockmax = reinterpret_cast<float*>(lex + LL.max);
    if (idx->timing) cudaEventRecord(idx->ev[0], st);
    idx->timed_lex = idx->timing;
    cudaError_t e = launch_bm25_matrix(sp, idx->n, q_indptr + c0, q_terms, qc, block, ld,
                                       blockmax, st);
    if (e != cudaSuccess) return cuda_fail(e, "BM25 kernel");
    const Fusion fu{block, ld, blockmax, alpha};
    if ((rc = run_search(idx, static_cast<const char*>(queries) + c0 * qrow, qc, k, fu,
                         out_ids + static_cast<size_t>(c0) * k,
                         out_scores + static_cast<size_t>(c0) * k, st)))
      return rc;
  }
  return end_call(idx, st);
}

int oprag_hybrid_search_dense_first(oprag_index* idx, const void* queries, int32_t q,
                                    const int32_t* q_indptr, const int32_t* q_terms, float alpha,
                                    int32_t n_cand, int32_t k, int64_t* out_ids,
                                    float* out_scores, void* stream) {
  int rc = check_search_args(idx, queries, q, k, out_ids, out_scores);
  if (rc) return rc;
  if (!idx->has_sparse) return fail(OPRAG_ERR_NOT_READY, "no sparse side: call oprag_index_set_sparse");
  if (n_cand < k || n_cand > kRerankMaxCand)
    return fail(OPRAG_ERR_INVALID_ARG, "need k <= n_cand <= %d (n_cand = %d, k = %d)",
                kRerankMaxCand, n_cand, k);
  if (q == 0) return ok();
  if (!q_indptr || !q_terms) return fail(OPRAG_ERR_INVALID_ARG, "NULL query terms");
  if (!std::isfinite(alpha)) return fail(OPRAG_ERR_INVALID_ARG, "alpha is not finite");
  // A corpus smaller than n_cand gives every chunk as a candidate.
  const int nc = static_cast<int>(std::min<int64_t>(n_cand, idx->n));
  DeviceGuard g(idx->device);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const size_t ids_bytes = static_cast<size_t>(q) * nc * sizeof(int64_t);
  if ((rc = idx->ensure(&idx->cand, &idx->cand_bytes,
                        ids_bytes + static_cast<size_t>(q) * nc * sizeof(float),
                        "dense-first candidates")))
    return rc;
  if ((rc = begin_call(idx, st))) return rc;
  int64_t* cid = static_cast<int64_t*>(idx->cand);
  float* csc = reinterpret_cast<float*>(static_cast<char*>(idx->cand) + ids_bytes);
  const Fusion none{nullptr, 0, nullptr, 0.f};
  if ((rc = run_search(idx, queries, q, nc, none, cid, csc, st))) return rc;
  const SparseIndex sp{idx->vocab,      idx->nnz,     idx->post_ptr, idx->post,
                       idx->dense_slot, idx->dense_w, idx->dense_ld, idx->tile_ptr,
                       idx->ntiles};
  cudaError_t e = launch_rerank(sp, q, nc, cid, csc, q_indptr, q_terms, alpha, k, out_ids,
                                out_scores, st);
  if (e != cudaSuccess) return cuda_fail(e, "rerank kernel");
  return end_call(idx, st);
}

int oprag_embed_pool(const void* hidden, int32_t hidden_dtype, int32_t batch, int32_t tokens,
                     int32_t dim, const uint8_t* mask, void* out, int32_t out_dtype,
                     void* stream) {
  if (hidden_dtype != OPRAG_F32 && hidden_dtype != OPRAG_BF16)
    return fail(OPRAG_ERR_INVALID_ARG, "hidden dtype %d", hidden_dtype);
  if (out_dtype != OPRAG_F32 && out_dtype != OPRAG_BF16)
    return fail(OPRAG_ERR_INVALID_ARG, "output dtype %d", out_dtype);
  if (batch < 0 || tokens < 1 || dim < 8 || dim % 8 != 0)
    return fail(OPRAG_ERR_INVALID_ARG, "need batch >= 0, tokens >= 1, dim a positive multiple of 8");
  if (dim > (hidden_dtype == OPRAG_BF16 ? 16384 : 8192))
    return fail(OPRAG_ERR_INVALID_ARG, "dim %d too large", dim);
  if (batch == 0) return ok();
  if (!hidden || !mask || !out) return fail(OPRAG_ERR_INVALID_ARG, "NULL argument");
  if ((reinterpret_cast<uintptr_t>(hidden) | reinterpret_cast<uintptr_t>(out)) % 16 != 0)
    return fail(OPRAG_ERR_INVALID_ARG, "hidden and out must be 16-byte aligned");
  cudaError_t e = launch_embed_pool(hidden_dtype == OPRAG_BF16 ? kBF16 : kF32, hidden, batch,
                                    tokens, dim, mask, out_dtype == OPRAG_BF16 ? kBF16 : kF32, out,
                                    static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "embedding tail kernel");
  return ok();
}

int oprag_index_check(oprag_index* idx) {
  if (!idx) return fail(OPRAG_ERR_INVALID_ARG, "index is NULL");
  DeviceGuard g(idx->device);
  cudaError_t e = idx->drain();
  if (e != cudaSuccess) return cuda_fail(e, "pending work");
  int flag = 0;
  e = cudaMemcpy(&flag, idx->dev_err, sizeof(int), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_fail(e, "reading the error word");
  if (flag != 0) {
    cudaMemset(idx->dev_err, 0, sizeof(int));
    return fail(OPRAG_ERR_DEVICE, "a kernel gave up a bounded wait (code %d)", flag);
  }
  return ok();
}

int oprag_index_set_option(oprag_index* idx, int32_t option, int32_t value) {
  if (!idx) return fail(OPRAG_ERR_INVALID_ARG, "index is NULL");
  ++idx->state_version;
  if (option == OPRAG_OPT_GRAPH) {
    if (value < 0 || value > 1) return fail(OPRAG_ERR_INVALID_ARG, "graph mode %d", value);
    idx->opt_graph = value;
    return ok();
  }
  if (option == OPRAG_OPT_PATH) {
    if (value < 0 || value > 2) return fail(OPRAG_ERR_INVALID_ARG, "path %d", value);
    if (value == 2 && idx->dtype != OPRAG_BF16)
      return fail(OPRAG_ERR_INVALID_ARG, "the tensor-core path needs a bf16 index");
    idx->opt_path = value;
    return ok();
  }
  if (option == OPRAG_OPT_TIMING) {
    if (value && !idx->ev[0]) {
      DeviceGuard g(idx->device);
      for (cudaEvent_t& ev : idx->ev) {
        cudaError_t e = cudaEventCreate(&ev);
        if (e != cudaSuccess) return cuda_fail(e, "timing events");
      }
    }
    idx->timing = value != 0;
    return ok();
  }
  if (option == OPRAG_OPT_LEX_GATHER) {
    if (value < 0 || value > 1) return fail(OPRAG_ERR_INVALID_ARG, "lexical form %d", value);
    idx->opt_lex_gather = value;
    return ok();
  }
  if (option == OPRAG_OPT_PHASES) {
    if (value < 0 || value > 1) return fail(OPRAG_ERR_INVALID_ARG, "phases %d", value);
    if (value) {
      DeviceGuard g(idx->device);
      // One stamp row per CTA of the largest grid (every SM, or pairs).
      const size_t need = static_cast<size_t>(2 * idx->num_sms) * kTcPhases * 8;
      int rc = idx->ensure(&idx->phases, &idx->phases_bytes, need, "phase stamps");
      if (rc) return rc;
    }
    idx->phases_on = value != 0;
    idx->phases_grid = 0;
    return ok();
  }
  if (option == OPRAG_OPT_WAIT_LIMIT) {
    if (value < 0) return fail(OPRAG_ERR_INVALID_ARG, "wait limit %d", value);
    idx->wait_limit = value;
    return ok();
  }
  if (option == OPRAG_OPT_BOUND_TAG) {
    idx->gen = static_cast<uint32_t>(value);
    return ok();
  }
  if (option == OPRAG_OPT_PAIR) {
    if (value < 0 || value > 3) return fail(OPRAG_ERR_INVALID_ARG, "pair mode %d", value);
    idx->opt_pair = value;
    return ok();
  }
  if (option == OPRAG_OPT_BLOCK_N) {
    if (value != 0 && value != 128 && value != 256)
      return fail(OPRAG_ERR_INVALID_ARG, "block_n %d", value);
    idx->opt_block_n = value;
    return ok();
  }
  return fail(OPRAG_ERR_INVALID_ARG, "unknown option %d", option);
}

int oprag_index_last_path(const oprag_index* idx) { return idx ? idx->last_path : 0; }

int oprag_index_last_launch(const oprag_index* idx, int32_t* grid, int32_t* cluster,
                            int32_t* block_n) {
  if (!idx) return fail(OPRAG_ERR_INVALID_ARG, "index is NULL");
  if (!idx->last_path) return fail(OPRAG_ERR_NOT_READY, "no search was issued");
  if (grid) *grid = idx->last_grid;
  if (cluster) *cluster = idx->last_cluster;
  if (block_n) *block_n = idx->last_block_n;
  return ok();
}

int oprag_plan_search(int64_t n, int32_t d, int32_t q, int32_t k, int32_t num_sms,
                      int32_t force_block_n, int32_t force_pair, int32_t pair_capacity,
                      int64_t* out) {
  if (!out) return fail(OPRAG_ERR_INVALID_ARG, "NULL out");
  if (n < 1 || d < 1 || q < 1 || k < 1 || num_sms < 1 || d % 8 != 0 || k > OPRAG_K_MAX)
    return fail(OPRAG_ERR_INVALID_ARG, "bad plan shape n=%lld d=%d q=%d k=%d sms=%d",
                (long long)n, d, q, k, num_sms);
  const SearchShape s{n, d, q, k};
  const TcPlan pl = tc_plan(s, num_sms, force_block_n, 1, force_pair, pair_capacity);
  const int64_t v[13] = {pl.grid,  pl.block_n, pl.pair,  pl.dual ? 1 : 0,
                         pl.qt,    pl.uqt,     pl.nt,    pl.win,
                         pl.pmax,  pl.stages,  static_cast<int64_t>(pl.smem),
                         static_cast<int64_t>(tc_scratch_bytes(s, pl)), pl.sets};
  for (int i = 0; i < 13; ++i) out[i] = v[i];
  return ok();
}

int oprag_index_last_tiles_per_cta(const oprag_index* idx, int32_t* tiles) {
  if (!idx) return fail(OPRAG_ERR_INVALID_ARG, "index is NULL");
  if (!idx->last_path) return fail(OPRAG_ERR_NOT_READY, "no search was issued");
  if (tiles) *tiles = idx->last_tiles;
  return ok();
}

int oprag_index_last_timing(oprag_index* idx, float* lexical_ms, float* sample_ms,
                            float* search_ms, float* merge_ms) {
  if (!idx) return fail(OPRAG_ERR_INVALID_ARG, "index is NULL");
  if (!idx->timed) return fail(OPRAG_ERR_NOT_READY, "no timed search was issued");
  DeviceGuard g(idx->device);
  cudaError_t e = cudaEventSynchronize(idx->ev[3]);
  if (e != cudaSuccess) return cuda_fail(e, "timing");
  float a = 0.f, b = 0.f, c = 0.f, m = 0.f;
  if (idx->timed_lex) e = cudaEventElapsedTime(&a, idx->ev[0], idx->ev[1]);
  if (e == cudaSuccess && idx->timed_sample) e = cudaEventElapsedTime(&b, idx->ev[1], idx->ev[4]);
  if (e == cudaSuccess)
    e = cudaEventElapsedTime(&c, idx->ev[idx->timed_sample ? 4 : 1], idx->ev[2]);
  if (e == cudaSuccess) e = cudaEventElapsedTime(&m, idx->ev[2], idx->ev[3]);
  if (e != cudaSuccess) return cuda_fail(e, "timing");
  if (lexical_ms) *lexical_ms = a;
  if (sample_ms) *sample_ms = b;
  if (search_ms) *search_ms = c;
  if (merge_ms) *merge_ms = m;
  return ok();
}

int oprag_index_last_phases(oprag_index* idx, int64_t* out, int32_t cap, int32_t* ctas) {
  if (!idx || !ctas) return fail(OPRAG_ERR_INVALID_ARG, "NULL argument");
  if (!idx->phases_on || idx->phases_grid == 0)
    return fail(OPRAG_ERR_NOT_READY, "no tensor-core search ran with phase stamps on");
  DeviceGuard g(idx->device);
  cudaError_t e = idx->drain();
  if (e != cudaSuccess) return cuda_fail(e, "pending work");
  *ctas = idx->phases_grid;
  const int64_t count = static_cast<int64_t>(idx->phases_grid) * kTcPhases;
  if (out == nullptr) return ok();
  if (cap < count) return fail(OPRAG_ERR_INVALID_ARG, "need room for %lld stamps", (long long)count);
  e = cudaMemcpy(out, idx->phases, count * 8, cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_fail(e, "reading phase stamps");
  return ok();
}

int oprag_index_buffer_bytes(const oprag_index* idx, int64_t* scratch, int64_t* bounds,
                             int64_t* lexical) {
  if (!idx) return fail(OPRAG_ERR_INVALID_ARG, "index is NULL");
  if (scratch) *scratch = static_cast<int64_t>(idx->scratch_bytes);
  if (bounds) *bounds = static_cast<int64_t>(idx->qfloor_bytes);
  if (lexical) *lexical = static_cast<int64_t>(idx->lex_bytes);
  return ok();
}

}  // extern "C"

// ---------------------------------------------------------------------------
// Search without device allocations.  The partial lists live in a statically
// sized device array instead of the index's lazily grown scratch buffer.  The
// paper has no counterpart; this serves callers that must not allocate device
// memory while serving a request.

namespace {

constexpr size_t kStaticScratchBytes = size_t(16) << 20;
constexpr int kMaxDevices = 64;

}  // namespace

// Shared by every call on a device; kept until the process exits.
static __device__ __align__(256) unsigned char g_static_scratch[kStaticScratchBytes];

namespace {

std::mutex g_static_mu;
void* g_static_ptr[kMaxDevices] = {};

// Device address of g_static_scratch on `device` (which must be current),
// resolved once per device.  The host-side name is only a stand-in.  The
// cached address belongs to the device's primary context: after a
// cudaDeviceReset it is stale (the header says so).
int static_scratch(int device, void** out) {
  if (device < 0 || device >= kMaxDevices)
    return fail(OPRAG_ERR_INVALID_ARG, "device %d out of range", device);
  std::lock_guard<std::mutex> lock(g_static_mu);
  if (g_static_ptr[device] == nullptr) {
    void* ptr = nullptr;
    cudaError_t e = cudaGetSymbolAddress(&ptr, g_static_scratch);
    if (e != cudaSuccess) return cuda_fail(e, "resolving the static scratch array");
    g_static_ptr[device] = ptr;
  }
  *out = g_static_ptr[device];
  return OPRAG_OK;
}

}  // namespace

extern "C" int oprag_search_noalloc(oprag_index* idx, const void* queries, int32_t q, int32_t k,
                                    int64_t* out_ids, float* out_scores, void* stream) {
  int rc = check_search_args(idx, queries, q, k, out_ids, out_scores);
  if (rc) return rc;
  if (q == 0) return ok();
  DeviceGuard g(idx->device);
  void* scratch = nullptr;
  if ((rc = static_scratch(idx->device, &scratch))) return rc;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  // The same passes as oprag_search (with the sampled first pass for k > 32
  // over many corpus tiles); its shared per-query bounds sit after the lists
  // and are cleared on every call, since the array is shared by all indexes.
  const SearchLayout L = search_layout(idx, q, k);
  const size_t floors = L.floors ? static_cast<size_t>(q) * sizeof(uint64_t) : 0;
  const size_t need = round256(L.total()) + floors;
  if (need > kStaticScratchBytes)
    return fail(OPRAG_ERR_INVALID_ARG,
                "this search needs %zu bytes of scratch but the static array holds %zu; use "
                "oprag_search or fewer queries / a smaller k",
                need, kStaticScratchBytes);
  if ((rc = begin_call(idx, st))) return rc;
  uint64_t* qf = nullptr;
  if (L.floors) {
    qf = reinterpret_cast<uint64_t*>(static_cast<char*>(scratch) + round256(L.total()));
    cudaError_t e = cudaMemsetAsync(qf, 0, floors, st);
    if (e != cudaSuccess) return cuda_fail(e, "clearing shared bounds");
  }
  const Fusion none{nullptr, 0, nullptr, 0.f};
  idx->timed_lex = false;
  if ((rc = launch_search(idx, L, queries, q, k, none, scratch, qf, 1u, out_ids, out_scores, st)))
    return rc;
  return end_call(idx, st);
}
