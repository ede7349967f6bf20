// Internal host-side interface between the C-ABI layer (oprag.cu) and the
// kernel translation units.  Not part of the public header.
#pragma once

#include <cstddef>
#include <cstdint>
#include <cuda_runtime.h>
#include <cuda_bf16.h>

namespace oprag {

enum Dtype : int { kF32 = 0, kBF16 = 1 };

// Kept-list length used for a requested k: 8, 16 or 32 (register lists), 128
// or 256 (buffered lists).
inline int list_len_for(int k) {
  return k <= 8 ? 8 : k <= 16 ? 16 : k <= 32 ? 32 : k <= 128 ? 128 : 256;
}

// Partial top-K lists written by a search kernel and read by the merge.  The
// list of query row `row` of query tile `tile` produced by producer `p` starts
// at keys + ((tile * P + p) * TH + row) * stride and is sorted best first,
// unless `counts` is set (see there).
struct ListSet {
  const uint64_t* keys;
  int P;
  int TH;
  int stride;
  // Tensor-core lists: only producers p < sets * (C - first_cta(tile / pair))
  // exist for a tile (see search_tc.cuh); C == 0 means all P lists exist.
  // C and qt count the kernel's schedule units: CTAs (pairs of CTAs) and
  // query tiles (pairs of query tiles) when pair == 1 (2).
  int C = 0;
  int qt = 0;
  int sets = 1;
  int pair = 1;
  int klen = 1 << 30;   // sorted keys held per list (the merge reads min(k, klen))
  // Search over two stacked corpora (oprag_search_two): ids >= split belong
  // to the second; the merge then writes id - split and out_src = 1 (else
  // the id and 0; -1 for an empty result).  out_src == nullptr: ids as kept.
  int64_t split = 0;
  int32_t* out_src = nullptr;
  // Buffered tensor-core lists (k > 32) are left as the search filled them:
  // list r (the index above without the stride) holds counts[r] <= stride
  // keys in no order.  nullptr: sorted lists of klen keys.
  const int* counts = nullptr;
  // With counts: the main pass's counted floors per query (kLevels each,
  // with one counter per band, see TcParams::levels).  A level whose band
  // counts up to it sum to k is a proven lower bound of the query's k-th
  // best score, so the merge drops keys below it.
  const float* levels = nullptr;
  const int* level_cnt = nullptr;
};

// Optional lexical part of the fused score (Sec. 4.4 weighted fusion):
// f = alpha * dense + (1 - alpha) * BM25(q, id) / max_q, zero lexical part when
// max_q <= 0.  Two forms:
//  * materialised (SIMT kernel): bm25 is a q x ld block of BM25 values;
//  * gathered in the tensor-core epilogue (bm25 == nullptr, lex_qcount set).
//    Each term of the sparse side has a class (lex_class):
//    - head (class s in [0, kLexHeadTerms)): one more K block of tensor-core
//      MMAs, lex_qcount (q x kLexK bf16: the query's count of each head
//      term, twice) times lex_wsplit (n x kLexK bf16: each chunk's head-term
//      weights split into a high and a low bf16 half), accumulated in fp32;
//    - mid (class -2 - r): row r of mid_w (fp32 weight per chunk, mid_ld
//      apart), read per chunk;
//    - tail (class -1): its postings (lex_post, chunks ascending), walked per
//      chunk with a cursor.
//    Per query the prep kernel lists up to kLexMidReg mid rows (lex_mid: row,
//    multiplicity bits) and kLexRegTerms tail terms (lex_terms: first
//    posting, end posting, multiplicity bits, term id); further terms of a
//    long query are handled by scanning its raw terms from lex_ovf[q] on.
// Neither (bm25 == nullptr and lex_qcount == nullptr) means a plain dense search.
constexpr int kLexHeadTerms = 32;              // head terms scored on tensor cores
constexpr int kLexK = 2 * kLexHeadTerms;       // one 64-element K block: high | low halves
constexpr int kLexRegTerms = 8;                // tail terms with a cursor per thread
constexpr int kLexMidReg = 2;                  // mid rows per query read with cp.async
struct Fusion {
  const float* bm25;      // q x ld, row-major
  int64_t ld;
  const float* bm25_max;  // q
  float alpha;
  const void* lex_qcount = nullptr;
  const void* lex_wsplit = nullptr;
  const int4* lex_terms = nullptr;    // q x kLexRegTerms
  const int* lex_term_cnt = nullptr;  // q
  const int2* lex_mid = nullptr;      // q x kLexMidReg
  const int* lex_mid_cnt = nullptr;   // q
  const int* lex_ovf = nullptr;       // q
  const int2* lex_post = nullptr;
  const float* mid_w = nullptr;
  int64_t mid_ld = 0;                 // multiple of 128, >= n
  // for the scan of long queries: the query CSR and the term tables
  const int32_t* q_indptr = nullptr;
  const int32_t* q_terms = nullptr;
  const int32_t* lex_class = nullptr;
  const int64_t* post_ptr = nullptr;
  int vocab = 0;
  bool gathered() const { return lex_qcount != nullptr; }
};

struct SearchShape {
  int64_t n;
  int d;
  int q;
  int k;
  // Rows of a second corpus searched after the first in the same launch
  // (its chunks get ids n + row); 0 for one corpus.
  int64_t n_second = 0;
  // The lexical part is gathered in the tensor-core epilogue: the plan uses
  // single CTAs with 128-row corpus tiles and one epilogue set.
  bool fused_lex = false;
};

// --- SIMT streaming search (fp32 or bf16; any q, meant for small q).
size_t simt_scratch_bytes(int dtype, const SearchShape& s, int grid);
int simt_grid(const SearchShape& s, int num_sms);
cudaError_t launch_simt_search(int dtype, const void* E, const void* Q, const SearchShape& s,
                               const Fusion& fu, void* scratch, int grid, ListSet* lists,
                               cudaStream_t st);

// --- tcgen05 tensor-core search (bf16).
struct TcPlan {
  int block_n;     // corpus rows per tile: 128 or 256
  int nt_first;    // corpus tiles of the first corpus (nt_first == tiles of all when one)
  int grid;        // CTAs (persistent)
  int pair;        // 2: clusters of two CTAs issue M = 256 MMAs together; 1: single CTAs
  bool dual;       // single CTAs that take two query tiles per unit (see search_tc.cuh)
  int qt;          // query tiles of 128
  int uqt;         // query tiles of the schedule: qt, or ceil(qt / 2) pairs of tiles
  int nt;          // corpus tiles
  int win;         // corpus tiles per L2 window
  int pmax;        // lists per query tile
  int sets;        // lists each CTA keeps per query tile (its epilogue sets; 1 in dual mode)
  int tile_stride; // corpus tiles skipped between scanned tiles (1 = all)
  int stages;
  size_t smem;
};
// tile_stride > 1 scans only corpus tiles t = 0, stride, 2 * stride, ...
// force_pair: 0 automatic, 1 single CTAs, 2 CTA pairs (needs 256-row tiles),
// 3 dual mode (single CTAs, two query tiles per unit; lists of 8 or 16).
// pair_capacity: clusters of two that fit on the device (0: no pair mode).
TcPlan tc_plan(const SearchShape& s, int num_sms, int force_block_n, int tile_stride = 1,
               int force_pair = 0, int pair_capacity = 0);
// Clusters of two pair-mode CTAs that fit on the current device at once.
int tc_pair_capacity();
size_t tc_scratch_bytes(const SearchShape& s, const TcPlan& p);
// init_floor (optional, q floats): a lower bound on each query's k-th best
// score; lists start with it as their admission floor.
// qfloor (optional, q entries, register lists only): per-query k-th score
// bounds shared by all lists, valid for entries tagged with gen (see
// search_tc.cuh); zero-filled memory is a valid initial state.
// levels / level_cnt (optional, q x kLevels, buffered lists only): candidate
// floors (non-increasing) and zeroed counters, one per band between floors;
// a floor becomes a shared bound once k pushed keys reach it.
// wait_limit: cycles an mbarrier wait may spin before the kernel gives up and
// sets *dev_err (<= 0: the default of about a second).
// phases (optional, grid x kTcPhases zeroed words): global-timer stamps of
// each CTA's run (entry, setup done, first and last stage landed, last MMA
// commit, epilogue sets done, exit), for measurement.
// E2 (s.n_second > 0): the second corpus, same d and dtype.
cudaError_t launch_tc_search(const void* E, const void* Q, const SearchShape& s, const Fusion& fu,
                             const TcPlan& plan, void* scratch, int* dev_err, ListSet* lists,
                             cudaStream_t st, const float* init_floor = nullptr,
                             uint64_t* qfloor = nullptr, uint32_t gen = 0,
                             const float* levels = nullptr, int* level_cnt = nullptr,
                             long long wait_limit = 0, unsigned long long* phases = nullptr,
                             const void* E2 = nullptr);
constexpr int kTcPhases = 8;

// --- final merge of partial lists into the sorted top-k per query.
// kth_out (optional, q floats): the k-th best merged score of every query
// (-inf when fewer than k candidates exist).  levels_out (optional, q x
// kLevels floats): the merged scores at ranks level_rank(k, i).
constexpr int kLevels = 4;
// Ranks k/16, k/8, k/4, k/2 (at least 1): candidate floors for a search of
// k > 32 that a first pass over a sample of the corpus tiles proposes.
inline __host__ __device__ int level_rank(int k, int i) {
  const int r = k >> (kLevels - i);
  return r < 1 ? 1 : r;
}
cudaError_t launch_merge(const ListSet& ls, int q, int k, int64_t* out_ids, float* out_scores,
                         cudaStream_t st, float* kth_out = nullptr, float* levels_out = nullptr);

// Two ranked lists per query (a: q x ka, b: q x kb, each sorted score
// descending then id ascending) into the top-k of both, score descending,
// then list a before list b, then id; out_src: 0 = a, 1 = b.
cudaError_t launch_merge_two(int q, const int64_t* a_ids, const float* a_sc, int ka,
                             const int64_t* b_ids, const float* b_sc, int kb, int k,
                             int64_t* out_ids, int32_t* out_src, float* out_scores,
                             cudaStream_t st);

// --- BM25 matrix pass (lexical part of the hybrid search).
// Per-posting weight w(t, d) = idf * tf (k1+1) / (tf + k1 (1 - b + b |d| / avgdl)).
// Terms held by more than half of the chunks are stored as dense rows of
// w(t, .) (zero where absent: 4 bytes per chunk instead of 8 per posting, and
// no scatter); the other terms as postings.
// Chunks per tile of the BM25 pass (one CTA per query and tile).
constexpr int kBm25DocTile = 8192;

struct SparseIndex {
  int vocab;
  int64_t nnz;               // postings of the sparse terms
  const int64_t* post_ptr;   // device, vocab + 1 (empty range for dense terms)
  const int2* post;          // device, nnz (chunk, weight bits), chunks ascending per term
  const int32_t* dense_slot; // device, vocab: row of a dense term, -1 otherwise
  const float* dense_w;      // device, rows x dense_ld
  int64_t dense_ld;          // multiple of 4, >= n; zero past n
  // device, vocab x (ntiles + 1): entry (t, b) is the first posting of term t
  // whose chunk is >= b * kBm25DocTile (post_ptr[t + 1] past the last).
  const int64_t* tile_ptr;
  int ntiles;
};
// out == nullptr computes only the per-query maxima (the gathered form).
cudaError_t launch_bm25_matrix(const SparseIndex& sp, int64_t n, const int32_t* q_indptr,
                               const int32_t* q_terms, int q, float* out, int64_t ld,
                               float* out_max, cudaStream_t st);

// Per-query operands of the gathered lexical part (see Fusion): qcount
// (q x kLexK bf16), terms (q x kLexRegTerms), mid (q x kLexMidReg) and the
// counts term_cnt, mid_cnt and ovf (q each), from the terms' classes.
struct LexPrep {
  void* qcount;
  int4* terms;
  int* term_cnt;
  int2* mid;
  int* mid_cnt;
  int* ovf;
};
cudaError_t launch_lex_prep(const int32_t* lex_class, const int64_t* post_ptr, int vocab,
                            const int32_t* q_indptr, const int32_t* q_terms, int q,
                            const LexPrep& out, cudaStream_t st);

// --- building the lexical index on the device (sparse_build.cu): from a
// term-major inverted index of (chunk, tf) pairs (term_start: vocab + 1
// offsets into inv), each chunk's token count and each term's idf, every
// per-posting weight, written to the postings (terms with slot < 0, at
// post_ptr[t]), the dense rows (slot >= 0), the split head-term operand
// (lex_class >= 0) and the mid rows (lex_class <= -2); then the per-tile
// postings table.  Destinations of dense rows, wsplit and mid_w must be
// zeroed beforehand.
struct LexBuild {
  int vocab;
  const int2* inv;
  const int64_t* term_start;
  const double* idf;
  const int32_t* doc_len;
  double avgdl, k1, b;
  const int32_t* slot;
  const int32_t* lex_class;
  const int64_t* post_ptr;
  int2* post;
  float* dense_w;
  int64_t dense_ld;
  __nv_bfloat16* wsplit;
  float* mid_w;
  int64_t mid_ld;
};
cudaError_t launch_lex_build(const LexBuild& lb, int ntiles, int64_t* tile_ptr, cudaStream_t st);

// --- lexical rerank of a dense top-N (dense-first hybrid), rerank.cu.
// cand_ids / cand_scores: q x ncand dense results (id -1 = none), ncand <=
// kRerankMaxCand; writes the fused top-k (k <= ncand) of each query.
constexpr int kRerankMaxCand = 256;
cudaError_t launch_rerank(const SparseIndex& sp, int q, int ncand, const int64_t* cand_ids,
                          const float* cand_scores, const int32_t* q_indptr,
                          const int32_t* q_terms, float alpha, int k, int64_t* out_ids,
                          float* out_scores, cudaStream_t st);

// --- embedding tail (embed.cu): masked mean pool + L2 normalisation of a
// batch x tokens x dim block of hidden states into batch x dim vectors.
// dim % 8 == 0 and dim <= 16384 (bf16 input) / 8192 (fp32 input).
cudaError_t launch_embed_pool(int hidden_dtype, const void* hidden, int batch, int tokens, int dim,
                              const uint8_t* mask, int out_dtype, void* out, cudaStream_t st);

// --- upsert / conversion.
cudaError_t launch_scatter_rows(int index_dtype, void* E, int d, const void* rows, int rows_dtype,
                                const int64_t* src_dst /* pairs: source row, destination row */,
                                int64_t count, cudaStream_t st);
cudaError_t launch_convert_f32_bf16(const float* src, void* dst, int64_t count, cudaStream_t st);

}  // namespace oprag
