/*
 * oprag.h -- C ABI of the GB300 retrieval hot path of OpRAG (arxiv 2608.08340).
 *
 * The library implements, on one GPU, the data-parallel core of the paper's
 * retrieval operator:
 *   - exact top-k inner-product search of a query batch against a chunk
 *     embedding index (Op_retrieve, Sec. 3.2: R_k = Op_retrieve(q, I), and the
 *     TopK display of Sec. 4.4);
 *   - hybrid dense + BM25 search with the weighted score fusion of Sec. 4.4;
 *   - in-place index upsert (Op_upsert, Sec. 3.2: I' = Op_upsert(I, E; b_u)).
 *
 * Conventions for every function below
 *   - Return value: OPRAG_OK (0) or a negative OPRAG_ERR_* code; the message
 *     of the last failure on the calling thread is oprag_last_error().  A
 *     failing call writes nothing to its outputs and leaves the index as it
 *     was, unless the code is OPRAG_ERR_CUDA.
 *   - "device" pointers are CUDA device memory of the GPU that was current when
 *     the index was created; "host" pointers are ordinary (pageable or pinned)
 *     host memory.  The caller keeps ownership of everything it passes in.
 *   - `stream` is a cudaStream_t passed as void* (NULL = the legacy default
 *     stream).  Asynchronous calls only enqueue work on it.  Calls on one index
 *     share its scratch memory: the library orders each call after the previous
 *     call on the same index (cross-stream calls wait on an event), but one
 *     index must not be used from two host threads at once.
 *   - Ranking: score descending, equal scores broken by the lower chunk id.
 *   - dtype codes: OPRAG_F32 (IEEE binary32) or OPRAG_BF16 (bfloat16, stored as
 *     the upper 16 bits of a binary32).
 *   - Inputs are finite.  Vectors are used as given: the index never
 *     normalises (normalisation belongs to embedding, Sec. 4.3).
 */
#ifndef OPRAG_H
#define OPRAG_H

#include <stdint.h>

#if defined(__GNUC__)
#define OPRAG_API __attribute__((visibility("default")))
#else
#define OPRAG_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

#define OPRAG_F32 0
#define OPRAG_BF16 1

#define OPRAG_OK 0
#define OPRAG_ERR_INVALID_ARG (-1) /* null pointer, bad size, k out of range, dtype mismatch */
#define OPRAG_ERR_RANGE (-2)       /* an upsert id outside [0, n) */
#define OPRAG_ERR_OOM (-3)         /* device or host allocation failed */
#define OPRAG_ERR_CUDA (-4)        /* a CUDA call or an earlier asynchronous launch failed */
#define OPRAG_ERR_NOT_READY (-5)   /* hybrid search before oprag_index_set_sparse */
#define OPRAG_ERR_DEVICE (-6)      /* a kernel gave up waiting (bounded wait expired) */

/* Largest k accepted by the search calls. */
#define OPRAG_K_MAX 256

typedef struct oprag_index oprag_index;

/*
 * Creates an index of n chunk embeddings of dimension d, stored on the current
 * GPU as dtype (OPRAG_F32 or OPRAG_BF16) in row-major n x d layout (the
 * "contiguous" vector buffer of Sec. 4.2).
 *   emb        n x d row-major, element type src_dtype; host memory if
 *              emb_on_device == 0, else device memory.  Copied; not retained.
 *   src_dtype  OPRAG_F32 or OPRAG_BF16.  F32 input into a BF16 index is
 *              rounded to nearest even; BF16 input into an F32 index is refused.
 *   d          1..8192, a multiple of 8.
 *   n          1 .. 2^31 - 1.
 * Synchronous.  *out receives the handle (NULL on failure).
 */
OPRAG_API int oprag_index_create(oprag_index **out, const void *emb, int64_t n, int32_t d, int32_t dtype,
                       int32_t src_dtype, int32_t emb_on_device);

/* Frees the index and all its device memory after its pending work is done.
 * NULL is allowed. */
OPRAG_API void oprag_index_destroy(oprag_index *idx);

/* Shape of the index: any out-pointer may be NULL. */
OPRAG_API int oprag_index_info(const oprag_index *idx, int64_t *n, int32_t *d, int32_t *dtype,
                     int32_t *device);

/* Device pointer of the n x d embedding matrix (read-only use; valid until
 * destroy).  For tests and zero-copy readers. */
OPRAG_API const void *oprag_index_data(const oprag_index *idx);

/*
 * Copies rows [first, first + count) of the index into host memory `out`
 * (count x d elements of the index dtype).  Synchronous.  For tests.
 */
OPRAG_API int oprag_index_get_rows(const oprag_index *idx, int64_t first, int64_t count, void *out);

/*
 * Pre-allocates the scratch memory that dense searches of up to q_max queries
 * and k_max results need -- partial lists, the sampled first pass of k > 32,
 * the per-query shared bounds (zeroed here) and, with a sparse side, the
 * lexical block of the hybrid search -- so that later searches of that size
 * allocate nothing and never synchronise the device.  Optional: search calls
 * grow the scratch on demand (which synchronises the device once).
 * Synchronous.
 */
OPRAG_API int oprag_index_reserve(oprag_index *idx, int32_t q_max, int32_t k_max);

/*
 * Upsert (Sec. 3.2 Op_upsert; Sec. 4.1: updates are coalesced and committed in
 * bulk).  Row i of `rows` overwrites chunk ids[i]; when an id repeats, the
 * later entry wins.
 *   ids              host, m int64 chunk ids in [0, n); validated before any
 *                    write (OPRAG_ERR_RANGE, nothing written).
 *   rows             m x d row-major of rows_dtype; device memory if
 *                    rows_on_device, else host memory (copied before return).
 *   rows_dtype       as for create: F32 rows into a BF16 index are rounded to
 *                    nearest even.
 * Asynchronous on `stream`; later searches on the same index see the new rows.
 */
OPRAG_API int oprag_upsert(oprag_index *idx, const int64_t *ids, const void *rows, int64_t m,
                 int32_t rows_dtype, int32_t rows_on_device, void *stream);

/*
 * Exact dense top-k search (Sec. 3.2 Op_retrieve; Sec. 4.4 dense scores by
 * matrix operations and partial top-k selection).  For each query i:
 * out[i][0..k) = the k chunks with the largest inner product <Q_i, E_c>.
 *   queries      device, q x d row-major, the index dtype, 16-byte aligned.
 *   q            >= 0 (0 is a no-op).
 *   k            1 .. min(n, OPRAG_K_MAX).
 *   out_ids      device, q x k int64, row-major, best first.
 *   out_scores   device, q x k float: the scores, accumulated in fp32.
 * Asynchronous on `stream`.
 */
OPRAG_API int oprag_search(oprag_index *idx, const void *queries, int32_t q, int32_t k, int64_t *out_ids,
                 float *out_scores, void *stream);

/*
 * Same search with host buffers: copies the q x d queries from host memory,
 * searches and copies ids and scores back to host memory.  Synchronous; also
 * reports a device-side wait failure of this call (OPRAG_ERR_DEVICE).
 */
OPRAG_API int oprag_search_host(oprag_index *idx, const void *queries, int32_t q, int32_t k,
                      int64_t *out_ids, float *out_scores, void *stream);

/*
 * Attaches the lexical side used by the hybrid search: the bag of term ids of
 * every chunk, as CSR on the host (doc_indptr[n + 1], doc_terms[doc_indptr[n]],
 * term ids in [0, vocab)).  BM25 statistics (document frequency, average
 * length, per-posting weights) are built here, in fp64 on the host, with the
 * Okapi form and idf(t) = ln(1 + (N - df + 0.5) / (df + 0.5)).  Synchronous;
 * replaces a previous sparse side.
 */
OPRAG_API int oprag_index_set_sparse(oprag_index *idx, const int32_t *doc_indptr, const int32_t *doc_terms,
                           int32_t vocab, float k1, float b);

/*
 * Hybrid search with the weighted score fusion of Sec. 4.4:
 *   score(d, q) = alpha * <q, e_d> + (1 - alpha) * BM25(q, d) / max_d' BM25(q, d'),
 * with the lexical part 0 for a query whose maximum BM25 is 0, followed by the
 * same top-k as oprag_search.
 *   queries      device, q x d (index dtype), 16-byte aligned.
 *   q_indptr     device, q + 1 int32 offsets into q_terms.
 *   q_terms      device, int32 term ids (repeats count again; ids outside
 *                [0, vocab) contribute nothing).
 *   alpha        dense weight w_d; the lexical weight is w_l = 1 - alpha.
 * Asynchronous on `stream`.  OPRAG_ERR_NOT_READY without a sparse side.
 */
OPRAG_API int oprag_hybrid_search(oprag_index *idx, const void *queries, int32_t q, const int32_t *q_indptr,
                        const int32_t *q_terms, float alpha, int32_t k, int64_t *out_ids,
                        float *out_scores, void *stream);

/*
 * Dense-first hybrid search (Sec. 4.1 Retrieval; Sec. 5.5): the exact dense
 * top-n_cand of each query (as oprag_search), then the fusion of
 * oprag_hybrid_search applied only to those candidates, with the BM25
 * maximum taken over the candidates (the paper does not name the maximum of a
 * rerank), and the top-k of the fused scores (score descending, chunk id
 * ascending).  With every chunk a candidate (n_cand >= n) the result equals
 * oprag_hybrid_search.
 *   queries, q_indptr, q_terms, alpha   as oprag_hybrid_search (device).
 *   n_cand       candidates per query, k <= n_cand <= 256 (fewer when n < n_cand).
 *   out_ids / out_scores   device, q x k.
 * Asynchronous on `stream`.  OPRAG_ERR_NOT_READY without a sparse side.
 */
OPRAG_API int oprag_hybrid_search_dense_first(oprag_index *idx, const void *queries, int32_t q,
                                              const int32_t *q_indptr, const int32_t *q_terms,
                                              float alpha, int32_t n_cand, int32_t k,
                                              int64_t *out_ids, float *out_scores, void *stream);

/*
 * Tail of Op_embed (Sec. 4.3: hidden states -> mean pool -> L2 normalise), for
 * a padded batch of chunks or queries:
 *   out[b] = m / ||m||,  m = (1 / c) * sum of hidden[b][t] over the c tokens t
 *   with mask[b][t] != 0  (a row with c = 0 or m = 0 gives zeros).
 *   hidden      device, batch x tokens x dim, OPRAG_BF16 or OPRAG_F32
 *               (hidden_dtype), 16-byte aligned; dim a multiple of 8, at most
 *               16384 (bf16) or 8192 (fp32).
 *   mask        device, batch x tokens uint8 (nonzero = a real token).
 *   out         device, batch x dim in out_dtype (OPRAG_BF16: round to nearest
 *               even of the fp32 result), 16-byte aligned; as queries it feeds
 *               oprag_search of an index of the same dim directly.
 * Accumulates in fp32.  Asynchronous on `stream`; needs no index.
 */
OPRAG_API int oprag_embed_pool(const void *hidden, int32_t hidden_dtype, int32_t batch,
                               int32_t tokens, int32_t dim, const uint8_t *mask, void *out,
                               int32_t out_dtype, void *stream);

/*
 * Appends m rows as chunks n, n + 1, ... (Op_upsert inserting, Sec. 3.2;
 * Sec. 4.4: the memory index grows by upserts).  The device buffer grows by
 * doubling (a reallocation: earlier oprag_index_data pointers become
 * invalid).  *first_id (optional) receives the id of the first new chunk.
 * With a sparse side attached, the new chunks hold no terms (see
 * oprag_index_update_sparse) and the BM25 statistics are rebuilt for the new
 * chunk count.  rows / rows_dtype / rows_on_device as oprag_upsert.
 * Synchronous when the buffer grows or a sparse side is attached.
 */
OPRAG_API int oprag_append(oprag_index *idx, const void *rows, int64_t m, int32_t rows_dtype,
                           int32_t rows_on_device, int64_t *first_id, void *stream);

/*
 * Replaces the token bags of chunks ids[0..m) (host, each in [0, n); a later
 * duplicate wins) by the host CSR bags bag_indptr[m + 1] / bag_terms, and
 * rebuilds df, avgdl and every BM25 weight so that the lexical scores stay
 * exact over the updated corpus (the lexical half of Op_upsert, Sec. 3.2).
 * Synchronous.  OPRAG_ERR_NOT_READY without a sparse side.
 */
OPRAG_API int oprag_index_update_sparse(oprag_index *idx, const int64_t *ids, int64_t m,
                                        const int32_t *bag_indptr, const int32_t *bag_terms);

/*
 * Dense top-k over a knowledge index and a memory index together (Sec. 3.6,
 * Sec. 4.4: both indices are searched the same way; one ranked result).  Same
 * dim and dtype on the same device.  out_ids: chunk id within its index;
 * out_src: 0 = knowledge, 1 = memory (device, q x k each, out_scores as
 * oprag_search).  Order: score descending, then knowledge before memory, then
 * chunk id.  k <= n_knowledge + n_memory.  Asynchronous on `stream`.
 * bf16 indices: one launch of the search kernel scans the knowledge rows
 * followed by the memory rows (plus its sampled first pass when k > 32 over
 * many tiles) and one merge writes the result, using the knowledge index's
 * scratch; fp32 indices: a search per index and a merge of the two lists.
 */
OPRAG_API int oprag_search_two(oprag_index *knowledge, oprag_index *memory, const void *queries,
                               int32_t q, int32_t k, int64_t *out_ids, int32_t *out_src,
                               float *out_scores, void *stream);

/*
 * Waits for the index's pending work and reports whether a kernel of it gave
 * up a bounded wait since the last check (OPRAG_ERR_DEVICE; the flag is then
 * cleared) or a CUDA error occurred (OPRAG_ERR_CUDA).
 */
OPRAG_API int oprag_index_check(oprag_index *idx);

/* Test hooks: 0 = automatic choice.  OPRAG_OPT_PATH: 1 forces the SIMT
 * streaming kernel, 2 the tensor-core kernel (bf16 only).  OPRAG_OPT_BLOCK_N:
 * corpus rows per tensor-core tile (128 or 256). */
#define OPRAG_OPT_PATH 1
#define OPRAG_OPT_BLOCK_N 2
OPRAG_API int oprag_index_set_option(oprag_index *idx, int32_t option, int32_t value);

/* OPRAG_OPT_PAIR (tensor-core path): 2 runs clusters of two CTAs that issue
 * M = 256 MMAs together, each CTA loading half of every corpus tile (needs
 * 256-row corpus tiles; ignored with 128-row tiles).  1 runs every CTA on its
 * own (M = 128 MMAs), one query tile per unit.  3 (dual mode) runs every CTA
 * on its own with two query tiles per unit that share each corpus tile
 * (128-row tiles; k <= 16 and more than 128 queries, ignored otherwise).
 * 0 (default) chooses dual mode when its units come to at most four per CTA,
 * CTA pairs for k > 32 with at least 1024 queries on 256-row tiles, single
 * CTAs otherwise. */
#define OPRAG_OPT_PAIR 4

/* OPRAG_OPT_BOUND_TAG (test hook): sets the 32-bit tag of the last search's
 * shared k-th score bounds (bit pattern of value); the next searches use the
 * following tags, so a test can make them wrap around (the bounds array is
 * then cleared). */
#define OPRAG_OPT_BOUND_TAG 5

/* OPRAG_OPT_GRAPH: 1 makes oprag_search capture its launches into a CUDA graph
 * when it is called again with the same queries / outputs pointers, q, k and
 * stream and the index has not changed (no growth, append or option change
 * since), and replay that graph on later identical calls (one launch instead
 * of several).  The stream must not be the legacy default stream; calls on
 * other streams keep their ordering through the index's completion event.
 * 0 (default) off. */
#define OPRAG_OPT_GRAPH 6

/* OPRAG_OPT_TIMING: 1 makes every later search record CUDA events, on the
 * call's stream, around its lexical (BM25) kernel, its sampled first pass,
 * its main search kernel and its merge kernel; oprag_index_last_timing()
 * reads them.  0 (default) off. */
#define OPRAG_OPT_TIMING 3

/* OPRAG_OPT_WAIT_LIMIT (test hook): the number of clock cycles a wait of the
 * tensor-core search kernel on one of its pipeline barriers may spin before
 * the kernel gives up, records OPRAG_ERR_DEVICE for oprag_index_check,
 * drains its copies and tensor-core work, frees its tensor memory and
 * returns (the results of that search are then undefined).  0 (default)
 * means about 2^31 cycles (about a second); a small value lets a test make
 * the waits of a real search run out. */
#define OPRAG_OPT_WAIT_LIMIT 7

/* OPRAG_OPT_LEX_GATHER (tensor-core path): how oprag_hybrid_search gets the
 * lexical half.  0 (default): a BM25 pass writes the q x n block of BM25
 * values (up to 2^28 values per pass) that the search's fused selection
 * reads.  1: nothing of that size is written -- a pass computes only each
 * query's BM25 maximum, and the search gathers BM25(q, d) in its epilogue:
 * the 32 commonest terms through one more tensor-core K block (the query's
 * term counts times each chunk's weights split into a high and a low bf16
 * half, within 2^-18 of the weight), terms in at least 1/32 of the chunks as
 * rows of fp32 weights, the others from their postings.  Same results
 * within the 1e-4 score bar; on 32768 x 768 with 1024 queries of 8 Zipf
 * terms the default measured 4x faster. */
#define OPRAG_OPT_LEX_GATHER 9

/* OPRAG_OPT_PHASES (measurement hook): 1 makes the main tensor-core pass of
 * every later search record, per CTA, the GPU global timer (nanoseconds) at
 * eight points of its run; oprag_index_last_phases() reads them.  Costs one
 * store per pipeline stage while on.  0 (default) off. */
#define OPRAG_OPT_PHASES 8

/*
 * Global-timer stamps (ns) of the last tensor-core main pass run with
 * OPRAG_OPT_PHASES on: *ctas receives its grid size; out (host, room for
 * cap >= *ctas * 8 values; NULL to ask the size only) receives, per CTA, in
 * order: entry, end of set-up (barriers, tensor memory), first pipeline
 * stage landed, last stage landed, last MMA committed (these three only on
 * the CTA that issues the MMAs), epilogue set 0 done, epilogue set 1 done
 * (0 with one set), exit.  Waits for the index's pending work.
 * OPRAG_ERR_NOT_READY when no such search ran.
 */
OPRAG_API int oprag_index_last_phases(oprag_index *idx, int64_t *out, int32_t cap,
                                      int32_t *ctas);

/*
 * Device durations (milliseconds) of the kernels of the last search issued
 * with timing on: lexical_ms (BM25 pass of a hybrid search, 0 for a dense
 * search), sample_ms (the first pass over every 32nd corpus tile and its
 * merge that a search with k > 32 over a large corpus runs first, else 0),
 * search_ms (main pass: score contraction + fused selection), merge_ms
 * (final top-k reduction).  Waits for that search to finish.  Any
 * out-pointer may be NULL.  OPRAG_ERR_NOT_READY if no timed search was issued.
 */
OPRAG_API int oprag_index_last_timing(oprag_index *idx, float *lexical_ms, float *sample_ms,
                                      float *search_ms, float *merge_ms);

/* Bytes currently held by the index's grow-on-demand buffers: the search
 * scratch (partial lists, sampled pass), the shared per-query k-th bounds
 * and the lexical block of the hybrid search.  Any out-pointer may be NULL.
 * For tests of oprag_index_reserve. */
OPRAG_API int oprag_index_buffer_bytes(const oprag_index *idx, int64_t *scratch, int64_t *bounds,
                                       int64_t *lexical);

/* Which kernel family served the last search on this index: 1 SIMT, 2 tensor
 * core, 0 none yet. */
OPRAG_API int oprag_index_last_path(const oprag_index *idx);

/* Launch shape of the last search's main tensor-core kernel: grid (CTAs),
 * cluster (1 single CTAs, 2 CTA pairs issuing M = 256 MMAs) and block_n
 * (corpus rows per tile); all 0 when the last search ran the SIMT kernel.
 * Out-pointers may be NULL.  OPRAG_ERR_NOT_READY before the first search. */
OPRAG_API int oprag_index_last_launch(const oprag_index *idx, int32_t *grid, int32_t *cluster,
                                      int32_t *block_n);

/* Query tiles (of 128 queries) that one CTA of the last search's main
 * tensor-core kernel takes per unit: 2 in dual mode (OPRAG_OPT_PAIR), else 1;
 * 0 for the SIMT kernel.  OPRAG_ERR_NOT_READY before the first search. */
OPRAG_API int oprag_index_last_tiles_per_cta(const oprag_index *idx, int32_t *tiles);

/* Host-side plan of a tensor-core search of q queries of dimension d over n
 * chunks with k results (bf16 index), for a device of num_sms SMs, without
 * any device work (usable without a GPU).  force_block_n (0, 128, 256) and
 * force_pair (0 automatic, 1 single CTAs, 2 CTA pairs, 3 dual mode) mean what
 * OPRAG_OPT_BLOCK_N and OPRAG_OPT_PAIR mean; pair_capacity is the number of
 * two-CTA clusters the device fits at once (0: no pair mode).  out[0..12]
 * receives, in order: CTAs launched, corpus rows per tile, CTAs per cluster
 * (1 or 2), dual mode (0 or 1), query tiles, query tiles of the schedule,
 * corpus tiles, corpus tiles per L2 window, list slots per query tile,
 * pipeline stages, dynamic shared memory per CTA in bytes, list scratch in
 * bytes, and list slots per producer and query tile.  OPRAG_ERR_INVALID_ARG
 * for n, d, q, k or num_sms < 1, d % 8 != 0, k > OPRAG_K_MAX, or a NULL out. */
OPRAG_API int oprag_plan_search(int64_t n, int32_t d, int32_t q, int32_t k, int32_t num_sms,
                                int32_t force_block_n, int32_t force_pair,
                                int32_t pair_capacity, int64_t *out);

/*
 * oprag_search without any device allocation.  The paper has no counterpart:
 * this entry point serves callers that must not allocate device memory while
 * answering a request -- a serving process whose memory pool has already
 * claimed the GPU, or a host that cannot afford the device-wide
 * synchronisation that cudaMalloc / cudaFree may cause.
 *
 * Same arguments, results and stream semantics as oprag_search, and the same
 * kernels (including the sampled first pass of k > 32 over a large corpus).
 * Instead of the index's scratch buffer (which oprag_search grows with
 * cudaMalloc), the partial top-k lists, the sampled pass and the per-query
 * shared bounds live in one statically sized device array of 16 MiB that the
 * library holds on every GPU that loads it until the process exits.
 *   - A search that needs more than 16 MiB is refused with
 *     OPRAG_ERR_INVALID_ARG and a message giving the required size; nothing
 *     is launched.  That covers k > 32 over thousands of queries and, since
 *     every CTA then keeps a 128-row list of 256 keys (256 KiB), k > 32 over
 *     a corpus of 128 or more tiles of 128 chunks: the searches for which
 *     oprag_search runs its sampled first pass.
 *   - The first call on a device resolves the array's device address (a
 *     runtime query, no allocation) and keeps it for the process; make that
 *     first call before any stream capture.  A cudaDeviceReset invalidates
 *     the kept address: do not call this entry point after one.
 *   - All calls share the array, so calls that overlap on the GPU (different
 *     indexes or streams without ordering between them) race; order them.
 *     The kernels initialise every list they use and each call clears its
 *     shared bounds, so nothing from an earlier call leaks into a later one.
 *   - With timing on (OPRAG_OPT_TIMING) it records the same events as
 *     oprag_search.
 */
OPRAG_API int oprag_search_noalloc(oprag_index *idx, const void *queries, int32_t q, int32_t k,
                                   int64_t *out_ids, float *out_scores, void *stream);

/* Message of the last failed call on this thread ("" if none). */
OPRAG_API const char *oprag_last_error(void);

#ifdef __cplusplus
}
#endif

#endif /* OPRAG_H */
