/*
 * oracle.c -- plain, slow, obviously correct CPU reference for the retrieval
 * hot path of OpRAG (arxiv 2608.08340).  TEST INFRASTRUCTURE ONLY: it is
 * called by tests/, by __graft_entry__.smoke() and by the cpu_baseline /
 * reference arm of bench.py, never by the product library.  It shares no
 * code, header or table with the CUDA path.
 *
 * Everything is computed in fp64 from the exact values the GPU sees:
 * inputs arrive either as fp32 or as bf16 bit patterns (uint16) and are
 * widened exactly to double here.
 *
 * What each function follows:
 *   oracle_dense_scores  -- dense inner-product scoring of a query against
 *                           every chunk embedding (the whole embedding
 *                           matrix scored at once, Sec. 4.4;
 *                           vectors are L2-normalised by Op_embed, Sec. 4.3,
 *                           so inner product == cosine).
 *   oracle_search        -- TopK over the whole index, Sec. 3.2 (Op_retrieve,
 *                           R_k = Op_retrieve(q, I)) and the TopK display of
 *                           Sec. 4.4.  Written as a FULL sort by (score desc,
 *                           chunk id asc) and truncation: Sec. 4.4 and Sec. 7
 *                           state that partial top-k selection must return the
 *                           same result as the full sort.
 *   oracle_bm25          -- Okapi BM25 by a document-wise scan (BM25 over the
 *                           whole corpus with exact statistics, Sec. 4.4 /
 *                           Sec. 7; the paper names BM25 but prints no formula, so the
 *                           textbook Okapi form with the non-negative idf
 *                           ln(1 + (N - df + 0.5)/(df + 0.5)) is used).
 *   oracle_hybrid_search -- weighted score fusion of Sec. 4.4:
 *                           score = w_d * s_dense + w_l * s_lex with
 *                           w_d = alpha, w_l = 1 - alpha and
 *                           s_lex = BM25 / max_d BM25 (per query), then TopK.
 *   oracle_rerank        -- the lexical rerank of the dense-first hybrid
 *                           policy (Sec. 4.1 Retrieval, Sec. 5.5): the same
 *                           fusion restricted to given candidates (a dense
 *                           top-N), with the BM25 maximum taken over those
 *                           candidates (the paper does not say which maximum
 *                           normalises a rerank; this is the reading used).
 *   oracle_embed_pool    -- the tail of Op_embed (Sec. 4.3: hidden states of
 *                           a chunk -> mean pool -> L2 normalise), with the
 *                           padded token positions of a batch masked out
 *                           (length-bucketed batches are padded, Sec. 4.3).
 *   oracle_upsert        -- Op_upsert of Sec. 3.2 (I' = Op_upsert(I, E; b_u)):
 *                           a literal row overwrite in the caller's order.
 *   oracle_round_bf16    -- fp32 -> bf16 round-to-nearest-even (the storage
 *                           precision of the index), from the IEEE definition.
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#include <unistd.h>

enum { ORACLE_F32 = 0, ORACLE_BF16 = 1 };

/* ---------------------------------------------------------------- widening */

static double bf16_bits_to_double(uint16_t bits)
{
    /* bf16 is the top half of an IEEE-754 binary32 word. */
    uint32_t w = ((uint32_t)bits) << 16;
    float f;
    memcpy(&f, &w, sizeof f);
    return (double)f;
}

static double load_elem(const void *base, int dtype, int64_t i)
{
    if (dtype == ORACLE_BF16)
        return bf16_bits_to_double(((const uint16_t *)base)[i]);
    return (double)((const float *)base)[i];
}

/* fp32 -> bf16, round to nearest, ties to even (finite inputs). */
uint16_t oracle_round_bf16_one(float x)
{
    uint32_t w;
    memcpy(&w, &x, sizeof w);
    uint32_t upper = w >> 16;
    uint32_t lower = w & 0xFFFFu;
    if (lower > 0x8000u || (lower == 0x8000u && (upper & 1u)))
        upper += 1u;
    return (uint16_t)upper;
}

void oracle_round_bf16(const float *x, int64_t count, uint16_t *out)
{
    for (int64_t i = 0; i < count; ++i)
        out[i] = oracle_round_bf16_one(x[i]);
}

/* ------------------------------------------------------------ thread pool */

typedef void (*row_fn)(void *ctx, int64_t row, double *work);

typedef struct {
    row_fn fn;
    void *ctx;
    int64_t rows;
    int64_t work_len;
    int tid, nthreads;
    int failed;
} job_t;

static void *job_main(void *arg)
{
    job_t *j = (job_t *)arg;
    double *work = NULL;
    if (j->work_len > 0) {
        work = (double *)malloc((size_t)j->work_len * sizeof(double));
        if (!work) { j->failed = 1; return NULL; }
    }
    for (int64_t r = j->tid; r < j->rows; r += j->nthreads)
        j->fn(j->ctx, r, work);
    free(work);
    return NULL;
}

/* Runs fn(ctx, row, work) for every row in [0, rows), rows striped over
 * nthreads threads (0 = all online cores).  Each thread owns a scratch array
 * of work_len doubles.  Returns the number of threads used, or -1. */
static int run_rows(row_fn fn, void *ctx, int64_t rows, int64_t work_len, int nthreads)
{
    if (nthreads <= 0) nthreads = (int)sysconf(_SC_NPROCESSORS_ONLN);
    if (nthreads < 1) nthreads = 1;
    if (rows < nthreads) nthreads = rows > 0 ? (int)rows : 1;
    pthread_t *th = (pthread_t *)calloc((size_t)nthreads, sizeof(pthread_t));
    job_t *jobs = (job_t *)calloc((size_t)nthreads, sizeof(job_t));
    if (!th || !jobs) { free(th); free(jobs); return -1; }
    int failed = 0;
    for (int t = 0; t < nthreads; ++t) {
        jobs[t] = (job_t){fn, ctx, rows, work_len, t, nthreads, 0};
        if (pthread_create(&th[t], NULL, job_main, &jobs[t]) != 0) {
            job_main(&jobs[t]);
            th[t] = 0;
        }
    }
    for (int t = 0; t < nthreads; ++t) {
        if (th[t]) pthread_join(th[t], NULL);
        failed |= jobs[t].failed;
    }
    free(th);
    free(jobs);
    return failed ? -1 : nthreads;
}

/* ------------------------------------------------------------ dense scores */

typedef struct {
    const void *E; int edtype; int64_t n; int d;
    const void *Q; int qdtype;
    double *S;
} dense_ctx;

/* s(q, c) = sum_j q_j * e_{c,j}, accumulated in fp64 in index order j. */
static double dot_row(const void *E, int edtype, int64_t c, const void *Q, int qdtype,
                      int64_t qi, int d)
{
    double acc = 0.0;
    for (int j = 0; j < d; ++j)
        acc += load_elem(Q, qdtype, qi * d + j) * load_elem(E, edtype, c * d + j);
    return acc;
}

static void dense_row(void *vctx, int64_t qi, double *work)
{
    (void)work;
    dense_ctx *c = (dense_ctx *)vctx;
    for (int64_t r = 0; r < c->n; ++r)
        c->S[qi * c->n + r] = dot_row(c->E, c->edtype, r, c->Q, c->qdtype, qi, c->d);
}

/* S[qi][c] for all q queries and n chunks (row-major q x n). */
int oracle_dense_scores(const void *E, int edtype, int64_t n, int d,
                        const void *Q, int qdtype, int q, double *S, int nthreads)
{
    dense_ctx c = {E, edtype, n, d, Q, qdtype, S};
    return run_rows(dense_row, &c, q, 0, nthreads);
}

/* ------------------------------------------------------------ full sort */

typedef struct { double s; int64_t id; } pair_t;

/* TopK order: higher score first; equal scores -> lower chunk id first. */
static int pair_cmp(const void *a, const void *b)
{
    const pair_t *x = (const pair_t *)a, *y = (const pair_t *)b;
    if (x->s > y->s) return -1;
    if (x->s < y->s) return 1;
    if (x->id < y->id) return -1;
    if (x->id > y->id) return 1;
    return 0;
}

/* Sorts all n (score, id) pairs of one query and keeps the first kout. */
static int sort_and_take(const double *scores, int64_t n, int64_t kout,
                         int64_t *ids_out, double *scores_out)
{
    pair_t *p = (pair_t *)malloc((size_t)n * sizeof(pair_t));
    if (!p) return -1;
    for (int64_t i = 0; i < n; ++i) { p[i].s = scores[i]; p[i].id = i; }
    qsort(p, (size_t)n, sizeof(pair_t), pair_cmp);
    for (int64_t i = 0; i < kout; ++i) { ids_out[i] = p[i].id; scores_out[i] = p[i].s; }
    free(p);
    return 0;
}

/* Top-kout of each row of a precomputed q x n score matrix. */
typedef struct {
    const double *S; int64_t n; int64_t kout; int64_t *ids; double *scores; int err;
} topk_ctx;

static void topk_row(void *vctx, int64_t qi, double *work)
{
    (void)work;
    topk_ctx *c = (topk_ctx *)vctx;
    if (sort_and_take(c->S + qi * c->n, c->n, c->kout, c->ids + qi * c->kout,
                      c->scores + qi * c->kout) != 0)
        c->err = 1;
}

int oracle_topk_rows(const double *S, int q, int64_t n, int64_t kout,
                     int64_t *ids, double *scores, int nthreads)
{
    if (kout < 0 || kout > n) return -1;
    topk_ctx c = {S, n, kout, ids, scores, 0};
    int r = run_rows(topk_row, &c, q, 0, nthreads);
    return c.err ? -1 : r;
}

/* Exact dense top-kout search without materialising the q x n matrix:
 * per query, all n scores in fp64 then a full sort. */
typedef struct {
    const void *E; int edtype; int64_t n; int d;
    const void *Q; int qdtype; int64_t kout;
    int64_t *ids; double *scores; int err;
} search_ctx;

static void search_row(void *vctx, int64_t qi, double *work)
{
    search_ctx *c = (search_ctx *)vctx;
    for (int64_t r = 0; r < c->n; ++r)
        work[r] = dot_row(c->E, c->edtype, r, c->Q, c->qdtype, qi, c->d);
    if (sort_and_take(work, c->n, c->kout, c->ids + qi * c->kout,
                      c->scores + qi * c->kout) != 0)
        c->err = 1;
}

int oracle_search(const void *E, int edtype, int64_t n, int d,
                  const void *Q, int qdtype, int q, int64_t kout,
                  int64_t *ids, double *scores, int nthreads)
{
    if (kout < 0 || kout > n) return -1;
    search_ctx c = {E, edtype, n, d, Q, qdtype, kout, ids, scores, 0};
    int r = run_rows(search_row, &c, q, n, nthreads);
    return c.err ? -1 : r;
}

/* ------------------------------------------------------------ BM25 */

/* Corpus statistics: document frequency per term and average length. */
typedef struct {
    const int32_t *doc_indptr; const int32_t *doc_terms; int64_t n; int vocab;
    double k1, b, avgdl;
    int64_t *df;
} corpus_stats;

static int build_stats(corpus_stats *cs)
{
    cs->df = (int64_t *)calloc((size_t)cs->vocab, sizeof(int64_t));
    int64_t *last_doc = (int64_t *)malloc((size_t)cs->vocab * sizeof(int64_t));
    if (!cs->df || !last_doc) { free(cs->df); free(last_doc); return -1; }
    for (int t = 0; t < cs->vocab; ++t) last_doc[t] = -1;
    double total = 0.0;
    for (int64_t dd = 0; dd < cs->n; ++dd) {
        int32_t lo = cs->doc_indptr[dd], hi = cs->doc_indptr[dd + 1];
        total += (double)(hi - lo);
        for (int32_t p = lo; p < hi; ++p) {
            int32_t t = cs->doc_terms[p];
            if (t < 0 || t >= cs->vocab) continue;
            if (last_doc[t] != dd) { last_doc[t] = dd; cs->df[t] += 1; }
        }
    }
    free(last_doc);
    cs->avgdl = cs->n > 0 ? total / (double)cs->n : 0.0;
    return 0;
}

/* idf(t) = ln(1 + (N - df + 0.5) / (df + 0.5)); a term no document holds
 * contributes nothing, so its idf is irrelevant and reported as 0. */
static double idf_of(const corpus_stats *cs, int32_t t)
{
    if (t < 0 || t >= cs->vocab || cs->df[t] == 0) return 0.0;
    double N = (double)cs->n, df = (double)cs->df[t];
    return log(1.0 + (N - df + 0.5) / (df + 0.5));
}

/* BM25(q, d) = sum over the query's term list (with repeats) of
 *   idf(t) * tf(t,d) * (k1 + 1) / (tf(t,d) + k1 * (1 - b + b * |d| / avgdl)).
 * tf is found by scanning the document's token list. */
static double bm25_pair(const corpus_stats *cs, int64_t dd, const int32_t *qt, int nq)
{
    int32_t lo = cs->doc_indptr[dd], hi = cs->doc_indptr[dd + 1];
    double len = (double)(hi - lo);
    double norm = 1.0 - cs->b + cs->b * (cs->avgdl > 0.0 ? len / cs->avgdl : 0.0);
    double score = 0.0;
    for (int i = 0; i < nq; ++i) {
        int32_t t = qt[i];
        int64_t tf = 0;
        for (int32_t p = lo; p < hi; ++p)
            if (cs->doc_terms[p] == t) ++tf;
        if (tf == 0) continue;
        double ftf = (double)tf;
        score += idf_of(cs, t) * ftf * (cs->k1 + 1.0) / (ftf + cs->k1 * norm);
    }
    return score;
}

typedef struct {
    const corpus_stats *cs;
    const int32_t *q_indptr; const int32_t *q_terms;
    double *out;
} bm25_ctx;

static void bm25_row(void *vctx, int64_t qi, double *work)
{
    (void)work;
    bm25_ctx *c = (bm25_ctx *)vctx;
    const int32_t *qt = c->q_terms + c->q_indptr[qi];
    int nq = c->q_indptr[qi + 1] - c->q_indptr[qi];
    for (int64_t dd = 0; dd < c->cs->n; ++dd)
        c->out[qi * c->cs->n + dd] = bm25_pair(c->cs, dd, qt, nq);
}

/* Full q x n BM25 matrix.  Also returns avgdl and (optionally) df. */
int oracle_bm25(const int32_t *doc_indptr, const int32_t *doc_terms, int64_t n, int vocab,
                double k1, double b, const int32_t *q_indptr, const int32_t *q_terms, int q,
                double *out, double *avgdl_out, int64_t *df_out, int nthreads)
{
    corpus_stats cs = {doc_indptr, doc_terms, n, vocab, k1, b, 0.0, NULL};
    if (build_stats(&cs) != 0) return -1;
    bm25_ctx c = {&cs, q_indptr, q_terms, out};
    int r = run_rows(bm25_row, &c, q, 0, nthreads);
    if (avgdl_out) *avgdl_out = cs.avgdl;
    if (df_out) memcpy(df_out, cs.df, (size_t)vocab * sizeof(int64_t));
    free(cs.df);
    return r;
}

/* ------------------------------------------------------------ hybrid */

typedef struct {
    const corpus_stats *cs;
    const void *E; int edtype; int d;
    const void *Q; int qdtype;
    const int32_t *q_indptr; const int32_t *q_terms;
    double alpha; int64_t kout;
    int64_t *ids; double *scores; double *max_bm25; int err;
} hybrid_ctx;

static void hybrid_row(void *vctx, int64_t qi, double *work)
{
    hybrid_ctx *c = (hybrid_ctx *)vctx;
    int64_t n = c->cs->n;
    const int32_t *qt = c->q_terms + c->q_indptr[qi];
    int nq = c->q_indptr[qi + 1] - c->q_indptr[qi];
    double *lex = work, *fused = work + n;
    double m = 0.0;
    for (int64_t dd = 0; dd < n; ++dd) {
        lex[dd] = bm25_pair(c->cs, dd, qt, nq);
        if (dd == 0 || lex[dd] > m) m = lex[dd];
    }
    c->max_bm25[qi] = m;
    for (int64_t dd = 0; dd < n; ++dd) {
        double dense = dot_row(c->E, c->edtype, dd, c->Q, c->qdtype, qi, c->d);
        double lexn = m > 0.0 ? lex[dd] / m : 0.0;
        fused[dd] = c->alpha * dense + (1.0 - c->alpha) * lexn;
    }
    if (sort_and_take(fused, n, c->kout, c->ids + qi * c->kout, c->scores + qi * c->kout) != 0)
        c->err = 1;
}

/* Fused top-kout: alpha * <q, e_d> + (1 - alpha) * BM25(q, d) / max_d' BM25(q, d'),
 * where a query whose maximum BM25 is not positive gets a zero lexical part. */
int oracle_hybrid_search(const void *E, int edtype, int64_t n, int d,
                         const void *Q, int qdtype, int q,
                         const int32_t *doc_indptr, const int32_t *doc_terms, int vocab,
                         double k1, double b,
                         const int32_t *q_indptr, const int32_t *q_terms,
                         double alpha, int64_t kout,
                         int64_t *ids, double *scores, double *max_bm25, int nthreads)
{
    if (kout < 0 || kout > n) return -1;
    corpus_stats cs = {doc_indptr, doc_terms, n, vocab, k1, b, 0.0, NULL};
    if (build_stats(&cs) != 0) return -1;
    hybrid_ctx c = {&cs, E, edtype, d, Q, qdtype, q_indptr, q_terms, alpha, kout,
                    ids, scores, max_bm25, 0};
    int r = run_rows(hybrid_row, &c, q, 2 * n, nthreads);
    free(cs.df);
    return c.err ? -1 : r;
}

/* ------------------------------------------------------------ rerank */

typedef struct {
    const corpus_stats *cs;
    const void *E; int edtype; int d;
    const void *Q; int qdtype;
    const int32_t *q_indptr; const int32_t *q_terms;
    const int64_t *cand; int64_t ncand;
    double alpha; int64_t kout;
    int64_t *ids; double *scores; int err;
} rerank_ctx;

static void rerank_row(void *vctx, int64_t qi, double *work)
{
    (void)work;
    rerank_ctx *c = (rerank_ctx *)vctx;
    const int32_t *qt = c->q_terms + c->q_indptr[qi];
    int nq = c->q_indptr[qi + 1] - c->q_indptr[qi];
    const int64_t *cd = c->cand + qi * c->ncand;
    pair_t *p = (pair_t *)malloc((size_t)(c->ncand > 0 ? c->ncand : 1) * sizeof(pair_t));
    double *lex = (double *)malloc((size_t)(c->ncand > 0 ? c->ncand : 1) * sizeof(double));
    if (!p || !lex) { free(p); free(lex); c->err = 1; return; }
    /* BM25 of every candidate and the maximum over the candidates. */
    int64_t m_valid = 0;
    double m = 0.0;
    for (int64_t i = 0; i < c->ncand; ++i) {
        if (cd[i] < 0 || cd[i] >= c->cs->n) continue;
        lex[i] = bm25_pair(c->cs, cd[i], qt, nq);
        if (m_valid == 0 || lex[i] > m) m = lex[i];
        ++m_valid;
    }
    int64_t np = 0;
    for (int64_t i = 0; i < c->ncand; ++i) {
        if (cd[i] < 0 || cd[i] >= c->cs->n) continue;
        double dense = dot_row(c->E, c->edtype, cd[i], c->Q, c->qdtype, qi, c->d);
        double lexn = m > 0.0 ? lex[i] / m : 0.0;
        p[np].s = c->alpha * dense + (1.0 - c->alpha) * lexn;
        p[np].id = cd[i];
        ++np;
    }
    if (np < c->kout) { c->err = 1; free(p); free(lex); return; }
    qsort(p, (size_t)np, sizeof(pair_t), pair_cmp);
    for (int64_t i = 0; i < c->kout; ++i) {
        c->ids[qi * c->kout + i] = p[i].id;
        c->scores[qi * c->kout + i] = p[i].s;
    }
    free(p);
    free(lex);
}

/* Rerank of given candidates (q x ncand chunk ids, -1 = none): fused top-kout
 * of alpha * <q, e_d> + (1 - alpha) * BM25(q, d) / max over the candidates d'
 * of BM25(q, d') (zero lexical part when that maximum is not positive).
 * Every row needs at least kout candidates. */
int oracle_rerank(const void *E, int edtype, int64_t n, int d,
                  const void *Q, int qdtype, int q,
                  const int32_t *doc_indptr, const int32_t *doc_terms, int vocab,
                  double k1, double b,
                  const int32_t *q_indptr, const int32_t *q_terms,
                  const int64_t *cand, int64_t ncand,
                  double alpha, int64_t kout,
                  int64_t *ids, double *scores, int nthreads)
{
    if (kout < 0 || kout > ncand) return -1;
    corpus_stats cs = {doc_indptr, doc_terms, n, vocab, k1, b, 0.0, NULL};
    if (build_stats(&cs) != 0) return -1;
    rerank_ctx c = {&cs, E, edtype, d, Q, qdtype, q_indptr, q_terms, cand, ncand, alpha, kout,
                    ids, scores, 0};
    int r = run_rows(rerank_row, &c, q, 0, nthreads);
    free(cs.df);
    return c.err ? -1 : r;
}

/* ------------------------------------------------------------ embedding tail */

/* out[b] = m / ||m|| with m = (1 / c) * sum of hidden[b][t] over the c tokens t
 * with mask[b][t] != 0 (hidden is batch x tokens x dim, fp32 or bf16 bits).
 * A row with no unmasked token or a zero mean gives a zero vector. */
int oracle_embed_pool(const void *hidden, int hdtype, int batch, int tokens, int dim,
                      const uint8_t *mask, double *out)
{
    if (batch < 0 || tokens < 0 || dim <= 0) return -1;
    for (int b = 0; b < batch; ++b) {
        double *o = out + (int64_t)b * dim;
        for (int j = 0; j < dim; ++j) o[j] = 0.0;
        int64_t c = 0;
        for (int t = 0; t < tokens; ++t) {
            if (!mask[(int64_t)b * tokens + t]) continue;
            ++c;
            int64_t row = ((int64_t)b * tokens + t) * dim;
            for (int j = 0; j < dim; ++j) o[j] += load_elem(hidden, hdtype, row + j);
        }
        if (c == 0) continue;
        double ss = 0.0;
        for (int j = 0; j < dim; ++j) {
            o[j] /= (double)c;
            ss += o[j] * o[j];
        }
        if (ss == 0.0) continue;
        double norm = sqrt(ss);
        for (int j = 0; j < dim; ++j) o[j] /= norm;
    }
    return 0;
}

/* ------------------------------------------------------------ upsert */

/* E[ids[i]] <- rows[i] for i = 0..m-1 in order (a later duplicate id wins).
 * Rows given as fp32 are stored into a bf16 index with round-to-nearest-even.
 * Returns -1 (and writes nothing) if any id lies outside [0, n). */
int oracle_upsert(void *E, int edtype, int64_t n, int d,
                  const int64_t *ids, const void *rows, int rdtype, int64_t m)
{
    for (int64_t i = 0; i < m; ++i)
        if (ids[i] < 0 || ids[i] >= n) return -1;
    if (edtype == ORACLE_F32 && rdtype == ORACLE_BF16) return -1;
    for (int64_t i = 0; i < m; ++i) {
        int64_t dst = ids[i];
        for (int j = 0; j < d; ++j) {
            int64_t si = i * d + j, di = dst * d + j;
            if (edtype == ORACLE_F32)
                ((float *)E)[di] = ((const float *)rows)[si];
            else if (rdtype == ORACLE_BF16)
                ((uint16_t *)E)[di] = ((const uint16_t *)rows)[si];
            else
                ((uint16_t *)E)[di] = oracle_round_bf16_one(((const float *)rows)[si]);
        }
    }
    return 0;
}
