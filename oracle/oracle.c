/*
 * oracle.c -- plain, slow, fp64 CPU oracle for the threshold-aware IVF search
 * of SieveIVF (arXiv 2608.03199).
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing on the product path may call, link or
 * load this file: only the tests, the smoke check and the benchmark's CPU
 * baseline leg use it.  It shares no code, header or constant with the CUDA
 * library; both sides see only the same input arrays.
 *
 * Every similarity is an fp64 inner product of the stored fp32 values
 * (cosine similarity of unit-norm vectors, Sec. 2.2 and Sec. 6.1).  Every
 * decision (rank order, tau test, top-k order) is taken on those fp64 values.
 *
 * Index representation (the oracle's own): the rows X[n][d] in any order,
 * their external ids, and assign[n] = the partition of each row (exact
 * centroid assignment, Sec. 4.4).  The oracle groups rows into partitions
 * itself, so it never consumes a layout built by the CUDA library.
 *
 * Readings of the paper used here (where it is silent):
 *   - qualifying means sim >= tau (the definition of R(q,tau), Sec. 2.2);
 *   - a row whose id equals the query's id is not a candidate (self-join
 *     deduplication with database-drawn queries); qids == NULL disables this;
 *   - centroid ties rank the lower centroid id first; top-k ties rank the
 *     lower row id first (a total order);
 *   - a partition with no rows is an empty probe;
 *   - W >= nprobe gives fixed probing (stop line min(W, nprobe) = nprobe).
 */
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#include <math.h>

#ifdef _OPENMP
#include <omp.h>
#endif

/* ------------------------------------------------------------------------ */
/* similarity: sim(q, x) = <q, x> in fp64 (Sec. 2.2, cosine on unit vectors) */
static double sim64(const float *a, const float *b, int d)
{
    double acc = 0.0;
    for (int t = 0; t < d; ++t)
        acc += (double)a[t] * (double)b[t];
    return acc;
}

/* ------------------------------------------------------------------------ */
/* bounded top-k under the total order (score desc, id asc)                  */
typedef struct {
    double score;
    int64_t id;
} cand_t;

static int ranks_before(double sa, int64_t ia, double sb, int64_t ib)
{
    return sa > sb || (sa == sb && ia < ib);
}

typedef struct {
    int k;       /* capacity */
    int n;       /* entries held, sorted best first */
    cand_t *e;
} topk_t;

static void topk_offer(topk_t *t, double s, int64_t id)
{
    if (t->n == t->k && !ranks_before(s, id, t->e[t->k - 1].score, t->e[t->k - 1].id))
        return;
    int i = (t->n < t->k) ? t->n++ : t->k - 1;
    while (i > 0 && ranks_before(s, id, t->e[i - 1].score, t->e[i - 1].id)) {
        t->e[i] = t->e[i - 1];
        --i;
    }
    t->e[i].score = s;
    t->e[i].id = id;
}

/* ------------------------------------------------------------------------ */
/* the oracle's partition lists: rows of partition p are                     */
/* rows[start[p] .. start[p+1]), in increasing row order                     */
typedef struct {
    int64_t nlist;
    int64_t *start; /* [nlist + 1] */
    int64_t *rows;  /* [n] */
} lists_t;

static int lists_build(lists_t *L, const int32_t *assign, int64_t n, int64_t nlist)
{
    L->nlist = nlist;
    L->start = (int64_t *)calloc((size_t)nlist + 1, sizeof(int64_t));
    L->rows = (int64_t *)malloc((size_t)(n > 0 ? n : 1) * sizeof(int64_t));
    if (!L->start || !L->rows)
        return -1;
    for (int64_t i = 0; i < n; ++i) {
        if (assign[i] < 0 || assign[i] >= nlist)
            return -2;
        L->start[assign[i] + 1]++;
    }
    for (int64_t p = 0; p < nlist; ++p)
        L->start[p + 1] += L->start[p];
    int64_t *fill = (int64_t *)malloc((size_t)nlist * sizeof(int64_t) + 1);
    if (!fill)
        return -1;
    memcpy(fill, L->start, (size_t)nlist * sizeof(int64_t));
    for (int64_t i = 0; i < n; ++i)
        L->rows[fill[assign[i]]++] = i;
    free(fill);
    return 0;
}

static void lists_free(lists_t *L)
{
    free(L->start);
    free(L->rows);
}

/* ------------------------------------------------------------------------ */
/* Centroid ranking (Sec. 2.3, Sec. 4.1): P_i lists the nprobe centroids     */
/* closest to q_i, closest first.  For unit vectors the closest centroid by  */
/* cosine is the one with the largest inner product; ties: lower id first.  */
typedef struct {
    double score;
    int32_t cid;
} cscore_t;

static int cscore_cmp(const void *a, const void *b)
{
    const cscore_t *x = (const cscore_t *)a, *y = (const cscore_t *)b;
    if (x->score > y->score) return -1;
    if (x->score < y->score) return 1;
    return (x->cid > y->cid) - (x->cid < y->cid);
}

/* fills order[0..nprobe) and, if cs != NULL, the fp64 scores of every
 * centroid in rank order cs[0..nlist) */
static void rank_one(const float *q, const float *C, int64_t nlist, int d, int nprobe,
                     cscore_t *scratch, int32_t *order, double *cs)
{
    for (int64_t c = 0; c < nlist; ++c) {
        scratch[c].score = sim64(q, C + c * (int64_t)d, d);
        scratch[c].cid = (int32_t)c;
    }
    qsort(scratch, (size_t)nlist, sizeof(cscore_t), cscore_cmp);
    for (int j = 0; j < nprobe; ++j)
        order[j] = scratch[j].cid;
    if (cs)
        for (int64_t c = 0; c < nlist; ++c)
            cs[c] = scratch[c].score;
}

int oracle_rank(const float *Q, int64_t nq, const float *C, int64_t nlist, int32_t d,
                int32_t nprobe, int32_t *order, double *scores_out, int32_t nthreads)
{
    if (nprobe < 1 || nprobe > nlist || d <= 0)
        return -1;
    int bad = 0;
#pragma omp parallel num_threads(nthreads > 0 ? nthreads : 1)
    {
        cscore_t *scratch = (cscore_t *)malloc((size_t)nlist * sizeof(cscore_t));
        double *cs = (double *)malloc((size_t)nlist * sizeof(double));
        if (!scratch || !cs) {
#pragma omp atomic write
            bad = 1;
        } else {
#pragma omp for schedule(dynamic, 16)
            for (int64_t i = 0; i < nq; ++i) {
                rank_one(Q + i * (int64_t)d, C, nlist, d, nprobe, scratch,
                         order + i * (int64_t)nprobe, cs);
                if (scores_out)
                    for (int j = 0; j < nprobe; ++j)
                        scores_out[i * (int64_t)nprobe + j] = cs[j];
            }
        }
        free(scratch);
        free(cs);
    }
    return bad ? -2 : 0;
}

/* ------------------------------------------------------------------------ */
/* Stopping rule.  A probe callback searches the partition at 1-based rank   */
/* j of the query's order and reports whether it held a qualifying           */
/* candidate (a "hit"; Sec. 4.1: empty means no candidate with sim >= tau).  */
typedef int (*probe_fn)(void *ctx, int rank);

/* Sequential form (Sec. 4.1 and the continuation of Algorithm 1): walk the
 * order one rank at a time; a hit clears the run of consecutive empties, an
 * empty lengthens it; the query stops once the run reaches W or the order is
 * exhausted.  Returns the number of partitions searched. */
static int stop_sequential(int nprobe, int64_t W, probe_fn f, void *ctx)
{
    int searched = 0;
    int64_t stale = 0;
    while (searched < nprobe && stale < W) {
        ++searched;
        if (f(ctx, searched))
            stale = 0;
        else
            ++stale;
    }
    return searched;
}

/* splitmix64 (Steele, Lea, Flood 2014): drives the completion order below */
static uint64_t splitmix64(uint64_t *x)
{
    uint64_t z = (*x += 0x9E3779B97F4A7C15ull);
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

/* Lookahead form (Sec. 4.3, Algorithm 2): the stop line s starts at
 * min(W, nprobe); every rank up to s is committed and is enqueued as soon as
 * it is committed (cursor e = first rank not yet enqueued).  Enqueued ranks
 * complete in an arbitrary order, modelled here by drawing the next
 * completion uniformly from the pending set with a seeded generator.  A hit
 * at rank j moves the stop line to max(s, min(j + W, nprobe)).  Returns the
 * final stop line; visits[j] counts the searches of rank j. */
static int stop_lookahead(int nprobe, int64_t W, probe_fn f, void *ctx, uint64_t seed,
                          int *pending, int *visits)
{
    int64_t s = W < nprobe ? W : nprobe;
    int e = 1, npend = 0;
    uint64_t rng = seed;
    while (e <= s)
        pending[npend++] = e++;
    while (npend > 0) {
        int pick = (int)(splitmix64(&rng) % (uint64_t)npend);
        int j = pending[pick];
        pending[pick] = pending[--npend];
        if (visits)
            visits[j]++;
        if (f(ctx, j)) {
            int64_t reach = (int64_t)j + W;
            if (reach > nprobe)
                reach = nprobe;
            if (reach > s)
                s = reach;
            while (e <= s)
                pending[npend++] = e++;
        }
    }
    return (int)s;
}

/* stopping rule over a given hit pattern (hits[j-1] for rank j), exported so
 * the tests can pin the state machines on hand-built patterns */
static int pattern_probe(void *ctx, int rank)
{
    return ((const uint8_t *)ctx)[rank - 1] != 0;
}

int oracle_stop_pattern(const uint8_t *hits, int32_t nprobe, int64_t W, int32_t mode,
                        uint64_t seed, int32_t *visits_out)
{
    if (nprobe < 1 || W < 1)
        return -1;
    if (mode == 0)
        return stop_sequential(nprobe, W, pattern_probe, (void *)hits);
    int *pending = (int *)malloc(sizeof(int) * (size_t)(nprobe + 1));
    int *visits = (int *)calloc((size_t)nprobe + 1, sizeof(int));
    int r = stop_lookahead(nprobe, W, pattern_probe, (void *)hits, seed, pending, visits);
    if (visits_out)
        for (int j = 1; j <= nprobe; ++j)
            visits_out[j - 1] = visits[j];
    free(pending);
    free(visits);
    return r;
}

/* ------------------------------------------------------------------------ */
/* Within-partition search (Sec. 4.1, Sec. 5): score every row of partition  */
/* p against q, keep the local top-k of the rows with sim >= tau (the query  */
/* itself excluded), and report whether any row qualified.                   */
typedef struct {
    const float *X;
    const int64_t *ids;
    const lists_t *L;
    int d;
    /* quantized local search (NULL codes: exact inner products) */
    const uint8_t *codes;   /* [n][d] RaBitQ-style codes of the rows */
    const float *factors;   /* [n] per-row factor f */
    const float *C;         /* [nlist][d] centroids */
    double mid;             /* (2^bits - 1) / 2 */
} index_t;

static int local_search(const index_t *ix, const float *q, int has_qid, int64_t qid, int32_t p,
                        double tau, topk_t *local)
{
    int hit = 0;
    local->n = 0;
    for (int64_t r = ix->L->start[p]; r < ix->L->start[p + 1]; ++r) {
        int64_t row = ix->L->rows[r];
        int64_t id = ix->ids[row];
        if (has_qid && id == qid)
            continue;
        double s = sim64(q, ix->X + row * (int64_t)ix->d, ix->d);
        if (s >= tau) {
            hit = 1;
            topk_offer(local, s, id);
        }
    }
    return hit;
}

/* The same local search on RaBitQ-style codes (the paper's IVF_RQ7 local  */
/* search, Sec. 3.1 and Sec. 6.1): the estimate of <q, x> for a row x of    */
/* partition p with codes u and factor f is                                   */
/*     <q, c_p> + f * (<u, q'> - mid * sum_i q'_i),   q' = P^T q,             */
/* the estimator of oracle_rq_encode's header.                                */
/* the estimate for one row, given qc = <q, c_p> */
static double rq_estimate(const index_t *ix, const double *qrot, double sq, double qc, int64_t row)
{
    const int d = ix->d;
    const uint8_t *u = ix->codes + row * (int64_t)d;
    double dot = 0.0;
    for (int t = 0; t < d; ++t)
        dot += (double)u[t] * qrot[t];
    return qc + (double)ix->factors[row] * (dot - ix->mid * sq);
}

/* q' = P^T q and the sum of its coordinates */
static double rq_rotate_query(const double *P, const float *q, int d, double *qrot)
{
    double sq = 0.0;
    for (int t = 0; t < d; ++t) {
        double acc = 0.0;
        for (int j = 0; j < d; ++j)
            acc += P[(int64_t)j * d + t] * (double)q[j];
        qrot[t] = acc;
        sq += acc;
    }
    return sq;
}

static int rq_local_search(const index_t *ix, const float *q, const double *qrot, double sq,
                           int has_qid, int64_t qid, int32_t p, double tau, topk_t *local)
{
    const int d = ix->d;
    const double qc = sim64(q, ix->C + (int64_t)p * d, d);
    int hit = 0;
    local->n = 0;
    for (int64_t r = ix->L->start[p]; r < ix->L->start[p + 1]; ++r) {
        int64_t row = ix->L->rows[r];
        int64_t id = ix->ids[row];
        if (has_qid && id == qid)
            continue;
        double s = rq_estimate(ix, qrot, sq, qc, row);
        if (s >= tau) {
            hit = 1;
            topk_offer(local, s, id);
        }
    }
    return hit;
}

/* per-query state for one search (the "results" of Table 2 kept per rank) */
typedef struct {
    const index_t *ix;
    const float *q;
    int has_qid;
    int64_t qid;
    const int32_t *order; /* this query's P_i */
    double tau;
    int k;
    cand_t *local_store;  /* [nprobe][k] */
    int *local_n;         /* [nprobe] entries kept per rank, -1 = not searched */
    const double *qrot;   /* quantized search: P^T q, and its coordinate sum */
    double sq;
} query_ctx_t;

static int search_probe(void *vctx, int rank)
{
    query_ctx_t *c = (query_ctx_t *)vctx;
    topk_t local = {c->k, 0, c->local_store + (int64_t)(rank - 1) * c->k};
    int hit = c->ix->codes
                  ? rq_local_search(c->ix, c->q, c->qrot, c->sq, c->has_qid, c->qid,
                                    c->order[rank - 1], c->tau, &local)
                  : local_search(c->ix, c->q, c->has_qid, c->qid, c->order[rank - 1], c->tau,
                                 &local);
    c->local_n[rank - 1] = local.n;
    return hit;
}

/*
 * oracle_search: the per-query result of SieveIVF for every query.
 *   mode 0: sequential stopping (Algorithm 1 semantics, one query at a time)
 *   mode 1: lookahead scheduling (Algorithm 2) with seeded completion orders
 * The final result merges the local results of every searched rank into the
 * top-k (MergeTopK of Algorithm 1).  Scores are fp64 similarities.
 * order: [nq][nprobe] 0-based centroid ids, or NULL to rank here.
 * Outputs: out_ids [nq][k] (-1 pad), out_scores [nq][k] (-inf pad),
 * out_count [nq], out_probes [nq] = partitions searched.
 * Returns 0, or <0 on bad arguments; returns -3 if the lookahead form ever
 * searched a rank twice or skipped a rank below its stop line.
 */
typedef struct {
    const uint8_t *codes;
    const float *factors;
    const double *P;   /* [d][d] rotation */
    int bits;
} rq_in_t;

static int search_impl(const float *X, const int64_t *ids, const int32_t *assign, int64_t n,
                       int32_t d, const float *C, int64_t nlist, const float *Q, int64_t nq,
                       const int64_t *qids, const int32_t *order_in, float tau, int32_t k,
                       int32_t nprobe, int64_t W, int32_t mode, uint64_t seed, int64_t *out_ids,
                       double *out_scores, int32_t *out_count, int32_t *out_probes,
                       int32_t nthreads, const rq_in_t *rq);

int oracle_search(const float *X, const int64_t *ids, const int32_t *assign, int64_t n, int32_t d,
                  const float *C, int64_t nlist, const float *Q, int64_t nq, const int64_t *qids,
                  const int32_t *order_in, float tau, int32_t k, int32_t nprobe, int64_t W,
                  int32_t mode, uint64_t seed, int64_t *out_ids, double *out_scores,
                  int32_t *out_count, int32_t *out_probes, int32_t nthreads)
{
    return search_impl(X, ids, assign, n, d, C, nlist, Q, nq, qids, order_in, tau, k, nprobe, W,
                       mode, seed, out_ids, out_scores, out_count, out_probes, nthreads, NULL);
}

/* oracle_search with the quantized local search of rq_local_search: codes
 * [n][d], factors [n] as made by oracle_rq_encode with the same rotation P. */
int oracle_rq_search(const float *X, const int64_t *ids, const int32_t *assign, int64_t n,
                     int32_t d, const float *C, int64_t nlist, const uint8_t *codes,
                     const float *factors, const double *P, int32_t bits, const float *Q,
                     int64_t nq, const int64_t *qids, const int32_t *order_in, float tau, int32_t k,
                     int32_t nprobe, int64_t W, int32_t mode, uint64_t seed, int64_t *out_ids,
                     double *out_scores, int32_t *out_count, int32_t *out_probes, int32_t nthreads)
{
    if (!codes || !factors || !P || bits < 1 || bits > 8)
        return -1;
    rq_in_t rq = {codes, factors, P, bits};
    return search_impl(X, ids, assign, n, d, C, nlist, Q, nq, qids, order_in, tau, k, nprobe, W,
                       mode, seed, out_ids, out_scores, out_count, out_probes, nthreads, &rq);
}

static int search_impl(const float *X, const int64_t *ids, const int32_t *assign, int64_t n,
                       int32_t d, const float *C, int64_t nlist, const float *Q, int64_t nq,
                       const int64_t *qids, const int32_t *order_in, float tau, int32_t k,
                       int32_t nprobe, int64_t W, int32_t mode, uint64_t seed, int64_t *out_ids,
                       double *out_scores, int32_t *out_count, int32_t *out_probes,
                       int32_t nthreads, const rq_in_t *rq)
{
    if (d <= 0 || k < 1 || nprobe < 1 || nprobe > nlist || W < 1 || isnan(tau))
        return -1;
    lists_t L;
    if (lists_build(&L, assign, n, nlist) != 0) {
        lists_free(&L);
        return -2;
    }
    index_t ix = {X, ids, &L, d, NULL, NULL, C, 0.0};
    if (rq) {
        ix.codes = rq->codes;
        ix.factors = rq->factors;
        ix.mid = ((double)(1 << rq->bits) - 1.0) / 2.0;
    }
    int bad = 0;
#pragma omp parallel num_threads(nthreads > 0 ? nthreads : 1)
    {
        cscore_t *scratch = (cscore_t *)malloc((size_t)nlist * sizeof(cscore_t));
        int32_t *order = (int32_t *)malloc((size_t)nprobe * sizeof(int32_t));
        cand_t *store = (cand_t *)malloc((size_t)nprobe * (size_t)k * sizeof(cand_t));
        int *local_n = (int *)malloc((size_t)nprobe * sizeof(int));
        int *pending = (int *)malloc((size_t)(nprobe + 1) * sizeof(int));
        int *visits = (int *)malloc((size_t)(nprobe + 1) * sizeof(int));
        cand_t *fin = (cand_t *)malloc((size_t)k * sizeof(cand_t));
        double *qrot = (double *)malloc((size_t)d * sizeof(double));
        if (!scratch || !order || !store || !local_n || !pending || !visits || !fin || !qrot) {
#pragma omp atomic write
            bad = -2;
        } else {
#pragma omp for schedule(dynamic, 4)
            for (int64_t i = 0; i < nq; ++i) {
                const float *q = Q + i * (int64_t)d;
                const int32_t *P = order;
                if (order_in)
                    P = order_in + i * (int64_t)nprobe;
                else
                    rank_one(q, C, nlist, d, nprobe, scratch, order, NULL);
                for (int j = 0; j < nprobe; ++j)
                    local_n[j] = -1;
                double sq = 0.0;
                if (rq)   /* q' = P^T q and its coordinate sum */
                    sq = rq_rotate_query(rq->P, q, d, qrot);
                query_ctx_t ctx = {&ix, q, qids != NULL, qids ? qids[i] : 0, P, (double)tau,
                                   k, store, local_n, qrot, sq};
                int probes;
                if (mode == 0) {
                    probes = stop_sequential(nprobe, W, search_probe, &ctx);
                } else {
                    memset(visits, 0, sizeof(int) * (size_t)(nprobe + 1));
                    uint64_t qseed = seed ^ (0xD1B54A32D192ED03ull * (uint64_t)(i + 1));
                    probes = stop_lookahead(nprobe, W, search_probe, &ctx, qseed, pending, visits);
                    for (int j = 1; j <= nprobe; ++j)
                        if (visits[j] != (j <= probes ? 1 : 0)) {
#pragma omp atomic write
                            bad = -3;
                        }
                }
                /* MergeTopK over the local results of the searched ranks */
                topk_t final = {k, 0, fin};
                for (int j = 0; j < nprobe; ++j)
                    for (int m = 0; m < (local_n[j] > 0 ? local_n[j] : 0); ++m)
                        topk_offer(&final, store[(int64_t)j * k + m].score,
                                   store[(int64_t)j * k + m].id);
                for (int m = 0; m < k; ++m) {
                    out_ids[i * (int64_t)k + m] = m < final.n ? fin[m].id : -1;
                    out_scores[i * (int64_t)k + m] = m < final.n ? fin[m].score : -INFINITY;
                }
                out_count[i] = final.n;
                out_probes[i] = probes;
            }
        }
        free(scratch); free(order); free(store); free(local_n);
        free(pending); free(visits); free(fin); free(qrot);
    }
    lists_free(&L);
    return bad;
}

/* ------------------------------------------------------------------------ */
/* hit matrix: hits[i][j] = 1 iff rank j+1 of query i holds a qualifying row */
/* (all nprobe ranks, regardless of stopping); used by tests to relate the   */
/* searched prefix to the hit pattern                                        */
int oracle_hit_matrix(const float *X, const int64_t *ids, const int32_t *assign, int64_t n,
                      int32_t d, int64_t nlist, const float *Q, int64_t nq, const int64_t *qids,
                      const int32_t *order, float tau, int32_t nprobe, uint8_t *hits,
                      int32_t nthreads)
{
    if (d <= 0 || nprobe < 1 || nprobe > nlist)
        return -1;
    lists_t L;
    if (lists_build(&L, assign, n, nlist) != 0) {
        lists_free(&L);
        return -2;
    }
    index_t ix = {X, ids, &L, d, NULL, NULL, NULL, 0.0};
#pragma omp parallel for schedule(dynamic, 4) num_threads(nthreads > 0 ? nthreads : 1)
    for (int64_t i = 0; i < nq; ++i) {
        cand_t one;
        for (int j = 0; j < nprobe; ++j) {
            topk_t local = {1, 0, &one};
            hits[i * (int64_t)nprobe + j] = (uint8_t)local_search(
                &ix, Q + i * (int64_t)d, qids != NULL, qids ? qids[i] : 0,
                order[i * (int64_t)nprobe + j], (double)tau, &local);
        }
    }
    lists_free(&L);
    return 0;
}

/* ------------------------------------------------------------------------ */
/* Fixed-probe IVF (Sec. 2.3): the filtered top-k over the union of the      */
/* first nprobe partitions of each query's order, in one plain loop.         */
int oracle_fixed_probe(const float *X, const int64_t *ids, const int32_t *assign, int64_t n,
                       int32_t d, int64_t nlist, const float *Q, int64_t nq, const int64_t *qids,
                       const int32_t *order, float tau, int32_t k, int32_t nprobe,
                       int64_t *out_ids, double *out_scores, int32_t *out_count,
                       int32_t nthreads)
{
    if (d <= 0 || k < 1 || nprobe < 1 || nprobe > nlist)
        return -1;
    lists_t L;
    if (lists_build(&L, assign, n, nlist) != 0) {
        lists_free(&L);
        return -2;
    }
#pragma omp parallel num_threads(nthreads > 0 ? nthreads : 1)
    {
        cand_t *fin = (cand_t *)malloc((size_t)k * sizeof(cand_t));
#pragma omp for schedule(dynamic, 4)
        for (int64_t i = 0; i < nq; ++i) {
            topk_t t = {k, 0, fin};
            const float *q = Q + i * (int64_t)d;
            for (int j = 0; j < nprobe; ++j) {
                int32_t p = order[i * (int64_t)nprobe + j];
                for (int64_t r = L.start[p]; r < L.start[p + 1]; ++r) {
                    int64_t row = L.rows[r];
                    if (qids && ids[row] == qids[i])
                        continue;
                    double s = sim64(q, X + row * (int64_t)d, d);
                    if (s >= (double)tau)
                        topk_offer(&t, s, ids[row]);
                }
            }
            for (int m = 0; m < k; ++m) {
                out_ids[i * (int64_t)k + m] = m < t.n ? fin[m].id : -1;
                out_scores[i * (int64_t)k + m] = m < t.n ? fin[m].score : -INFINITY;
            }
            out_count[i] = t.n;
        }
        free(fin);
    }
    lists_free(&L);
    return 0;
}

/* ------------------------------------------------------------------------ */
/* Exhaustive filtered top-k over all n rows (the ground truth G_{tau,k} of  */
/* Sec. 6.1).  Also the expected result of nprobe = nlist with W = infinity. */
int oracle_bruteforce(const float *X, const int64_t *ids, int64_t n, int32_t d, const float *Q,
                      int64_t nq, const int64_t *qids, float tau, int32_t k, int64_t *out_ids,
                      double *out_scores, int32_t *out_count, int32_t nthreads)
{
    if (d <= 0 || k < 1)
        return -1;
#pragma omp parallel num_threads(nthreads > 0 ? nthreads : 1)
    {
        cand_t *fin = (cand_t *)malloc((size_t)k * sizeof(cand_t));
#pragma omp for schedule(dynamic, 4)
        for (int64_t i = 0; i < nq; ++i) {
            topk_t t = {k, 0, fin};
            for (int64_t row = 0; row < n; ++row) {
                if (qids && ids[row] == qids[i])
                    continue;
                double s = sim64(Q + i * (int64_t)d, X + row * (int64_t)d, d);
                if (s >= (double)tau)
                    topk_offer(&t, s, ids[row]);
            }
            for (int m = 0; m < k; ++m) {
                out_ids[i * (int64_t)k + m] = m < t.n ? fin[m].id : -1;
                out_scores[i * (int64_t)k + m] = m < t.n ? fin[m].score : -INFINITY;
            }
            out_count[i] = t.n;
        }
        free(fin);
    }
    return 0;
}

/* ------------------------------------------------------------------------ */
/* Fragility tags: how close a query's decisions sit to a rounding flip.     */
/* For query i and its first upto[i] ranks (order[i][.]):                    */
/*   tau_gap[i]  = min |sim - tau| over the non-self rows of those partitions */
/*   kth_gap[i]  = sim(k-th) - sim(k+1-th) among their qualifying rows        */
/*                 (+inf when fewer than k+1 qualify)                         */
/*   cen_gap[i]  = min gap between consecutive fp64 centroid scores among     */
/*                 ranks 1..min(nprobe+1, nlist)                              */
static int fragility_impl(const float *X, const int64_t *ids, const int32_t *assign, int64_t n,
                          int32_t d, const float *C, int64_t nlist, const float *Q, int64_t nq,
                          const int64_t *qids, const int32_t *order, const int32_t *upto,
                          float tau, int32_t k, int32_t nprobe, double *tau_gap, double *kth_gap,
                          double *cen_gap, int32_t nthreads, const rq_in_t *rq)
{
    if (d <= 0 || k < 1 || nprobe < 1 || nprobe > nlist)
        return -1;
    lists_t L;
    if (lists_build(&L, assign, n, nlist) != 0) {
        lists_free(&L);
        return -2;
    }
    index_t ix = {X, ids, &L, d, NULL, NULL, C, 0.0};
    if (rq) {
        ix.codes = rq->codes;
        ix.factors = rq->factors;
        ix.mid = ((double)(1 << rq->bits) - 1.0) / 2.0;
    }
#pragma omp parallel num_threads(nthreads > 0 ? nthreads : 1)
    {
        cand_t *fin = (cand_t *)malloc((size_t)(k + 1) * sizeof(cand_t));
        cscore_t *scratch = (cscore_t *)malloc((size_t)nlist * sizeof(cscore_t));
        int32_t *ord = (int32_t *)malloc((size_t)nprobe * sizeof(int32_t));
        double *cs = (double *)malloc((size_t)nlist * sizeof(double));
        double *qrot = (double *)malloc((size_t)d * sizeof(double));
#pragma omp for schedule(dynamic, 4)
        for (int64_t i = 0; i < nq; ++i) {
            const float *q = Q + i * (int64_t)d;
            topk_t t = {k + 1, 0, fin};
            double tg = INFINITY;
            int lim = upto[i] < nprobe ? upto[i] : nprobe;
            const double sq = rq ? rq_rotate_query(rq->P, q, d, qrot) : 0.0;
            for (int j = 0; j < lim; ++j) {
                int32_t p = order[i * (int64_t)nprobe + j];
                const double qc = rq ? sim64(q, C + (int64_t)p * d, d) : 0.0;
                for (int64_t r = L.start[p]; r < L.start[p + 1]; ++r) {
                    int64_t row = L.rows[r];
                    if (qids && ids[row] == qids[i])
                        continue;
                    double s = rq ? rq_estimate(&ix, qrot, sq, qc, row)
                                  : sim64(q, X + row * (int64_t)d, d);
                    double g = fabs(s - (double)tau);
                    if (g < tg)
                        tg = g;
                    if (s >= (double)tau)
                        topk_offer(&t, s, ids[row]);
                }
            }
            tau_gap[i] = tg;
            kth_gap[i] = (t.n > k) ? fin[k - 1].score - fin[k].score : INFINITY;
            rank_one(q, C, nlist, d, nprobe, scratch, ord, cs);
            double cg = INFINITY;
            int64_t top = (int64_t)nprobe + 1 < nlist ? (int64_t)nprobe + 1 : nlist;
            for (int64_t j = 0; j + 1 < top; ++j) {
                double g = cs[j] - cs[j + 1];
                if (g < cg)
                    cg = g;
            }
            cen_gap[i] = cg;
        }
        free(fin); free(scratch); free(ord); free(cs); free(qrot);
    }
    lists_free(&L);
    return 0;
}

int oracle_fragility(const float *X, const int64_t *ids, const int32_t *assign, int64_t n,
                     int32_t d, const float *C, int64_t nlist, const float *Q, int64_t nq,
                     const int64_t *qids, const int32_t *order, const int32_t *upto, float tau,
                     int32_t k, int32_t nprobe, double *tau_gap, double *kth_gap,
                     double *cen_gap, int32_t nthreads)
{
    return fragility_impl(X, ids, assign, n, d, C, nlist, Q, nq, qids, order, upto, tau, k, nprobe,
                          tau_gap, kth_gap, cen_gap, nthreads, NULL);
}

/* oracle_fragility with the quantized estimates (codes and factors as for
 * oracle_rq_search): the gaps of the estimates the quantized search decides on */
int oracle_rq_fragility(const float *X, const int64_t *ids, const int32_t *assign, int64_t n,
                        int32_t d, const float *C, int64_t nlist, const uint8_t *codes,
                        const float *factors, const double *P, int32_t bits, const float *Q,
                        int64_t nq, const int64_t *qids, const int32_t *order, const int32_t *upto,
                        float tau, int32_t k, int32_t nprobe, double *tau_gap, double *kth_gap,
                        double *cen_gap, int32_t nthreads)
{
    if (!codes || !factors || !P || bits < 1 || bits > 8)
        return -1;
    rq_in_t rq = {codes, factors, P, bits};
    return fragility_impl(X, ids, assign, n, d, C, nlist, Q, nq, qids, order, upto, tau, k, nprobe,
                          tau_gap, kth_gap, cen_gap, nthreads, &rq);
}

/* ------------------------------------------------------------------------ */
/* In-call window calibration (Appendix A, Algorithm 3).                      */
/*                                                                            */
/* The sample Q_s is given as ns sorted, distinct row indices into Q (the     */
/* paper draws it uniformly without replacement; here the caller does).      */
/*  1. nq < min_queries or ns == 0: W* = fallback and every query runs the   */
/*     W*-rule (the paper's fallback for small calls).                        */
/*  2. FullProbeByPartition: each sampled query searches all nprobe ranks of */
/*     its order; L_s = the local result of every rank.                       */
/*  3. A_fixed = MergeTopK(L_s, k); each neighbour keeps the rank it came    */
/*     from (every row sits in exactly one partition).                        */
/*  4. RequiredWindowHistogram: window W reaches rank j iff no run of W      */
/*     consecutive empty ranks ends before j (the stop rule of Sec. 4.1), so */
/*     a neighbour found at rank j needs W >= 1 + (longest run of empty      */
/*     ranks before j); H[W] counts neighbours by that required window.      */
/*  5. Z = sum |A_fixed(q)|; W* = the smallest W < nprobe with               */
/*     1 - (H[1] + ... + H[W]) / Z < eps, else nprobe; Z == 0: W* = fallback.*/
/*  6. Every other query runs the W*-rule (sequential form); the sampled     */
/*     queries keep A_fixed and report nprobe probes.                         */
/* hist: [nprobe + 1] (H[0] unused); outputs as oracle_search.                */
int oracle_calibrate(const float *X, const int64_t *ids, const int32_t *assign, int64_t n,
                     int32_t d, const float *C, int64_t nlist, const float *Q, int64_t nq,
                     const int64_t *qids, const int64_t *sample, int64_t ns, float tau, int32_t k,
                     int32_t nprobe, double eps, int64_t min_queries, int64_t fallback,
                     int64_t *out_ids, double *out_scores, int32_t *out_count,
                     int32_t *out_probes, int64_t *W_out, int64_t *hist, int64_t *Z_out,
                     int32_t nthreads)
{
    if (d <= 0 || k < 1 || nprobe < 1 || nprobe > nlist || fallback < 1 || isnan(tau) || ns < 0)
        return -1;
    for (int64_t s = 0; s < ns; ++s)
        if (sample[s] < 0 || sample[s] >= nq || (s > 0 && sample[s] <= sample[s - 1]))
            return -1;
    for (int w = 0; w <= nprobe; ++w)
        hist[w] = 0;
    *Z_out = 0;
    if (nq < min_queries || ns == 0) {
        *W_out = fallback;
        return oracle_search(X, ids, assign, n, d, C, nlist, Q, nq, qids, NULL, tau, k, nprobe,
                             fallback, 0, 0, out_ids, out_scores, out_count, out_probes, nthreads);
    }
    lists_t L;
    if (lists_build(&L, assign, n, nlist) != 0) {
        lists_free(&L);
        return -2;
    }
    index_t ix = {X, ids, &L, d, NULL, NULL, C, 0.0};
    int64_t Z = 0;
    int bad = 0;
    /* steps 2-4 for every sampled query */
#pragma omp parallel num_threads(nthreads > 0 ? nthreads : 1)
    {
        cscore_t *scratch = (cscore_t *)malloc((size_t)nlist * sizeof(cscore_t));
        int32_t *order = (int32_t *)malloc((size_t)nprobe * sizeof(int32_t));
        cand_t *store = (cand_t *)malloc((size_t)nprobe * (size_t)k * sizeof(cand_t));
        int *local_n = (int *)malloc((size_t)nprobe * sizeof(int));
        cand_t *fin = (cand_t *)malloc((size_t)k * sizeof(cand_t));
        int64_t *h = (int64_t *)calloc((size_t)nprobe + 1, sizeof(int64_t));
        int64_t z = 0;
        if (!scratch || !order || !store || !local_n || !fin || !h) {
#pragma omp atomic write
            bad = -2;
        } else {
#pragma omp for schedule(dynamic, 4)
            for (int64_t s = 0; s < ns; ++s) {
                const int64_t i = sample[s];
                const float *q = Q + i * (int64_t)d;
                rank_one(q, C, nlist, d, nprobe, scratch, order, NULL);
                /* FullProbeByPartition: L_s, rank by rank */
                query_ctx_t ctx = {&ix, q, qids != NULL, qids ? qids[i] : 0, order, (double)tau,
                                   k, store, local_n};
                for (int j = 1; j <= nprobe; ++j)
                    search_probe(&ctx, j);
                /* MergeTopK */
                topk_t final = {k, 0, fin};
                for (int j = 0; j < nprobe; ++j)
                    for (int m = 0; m < local_n[j]; ++m)
                        topk_offer(&final, store[(int64_t)j * k + m].score,
                                   store[(int64_t)j * k + m].id);
                /* RequiredWindowHistogram: walk the ranks in order */
                int run = 0, longest = 0;
                for (int j = 1; j <= nprobe; ++j) {
                    for (int m = 0; m < final.n; ++m) {   /* neighbours found at rank j */
                        int from_j = 0;
                        for (int t = 0; t < local_n[j - 1]; ++t)
                            if (store[(int64_t)(j - 1) * k + t].id == fin[m].id)
                                from_j = 1;
                        if (from_j)
                            h[1 + longest]++;
                    }
                    run = local_n[j - 1] > 0 ? 0 : run + 1;   /* a hit has a local result */
                    if (run > longest)
                        longest = run;
                }
                z += final.n;
                for (int m = 0; m < k; ++m) {
                    out_ids[i * (int64_t)k + m] = m < final.n ? fin[m].id : -1;
                    out_scores[i * (int64_t)k + m] = m < final.n ? fin[m].score : -INFINITY;
                }
                out_count[i] = final.n;
                out_probes[i] = nprobe;
            }
#pragma omp critical
            {
                for (int w = 0; w <= nprobe; ++w)
                    hist[w] += h[w];
                Z += z;
            }
        }
        free(scratch); free(order); free(store); free(local_n); free(fin); free(h);
    }
    lists_free(&L);
    if (bad)
        return bad;
    /* step 5: the smallest pruned window under the loss target */
    int64_t Wstar = nprobe;
    if (Z == 0) {
        Wstar = fallback;
    } else {
        int64_t retained = 0;
        for (int w = 1; w < nprobe; ++w) {
            retained += hist[w];
            double loss = 1.0 - (double)retained / (double)Z;
            if (loss < eps) {
                Wstar = w;
                break;
            }
        }
    }
    *W_out = Wstar;
    *Z_out = Z;
    /* step 6: the rest of the batch under W* */
    int64_t nr = nq - ns;
    if (nr == 0)
        return 0;
    float *Qr = (float *)malloc((size_t)nr * (size_t)d * sizeof(float));
    int64_t *qr = qids ? (int64_t *)malloc((size_t)nr * sizeof(int64_t)) : NULL;
    int64_t *idx = (int64_t *)malloc((size_t)nr * sizeof(int64_t));
    int64_t *oi = (int64_t *)malloc((size_t)nr * (size_t)k * sizeof(int64_t));
    double *os = (double *)malloc((size_t)nr * (size_t)k * sizeof(double));
    int32_t *oc = (int32_t *)malloc((size_t)nr * sizeof(int32_t));
    int32_t *op = (int32_t *)malloc((size_t)nr * sizeof(int32_t));
    int rc = -2;
    if (Qr && (qr || !qids) && idx && oi && os && oc && op) {
        int64_t r = 0, s = 0;
        for (int64_t i = 0; i < nq; ++i) {
            if (s < ns && sample[s] == i) {
                ++s;
                continue;
            }
            idx[r] = i;
            memcpy(Qr + r * (int64_t)d, Q + i * (int64_t)d, (size_t)d * sizeof(float));
            if (qids)
                qr[r] = qids[i];
            ++r;
        }
        rc = oracle_search(X, ids, assign, n, d, C, nlist, Qr, nr, qr, NULL, tau, k, nprobe, Wstar,
                           0, 0, oi, os, oc, op, nthreads);
        if (rc == 0)
            for (int64_t r2 = 0; r2 < nr; ++r2) {
                int64_t i = idx[r2];
                memcpy(out_ids + i * (int64_t)k, oi + r2 * (int64_t)k, (size_t)k * sizeof(int64_t));
                memcpy(out_scores + i * (int64_t)k, os + r2 * (int64_t)k, (size_t)k * sizeof(double));
                out_count[i] = oc[r2];
                out_probes[i] = op[r2];
            }
    }
    free(Qr); free(qr); free(idx); free(oi); free(os); free(oc); free(op);
    return rc;
}


/* ------------------------------------------------------------------------ */
/* RaBitQ-style codes of the rows (the paper's IVF_RQ7, Sec. 3.1: RaBitQ     */
/* configured with 7 bits), given a d x d orthogonal rotation P (row-major). */
/* For a row x of partition p, with r = x - c_p:                             */
/*   o  = r / |r|,  o' = P^T o   (o'_i = sum_j P[j][i] o_j)                   */
/*   D  = 2 max_i |o'_i| / (2^bits - 1),  mid = (2^bits - 1) / 2             */
/*   u_i = rint(o'_i / D + mid) clamped to [0, 2^bits - 1]  (the codes)      */
/*   f  = |r| / <u - mid, o'>  (stored as fp32)                               */
/* and the estimate of <q, x> is <q, c_p> + f (<u, q'> - mid sum_i q'_i),    */
/* q' = P^T q: RaBitQ's estimator <o', q'> ~ <o_bar, q'> / <o_bar, o'> with   */
/* o_bar the normalised code vector, scaled back by |r| and shifted by the   */
/* centroid term.  A row equal to its centroid gets codes rint(mid), f = 0.  */
/* Every sum runs in fp64 in index order with fused multiply-adds, so an     */
/* implementation that does the same gets the same codes and factors.        */
int oracle_rq_encode(const float *X, const int32_t *assign, int64_t n, int32_t d, const float *C,
                     int64_t nlist, const double *P, int32_t bits, uint8_t *codes, float *factors,
                     int32_t nthreads)
{
    if (d <= 0 || bits < 1 || bits > 8 || !P)
        return -1;
    const double top = (double)((1 << bits) - 1), mid = top / 2.0;
    int bad = 0;
#pragma omp parallel num_threads(nthreads > 0 ? nthreads : 1)
    {
        double *o = (double *)malloc((size_t)d * sizeof(double));
        double *rot = (double *)malloc((size_t)d * sizeof(double));
        if (!o || !rot) {
#pragma omp atomic write
            bad = -2;
        } else {
#pragma omp for schedule(static)
            for (int64_t i = 0; i < n; ++i) {
                const int32_t p = assign[i];
                uint8_t *u = codes + i * (int64_t)d;
                if (p < 0 || p >= nlist) {
#pragma omp atomic write
                    bad = -1;
                    continue;
                }
                const float *x = X + i * (int64_t)d, *c = C + (int64_t)p * d;
                double nn = 0.0;
                for (int j = 0; j < d; ++j) {
                    o[j] = (double)x[j] - (double)c[j];
                    nn = fma(o[j], o[j], nn);
                }
                const double norm = sqrt(nn);
                if (norm == 0.0) {
                    for (int t = 0; t < d; ++t)
                        u[t] = (uint8_t)rint(mid);
                    factors[i] = 0.0f;
                    continue;
                }
                for (int j = 0; j < d; ++j)
                    o[j] = o[j] / norm;
                double mx = 0.0;
                for (int t = 0; t < d; ++t) {
                    double acc = 0.0;
                    for (int j = 0; j < d; ++j)
                        acc = fma(P[(int64_t)j * d + t], o[j], acc);
                    rot[t] = acc;
                    if (fabs(acc) > mx)
                        mx = fabs(acc);
                }
                const double delta = 2.0 * mx / top;
                double dot = 0.0;
                for (int t = 0; t < d; ++t) {
                    double v = rint(rot[t] / delta + mid);
                    v = v < 0.0 ? 0.0 : (v > top ? top : v);
                    u[t] = (uint8_t)v;
                    dot = fma(v - mid, rot[t], dot);
                }
                factors[i] = (float)(norm / dot);
            }
        }
        free(o);
        free(rot);
    }
    return bad;
}
