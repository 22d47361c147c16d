/*
 * CPU oracle for region-conditional sparse retrieval (RCSR).
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the plain, slow, obviously correct
 * statement of what the GPU path computes.  Only the tests, the smoke check
 * and the benchmark's CPU-baseline leg may load it; the product path never
 * does.  It shares no code, header, table or helper with the CUDA library.
 *
 * What it computes (paper §3.3 Eq. rcsr; App. B.2 Def. B.2; Alg. 1 "RCSR"
 * loop and "Dedup" step):
 *
 *   1. score      s(r, i) = sum_j q_{r,j} * x_{i,j}            (MIPS, Def. B.2)
 *                 q = bf16 region query, x = dequantised corpus row
 *                 (bf16, or e4m3 times the row's fp32 scale); fp64, j order.
 *   2. per region L_r = the first k_region ids of {0..N-1} ordered by
 *                 (s(r, i) descending, i ascending)       (top-k', Eq. rcsr)
 *   3. per question q with regions r in [off[q], off[q+1]):
 *                 U_q = union of L_r; m(i) = max over those r with i in L_r
 *                 of s(r, i); output the first K of U_q ordered by
 *                 (m descending, id ascending); pad with (-1, -inf).
 *                 (§3.3 "deduplicate the union of K_r"; Def. B.2 Dedup.)
 *
 * Readings where the paper is silent: duplicate ids keep their maximum
 * score; ties go to the lower id at both stages; slots past the number of
 * unique candidates are padded with id -1 and score -inf; the region count
 * per question is whatever the offsets say.
 *
 * Pins (tests/test_oracle_pins.py): a hand-worked integer example, brute
 * force by full sort, one-hot and self-score closed forms, planted nearest
 * neighbours, duplicate-row ties, merge invariants and the e4m3 decode.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

/* ---- number formats -------------------------------------------------- */

/* bf16 is the upper half of an IEEE-754 binary32. */
static double bf16_value(uint16_t h)
{
    uint32_t u = (uint32_t)h << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

/* OCP FP8 E4M3 ("FN"): sign, 4 exponent bits with bias 7, 3 mantissa bits;
 * exponent field 0 holds subnormals m * 2^-9; S.1111.111 is NaN; there are no
 * infinities. */
static double e4m3_value(uint8_t b)
{
    int s = (b >> 7) & 1, e = (b >> 3) & 15, m = b & 7;
    double v;
    if (e == 15 && m == 7)
        return NAN;
    if (e == 0)
        v = ldexp((double)m, -9);
    else
        v = ldexp(1.0 + (double)m / 8.0, e - 7);
    return s ? -v : v;
}

double skip_oracle_bf16_value(uint16_t h) { return bf16_value(h); }
double skip_oracle_e4m3_value(uint8_t b) { return e4m3_value(b); }

/* ---- scoring (Def. B.2: maximum inner product) ----------------------- */

typedef struct {
    const uint16_t *bf16; /* [N, d] bf16 bits, or NULL */
    const uint8_t *e4m3;  /* [N, d] e4m3 bytes, or NULL */
    const float *scale;   /* [N] row scales (e4m3 only) */
    int64_t N;
    int d;
} corpus_t;

static double e4m3_table[256];

static void init_tables(void)
{
    for (int b = 0; b < 256; ++b)
        e4m3_table[b] = e4m3_value((uint8_t)b);
}

/* s(r, i) = sum_j q_j * x_{i,j}, in fp64, in j order. */
static double score(const corpus_t *c, const double *q, int64_t i)
{
    double s = 0.0;
    if (c->bf16) {
        const uint16_t *x = c->bf16 + i * (int64_t)c->d;
        for (int j = 0; j < c->d; ++j)
            s += q[j] * bf16_value(x[j]);
    } else {
        const uint8_t *x = c->e4m3 + i * (int64_t)c->d;
        double sc = (double)c->scale[i];
        for (int j = 0; j < c->d; ++j)
            s += q[j] * (e4m3_table[x[j]] * sc);
    }
    return s;
}

/* ---- candidates ordered by (score desc, id asc) ----------------------- */

typedef struct {
    double s;
    int64_t id;
} cand_t;

/* a ranks before b */
static int ranks_before(cand_t a, cand_t b)
{
    return a.s > b.s || (a.s == b.s && a.id < b.id);
}

static int cmp_rank(const void *pa, const void *pb)
{
    cand_t a = *(const cand_t *)pa, b = *(const cand_t *)pb;
    if (ranks_before(a, b))
        return -1;
    if (ranks_before(b, a))
        return 1;
    return 0;
}

/* (id asc, score desc): the first entry of each id run holds its max. */
static int cmp_id_then_score(const void *pa, const void *pb)
{
    cand_t a = *(const cand_t *)pa, b = *(const cand_t *)pb;
    if (a.id != b.id)
        return a.id < b.id ? -1 : 1;
    if (a.s != b.s)
        return a.s > b.s ? -1 : 1;
    return 0;
}

/* Bounded heap holding the best `cap` candidates seen; the root is the one
 * that ranks last, so a newcomer only has to beat the root. */
static void heap_sift_down(cand_t *h, int n, int at)
{
    for (;;) {
        int l = 2 * at + 1, r = l + 1, w = at;
        if (l < n && ranks_before(h[w], h[l]))
            w = l;
        if (r < n && ranks_before(h[w], h[r]))
            w = r;
        if (w == at)
            return;
        cand_t t = h[at];
        h[at] = h[w];
        h[w] = t;
        at = w;
    }
}

static void heap_sift_up(cand_t *h, int at)
{
    while (at > 0) {
        int p = (at - 1) / 2;
        if (!ranks_before(h[p], h[at]))
            return;
        cand_t t = h[at];
        h[at] = h[p];
        h[p] = t;
        at = p;
    }
}

/* Step 2 for one region: the exact top-kk of the corpus by (s desc, id asc). */
static void region_topk_one(const corpus_t *c, const uint16_t *qbits, int kk, cand_t *heap,
                            double *q, int64_t *out_ids, double *out_scores)
{
    for (int j = 0; j < c->d; ++j)
        q[j] = bf16_value(qbits[j]);
    int n = 0;
    for (int64_t i = 0; i < c->N; ++i) {
        cand_t x = {score(c, q, i), i};
        if (n < kk) {
            heap[n] = x;
            heap_sift_up(heap, n);
            ++n;
        } else if (ranks_before(x, heap[0])) {
            heap[0] = x;
            heap_sift_down(heap, n, 0);
        }
    }
    qsort(heap, (size_t)n, sizeof(cand_t), cmp_rank);
    for (int t = 0; t < kk; ++t) {
        out_ids[t] = t < n ? heap[t].id : -1;
        out_scores[t] = t < n ? heap[t].s : -INFINITY;
    }
}

static int resolve_threads(int nthreads)
{
#ifdef _OPENMP
    return nthreads > 0 ? nthreads : omp_get_max_threads();
#else
    (void)nthreads;
    return 1;
#endif
}

/*
 * Step 1 + 2 for every region: out_ids/out_scores [R x kk], row r sorted by
 * (score desc, id asc); slots beyond N are (-1, -inf).  Regions are spread
 * over `nthreads` OpenMP threads (0 = all); each region is computed by one
 * thread exactly as written above.
 */
int skip_oracle_region_topk(const uint16_t *corpus_bf16, const uint8_t *corpus_e4m3,
                            const float *row_scale, int64_t N, int d,
                            const uint16_t *regions, int64_t R, int kk,
                            int64_t *out_ids, double *out_scores, int nthreads)
{
    if ((corpus_bf16 == NULL) == (corpus_e4m3 == NULL) || (corpus_e4m3 && !row_scale) ||
        N < 0 || d <= 0 || R < 0 || kk <= 0)
        return 1;
    init_tables();
    corpus_t c = {corpus_bf16, corpus_e4m3, row_scale, N, d};
    int nt = resolve_threads(nthreads);
    int failed = 0;
#ifdef _OPENMP
#pragma omp parallel num_threads(nt)
#endif
    {
        cand_t *heap = (cand_t *)malloc(sizeof(cand_t) * (size_t)kk);
        double *q = (double *)malloc(sizeof(double) * (size_t)d);
        if (!heap || !q) {
            failed = 1;
        } else {
#ifdef _OPENMP
#pragma omp for schedule(dynamic, 1)
#endif
            for (int64_t r = 0; r < R; ++r)
                region_topk_one(&c, regions + r * (int64_t)d, kk, heap, q, out_ids + r * kk,
                                out_scores + r * kk);
        }
        free(heap);
        free(q);
    }
    (void)nt;
    return failed ? 2 : 0;
}

/*
 * Step 3: per-question union, dedup by id keeping the max score, then the
 * first K by (score desc, id asc), padded with (-1, -inf).
 * reg_ids/reg_scores: [R x ld] per-region lists; the first k of each row are
 * the region's list (entries with id -1 are ignored).
 */
int skip_oracle_merge(const int64_t *reg_ids, const double *reg_scores, int ld, int k,
                      const int32_t *offsets, int Q, int K, int64_t *out_ids,
                      double *out_scores)
{
    if (k <= 0 || ld < k || Q < 0 || K <= 0)
        return 1;
    for (int q = 0; q < Q; ++q) {
        int64_t r0 = offsets[q], r1 = offsets[q + 1];
        if (r1 < r0)
            return 1;
        size_t cap = (size_t)(r1 - r0) * (size_t)k;
        cand_t *u = (cand_t *)malloc(sizeof(cand_t) * (cap ? cap : 1));
        if (!u)
            return 2;
        size_t n = 0;
        for (int64_t r = r0; r < r1; ++r)
            for (int t = 0; t < k; ++t) {
                int64_t id = reg_ids[r * ld + t];
                if (id < 0)
                    continue;
                u[n].id = id;
                u[n].s = reg_scores[r * ld + t];
                ++n;
            }
        qsort(u, n, sizeof(cand_t), cmp_id_then_score);
        size_t m = 0;
        for (size_t t = 0; t < n; ++t)
            if (t == 0 || u[t].id != u[t - 1].id)
                u[m++] = u[t];
        qsort(u, m, sizeof(cand_t), cmp_rank);
        for (int t = 0; t < K; ++t) {
            out_ids[(int64_t)q * K + t] = (size_t)t < m ? u[t].id : -1;
            out_scores[(int64_t)q * K + t] = (size_t)t < m ? u[t].s : -INFINITY;
        }
        free(u);
    }
    return 0;
}

/* The whole path: steps 1-3.  reg_* [R x k] and out_* [Q x K]. */
int skip_oracle_retrieve(const uint16_t *corpus_bf16, const uint8_t *corpus_e4m3,
                         const float *row_scale, int64_t N, int d, const uint16_t *regions,
                         const int32_t *offsets, int Q, int64_t R, int k, int K,
                         int64_t *reg_ids, double *reg_scores, int64_t *out_ids,
                         double *out_scores, int nthreads)
{
    if (Q < 0 || offsets[0] != 0 || offsets[Q] != R)
        return 1;
    int rc = skip_oracle_region_topk(corpus_bf16, corpus_e4m3, row_scale, N, d, regions, R, k,
                                     reg_ids, reg_scores, nthreads);
    if (rc)
        return rc;
    return skip_oracle_merge(reg_ids, reg_scores, k, k, offsets, Q, K, out_ids, out_scores);
}

/*
 * Brute force for tiny inputs: every score s(r, i) into an [R x N] matrix
 * (fp64), used by the pins to rank by a full sort instead of the heap.
 */
int skip_oracle_score_matrix(const uint16_t *corpus_bf16, const uint8_t *corpus_e4m3,
                             const float *row_scale, int64_t N, int d,
                             const uint16_t *regions, int64_t R, double *out)
{
    if ((corpus_bf16 == NULL) == (corpus_e4m3 == NULL) || (corpus_e4m3 && !row_scale))
        return 1;
    init_tables();
    corpus_t c = {corpus_bf16, corpus_e4m3, row_scale, N, d};
    double *q = (double *)malloc(sizeof(double) * (size_t)(d > 0 ? d : 1));
    if (!q)
        return 2;
    for (int64_t r = 0; r < R; ++r) {
        for (int j = 0; j < d; ++j)
            q[j] = bf16_value(regions[r * (int64_t)d + j]);
        for (int64_t i = 0; i < N; ++i)
            out[r * N + i] = score(&c, q, i);
    }
    free(q);
    return 0;
}

/* s(r, ids[t]) for a list of (region, id) pairs: the oracle's value of
 * chosen scores, used to check scores reported for ids outside a list. */
int skip_oracle_scores_at(const uint16_t *corpus_bf16, const uint8_t *corpus_e4m3,
                          const float *row_scale, int64_t N, int d, const uint16_t *regions,
                          const int64_t *region_idx, const int64_t *ids, int64_t n, double *out)
{
    if ((corpus_bf16 == NULL) == (corpus_e4m3 == NULL) || (corpus_e4m3 && !row_scale))
        return 1;
    init_tables();
    corpus_t c = {corpus_bf16, corpus_e4m3, row_scale, N, d};
    double *q = (double *)malloc(sizeof(double) * (size_t)(d > 0 ? d : 1));
    if (!q)
        return 2;
    for (int64_t t = 0; t < n; ++t) {
        if (ids[t] < 0 || ids[t] >= N) {
            out[t] = NAN;
            continue;
        }
        for (int j = 0; j < d; ++j)
            q[j] = bf16_value(regions[region_idx[t] * (int64_t)d + j]);
        out[t] = score(&c, q, ids[t]);
    }
    free(q);
    return 0;
}

int skip_oracle_threads(void) { return resolve_threads(0); }
