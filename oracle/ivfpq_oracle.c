/*
 * CPU oracle for the IVF-PQ approximate variant of the per-region search.
 *
 * TEST INFRASTRUCTURE ONLY.  The plain, slow statement of what the GPU index
 * build and search compute; only the tests, the smoke check and the
 * benchmark's CPU leg load it.  It shares no code, header, table or helper
 * with the CUDA library.
 *
 * The paper retrieves from a FAISS IVF-PQ index (§4.1 "Implementation":
 * 768-d vectors, 1,024 IVF centroids; App. I.4: IVF4096-PQ64) and names no
 * further parameter.  The index and its search follow the published method
 * (Jegou, Douze, Schmid, "Product quantization for nearest neighbor search",
 * IEEE TPAMI 33(1), 2011: the inverted file with asymmetric distance
 * computation on residuals), here with inner-product scores:
 *
 *   coarse:  list(i) = argmax_l <x_i, c_l>                  (ties: lower l)
 *   residual r_i = x_i - c_list(i), cut into M sub-vectors of d/M values
 *   code:    code_{i,m} = argmin_j || r_{i,m} - p_{m,j} ||^2 (ties: lower j)
 *   lists:   list l holds the ids i with list(i) = l
 *   search:  probes(q) = the nprobe lists with the largest <q, c_l>
 *            (ties: lower l); for every id i in a probed list
 *            s^(q, i) = <q, c_list(i)> + sum_m <q_m, p_{m, code_{i,m}}>
 *            L_q = the first k of those ids by (s^ desc, id asc), padded
 *            with (-1, -inf) when the probed lists hold fewer than k ids.
 *
 * x, c and q are bf16, the codebooks p fp32; everything here is fp64.
 *
 * Pins (tests/test_ivfpq_oracle.py): a hand-worked example, brute-force
 * argmax / argmin, the closed form when every residual sub-vector is a
 * codeword and all lists are probed (then s^ is the exact inner product and
 * the search equals exact MIPS), and the probe count's monotonicity.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

static double bf(uint16_t h)
{
    uint32_t u = (uint32_t)h << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

static double dot_bf(const uint16_t *a, const uint16_t *b, int d)
{
    double s = 0.0;
    for (int t = 0; t < d; ++t)
        s += bf(a[t]) * bf(b[t]);
    return s;
}

/* list[i] = argmax_l <x_i, c_l>, ties to the lower l. */
int skip_oracle_ivf_assign(const uint16_t *corpus, int64_t N, int d, const uint16_t *centroids, int C,
                           int32_t *list)
{
    if (N < 0 || d < 1 || C < 1)
        return -1;
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < N; ++i) {
        const uint16_t *x = corpus + i * (int64_t)d;
        int best = 0;
        double bs = dot_bf(x, centroids, d);
        for (int l = 1; l < C; ++l) {
            double s = dot_bf(x, centroids + (int64_t)l * d, d);
            if (s > bs) {
                bs = s;
                best = l;
            }
        }
        list[i] = best;
    }
    return 0;
}

/* codes[i][m] = argmin_j ||(x_i - c_list[i])_m - p_{m,j}||^2, ties to the lower j.
 * codebook fp32 [M][ksub][d/M]. */
int skip_oracle_pq_encode(const uint16_t *corpus, int64_t N, int d, const uint16_t *centroids,
                          const int32_t *list, const float *codebook, int M, int ksub, uint8_t *codes)
{
    if (N < 0 || d < 1 || M < 1 || d % M != 0 || ksub < 1 || ksub > 256)
        return -1;
    const int ds = d / M;
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < N; ++i) {
        const uint16_t *x = corpus + i * (int64_t)d;
        const uint16_t *c = centroids + (int64_t)list[i] * d;
        for (int m = 0; m < M; ++m) {
            int best = 0;
            double bd = INFINITY;
            for (int j = 0; j < ksub; ++j) {
                const float *p = codebook + ((int64_t)m * ksub + j) * ds;
                double dist = 0.0;
                for (int t = 0; t < ds; ++t) {
                    double r = bf(x[m * ds + t]) - bf(c[m * ds + t]);
                    double e = r - (double)p[t];
                    dist += e * e;
                }
                if (dist < bd) {
                    bd = dist;
                    best = j;
                }
            }
            codes[i * (int64_t)M + m] = (uint8_t)best;
        }
    }
    return 0;
}

typedef struct {
    double s;
    int64_t id;
} cand_t;

static int before(cand_t a, cand_t b) { return a.s > b.s || (a.s == b.s && a.id < b.id); }

static int cmp_cand(const void *pa, const void *pb)
{
    cand_t a = *(const cand_t *)pa, b = *(const cand_t *)pb;
    return before(a, b) ? -1 : before(b, a) ? 1 : 0;
}

/* The lookup table of one query: T[m][j] = <q_m, p_{m,j}>. */
static void adc_table(const uint16_t *q, int d, const float *codebook, int M, int ksub, double *T)
{
    const int ds = d / M;
    for (int m = 0; m < M; ++m)
        for (int j = 0; j < ksub; ++j) {
            const float *p = codebook + ((int64_t)m * ksub + j) * ds;
            double s = 0.0;
            for (int t = 0; t < ds; ++t)
                s += bf(q[m * ds + t]) * (double)p[t];
            T[m * ksub + j] = s;
        }
}

/*
 * Search.  list_offsets int64 [C+1] and list_ids int64 [N] describe the
 * lists; codes_by_id uint8 [N x M] holds each id's code (in id order).
 * Outputs: ids int64 [R x k], scores fp64 [R x k], probes int32 [R x nprobe].
 */
int skip_oracle_ivfpq_search(const uint16_t *centroids, int C, int d, const int64_t *list_offsets,
                             const int64_t *list_ids, const uint8_t *codes_by_id, const float *codebook,
                             int M, int ksub, const uint16_t *regions, int R, int nprobe, int k,
                             int64_t *out_ids, double *out_scores, int32_t *out_probes)
{
    if (C < 1 || d < 1 || M < 1 || d % M != 0 || nprobe < 1 || nprobe > C || k < 1 || ksub < 1 ||
        ksub > 256)
        return -1;
    int rc = 0;
#pragma omp parallel
    {
        double *T = (double *)malloc(sizeof(double) * M * ksub);
        cand_t *cs = (cand_t *)malloc(sizeof(cand_t) * C);
        int64_t cap = 0;
        cand_t *pool = NULL;
#pragma omp for schedule(dynamic, 1)
        for (int r = 0; r < R; ++r) {
            const uint16_t *q = regions + (int64_t)r * d;
            if (!T || !cs) {
                rc = -1;
                continue;
            }
            for (int l = 0; l < C; ++l) {
                cs[l].s = dot_bf(q, centroids + (int64_t)l * d, d);
                cs[l].id = l;
            }
            qsort(cs, C, sizeof(cand_t), cmp_cand);
            int64_t total = 0;
            for (int p = 0; p < nprobe; ++p)
                total += list_offsets[cs[p].id + 1] - list_offsets[cs[p].id];
            if (total > cap) {
                free(pool);
                cap = total;
                pool = (cand_t *)malloc(sizeof(cand_t) * (cap > 0 ? cap : 1));
                if (!pool) {
                    rc = -1;
                    cap = 0;
                    continue;
                }
            }
            adc_table(q, d, codebook, M, ksub, T);
            int64_t n = 0;
            for (int p = 0; p < nprobe; ++p) {
                const int l = (int)cs[p].id;
                out_probes[(int64_t)r * nprobe + p] = l;
                for (int64_t e = list_offsets[l]; e < list_offsets[l + 1]; ++e) {
                    const int64_t id = list_ids[e];
                    const uint8_t *code = codes_by_id + id * (int64_t)M;
                    double s = cs[p].s;
                    for (int m = 0; m < M; ++m)
                        s += T[m * ksub + code[m]];
                    pool[n].s = s;
                    pool[n].id = id;
                    ++n;
                }
            }
            qsort(pool, n, sizeof(cand_t), cmp_cand);
            for (int t = 0; t < k; ++t) {
                out_ids[(int64_t)r * k + t] = t < n ? pool[t].id : -1;
                out_scores[(int64_t)r * k + t] = t < n ? pool[t].s : -INFINITY;
            }
        }
        free(T);
        free(cs);
        free(pool);
    }
    return rc;
}

/* s^(q_r, i) for chosen (region, id) pairs: <q, c_list(i)> + sum_m T[m][code].
 * list_of_id int32 [N]; NaN for ids outside [0, N). */
int skip_oracle_ivfpq_scores_at(const uint16_t *centroids, int d, const int32_t *list_of_id,
                                const uint8_t *codes_by_id, int64_t N, const float *codebook, int M, int ksub,
                                const uint16_t *regions, const int64_t *region_idx, const int64_t *ids,
                                int64_t n, double *out)
{
    if (d < 1 || M < 1 || d % M != 0)
        return -1;
    const int ds = d / M;
    for (int64_t t = 0; t < n; ++t) {
        const int64_t i = ids[t];
        if (i < 0 || i >= N) {
            out[t] = NAN;
            continue;
        }
        const uint16_t *q = regions + region_idx[t] * (int64_t)d;
        double s = dot_bf(q, centroids + (int64_t)list_of_id[i] * d, d);
        for (int m = 0; m < M; ++m) {
            const float *p = codebook + ((int64_t)m * ksub + codes_by_id[i * (int64_t)M + m]) * ds;
            for (int u = 0; u < ds; ++u)
                s += bf(q[m * ds + u]) * (double)p[u];
        }
        out[t] = s;
    }
    return 0;
}
