/*
 * CPU oracle for the SKV passage gate (Speculative Knowledge Verification).
 *
 * TEST INFRASTRUCTURE ONLY.  The plain, slow statement of what the GPU gate
 * computes; only the tests, the smoke check and the benchmark's CPU leg load
 * it.  It shares no code, header, table or helper with the CUDA library.
 *
 * What it computes (App. B.4 Def. B.4, Eq. skv_score; Alg. 1, the "SKV:
 * verify" step and the TopK that follows it):
 *
 *   for each question q with candidate passages k_j (the merged, deduplicated
 *   retrieval list; id -1 marks an empty slot):
 *     f_j  = [ qbar ; vbar ; e_j ; e_j (.) qbar ; |e_j - qbar| ]   (5d inputs)
 *     h_j  = relu(W1 f_j + b1)                       (layer 1 of h_psi, H units)
 *     nu_j = sigmoid(w2 . h_j + b2)                  (layer 2, one logit)
 *     gated   = { j : nu_j >= tau }                  (Def. B.4, verified set)
 *     n       = ceil(rho * K' - 1e-3), K' = number of non-empty slots
 *     output  = the first min(n, |gated|) of gated ordered by
 *               (nu desc, id asc); pad with (id -1, nu -inf)
 *
 *   e_j is the passage embedding: the corpus row of id k_j (bf16).  qbar is
 *   the question embedding and vbar the mean-pooled visual tokens, both given
 *   as bf16 vectors of the corpus dimension d.
 *
 * Readings where the paper is silent (each one listed in the design notes):
 *  - the MLP input is held in bf16: the two interaction features e (.) qbar
 *    and |e - qbar| are rounded to the nearest bf16 (ties to even) before the
 *    first layer; everything after that is exact here (fp64);
 *  - the hidden activation is ReLU; W1 is [H x 5d] with its columns in the
 *    order of the concatenation above;
 *  - ceil(rho * |K|) is taken with a 1e-3 slack so that two-decimal ratios
 *    such as 0.6 * 5 give 3, and |K| counts the non-empty slots;
 *  - ties in nu go to the lower id.
 *
 * Alongside each nu the oracle reports how far an fp32 evaluation (any
 * summation order, bf16 x bf16 products exact, fp32 sums) may land from the
 * exact value, and the tests use it as the tolerance.  It is the
 * probabilistic rounding-error bound of Higham and Mary (SIAM J. Sci.
 * Comput. 41(5), 2019): an n-term sum is off by at most
 * lambda * sqrt(n) * u * sum|terms|, with u = 2^-24, here with lambda = 6
 * (the bound fails with probability below 2 exp(-lambda^2 / 2) ~ 3e-8 per
 * sum under that model); it is at least the worst-case n * u * sum|terms|
 * for n <= 36.  It is carried through ReLU (1-Lipschitz), the second layer
 * and the sigmoid (1/4-Lipschitz).
 *
 * Pins (tests/test_skv_oracle.py): bf16 rounding against torch, a hand-worked
 * example whose logits are the integers -2..2 (tests/golden/
 * skv_hand_example.txt; it has a passage exactly at the gate, nu = 1/2, and
 * a tie broken by id), one-hot weights that read out each feature block, the
 * count rule, and brute-force selection.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

static double bf16_to_double(uint16_t h)
{
    uint32_t u = (uint32_t)h << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

/* Round-to-nearest-integer, ties to even, of a non-negative finite y. */
static double rne_int(double y)
{
    double t = floor(y);
    double frac = y - t;
    if (frac > 0.5)
        return t + 1.0;
    if (frac < 0.5)
        return t;
    return fmod(t, 2.0) == 0.0 ? t : t + 1.0;
}

/* x rounded to bf16 (8 significant bits, exponent range of binary32, ties to
 * even), returned as its bit pattern.  x must be exact in double. */
static uint16_t bf16_round(double x)
{
    if (isnan(x))
        return 0x7FC0;
    const int neg = signbit(x) ? 1 : 0;
    double a = fabs(x);
    uint16_t sign = neg ? 0x8000 : 0;
    if (a == 0.0)
        return sign;
    if (isinf(a))
        return sign | 0x7F80;
    int e;
    frexp(a, &e); /* a = m * 2^e, m in [0.5, 1) */
    /* quantum: 2^(e - 8) for normals, 2^-133 below 2^-126 */
    int qe = e - 8;
    if (qe < -133)
        qe = -133;
    double r = ldexp(rne_int(ldexp(a, -qe)), qe);
    /* largest finite bf16 is (2 - 2^-7) * 2^127; anything rounding past it is inf */
    if (r >= ldexp(1.0, 128))
        return sign | 0x7F80;
    float f = (float)r; /* exact */
    uint32_t u;
    memcpy(&u, &f, sizeof u);
    return (uint16_t)(sign | ((u >> 16) & 0x7FFF));
}

uint16_t skip_oracle_bf16_round(double x) { return bf16_round(x); }

typedef struct {
    double nu;
    int64_t id;
} gated_t;

static int cmp_gated(const void *pa, const void *pb)
{
    const gated_t *a = (const gated_t *)pa, *b = (const gated_t *)pb;
    if (a->nu != b->nu)
        return a->nu > b->nu ? -1 : 1;
    if (a->id != b->id)
        return a->id < b->id ? -1 : 1;
    return 0;
}

/* Relative error allowance of an n-term fp32 sum (see the header). */
static double sum_err(double n, double u) { return 6.0 * sqrt(n) * u; }

int skip_oracle_skv_count(int n_nonempty, double rho)
{
    double v = ceil(rho * (double)n_nonempty - 1e-3);
    if (v < 0.0)
        v = 0.0;
    if (v > (double)n_nonempty)
        v = (double)n_nonempty;
    return (int)v;
}

/*
 * corpus   bf16 bits [N x d]; ids int64 [Q x K] (-1 = empty slot);
 * qbar, vbar bf16 bits [Q x d]; w1 bf16 bits [H x 5d]; b1, w2 fp32 [H].
 * Outputs: nu_all [Q x K] (nu of every slot, -inf for empty ones),
 * bound [Q x K] (fp32-evaluation bound on |nu - exact|, 0 for empty ones),
 * out_ids [Q x K], out_nu [Q x K], out_count [Q].
 * Returns 0, or -1 for a bad argument (an id outside [0, N), bad sizes).
 */
int skip_oracle_skv(const uint16_t *corpus, int64_t N, int d, const int64_t *ids, int Q, int K,
                    const uint16_t *qbar, const uint16_t *vbar, const uint16_t *w1, const float *b1,
                    const float *w2, float b2, int H, double tau, double rho, double *nu_all,
                    double *bound, int64_t *out_ids, double *out_nu, int *out_count)
{
    if (N < 1 || d < 1 || Q < 0 || K < 1 || H < 1)
        return -1;
    const int D5 = 5 * d;
    const double u = ldexp(1.0, -24); /* fp32 unit roundoff */
    double *f = (double *)malloc(sizeof(double) * D5);
    double *c = (double *)malloc(sizeof(double) * H);
    double *cabs = (double *)malloc(sizeof(double) * H);
    gated_t *g = (gated_t *)malloc(sizeof(gated_t) * K);
    if (!f || !c || !cabs || !g) {
        free(f), free(c), free(cabs), free(g);
        return -1;
    }
    int rc = 0;
    for (int q = 0; q < Q && rc == 0; ++q) {
        const uint16_t *qb = qbar + (int64_t)q * d, *vb = vbar + (int64_t)q * d;
        /* per-question part of layer 1: b1 + W1[:, q-block] qbar + W1[:, v-block] vbar */
        for (int i = 0; i < H; ++i) {
            const uint16_t *w = w1 + (int64_t)i * D5;
            double s = (double)b1[i], sa = fabs((double)b1[i]);
            for (int t = 0; t < d; ++t) {
                double p = bf16_to_double(w[t]) * bf16_to_double(qb[t]);
                s += p, sa += fabs(p);
            }
            for (int t = 0; t < d; ++t) {
                double p = bf16_to_double(w[d + t]) * bf16_to_double(vb[t]);
                s += p, sa += fabs(p);
            }
            c[i] = s;
            cabs[i] = sa;
        }
        int nonempty = 0, ng = 0;
        for (int j = 0; j < K; ++j) {
            const int64_t id = ids[(int64_t)q * K + j];
            double *nu_out = nu_all + (int64_t)q * K + j, *b_out = bound + (int64_t)q * K + j;
            if (id < 0) {
                *nu_out = -INFINITY;
                *b_out = 0.0;
                continue;
            }
            if (id >= N) {
                rc = -1;
                break;
            }
            ++nonempty;
            const uint16_t *e = corpus + id * (int64_t)d;
            for (int t = 0; t < d; ++t) {
                double et = bf16_to_double(e[t]), qt = bf16_to_double(qb[t]);
                f[2 * d + t] = et;
                f[3 * d + t] = bf16_to_double(bf16_round(et * qt));
                f[4 * d + t] = bf16_to_double(bf16_round(fabs(et - qt)));
            }
            double logit = (double)b2, lsum = fabs((double)b2), lerr = 0.0;
            for (int i = 0; i < H; ++i) {
                const uint16_t *w = w1 + (int64_t)i * D5;
                double s = 0.0, sa = 0.0;
                for (int t = 2 * d; t < D5; ++t) {
                    double p = bf16_to_double(w[t]) * f[t];
                    s += p, sa += fabs(p);
                }
                double h = c[i] + s;
                /* fp32: c (2d + 1 terms), the passage part (3d terms), their sum */
                double herr = sum_err(2.0 * d + 1.0, u) * cabs[i] + sum_err(3.0 * d, u) * sa +
                              u * (fabs(c[i]) + fabs(s));
                double a = h > 0.0 ? h : 0.0;
                double t2 = (double)w2[i] * a;
                logit += t2;
                lsum += fabs(t2);
                lerr += fabs((double)w2[i]) * herr;
            }
            lerr += sum_err((double)H + 1.0, u) * (lsum + lerr);
            const double nu = 1.0 / (1.0 + exp(-logit));
            *nu_out = nu;
            /* sigmoid is 1/4-Lipschitz; plus the rounding of exp, add, divide */
            *b_out = lerr / 4.0 + 16.0 * u;
            if (nu >= tau) {
                g[ng].nu = nu;
                g[ng].id = id;
                ++ng;
            }
        }
        if (rc)
            break;
        qsort(g, ng, sizeof(gated_t), cmp_gated);
        int n = skip_oracle_skv_count(nonempty, rho);
        if (n > ng)
            n = ng;
        for (int j = 0; j < K; ++j) {
            out_ids[(int64_t)q * K + j] = j < n ? g[j].id : -1;
            out_nu[(int64_t)q * K + j] = j < n ? g[j].nu : -INFINITY;
        }
        out_count[q] = n;
    }
    free(f), free(c), free(cabs), free(g);
    return rc;
}
