/*
 * CPU oracle for QVS, question-guided visual token pruning.
 *
 * TEST INFRASTRUCTURE ONLY.  The plain, slow statement of what the GPU QVS
 * kernel computes; only the tests, the smoke check and the benchmark's CPU
 * leg load it.  It shares no code, header, table or helper with the CUDA
 * library.
 *
 * What it computes (App. B.1 Def. B.1, Eq. qvs_score; Alg. 1, the "QVS:
 * prune" step): for each image b with visual tokens v_1..v_L and the
 * question's projected representation f_q (d_k values),
 *
 *     f_v(v)   = W_v v + b_v                     (W_v [d_k x d], b_v [d_k])
 *     logit_i  = <f_q, f_v(v_i)> / sqrt(d_k) + <w_b, v_i>
 *     s_i      = sigmoid(logit_i)
 *     kept     = the n = ceil(rho_v L - 1e-3) tokens with the largest s_i,
 *                ordered by (s desc, token index asc)
 *
 * Readings where the paper is silent (listed in the design notes): f_v is a
 * linear layer with bias; f_q(Q) is given per image as d_k values; ranking by
 * s is ranking by the logit (the sigmoid is increasing), ties to the lower
 * token index; ceil(rho L) is taken with a 1e-3 slack as for the SKV count.
 * Tokens, W_v and f_q are bf16; b_v and w_b fp32; everything here is fp64.
 *
 * Pins (tests/test_qvs_oracle.py): a hand-worked example, the closed form
 * with W_v = 0 (logit = <w_b, v>) against a brute-force sort, and the count.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

static double bfq(uint16_t h)
{
    uint32_t u = (uint32_t)h << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

typedef struct {
    double logit;
    int idx;
} tok_t;

static int cmp_tok(const void *pa, const void *pb)
{
    const tok_t *a = (const tok_t *)pa, *b = (const tok_t *)pb;
    if (a->logit != b->logit)
        return a->logit > b->logit ? -1 : 1;
    return a->idx < b->idx ? -1 : (a->idx > b->idx);
}

int skip_oracle_qvs_count(int L, double rho)
{
    double v = ceil(rho * (double)L - 1e-3);
    if (v < 0.0)
        v = 0.0;
    if (v > (double)L)
        v = (double)L;
    return (int)v;
}

/*
 * tokens bf16 [B x L x d]; fq bf16 [B x dk]; wv bf16 [dk x d]; bv fp32 [dk]
 * (nullable: zero); wb fp32 [d].
 * Outputs: logits [B x L]; idx int32 [B x n]; score [B x n] (sigmoid).
 */
int skip_oracle_qvs(const uint16_t *tokens, int B, int L, int d, const uint16_t *fq, const uint16_t *wv,
                    const float *bv, const float *wb, int dk, double rho, double *logits, int32_t *out_idx,
                    double *out_score)
{
    if (B < 0 || L < 1 || d < 1 || dk < 1)
        return -1;
    const int n = skip_oracle_qvs_count(L, rho);
    const double inv = 1.0 / sqrt((double)dk);
    int rc = 0;
#pragma omp parallel for schedule(dynamic, 1)
    for (int b = 0; b < B; ++b) {
        tok_t *t = (tok_t *)malloc(sizeof(tok_t) * L);
        if (!t) {
            rc = -1;
            continue;
        }
        const uint16_t *f = fq + (int64_t)b * dk;
        double c = 0.0; /* <f_q, b_v> / sqrt(dk) */
        for (int k = 0; k < dk; ++k)
            c += bfq(f[k]) * (bv ? (double)bv[k] : 0.0);
        c *= inv;
        for (int i = 0; i < L; ++i) {
            const uint16_t *v = tokens + ((int64_t)b * L + i) * d;
            double s = 0.0;
            for (int k = 0; k < dk; ++k) {
                double proj = 0.0; /* (W_v v)_k */
                for (int j = 0; j < d; ++j)
                    proj += bfq(wv[(int64_t)k * d + j]) * bfq(v[j]);
                s += bfq(f[k]) * proj;
            }
            double bias = 0.0;
            for (int j = 0; j < d; ++j)
                bias += (double)wb[j] * bfq(v[j]);
            t[i].logit = s * inv + c + bias;
            t[i].idx = i;
            logits[(int64_t)b * L + i] = t[i].logit;
        }
        qsort(t, L, sizeof(tok_t), cmp_tok);
        for (int r = 0; r < n; ++r) {
            out_idx[(int64_t)b * n + r] = t[r].idx;
            out_score[(int64_t)b * n + r] = 1.0 / (1.0 + exp(-t[r].logit));
        }
        free(t);
    }
    return rc;
}
