/*
 * CPU oracle for BSCA, bipartite sparse cross-attention.
 *
 * TEST INFRASTRUCTURE ONLY.  The plain, slow statement of what the GPU BSCA
 * kernels compute; only the tests, the smoke check and the benchmark's CPU
 * leg load it.  It shares no code, header, table or helper with the CUDA
 * library.
 *
 * What it computes (App. B.3 Def. B.3, Eq. bsca_edges and bsca_attn; §3.3
 * "BSCA"; Alg. 1 "BSCA: graph" and "BSCA: fuse"), per question q with
 * retained visual tokens i in [vo[q], vo[q+1]) and verified chunks j in
 * [co[q], co[q+1]), given their projections (h_v(v_i), W_Q v_i) and
 * (h_k(k_j), W_K k_j, W_V k_j):
 *
 *   cos_ij  = <h_v(v_i), h_k(k_j)> / (||h_v(v_i)|| ||h_k(k_j)||)   (0 if a norm is 0)
 *   tau_e   = the m-th largest cos_ij of the question, m = ceil(dbar * P_q - 1e-3)
 *             (all pairs if m >= P_q R_q; no edge if m < 1)
 *   E       = { (i, j) : cos_ij >= tau_e }                    (Eq. bsca_edges)
 *   e_ij    = <W_Q v_i, W_K k_j> / sqrt(d_h)
 *   out_i   = sum_{j in N(i)} exp(e_ij) W_V k_j / sum_{j in N(i)} exp(e_ij)
 *             (Eq. bsca_attn); out_i = 0 when N(i) is empty.
 *
 * Readings where the paper is silent (listed in the design notes): tau_e
 * "set dynamically to keep the mean degree near dbar" is the m-th largest
 * cosine of the question with ties at tau_e all kept; an isolated token gets
 * a zero update.  Inputs are bf16, everything here is fp64.
 *
 * Pins (tests/test_bsca_oracle.py): a hand-worked example, dense attention
 * (dbar = R) against torch's scaled_dot_product_attention, a single edge
 * (out = W_V k_j), and the edge count.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

static double bfb(uint16_t h)
{
    uint32_t u = (uint32_t)h << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

static int cmp_desc(const void *pa, const void *pb)
{
    double a = *(const double *)pa, b = *(const double *)pb;
    return a > b ? -1 : a < b ? 1 : 0;
}

int skip_oracle_bsca_edges_count(int P, double dbar)
{
    double v = ceil(dbar * (double)P - 1e-3);
    return v < 0.0 ? 0 : (int)v;
}

/* Cosines of one question: cs [P x R]. */
static void cosines(const uint16_t *hv, const uint16_t *hk, int P, int R, int dp, double *cs)
{
    for (int i = 0; i < P; ++i) {
        double na = 0.0;
        for (int t = 0; t < dp; ++t)
            na += bfb(hv[(int64_t)i * dp + t]) * bfb(hv[(int64_t)i * dp + t]);
        for (int j = 0; j < R; ++j) {
            double nb = 0.0, s = 0.0;
            for (int t = 0; t < dp; ++t) {
                nb += bfb(hk[(int64_t)j * dp + t]) * bfb(hk[(int64_t)j * dp + t]);
                s += bfb(hv[(int64_t)i * dp + t]) * bfb(hk[(int64_t)j * dp + t]);
            }
            cs[(int64_t)i * R + j] = (na > 0.0 && nb > 0.0) ? s / (sqrt(na) * sqrt(nb)) : 0.0;
        }
    }
}

/* Attention of token i over the chunks with mask[j] != 0: out [d_o]. */
static void attend(const uint16_t *qh_i, const uint16_t *kh, const uint16_t *vh, int R, int dh, int dout,
                   const unsigned char *mask, double *out)
{
    double mx = -INFINITY;
    double *e = (double *)malloc(sizeof(double) * (R > 0 ? R : 1));
    for (int j = 0; j < R; ++j) {
        e[j] = -INFINITY;
        if (!mask[j])
            continue;
        double s = 0.0;
        for (int t = 0; t < dh; ++t)
            s += bfb(qh_i[t]) * bfb(kh[(int64_t)j * dh + t]);
        e[j] = s / sqrt((double)dh);
        if (e[j] > mx)
            mx = e[j];
    }
    for (int c = 0; c < dout; ++c)
        out[c] = 0.0;
    double den = 0.0;
    for (int j = 0; j < R; ++j) {
        if (!mask[j])
            continue;
        const double w = exp(e[j] - mx); /* the common factor exp(-mx) cancels */
        den += w;
        for (int c = 0; c < dout; ++c)
            out[c] += w * bfb(vh[(int64_t)j * dout + c]);
    }
    if (den > 0.0)
        for (int c = 0; c < dout; ++c)
            out[c] /= den;
    free(e);
}

/*
 * vo, co int32 [Q+1]; hv bf16 [Nv x dp], qh [Nv x dh]; hk [Nc x dp], kh [Nc x dh],
 * vh [Nc x dout].  Outputs: cos [Nv x Rmax] (row i: its question's chunks,
 * the rest 0), tau [Q], degree int32 [Nv], out [Nv x dout].
 * If edge_mask (uint8 [Nv x Rmax]) is given, it replaces the threshold rule
 * (for checking a given edge set); tau is then left as computed.
 */
int skip_oracle_bsca(const int32_t *vo, const int32_t *co, int Q, const uint16_t *hv, const uint16_t *qh,
                     const uint16_t *hk, const uint16_t *kh, const uint16_t *vh, int dp, int dh, int dout, int Rmax,
                     double dbar, const unsigned char *edge_mask, double *cos_out, double *tau, int32_t *degree,
                     double *out)
{
    if (Q < 0 || dp < 1 || dh < 1 || dout < 1 || Rmax < 1)
        return -1;
    for (int q = 0; q < Q; ++q) {
        const int i0 = vo[q], P = vo[q + 1] - vo[q], j0 = co[q], R = co[q + 1] - co[q];
        if (P < 0 || R < 0 || R > Rmax)
            return -1;
        double *cs = (double *)malloc(sizeof(double) * ((int64_t)P * R + 1));
        double *sorted = (double *)malloc(sizeof(double) * ((int64_t)P * R + 1));
        unsigned char *mask = (unsigned char *)malloc((size_t)Rmax + 1);
        if (!cs || !sorted || !mask) {
            free(cs), free(sorted), free(mask);
            return -1;
        }
        cosines(hv + (int64_t)i0 * dp, hk + (int64_t)j0 * dp, P, R, dp, cs);
        memcpy(sorted, cs, sizeof(double) * (int64_t)P * R);
        qsort(sorted, (size_t)P * R, sizeof(double), cmp_desc);
        const int m = skip_oracle_bsca_edges_count(P, dbar);
        double t;
        if (m < 1 || (int64_t)P * R == 0)
            t = INFINITY;
        else if ((int64_t)m >= (int64_t)P * R)
            t = -INFINITY;
        else
            t = sorted[m - 1];
        tau[q] = t;
        for (int i = 0; i < P; ++i) {
            const int gi = i0 + i;
            int deg = 0;
            for (int j = 0; j < Rmax; ++j) {
                const double c = j < R ? cs[(int64_t)i * R + j] : 0.0;
                cos_out[(int64_t)gi * Rmax + j] = c;
                unsigned char e = 0;
                if (j < R)
                    e = edge_mask ? edge_mask[(int64_t)gi * Rmax + j] != 0 : (c >= t);
                mask[j] = e;
                deg += e;
            }
            degree[gi] = deg;
            attend(qh + (int64_t)gi * dh, kh + (int64_t)j0 * dh, vh + (int64_t)j0 * dout, R, dh, dout, mask,
                   out + (int64_t)gi * dout);
        }
        free(cs), free(sorted), free(mask);
    }
    return 0;
}
