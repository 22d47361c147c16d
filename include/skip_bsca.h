/*
 * skip_bsca.h -- C ABI of BSCA, bipartite sparse cross-attention.
 *
 * The operation (paper App. B.3 Def. B.3, Eq. bsca_edges and bsca_attn;
 * §3.3 "BSCA"; Alg. 1 "BSCA: graph" and "BSCA: fuse"): per question, the
 * retained visual tokens v_i and the verified chunks k_j form a bipartite
 * graph whose edges are the pairs with cos(h_v(v_i), h_k(k_j)) >= tau_e,
 * tau_e set so that the mean degree of a visual token is dbar (the paper
 * uses 4, App. I.4); every visual token then attends over its neighbours
 * only:
 *
 *   tau_e  = the m-th largest cosine of the question, m = ceil(dbar P - 1e-3)
 *            (every pair if m >= P R, none if m < 1; ties at tau_e kept)
 *   out_i  = sum_{j in N(i)} exp(e_ij) W_V k_j / sum_{j in N(i)} exp(e_ij),
 *   e_ij   = <W_Q v_i, W_K k_j> / sqrt(d_h);  out_i = 0 if N(i) is empty.
 *
 * The inputs are the projections, computed upstream by the model's linear
 * layers: hv = h_v(v) [Nv x d_p], qh = W_Q v [Nv x d_h], hk = h_k(k)
 * [Nc x d_p], kh = W_K k [Nc x d_h], vh = W_V k [Nc x d_o], all bf16.
 * Questions own consecutive rows: question q's tokens are
 * [vis_offsets[q], vis_offsets[q+1]) and its chunks [chunk_offsets[q],
 * chunk_offsets[q+1]) (device int32 [Q + 1] each), with vis_offsets[0] = 0
 * and vis_offsets[Q] = total_tokens (rows outside every question's range
 * are not written).  Sums and outputs fp32.
 *
 * Device pointers; asynchronous and stream ordered; errors found by kernels
 * latched in the handle (skip_bsca_sync_status); no CPU fallback.  Limits:
 * at most 64 chunks and 32,768 (token, chunk) pairs per question (a
 * question beyond either latches SKIP_EINVAL and gets zero outputs), d_p and
 * d_h at most 256, d_o even and at most 2048.
 */
#ifndef SKIP_BSCA_H
#define SKIP_BSCA_H

#include "skip_retrieve.h"

#ifdef __cplusplus
extern "C" {
#endif

typedef struct skip_bsca *skip_bsca_t; /* opaque: workspace and error word */

/* Sizes the workspace for up to max_questions questions and max_tokens
 * visual tokens in all.  Errors: SKIP_EINVAL, SKIP_EUNSUPPORTED (widths
 * beyond the limits, or no sm_103 device), SKIP_ENOMEM. */
SKIP_API skip_status_t skip_bsca_create(int32_t d_p, int32_t d_h, int32_t d_o, int32_t max_questions,
                                        int32_t max_tokens, skip_bsca_t *out);

SKIP_API skip_status_t skip_bsca_free(skip_bsca_t bsca);

/*
 * skip_bsca_run -- graph and attention for Q questions.
 *  out     device fp32 [total_tokens x d_o].
 *  degree  optional (NULL) device int32 [total_tokens]: |N(i)|.
 *  edges   optional (NULL) device uint64 [total_tokens]: bit j set when the
 *          question's chunk j (counted from chunk_offsets[q]) is in N(i).
 *  tau_e   optional (NULL) device fp32 [Q]: each question's threshold
 *          (+inf: no edge, -inf: every pair).
 * Asynchronous on `stream`.  Errors: SKIP_EINVAL (null pointers, sizes
 * beyond the handle's maxima, dbar < 0), SKIP_ECUDA.
 */
SKIP_API skip_status_t skip_bsca_run(skip_bsca_t bsca, int32_t Q, const int32_t *vis_offsets,
                                     const int32_t *chunk_offsets, int32_t total_tokens, const uint16_t *hv,
                                     const uint16_t *qh, const uint16_t *hk, const uint16_t *kh, const uint16_t *vh,
                                     float dbar, float *out, int32_t *degree, uint64_t *edges, float *tau_e,
                                     void *stream);

/* Synchronises `stream`, then reports and clears the handle's error word
 * (SKIP_EINVAL for a question with too many chunks). */
SKIP_API skip_status_t skip_bsca_sync_status(skip_bsca_t bsca, void *stream);

#ifdef __cplusplus
}
#endif

#endif /* SKIP_BSCA_H */
