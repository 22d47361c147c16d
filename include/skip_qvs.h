/*
 * skip_qvs.h -- C ABI of QVS, question-guided visual token pruning.
 *
 * The operation (paper App. B.1 Def. B.1, Eq. qvs_score; Alg. 1, the
 * "QVS: prune" step): for each image b with visual tokens v_1..v_L (d values
 * each) and the question's projected representation f_q = f_q(Q) (d_k
 * values), every token is scored
 *
 *   s_i = sigmoid( <f_q, W_v v_i + b_v> / sqrt(d_k) + <w_b, v_i> )
 *
 * (f_v(v) = W_v v + b_v, a linear layer; w_b the content bias) and the
 * n = ceil(rho_v L - 1e-3) tokens with the largest s are kept, ordered by
 * (s desc, token index asc).  The paper uses L = 576 and rho_v = 0.40
 * (App. I.4) or 0.11 (main text).
 *
 * Tokens, f_q and W_v are bf16; b_v, w_b, the sums and s are fp32.  Ranking
 * by s is ranking by its argument (the sigmoid is increasing), so ties in s
 * that fp32 rounding creates near 1 do not reorder tokens.
 *
 * Device pointers; calls are asynchronous and stream ordered; no CPU
 * fallback.  W_v^T f_q for all images is one bf16 GEMM with fp32 results on
 * the library's own tensor-core kernel (the handle keeps W_v^T so that both
 * operands are K-major); every step runs in the library's kernels.  Limits:
 * d a multiple of 8 and at most 8192, 1 <= d_k <= 4096, 1 <= L <= 4096.
 */
#ifndef SKIP_QVS_H
#define SKIP_QVS_H

#include "skip_retrieve.h"

#ifdef __cplusplus
extern "C" {
#endif

typedef struct skip_qvs *skip_qvs_t; /* opaque: a copy of the QVS head and its workspace */

/*
 * skip_qvs_create -- copies the head's weights (device pointers): wv bf16
 * [d_k x d] row-major (kept transposed), bv fp32 [d_k] (NULL: zero), wb fp32
 * [d]; sizes the
 * workspace for up to max_images images of up to max_tokens tokens.
 * Returns after the copies.  Errors: SKIP_EINVAL, SKIP_EUNSUPPORTED (sizes
 * beyond the limits, or no sm_103 device), SKIP_ENOMEM, SKIP_ECUDA.
 */
SKIP_API skip_status_t skip_qvs_create(const uint16_t *wv, const float *bv, const float *wb, int32_t d,
                                       int32_t dk, int32_t max_images, int32_t max_tokens, void *stream,
                                       skip_qvs_t *out);

SKIP_API skip_status_t skip_qvs_free(skip_qvs_t qvs);

/* Tokens kept per image: ceil(rho_v * L - 1e-3), clamped to [0, L]. */
SKIP_API int32_t skip_qvs_count(int32_t L, float rho_v);

/*
 * skip_qvs_prune -- scores and prunes a batch.
 *  tokens     device bf16 [B x L x d]; fq device bf16 [B x d_k].
 *  out_idx    device int32 [B x n]: kept token indices, best first.
 *  out_score  device fp32 [B x n]: their s.
 *  out_tokens optional (NULL) device bf16 [B x n x d]: the kept tokens.
 *  logits     optional (NULL) device fp32 [B x L]: every token's argument of
 *             the sigmoid.
 * tokens must start on a 16-byte boundary.
 * Asynchronous on `stream`.  Errors: SKIP_EINVAL (null or misaligned
 * pointers, B or L beyond the handle's maxima, rho_v outside [0, 1]),
 * SKIP_ECUDA.
 */
SKIP_API skip_status_t skip_qvs_prune(skip_qvs_t qvs, const uint16_t *tokens, int32_t B, int32_t L,
                                      const uint16_t *fq, float rho_v, int32_t *out_idx, float *out_score,
                                      uint16_t *out_tokens, float *logits, void *stream);

/* Synchronises `stream`, then reports and clears the handle's error word:
 * SKIP_ETIMEOUT if a bounded wait of the projection GEMM gave up since the
 * last check, SKIP_ECUDA if the stream reported an error, else SKIP_OK. */
SKIP_API skip_status_t skip_qvs_sync_status(skip_qvs_t qvs, void *stream);

#ifdef __cplusplus
}
#endif

#endif /* SKIP_QVS_H */
