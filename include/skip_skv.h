/*
 * skip_skv.h -- C ABI of the SKV passage gate (Speculative Knowledge
 * Verification), run on the merged retrieval lists.
 *
 * The operation (paper App. B.4 Def. B.4, Eq. skv_score; Alg. 1, the
 * "SKV: verify" step and the TopK after it): every candidate passage k_j of
 * a question is scored by a two-layer MLP h_psi over the question embedding
 * qbar, the mean-pooled visual tokens vbar and the passage embedding e_j,
 * and the question keeps the best ceil(rho_r |K|) passages among those whose
 * score reaches tau_nu:
 *
 *   f_j   = [qbar; vbar; e_j; e_j (.) qbar; |e_j - qbar|]        (5d inputs)
 *   nu_j  = sigmoid(w2 . relu(W1 f_j + b1) + b2)
 *   keep  = the first min(n, |{j : nu_j >= tau_nu}|) of {j : nu_j >= tau_nu}
 *           ordered by (nu desc, id asc), n = ceil(rho_r * |K| - 1e-3),
 *           |K| = the question's non-empty candidate slots
 *
 * e_j is the corpus row of passage k_j (the passage's index embedding).
 * Precision: qbar, vbar, e_j and W1 are bf16; the interaction features
 * e (.) qbar and |e - qbar| are rounded to the nearest bf16 (ties to even)
 * and enter the first layer as bf16 operands of the tensor cores; sums,
 * b1, w2, b2 and nu are fp32.  Padded slots (id -1) are skipped.
 *
 * Conventions as in skip_retrieve.h (device pointers, asynchronous and
 * stream ordered, errors latched in the handle and reported by
 * skip_sync_status, no CPU fallback).  The gate needs a bf16 corpus with
 * d a multiple of 64 and at most 1024 (SKIP_EUNSUPPORTED otherwise) and
 * hidden a positive multiple of 128.
 */
#ifndef SKIP_SKV_H
#define SKIP_SKV_H

#include "skip_retrieve.h"

#ifdef __cplusplus
extern "C" {
#endif

/* The gate MLP h_psi (device buffers owned by the caller). */
typedef struct {
    int32_t hidden;        /* H, a positive multiple of 128 (the paper uses 512) */
    const uint16_t *w1;    /* bf16 bits [H x 5d] row-major; columns in the order
                              qbar | vbar | e | e (.) qbar | |e - qbar|, d each */
    const float *b1;       /* fp32 [H] */
    const float *w2;       /* fp32 [H] */
    float b2;              /* output bias */
} skip_skv_mlp_t;

/*
 * skip_skv_gate -- the gate on given candidate lists.
 *
 *  cand_ids   device int64 [num_questions x K]: passage ids (corpus rows),
 *             -1 for an empty slot.  An id >= N is treated as an empty
 *             slot and latches SKIP_EINVAL in the handle (skip_sync_status).
 *  qbar, vbar device bf16 bits [num_questions x d].
 *  mlp        host struct pointing at device weights.
 *  tau_nu     gate threshold (the paper uses 0.5); rho_r in [0, 1] (0.6).
 *  out_ids    device int64 [num_questions x K]: kept passages in order,
 *             then -1.
 *  out_nu     device fp32 [num_questions x K]: their nu, then -inf.
 *  out_count  device int32 [num_questions]: passages kept.
 *  nu_all     optional (NULL) device fp32 [num_questions x K]: nu of every
 *             input slot (-inf for empty ones).
 * Uses the handle's gate workspace (grown on demand, which synchronises the
 * device once).  Asynchronous on `stream`.  In skip_retrieve_skv the
 * per-question half of the first layer (which needs no candidate) runs on a
 * second stream of the handle, forked from `stream` once the retrieval's
 * score kernel is queued.  A flag in device memory tells the gate's MLP
 * kernel when that half is ready (a bounded wait), and the second stream is
 * joined back into `stream` after the gate's last kernel.  The call thus
 * stays ordered on `stream` as a whole, and can be captured into a CUDA
 * graph.
 * qbar, vbar and the mlp's w1 must start on 16-byte boundaries.
 * Errors: SKIP_EINVAL (null or misaligned pointers, K < 1 or > SKIP_MAX_K,
 * bad hidden, tau or rho), SKIP_EUNSUPPORTED (e4m3 corpus, d % 64 != 0,
 * d > 1024), SKIP_ENOMEM, SKIP_ECUDA.
 */
SKIP_API skip_status_t skip_skv_gate(skip_corpus_t corpus, const int64_t *cand_ids, int32_t num_questions,
                                     int32_t K, const uint16_t *qbar, const uint16_t *vbar,
                                     const skip_skv_mlp_t *mlp, float tau_nu, float rho_r, int64_t *out_ids,
                                     float *out_nu, int32_t *out_count, float *nu_all, void *stream);

/*
 * skip_retrieve_skv -- retrieval and gate in one call: skip_retrieve's
 * merged top-K lists go straight into skip_skv_gate.  Arguments as the two
 * calls; outputs as skip_skv_gate, and merged_ids / merged_scores
 * (optional, NULL: kept in the gate workspace) receive the merged lists.
 */
SKIP_API skip_status_t skip_retrieve_skv(skip_corpus_t corpus, const void *regions,
                                         const int32_t *region_offsets, int32_t num_questions,
                                         int32_t R_total, int32_t k_region, int32_t K, const uint16_t *qbar,
                                         const uint16_t *vbar, const skip_skv_mlp_t *mlp, float tau_nu,
                                         float rho_r, int64_t *out_ids, float *out_nu, int32_t *out_count,
                                         int64_t *merged_ids, float *merged_scores, void *stream);

#ifdef __cplusplus
}
#endif

#endif /* SKIP_SKV_H */
