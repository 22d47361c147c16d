/*
 * skip_ivfpq.h -- C ABI of the IVF-PQ approximate variant of the per-region
 * search.
 *
 * The paper retrieves from a FAISS IVF-PQ index (§4.1 "Implementation":
 * 1,024 IVF centroids over 768-d vectors; App. I.4: IVF4096-PQ64).  This is
 * that index, built and searched on the GPU as in the published method
 * (Jegou, Douze, Schmid, IEEE TPAMI 33(1), 2011), with inner products:
 *
 *   coarse   list(i) = argmax_l <x_i, c_l>                 (ties: lower l)
 *   code     code_{i,m} = argmin_j ||(x_i - c_list(i))_m - p_{m,j}||^2
 *            over M sub-spaces of d/M values, 256 codewords each (ties: lower j)
 *   search   probes(q) = the nprobe lists with the largest <q, c_l>;
 *            s^(q, i) = <q, c_list(i)> + sum_m <q_m, p_{m, code_{i,m}}> over
 *            the ids of the probed lists; the k_region best by
 *            (s^ desc, id asc), padded with (-1, -inf); questions then merge
 *            their regions' lists as skip_retrieve does.
 *
 * Centroids are bf16 [C x d], the codebook fp32 [M x 256 x d/M] (both given:
 * training them is not part of this library).  Codes are one byte per
 * sub-space.  Conventions as in skip_retrieve.h (device pointers,
 * asynchronous and stream ordered, no CPU fallback).  Limits: bf16 corpus,
 * M a multiple of 16, at most 128, with d / M <= 32, 1 <= nprobe <= min(C, 1024),
 * 1 <= k_region <= 1024, C <= 2^20.
 */
#ifndef SKIP_IVFPQ_H
#define SKIP_IVFPQ_H

#include "skip_retrieve.h"

#ifdef __cplusplus
extern "C" {
#endif

typedef struct skip_ivfpq *skip_ivfpq_t; /* opaque; owns its device arrays */

/*
 * skip_ivfpq_build -- the index of a loaded corpus: coarse assignment (on the
 * exact MIPS path, centroids as the searched set), residual PQ encoding and
 * the inverted lists.  centroids device bf16 [C x d]; codebook device fp32
 * [M x 256 x d/M].  The corpus handle must outlive nothing: the index keeps
 * only its own arrays.  Returns after the build has finished on `stream`.
 * Errors: SKIP_EINVAL (null pointers, sizes), SKIP_EUNSUPPORTED (e4m3 corpus,
 * M or d/M outside the limits), SKIP_ENOMEM, SKIP_ECUDA, SKIP_ETIMEOUT.
 */
SKIP_API skip_status_t skip_ivfpq_build(skip_corpus_t corpus, const void *centroids, int32_t C,
                                        const float *codebook, int32_t M, void *stream, skip_ivfpq_t *out);

/*
 * skip_ivfpq_load -- an index from existing arrays (device pointers, copied):
 * list_offsets int64 [C + 1] (list l holds entries [off[l], off[l+1])),
 * ids int32 [N] and codes uint8 [N x M] in list order, centroids bf16
 * [C x d], codebook fp32 [M x 256 x d/M].  Returns after the copies.
 * The index stores the codes in its own layout (blocks of 32 entries of a
 * list, grouped by sub-space); skip_ivfpq_lists returns them in the row
 * layout above.  Errors: SKIP_EINVAL also when the offsets are not
 * 0 = off[0] <= off[1] <= ... <= off[C] = N.
 */
SKIP_API skip_status_t skip_ivfpq_load(const void *centroids, int32_t C, int32_t d, const float *codebook,
                                       int32_t M, const int64_t *list_offsets, const int32_t *ids,
                                       const uint8_t *codes, int64_t N, void *stream, skip_ivfpq_t *out);

/* Copies the index's lists out (device pointers, sizes as in
 * skip_ivfpq_load; any may be NULL).  Ids inside a list are in no particular
 * order.  Returns after the copies. */
SKIP_API skip_status_t skip_ivfpq_lists(skip_ivfpq_t index, int64_t *list_offsets, int32_t *ids, uint8_t *codes,
                                        void *stream);

/* Index sizes: any pointer may be NULL. */
SKIP_API skip_status_t skip_ivfpq_info(skip_ivfpq_t index, int64_t *N, int32_t *d, int32_t *C, int32_t *M);

SKIP_API skip_status_t skip_ivfpq_free(skip_ivfpq_t index);

/*
 * skip_ivfpq_search_regions -- per region: reg_ids int64 / reg_scores fp32,
 * both device [R_total x k_region], sorted by (s^ desc, id asc); with
 * SKIP_OPT_IVF_REFINE = r >= 2 (an option beyond the paper's IVF-PQ, the
 * usual exact re-rank), the best min(r k_region, 1024) entries by s^ are
 * re-scored exactly (fp32 sums of the bf16 products) and the k_region best by
 * (exact score desc, id asc) are returned with their exact scores.
 */
SKIP_API skip_status_t skip_ivfpq_search_regions(skip_ivfpq_t index, const void *regions, int32_t R_total,
                                                 int32_t nprobe, int32_t k_region, int64_t *reg_ids,
                                                 float *reg_scores, void *stream);

/*
 * skip_ivfpq_search -- per region, then the per-question merge as in
 * skip_retrieve (union, max per id, top-K by (score desc, id asc), padded).
 * out_ids int64 / out_scores fp32, device [num_questions x K].
 */
SKIP_API skip_status_t skip_ivfpq_search(skip_ivfpq_t index, const void *regions, const int32_t *region_offsets,
                                         int32_t num_questions, int32_t R_total, int32_t nprobe, int32_t k_region,
                                         int32_t K, int64_t *out_ids, float *out_scores, void *stream);

/* As skip_sync_status, for the index's kernels. */
SKIP_API skip_status_t skip_ivfpq_sync_status(skip_ivfpq_t index, void *stream);

/* Sets an option of the index: SKIP_OPT_IVF_SPLIT for its list scan,
 * SKIP_OPT_IVF_REFINE for the exact re-rank of a shortlist; any
 * other skip_option_t of skip_retrieve.h applies to its centroid set, which
 * the exact MIPS path searches for the build's coarse assignment and, with
 * more than 4,096 centroids, for the search's coarse probe (with at most
 * 4,096 the probe is one bf16 GEMM and a per-region sort).  SKIP_OPT_TIMING
 * records the index's kernels, reported by skip_ivfpq_timing_report.
 * Apart from SKIP_OPT_IVF_REFINE, results do not depend on the options. */
SKIP_API skip_status_t skip_ivfpq_set_option(skip_ivfpq_t index, int option, int64_t value);
SKIP_API skip_status_t skip_ivfpq_timing_report(skip_ivfpq_t index, char *buf, int32_t len);

#ifdef __cplusplus
}
#endif

#endif /* SKIP_IVFPQ_H */
