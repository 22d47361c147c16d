/*
 * skip_retrieve.h -- C ABI of the GB300 (sm_103a) region-conditional sparse
 * retrieval library.
 *
 * The operation (paper §3.3 Eq. rcsr; App. B.2 Def. B.2; Alg. 1, the RCSR
 * loop and the Dedup step): every region query q_r of a question is scored
 * against every corpus row x_i by inner product (maximum inner product
 * search), the exact top-k_region ids are kept per region, and each
 * question's region lists are merged into one deduplicated top-K list.
 *
 *   s(r, i)  = sum_j q_{r,j} x_{i,j}        x = bf16 row, or e4m3 row * scale_i
 *   L_r      = top-k_region of {0..N-1} by (s desc, id asc)
 *   out_q    = top-K of union_{r in q} L_r by (max_r s desc, id asc),
 *              one entry per id, padded with (id -1, score -inf)
 *
 * Conventions shared by every entry point:
 *  - Corpus rows are row-major [N x d]; d must be a multiple of 16 and
 *    N < 2^31.  Ids are corpus row indices.
 *  - Region queries are bf16, row-major [R_total x d].  Questions own
 *    consecutive regions: question q owns rows [offsets[q], offsets[q+1]);
 *    offsets has Q + 1 int32 entries with offsets[0] = 0 and
 *    offsets[Q] = R_total; a question may own zero regions.
 *  - Scores are returned as fp32, ids as int64.  Lists are sorted by
 *    (score desc, id asc).  Ties go to the lower id.
 *  - Device pointers are CUDA device (or managed) addresses; host pointers
 *    are ordinary host memory.  Streams are cudaStream_t values passed as
 *    void* (NULL = the legacy default stream).
 *  - Calls on device buffers are asynchronous and stream ordered: they
 *    enqueue work on `stream` and return.  Argument errors are reported
 *    synchronously; errors found by kernels (a bounded wait that gave up)
 *    are latched in the corpus handle and reported by skip_sync_status.
 *  - A handle is not thread safe: serialise calls that share one.
 *  - Nothing here falls back to the CPU.  Without a usable sm_103 device,
 *    skip_corpus_load returns SKIP_EUNSUPPORTED.
 */
#ifndef SKIP_RETRIEVE_H
#define SKIP_RETRIEVE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#if defined(__GNUC__)
#define SKIP_API __attribute__((visibility("default")))
#else
#define SKIP_API
#endif

typedef struct skip_corpus *skip_corpus_t; /* opaque; owns the device copy */

typedef enum {
    SKIP_BF16 = 0, /* bf16 rows, 2 bytes per element */
    SKIP_E4M3 = 1  /* OCP float8 e4m3fn rows with one fp32 scale per row */
} skip_dtype_t;

typedef enum {
    SKIP_OK = 0,
    SKIP_EINVAL = 1,        /* bad argument (null pointer, size or range) */
    SKIP_ENOMEM = 2,        /* device or pinned allocation failed */
    SKIP_EUNSUPPORTED = 3,  /* no sm_103 device, or a size beyond a stated limit */
    SKIP_ETIMEOUT = 4,      /* a kernel's bounded wait gave up; results invalid */
    SKIP_ECUDA = 5,         /* a CUDA runtime/driver call failed */
    SKIP_ECANARY = 6        /* SKIP_OPT_CANARY: guard bytes after a buffer of the
                               handle were overwritten (a kernel wrote past its end) */
} skip_status_t;

typedef enum {
    SKIP_OPT_PATH = 0,            /* score kernel: 0 auto, 1 tensor core, 2 warp-dot, 3 small-batch tensor */
    SKIP_OPT_WAIT_TIMEOUT_NS = 1, /* cap on each in-kernel wait (default 2e9 ns) */
    SKIP_OPT_GRID = 2,            /* score-kernel CTAs (0 = one per SM) */
    SKIP_OPT_TIMING = 3,          /* 1: time each kernel with CUDA events */
    SKIP_OPT_CLUSTER = 4,         /* accepts 0 or 1 only: single-CTA tensor launches use no
                                     thread-block clusters (each CTA loads its own corpus tiles) */
    SKIP_OPT_MMA = 5,             /* tensor path MMA: 0 pick, 1 single CTA, 2 CTA pair */
    SKIP_OPT_BOUND = 6,           /* bf16 tensor path: 0 auto (a bounding pass over every 48th
                                     corpus tile first when the corpus has at least 2,048
                                     tiles and the full pass would admit about one key per
                                     thousand scores or more), 1 never, 2 always */
    SKIP_OPT_IVF_SPLIT = 7,       /* IVF-PQ index only (skip_ivfpq_set_option): parts each
                                     region's probed lists are cut into for the list scan,
                                     0 pick (1, 2 or 4: doubled while twice the parts
                                     still fit in the resident CTAs), else 1..8 */
    SKIP_OPT_CANARY = 8,          /* debugging aid (no counterpart in the paper): 1 places
                                     4 KiB of guard bytes after the handle's workspace,
                                     host staging and gate buffers (reallocating them now);
                                     skip_sync_status then also checks them and returns
                                     SKIP_ECANARY if any changed.  0 (default) off. */
    SKIP_OPT_RESIDENT = 9,        /* bf16 tensor path with CTA pairs, d <= 512, after a
                                     bounding pass: 0 auto (each CTA keeps its query block in
                                     shared memory for a work item and the per-row sets in
                                     global memory when the items can be sized so that about
                                     16 keys or fewer reach a set), 1 never, 2 whenever the
                                     shape allows (for tests) */
    SKIP_OPT_IVF_REFINE = 10      /* IVF-PQ index built from a corpus (skip_ivfpq_set_option):
                                     0 or 1 off; r >= 2 keeps the best min(r k_region, 1024)
                                     entries of each region by s^ and re-ranks them by the
                                     exact inner product with the corpus rows (the corpus
                                     handle must stay alive); SKIP_EUNSUPPORTED for an index
                                     made by skip_ivfpq_load */
} skip_option_t;

enum { SKIP_PATH_AUTO = 0, SKIP_PATH_TENSOR = 1, SKIP_PATH_WARP = 2, SKIP_PATH_LATENCY = 3 };

/* Limits checked by every retrieval call. */
#define SKIP_MAX_K_REGION 1024
#define SKIP_MAX_K 2048

/*
 * skip_corpus_load -- lay the corpus D (paper Def. B.2, the searched set;
 * §4.1 "Knowledge corpora") out in device memory for retrieval.
 *
 *  rows            [N x d] row-major elements: uint16 bf16 bits for
 *                  SKIP_BF16, bytes for SKIP_E4M3.
 *  rows_on_device  nonzero: `rows` and `row_scale` are device pointers and
 *                  are copied device-to-device; zero: host pointers.
 *  row_scale       [N] fp32 per-row dequantisation scales; required for
 *                  SKIP_E4M3 (each element's value is e4m3 * scale), must
 *                  be NULL for SKIP_BF16.
 *  stream          stream for the copies; the call returns after they finish.
 *  out             receives the handle.
 * The library owns the copy until skip_corpus_free; the caller's buffers
 * can be reused as soon as the call returns.
 * Errors: SKIP_EINVAL (null pointers, N < 1, N >= 2^31, d % 16 != 0,
 * scale missing or unexpected), SKIP_ENOMEM, SKIP_EUNSUPPORTED (no
 * sm_103 device), SKIP_ECUDA.
 */
SKIP_API skip_status_t skip_corpus_load(const void *rows, int rows_on_device, int64_t N, int32_t d,
                               skip_dtype_t dtype, const float *row_scale, void *stream,
                               skip_corpus_t *out);

/* Frees the corpus copy and the handle's workspace after synchronising the
 * device.  NULL is accepted. */
SKIP_API skip_status_t skip_corpus_free(skip_corpus_t corpus);

/* Sets a per-handle option (skip_option_t); SKIP_EINVAL for an unknown
 * option or a value out of range. */
SKIP_API skip_status_t skip_corpus_set_option(skip_corpus_t corpus, int option, int64_t value);

/*
 * skip_retrieve -- the whole path on device buffers: per-region MIPS top-k
 * (Def. B.2, Eq. rcsr), then the per-question Dedup of the union cut to K
 * (§3.3, Def. B.2, Alg. 1).
 *
 *  regions         device bf16 [R_total x d] (uint16 bits), row-major.
 *  region_offsets  device int32 [num_questions + 1] prefix offsets; the
 *                  library never reads them on the host, so R_total must
 *                  equal region_offsets[num_questions].
 *  k_region        1 <= k_region <= min(N, SKIP_MAX_K_REGION).
 *  K               1 <= K <= SKIP_MAX_K.
 *  out_ids         device int64 [num_questions x K].
 *  out_scores      device fp32  [num_questions x K].
 * Uses a workspace owned by the handle (grown on demand, which
 * synchronises the device once).  Asynchronous on `stream`.
 * Errors: SKIP_EINVAL, SKIP_ENOMEM, SKIP_ECUDA.
 */
SKIP_API skip_status_t skip_retrieve(skip_corpus_t corpus, const void *regions,
                            const int32_t *region_offsets, int32_t num_questions,
                            int32_t R_total, int32_t k_region, int32_t K, int64_t *out_ids,
                            float *out_scores, void *stream);

/*
 * skip_retrieve_regions -- only the per-region step (Def. B.2
 * MIPS(q_r, D; k_r)): reg_ids int64 and reg_scores fp32, both device
 * [R_total x k_region], each row sorted by (score desc, id asc).
 * Same argument rules as skip_retrieve.
 */
SKIP_API skip_status_t skip_retrieve_regions(skip_corpus_t corpus, const void *regions, int32_t R_total,
                                    int32_t k_region, int64_t *reg_ids, float *reg_scores,
                                    void *stream);

/*
 * skip_retrieve_host -- skip_retrieve on HOST buffers: copies regions and
 * offsets to the device, runs the path and copies the results back, all on
 * `stream`, and returns after the stream has drained (so the kernels'
 * error word is also checked).  Shapes as in skip_retrieve.
 * Errors: as skip_retrieve, plus SKIP_ETIMEOUT.
 */
SKIP_API skip_status_t skip_retrieve_host(skip_corpus_t corpus, const uint16_t *regions,
                                 const int32_t *region_offsets, int32_t num_questions,
                                 int32_t R_total, int32_t k_region, int32_t K, int64_t *out_ids,
                                 float *out_scores, void *stream);

/*
 * skip_retrieve_regions_noalloc -- the per-region step for callers that
 * cannot allocate device memory.  The paper has no counterpart: this entry
 * point exists for callers whose device memory is owned by a host framework
 * (every allocation must come from its pool) and for serving loops that
 * cannot afford the device-wide synchronisation of cudaMalloc/cudaFree.
 *
 * It takes the corpus as device pointers instead of a handle and allocates
 * nothing: its scratch is one 16 MiB array in the library's device memory,
 * created once per device that loads the library and kept until the process
 * exits.  The first call on a device looks that array's address up (make it
 * before any stream capture).  All calls on a device share the array, so
 * calls that overlap on the GPU race; calls ordered on one stream do not.
 *
 *  corpus_rows     device [N x d] row-major, bf16 bits or e4m3 bytes (dtype);
 *                  row_scale device [N] fp32 for SKIP_E4M3, NULL for bf16.
 *  regions         device bf16 [R_total x d].
 *  reg_ids/scores  device int64 / fp32 [R_total x k_region], each row sorted
 *                  by (score desc, id asc) -- the same result as
 *                  skip_retrieve_regions.
 * Alignment (SKIP_EINVAL otherwise, checked before anything is launched):
 * corpus_rows on a 16-byte boundary, row_scale and reg_scores on 4 bytes,
 * regions on 2, reg_ids on 8.
 * Limits as skip_retrieve_regions, plus: with G = min(#SMs, 512,
 * ceil(N / 256)) score-kernel blocks, the scratch of
 * 8 * k_region * (G * R_total + G * 64) bytes (the first term rounded up to
 * 256) must fit in 16 MiB, else SKIP_EUNSUPPORTED; the limit on R_total *
 * k_region therefore depends on the GPU's SM count and on N.
 * Asynchronous on `stream`.
 */
SKIP_API skip_status_t skip_retrieve_regions_noalloc(const void *corpus_rows, int64_t N, int32_t d,
                                                     skip_dtype_t dtype, const float *row_scale,
                                                     const void *regions, int32_t R_total,
                                                     int32_t k_region, int64_t *reg_ids,
                                                     float *reg_scores, void *stream);

/* Synchronises `stream`, then reports and clears the handle's error word:
 * SKIP_ETIMEOUT if a kernel's bounded wait gave up since the last check,
 * SKIP_EINVAL if region offsets were inconsistent with R_total (clamped),
 * SKIP_ECUDA if the stream reported an error, with SKIP_OPT_CANARY on
 * SKIP_ECANARY if a guard region was overwritten, else SKIP_OK.
 *
 * Fault injection (a debugging aid with no counterpart in the paper): with
 * the environment variable SKIP_FAULT_INJECT=alloc every device allocation
 * the library makes fails as on an exhausted device, and the call that needed
 * it returns SKIP_ENOMEM; SKIP_FAULT_INJECT=alloc:<kind> limits this to one
 * kind (corpus, workspace, staging, gate, ivfpq, qvs, bsca).  The variable
 * is read at every allocation; a handle whose workspace growth failed stays
 * usable and allocates again on its next call. */
SKIP_API skip_status_t skip_sync_status(skip_corpus_t corpus, void *stream);

/* Describes the last retrieval call's launch plan as a short JSON object
 * (path, grid, corpus chunks, kernels launched) and, when SKIP_OPT_TIMING is
 * on, the device time of each kernel in ms (this synchronises on the
 * events).  Writes at most `len` bytes including the terminator. */
SKIP_API skip_status_t skip_last_plan(skip_corpus_t corpus, char *buf, int32_t len);

/* Infrastructure (no counterpart in the paper): with SKIP_OPT_TIMING on,
 * every retrieval call records CUDA events on its stream around each kernel
 * it launches.  This call waits for the last event, writes a JSON object
 * {"<kernel>": {"launches": n, "ms": total device time}, ...} accumulated
 * over all calls since the previous report, and clears the record.
 * SKIP_EINVAL if `len` is too small. */
SKIP_API skip_status_t skip_timing_report(skip_corpus_t corpus, char *buf, int32_t len);

/* Static description of a status code. */
SKIP_API const char *skip_status_string(skip_status_t status);

#ifdef __cplusplus
}
#endif

#endif /* SKIP_RETRIEVE_H */
