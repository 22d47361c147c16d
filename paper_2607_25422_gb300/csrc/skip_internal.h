// Host-side declarations shared by the C-ABI layer and the kernel files.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace skipk {

// Bits of the per-handle device error word.
enum : int { kErrTimeout = 1, kErrConfig = 2 };

// ---- warp-dot score + top-k (small region batches) -------------------
struct WarpDotParams {
    const uint8_t *corpus;   // [N x d] rows, d * elem_bytes bytes apart
    const float *scale;      // [N] (e4m3 only)
    int64_t N;
    int d;
    const uint16_t *regions; // bf16 bits; rows [q0, q0 + nq) of the batch
    int nq;                  // queries in this launch (<= 8)
    int k;
    uint64_t *warp_lists;    // [grid][kWarpDotWarps][nq][k] scratch
    uint64_t *lists;         // [grid][R_pad][k]; this launch writes rows q0..q0+nq
    int64_t list_g_stride;   // elements between consecutive grid lists (R_pad * k)
    int q0;
};
constexpr int kWarpDotWarps = 8;
constexpr int kWarpDotThreads = kWarpDotWarps * 32;
cudaError_t launch_warpdot(const WarpDotParams &p, bool e4m3, int grid, cudaStream_t s);

// ---- tensor-core score + top-k -----------------------------------------
struct TcParams {
    int64_t N;
    int d;
    int R;            // region rows
    int R_pad;        // padded query blocks * 128
    int k;
    int MB;           // query blocks of 128 rows holding region rows
    int CL;           // CTAs per cluster: 1, or 2 for a CTA pair (one query block each)
    int QG;           // query groups: ceil(MB / CL)
    int G;            // corpus chunks (lists per row)
    int64_t tiles;    // corpus tiles of kTcTileN rows this launch visits
    int tile_stride;  // bf16 kernel: item tile t is corpus tile t * tile_stride (1, or the
                      // sample stride of a bounding pass)
    int share;        // bf16 kernel: 1 = the chunks of a row share their k-th score through
                      // tau; 0 in a bounding pass (its lists are shorter than the caller's k)
    int dense;        // bf16 kernel, bounding pass with k == 4: each row's four largest scores
                      // of the chunk kept in registers (no ids; keys with stand-in ids)
    uint64_t *lists;  // [G][R_pad][k]
    uint32_t *tau;    // [R_pad] shared per-row threshold (order-preserving ints), zeroed
    int *err;
    uint64_t timeout_ns;
    int stages;       // operand pipeline depth
    int list_in_smem; // per-row lists in shared memory (else global)
    const float *scale;  // [N] row scales (e4m3 corpus only)
    int raw_stages;      // e4m3 corpus: depth of the raw-slice ring
    int *sched;          // bf16 kernel: work-item counter, zero at launch
    int a_res;           // bf16 pair kernel: the query block stays resident in shared memory for
                         // the whole item and the ring carries corpus slices only (sets in global
                         // memory; d <= 64 * kMaxResidentSlices)
};
constexpr int kTcTileM = 128;   // region rows per tile (TMEM lanes)
constexpr int kTcTileN = 256;   // corpus rows per tile (TMEM columns)
constexpr int kTcTileK = 64;    // bf16 elements per stage row (128 bytes)
constexpr int kTcThreads = 192; // producer warp, MMA warp, 4 epilogue warps
constexpr int kBoundStride = 48;     // bounding pass: every 48th corpus tile (2% more MMA work)
constexpr int kBoundMinTiles = 2048; // ... on corpora of at least 2,048 tiles (524,288 rows)
constexpr int kMaxResidentSlices = 8;  // resident query block: d <= 512
constexpr int kTcChunkTiles = 200;     // corpus tiles per work item at most (chunks of a large corpus)
// pair: CTA-pair MMA (cta_group::2, clusters of 2); else single-CTA MMA.
// a_res_slices: 64-element slices of a resident query block (0: none).
size_t tc_smem_bytes(bool pair, int stages, int k, bool list_in_smem, int a_res_slices);
// Deepest pipeline that fits next to shared-memory lists, else global lists.
void tc_pick_layout(bool pair, int k, int max_smem, int *stages, bool *list_in_smem);
// Pair kernel with a resident query block of width d (sets in global
// memory): the ring depth that fits, 0 if d is too wide.
int tc_pick_resident_stages(int d, int max_smem);
// Clusters of CL CTAs that can be resident at once with this layout.
int tc_max_clusters(bool pair, int CL, int stages, int k, bool list_in_smem, int a_res_slices);
// pdl: launched as the programmatic dependent of the kernel before it in the
// stream (the epilogue waits for it before reading the shared thresholds).
cudaError_t launch_tc(bool pair, const CUtensorMap &tq, const CUtensorMap &tx, const TcParams &p, int grid,
                      cudaStream_t s, bool pdl = false);

// e4m3 corpus (single-CTA MMA, corpus widened to bf16 in shared memory).
void tc_fp8_pick_layout(int k, int max_smem, int *stages, int *raw_stages, bool *list_in_smem);
cudaError_t launch_tc_fp8(const CUtensorMap &tq, const CUtensorMap &traw, const TcParams &p, int grid,
                          cudaStream_t s);

// ---- small batches on the tensor cores (corpus tile = A, queries = B) ----
constexpr int kLatMaxR = 32;
struct LatParams {
    int64_t N;
    int d;
    int R;                    // region rows (<= kLatMaxR)
    int k;
    int Npad;                 // MMA N: 96 (e4m3, three query parts) or R rounded up to 16
    int slices;               // 128-byte K slices per row
    int stages;               // corpus ring depth
    int64_t tiles;            // 128-row corpus tiles
    int G;                    // corpus chunks (lists per query)
    const float *corpus_scale;  // [N] (e4m3)
    const float *qscale;        // [3][R] scales of the query parts (e4m3)
    uint64_t *lists;          // [G][R][k]
    uint32_t *tau;            // [R] shared thresholds, zero at launch
    uint32_t *tau_clear;      // [kLatMaxR] the next call's thresholds, cleared by this kernel
    int *err;
    uint64_t timeout_ns;
};
bool lat_pick_layout(bool fp8, int R, int d, int k, int max_smem, int *Npad, int *slices, int *stages);
// e4m3 query parts: parts [96 x d] bytes (all 96 rows written: rows of slots past R are zero), qscale [3][R].
cudaError_t launch_split_queries(const uint16_t *regions, int R, int d, uint8_t *parts, float *qscale,
                                 cudaStream_t s);
cudaError_t launch_latency(bool fp8, const CUtensorMap &ta, const CUtensorMap &tb, const LatParams &p, int grid,
                           cudaStream_t s);

// ---- small dense GEMM with fp32 results (k_gemm.cu) ------------------------
// D [M x N] (leading dimension ldd) = alpha * A [M x K] B [N x K]^T, bf16
// operands row-major with K contiguous (K % 8 == 0).  ta: tensor map over A,
// box 128 rows x 64 elements; tb: over B, box tile_n rows x 64 elements; both
// 128-byte swizzle.  err (nullable) receives kErrTimeout if a wait gives up.
// gemm_tile_n: the tile width (32 or 64) to use for an M x N product.
// splits > 1: K is split over that many CTAs per tile, each writing its
// partial product to D + z * split_stride (split_stride >= M * ldd); the
// caller sums the slabs.  gemm_splits: the split count that fills the SMs
// once (1 when the tiles already do).
int gemm_tile_n(int M, int N, int sms);
int gemm_splits(int M, int N, int K, int tile_n, int sms);
cudaError_t launch_gemm_bf16_f32(const CUtensorMap &ta, const CUtensorMap &tb, int tile_n, int M, int N, int K,
                                 float alpha, float *D, int64_t ldd, int *err, uint64_t timeout_ns, cudaStream_t s,
                                 int splits = 1, int64_t split_stride = 0);
// D = alpha * (A B^T + A2 B2^T) + bias (per column n; nullable); ta2 / tb2
// over A2 [M x K2] / B2 [N x K2] with the same boxes (K2 = 0: one product).
cudaError_t launch_gemm2_bf16_f32(const CUtensorMap &ta, const CUtensorMap &tb, const CUtensorMap *ta2,
                                  const CUtensorMap *tb2, int tile_n, int M, int N, int K, int K2, float alpha,
                                  const float *bias, float *D, int64_t ldd, int *err, uint64_t timeout_ns,
                                  cudaStream_t s, int splits = 1, int64_t split_stride = 0);

// ---- merges -------------------------------------------------------------
// Per-region merge of G sorted lists into the exact top-k (keys and/or
// decoded ids/scores).  pdl (here and below): launched as the programmatic
// dependent of the kernel just before it in the stream (the merge waits for
// it before reading, and lets the next kernel launch early).
int question_merge_capacity();
// Both merges in one launch (small batches): per question, the k-way merge
// of each of its region rows' G lists, then dedup / rank / cut to K.
// Requires R k <= question_merge_capacity(), K <= the same, G <= 512.
cudaError_t launch_merge_regions_questions(const uint64_t *lists, int G, int64_t g_stride, int R, int k,
                                           const int32_t *offsets, int Q, int K, int64_t *out_ids,
                                           float *out_scores, int *err, cudaStream_t s, bool pdl);
cudaError_t launch_merge_lists(const uint64_t *lists, int G, int64_t g_stride, int R, int k,
                               uint64_t *reg_keys, int64_t *reg_ids, float *reg_scores,
                               cudaStream_t s, bool pdl = false);
// The same over lists of `len` keys each (len may differ from the k kept);
// with tau, also tau[row] = max(tau[row], the order-preserving integer of the
// score of the row's k-th merged key) when it has one: a sample's k-th best
// score bounds the row's k-th best score over the whole corpus from below.
cudaError_t launch_merge_lists_len(const uint64_t *lists, int G, int64_t g_stride, int len, int R, int k,
                                   uint64_t *reg_keys, int64_t *reg_ids, float *reg_scores, uint32_t *tau,
                                   cudaStream_t s, bool pdl = false);
// Per-question union + dedup (max score) + top-K.
// Offsets are clamped to [0, R]; a clamp sets kErrConfig in *err.
cudaError_t launch_question_merge(const uint64_t *reg_keys, int k, const int32_t *offsets, int Q,
                                  int R, int K, int64_t *out_ids, float *out_scores, int *err,
                                  cudaStream_t s, bool pdl = false);

// ---- SKV passage gate (k_skv.cu) ------------------------------------------
constexpr int kSkvHidden = 128;  // the gate MLP's hidden width is a multiple of this
constexpr int kSkvMaxK = 2048;   // candidate slots per question (SKIP_MAX_K)
struct SkvParams {
    const uint16_t *rows;  // bf16 corpus [N x d]
    int64_t N;
    int d;                 // multiple of 64, at most 1024
    const int64_t *ids;    // [Q x K] candidate ids, -1 = empty
    int64_t P;             // Q * K slots
    int K;
    int Q;
    const uint16_t *qbar;  // bf16 [Q x d]
    const uint16_t *vbar;  // bf16 [Q x d]
    const uint16_t *w1;    // bf16 [H x 5d]
    const float *b1;       // [H]
    const float *w2;       // [H]
    float b2;
    int H;                 // multiple of kSkvHidden
    float tau, rho;
    float *cq;             // [cq_splits x Q x H] workspace: partial sums of b1 + W1 qbar-part + W1 vbar-part
    int cq_splits;         // K splits of the c_q GEMM (the slabs are summed in k_skv_mlp)
    const int *cq_flag;    // null, or raised to cq_epoch when c_q (from another stream) is complete
    int cq_epoch;
    float *partial;        // [nparts][P] workspace: partial logits
    int nparts;            // partial-logit slabs: H / BN * S * 2 (skv_mlp_shape)
    int64_t *out_ids;      // [Q x K]
    float *out_nu;         // [Q x K]
    int32_t *out_count;    // [Q]
    float *nu_all;         // [Q x K] or null
    int *err;
    uint64_t timeout_ns;
};
size_t skv_mlp_smem_bytes(int BN, int S);  // dynamic shared memory of k_skv_mlp
// Tile shape of the gate MLP for P slots and H hidden units: BN hidden units
// per CTA pair (128 or 256) and S K parts (1 or 2; clusters of 2 S CTAs).
void skv_mlp_shape(int64_t P, int H, int *BN, int *S);
// The gate in four launches: per-question bias (the library GEMM), the
// passage features F [P x 3d] bf16, the tensor-core layer 1 + ReLU + w2
// partial dots, and the sigmoid / gate / selection.
// tf: tensor map over F [P x 3d], box 64 columns x 128 rows; tw: over W1
// [H x 5d], box 64 columns x BN / 2 rows; both bf16, 128-byte swizzle.
// The features kernel waits for the grid before it (the candidate ids)
// before it reads; the MLP reads c_q, which must be complete when it starts.
cudaError_t launch_skv_features(const SkvParams &p, uint16_t *F, cudaStream_t s);
cudaError_t launch_skv_mlp(const CUtensorMap &tf, const CUtensorMap &tw, const SkvParams &p, int BN, int S,
                           cudaStream_t s);
cudaError_t launch_skv_select(const SkvParams &p, cudaStream_t s);
// One thread stores `epoch` to *flag (release, GPU scope).
cudaError_t launch_skv_cq_ready(int *flag, int epoch, cudaStream_t s);

// ---- IVF-PQ variant (k_ivfpq.cu) ------------------------------------------
constexpr int kIvfMaxDs = 32;   // largest sub-space width d / M
constexpr int kIvfMaxM = 128;   // most sub-spaces (code bytes)
struct IvfParams {
    const void *rows;       // bf16 corpus [N x d] (build only)
    int64_t N;
    int d;
    const void *centroids;  // bf16 [C x d]
    int C;
    const float *codebook;  // [M][256][ds]
    const float *cbT;       // [256][ds][Mp]: codebook with the sub-space fastest, 0 past M
    int M;                  // sub-spaces, a multiple of 16
    int ds;                 // d / M
    const int64_t *offsets; // [C + 1] list starts (entries)
    const int64_t *boff;    // [C + 1] list starts (blocks of 32 entries)
    const int32_t *ids;     // [N] ids in list order
    const uint8_t *codes;   // [boff[C]][M * 32] codes in blocks of 32 entries (k_ivfpq.cu: il_offset)
};
// M rounded up to a whole number of warps: the row stride of the lookup table.
inline int ivf_padded_m(int M) { return (M + 31) / 32 * 32; }
cudaError_t launch_pq_encode(const IvfParams &p, const int64_t *row_list, uint8_t *codes, cudaStream_t s);
// counts, cursor: [C] scratch; offsets [C + 1]; ids [N]; codes [N x M] (list order, one row per entry).
cudaError_t launch_ivf_lists(const IvfParams &p, const int64_t *row_list, const uint8_t *codes_rows,
                             int64_t *counts, int64_t *cursor, int64_t *offsets, int32_t *ids, uint8_t *codes,
                             int *err, int sms, cudaStream_t s);
// rows [N x M] in list order <-> p.codes (p.offsets, p.boff valid).
cudaError_t launch_ivf_interleave(const IvfParams &p, const uint8_t *rows, uint8_t *il, int sms, cudaStream_t s);
cudaError_t launch_ivf_deinterleave(const IvfParams &p, uint8_t *rows, int sms, cudaStream_t s);
// cbT [256 x ds x ivf_padded_m(M)] from codebook [M x 256 x ds].
cudaError_t launch_pq_codebook_t(const float *codebook, int M, int ds, float *cbT, cudaStream_t s);
// Coarse probe over at most kIvfCoarseMaxC centroids: scores [R x C] (a
// GEMM) -> per region the nprobe best (id, score), sorted (score desc, id asc).
constexpr int kIvfCoarseMaxC = 4096;
cudaError_t launch_ivf_probe_select(const float *scores, int R, int C, int nprobe, int64_t *probe_ids,
                                    float *probe_sc, cudaStream_t s);
size_t ivfpq_scan_smem(int M, int nprobe);
// Exact re-rank: per region, the ks shortlisted keys cand [R x ks] scored
// exactly against the bf16 rows [N x d], the k best written as keys [R x k].
constexpr int kIvfMaxRefine = 1024;  // shortlist length at most
cudaError_t launch_ivf_refine(const uint16_t *rows, int64_t N, int d, const uint16_t *regions, int R,
                              const uint64_t *cand, int ks, int k, uint64_t *out, cudaStream_t s);
constexpr int kIvfMaxSplit = 8;  // most parts a region's probed blocks are cut into
// Parts per region of the list scan: `requested` if > 0, else 1, 2 or 4,
// doubling while twice the items still fit in the resident CTAs.
cudaError_t ivfpq_scan_split(int M, int nprobe, int R, int sms, int requested, int *G);
// Per part g of region r: keys (ordered score << 32 | ~id, 0 = empty) of its
// top k at out_keys[(g * R + r) * k], sorted descending [G x R x k].
cudaError_t launch_ivfpq_scan(const IvfParams &p, const uint16_t *regions, int R, const int64_t *probe_ids,
                              const float *probe_scores, int nprobe, int k, int G, uint64_t *out_keys, int sms,
                              cudaStream_t s);

// ---- QVS visual token pruning (k_qvs.cu) -----------------------------------
constexpr int kQvsMaxDk = 4096;  // projection width d_k
constexpr int kQvsMaxL = 4096;   // tokens per image
constexpr int kQvsUSplits = 4;   // K splits of the projected-query GEMM
constexpr int kSkvCqSplits = 4;  // K splits of the SKV gate's c_q GEMM
struct QvsParams {
    const void *tokens;     // bf16 [B x L x d]
    const void *fq;         // bf16 [B x dk]
    const void *wvt;        // bf16 [d x dk]: W_v^T
    const float *bv;        // [dk] or null
    const float *wb;        // [d]
    int B, L, d, dk, n;     // n tokens kept per image
    float *u;               // [u_splits x B x d] partial sums of W_v^T f_q / sqrt(d_k) (split-K GEMM)
    int u_splits;
    float *logits;          // [B x L] workspace
    int32_t *out_idx;       // [B x n]
    float *out_score;       // [B x n]
    void *out_tokens;       // bf16 [B x n x d] or null
};
cudaError_t launch_qvs_logits(const QvsParams &p, int sms, cudaStream_t s);
// wt [cols x ldt] (first `rows` of each row) = w^T for a bf16 w [rows x cols].
cudaError_t launch_transpose_bf16(const uint16_t *w, int rows, int cols, uint16_t *wt, int ldt, cudaStream_t s);
// Ranks every token by counting the larger logits and writes the kept ones
// (rank < n) in rank order, with their rows when out_tokens is set.
cudaError_t launch_qvs_select(const QvsParams &p, cudaStream_t s);

// ---- BSCA bipartite sparse cross-attention (k_bsca.cu) --------------------
constexpr int kBscaMaxR = 64;     // chunks per question
constexpr int kBscaMaxDp = 256;   // width of h_v / h_k
constexpr int kBscaMaxDh = 256;   // width of W_Q / W_K
constexpr int kBscaMaxDo = 2048;  // width of W_V
constexpr int kBscaMaxPairs = 32768;  // (visual token, chunk) pairs per question
constexpr int kBscaBins = 4096;       // cosine histogram bins per question (over [-1, 1])
struct BscaParams {
    int Q;
    const int32_t *vis_offsets;    // [Q + 1]
    const int32_t *chunk_offsets;  // [Q + 1]
    int64_t Nv;                    // visual tokens in all
    const uint16_t *hv, *qh;       // bf16 [Nv x dp], [Nv x dh]
    const uint16_t *hk, *kh, *vh;  // bf16 [Nc x dp], [Nc x dh], [Nc x dout]
    int dp, dh, dout;              // dout even
    float dbar;
    float *cos;                    // [Nv x kBscaMaxR] workspace
    uint32_t *hist;                // [Q x kBscaBins] workspace, all zero between calls
    float *tau;                    // [Q]
    int32_t *degree;               // [Nv] or null
    uint64_t *edges;               // [Nv] neighbour bit masks or null
    float *out;                    // [Nv x dout]
    int *err;
};
cudaError_t launch_bsca(const BscaParams &p, cudaStream_t s);

}  // namespace skipk
