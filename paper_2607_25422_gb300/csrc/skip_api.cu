// C-ABI layer of the retrieval library: argument checks, the corpus copy and
// its TMA descriptor, the per-handle workspace, the launch plan for each
// regime and the error word.  The arithmetic lives in the kernels
// (k_tc.cu, k_warpdot.cu, k_merge.cu and the others); this file only decides
// what to launch.  No vendor library is called: the two plain products (QVS's
// projected query and the IVF-PQ coarse probe) run on k_gemm.cu.
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include <algorithm>
#include <cmath>
#include <functional>
#include <map>
#include <mutex>
#include <string>
#include <vector>

#include "../../include/skip_retrieve.h"
#include "../../include/skip_skv.h"
#include "../../include/skip_ivfpq.h"
#include "../../include/skip_qvs.h"
#include "../../include/skip_bsca.h"
#include "skip_internal.h"

using namespace skipk;

namespace {

constexpr uint64_t kDefaultTimeoutNs = 2000000000ull;
constexpr int kMaxD = 4096;
constexpr size_t kMaxEvents = 1 << 20;

typedef CUresult (*EncodeTiledFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *,
                                  const cuuint64_t *, const cuuint64_t *, const cuuint32_t *,
                                  const cuuint32_t *, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
    static EncodeTiledFn fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(p);
    });
    return fn;
}

// 2D bf16 tensor map over a row-major [rows x d] matrix, box = box_rows x 64
// elements (128 bytes), 128-byte swizzle, zero fill out of bounds.
bool encode_bf16_rows(CUtensorMap *map, const void *base, int64_t rows, int d, int box_rows) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return false;
    cuuint64_t dims[2] = {(cuuint64_t)d, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)d * 2};
    cuuint32_t box[2] = {(cuuint32_t)kTcTileK, (cuuint32_t)box_rows};
    cuuint32_t estr[2] = {1, 1};
    return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(base), dims, strides, box,
              estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// 2D bf16 tensor map over `cols` columns of a row-major matrix whose rows
// are `ld` elements apart (a column block of a wider matrix), box
// box_rows x 64 elements, 128-byte swizzle.
bool encode_bf16_block(CUtensorMap *map, const void *base, int64_t rows, int cols, int64_t ld, int box_rows) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return false;
    cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)ld * 2};
    cuuint32_t box[2] = {(cuuint32_t)kTcTileK, (cuuint32_t)box_rows};
    cuuint32_t estr[2] = {1, 1};
    return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(base), dims, strides, box, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// 2D byte tensor map over the e4m3 corpus [rows x d], box 256 rows x 128
// elements (128 bytes), 128-byte swizzle, zero fill out of bounds.
bool encode_e4m3_rows(CUtensorMap *map, const void *base, int64_t rows, int d, int box_rows = kTcTileN) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return false;
    cuuint64_t dims[2] = {(cuuint64_t)d, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)d};
    cuuint32_t box[2] = {128, (cuuint32_t)box_rows};
    cuuint32_t estr[2] = {1, 1};
    return fn(map, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<void *>(base), dims, strides, box, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

struct skip_corpus {
    int device = 0;
    int sm_count = 0;
    int max_smem = 0;          // opt-in shared memory per block
    int64_t N = 0;
    int d = 0;
    skip_dtype_t dtype = SKIP_BF16;
    void *rows = nullptr;      // device [N x d]
    float *scale = nullptr;    // device [N] (e4m3)
    int *err = nullptr;        // device error word
    CUtensorMap tmap_x;        // corpus rows, box 256 x 64 (bf16 only)
    bool tmap_ok = false;
    void *ws = nullptr;        // workspace
    size_t ws_bytes = 0;
    void *io = nullptr;        // device staging for skip_retrieve_host
    size_t io_bytes = 0;
    void *gws = nullptr;       // SKV gate workspace
    size_t gws_bytes = 0;
    int path = SKIP_PATH_AUTO;
    uint64_t timeout_ns = kDefaultTimeoutNs;
    int grid = 0;
    int mma = 0;               // 0 = pick, 1 = single-CTA MMA, 2 = CTA-pair MMA
    int bound = 0;             // bounding pass: 0 = by corpus size, 1 = never, 2 = always
    bool canary = false;       // guard bytes after the growable buffers (SKIP_OPT_CANARY)
    int resident = 0;          // resident query blocks: 0 by the rule, 1 never, 2 whenever possible
    std::map<int, int> cluster_cache;  // resident clusters per (size, stages, list place)
    int timing = 0;
    // Timing: events recorded on the launching stream before each kernel and
    // after the last one, kept across calls until skip_timing_report.
    std::vector<cudaEvent_t> ev_pool;
    std::vector<const char *> ev_name;
    std::vector<int> ev_call;
    size_t ev_used = 0;
    int call_id = 0;
    char plan[384] = "{}";
    // Second stream for work that needs no retrieval result (the SKV gate's
    // per-question bias), forked from and joined back to the caller's stream.
    cudaStream_t aux = nullptr;
    cudaEvent_t ev_fork = nullptr, ev_join = nullptr;
    int *cq_flag = nullptr;  // device: epoch of the last completed bias GEMM on aux
    int cq_epoch = 0;
    // Small-batch kernel thresholds, two sets of kLatMaxR: a call uses one
    // and its kernel clears the other for the next call (no clearing launch).
    uint32_t *lat_tau = nullptr;
    int lat_parity = 0;
};

namespace {

skip_status_t cuda_status(cudaError_t e) {
    if (e == cudaSuccess) return SKIP_OK;
    if (e == cudaErrorMemoryAllocation) return SKIP_ENOMEM;
    return SKIP_ECUDA;
}

// Every device allocation of the library goes through dev_alloc.  Host-side
// fault injection (no counterpart in the paper; it stands in for a device
// that runs out of memory, without touching the GPU): with the environment
// variable SKIP_FAULT_INJECT=alloc every allocation fails as cudaMalloc does
// when memory is exhausted, with SKIP_FAULT_INJECT=alloc:<kind> only the
// allocations of that kind (corpus, workspace, staging, gate, ivfpq, qvs,
// bsca).  The variable is read at each allocation.
cudaError_t dev_alloc(void **p, size_t bytes, const char *kind) {
    const char *e = getenv("SKIP_FAULT_INJECT");
    if (e && strncmp(e, "alloc", 5) == 0 && (e[5] == 0 || (e[5] == ':' && strcmp(e + 6, kind) == 0))) {
        *p = nullptr;
        return cudaErrorMemoryAllocation;
    }
    return cudaMalloc(p, bytes);
}

// Guard bytes after a handle's growable buffers (SKIP_OPT_CANARY): a kernel
// that writes past the end of its workspace changes them, and
// skip_sync_status reports it.
constexpr size_t kCanaryBytes = 4096;
constexpr unsigned char kCanaryByte = 0xA5;

// Grows a device buffer to at least `bytes` (25% headroom; none with
// guard bytes, which then follow the `bytes` usable ones); a buffer in use
// by queued work is freed only after the device has drained.  A failed
// allocation leaves the buffer empty, so the next call allocates again.
skip_status_t ensure_buf(void *&buf, size_t &have, size_t bytes, const char *kind, bool canary) {
    if (bytes <= have) return SKIP_OK;
    if (buf) {
        cudaError_t e = cudaDeviceSynchronize();
        if (e != cudaSuccess) return SKIP_ECUDA;
        cudaFree(buf);
        buf = nullptr;
        have = 0;
    }
    const size_t want = canary ? bytes : bytes + bytes / 4;
    if (dev_alloc(&buf, want + (canary ? kCanaryBytes : 0), kind) != cudaSuccess) {
        cudaGetLastError();
        buf = nullptr;
        return SKIP_ENOMEM;
    }
    if (canary && (cudaMemset((char *)buf + want, kCanaryByte, kCanaryBytes) != cudaSuccess ||
                   cudaDeviceSynchronize() != cudaSuccess)) {
        cudaFree(buf);
        buf = nullptr;
        return SKIP_ECUDA;
    }
    have = want;
    return SKIP_OK;
}

skip_status_t ensure_ws(skip_corpus *c, size_t bytes) {
    return ensure_buf(c->ws, c->ws_bytes, bytes, "workspace", c->canary);
}

// SKIP_OPT_CANARY: true when the guard bytes after every allocated
// growable buffer of the handle are intact.
bool canaries_intact(skip_corpus *c, bool *ok) {
    unsigned char h[kCanaryBytes];
    const std::pair<void *, size_t> bufs[3] = {{c->ws, c->ws_bytes}, {c->io, c->io_bytes}, {c->gws, c->gws_bytes}};
    *ok = true;
    for (const auto &b : bufs) {
        if (!b.first) continue;
        if (cudaMemcpy(h, (char *)b.first + b.second, kCanaryBytes, cudaMemcpyDeviceToHost) != cudaSuccess)
            return false;
        for (size_t i = 0; i < kCanaryBytes; ++i)
            if (h[i] != kCanaryByte) *ok = false;
    }
    return true;
}

void record(skip_corpus *c, cudaStream_t s, const char *name) {
    if (!c->timing || c->ev_used >= kMaxEvents) return;
    if (c->ev_used == c->ev_pool.size()) {
        cudaEvent_t e;
        if (cudaEventCreate(&e) != cudaSuccess) return;
        c->ev_pool.push_back(e);
        c->ev_name.push_back(nullptr);
        c->ev_call.push_back(0);
    }
    c->ev_name[c->ev_used] = name;
    c->ev_call[c->ev_used] = c->call_id;
    cudaEventRecord(c->ev_pool[c->ev_used], s);
    ++c->ev_used;
}

size_t align_up(size_t v, size_t a) { return (v + a - 1) / a * a; }

struct Plan {
    bool tensor = false;
    int grid = 0;
    int G = 0;          // lists per region row
    int MB = 0;
    int R_pad = 0;
    int64_t tiles = 0;
    int launches = 0;
    int stages = 0;
    bool list_in_smem = false;
    bool bound = false;  // bounding pass over a sample of corpus tiles first
    int CL = 1;
    bool pair = false;
    bool latency = false;
    bool resident = false;  // query blocks resident in shared memory (pair kernel)
};

// Corpus chunks G for the tensor path: make MB * G a whole number of waves of
// `ctas` while keeping at least 4 tiles per item where the corpus allows, and
// at least gmin chunks.
int pick_chunks(int MB, int64_t tiles, int ctas, int gmin = 1) {
    int best = std::max(1, std::min(gmin, 512));
    double best_eff = -1.0;
    // At least 4 tiles per item, unless that leaves most CTAs idle (a small
    // corpus, e.g. IVF centroids): then down to one tile per item.
    const int64_t per = (int64_t)MB * std::max<int64_t>(1, tiles / 4) < ctas ? 1 : 4;
    const int gmax = (int)std::min<int64_t>(512, std::max<int64_t>(best, tiles / per));
    for (int G = best; G <= gmax; ++G) {
        const int64_t items = (int64_t)MB * G;
        const int64_t waves = (items + ctas - 1) / ctas;
        const double eff = (double)items / (double)(waves * ctas);
        if (eff > best_eff + 1e-9) {
            best_eff = eff;
            best = G;
        }
        if (items >= 8LL * ctas) break;
    }
    return best;
}

skip_status_t check_common(skip_corpus *c, const void *regions, int32_t R_total, int32_t k_region) {
    if (!c || R_total < 0) return SKIP_EINVAL;
    if (R_total > 0 && !regions) return SKIP_EINVAL;
    if (k_region < 1 || k_region > SKIP_MAX_K_REGION || (int64_t)k_region > c->N) return SKIP_EINVAL;
    return SKIP_OK;
}

// Per-region step into reg_keys (or decoded ids/scores).  Shared by
// skip_retrieve and skip_retrieve_regions.
// When keys_out is non-null the keys go to the head of the workspace (the
// first ws_extra bytes) and *keys_out receives their address.
// The question merge that run_regions may do itself (small batches: one
// launch for both merges); `done` tells the caller whether it did.
struct QuestionMerge {
    const int32_t *offsets;
    int Q, K;
    int64_t *out_ids;
    float *out_scores;
    bool done = false;
    // called once the score kernel is queued (work that needs no retrieval
    // result and should not compete with that kernel for SMs)
    std::function<skip_status_t()> after_score;
};

skip_status_t run_regions(skip_corpus *c, const uint16_t *regions, int R, int k, uint64_t **keys_out,
                          int64_t *reg_ids, float *reg_scores, cudaStream_t s, Plan &pl,
                          size_t ws_extra, QuestionMerge *qm = nullptr) {
    uint64_t *reg_keys = nullptr;
    const bool e4m3 = c->dtype == SKIP_E4M3;
    const int ctas = c->grid > 0 ? c->grid : c->sm_count;
    bool tensor;
    if (c->path == SKIP_PATH_TENSOR)
        tensor = true;
    else if (c->path == SKIP_PATH_WARP)
        tensor = false;
    else
        tensor = e4m3 ? R > 4 : R > 8;
    if (!e4m3 && !c->tmap_ok) tensor = false;
    // Small batches: corpus tile as the streamed MMA operand, queries resident.
    int lat_npad = 0, lat_slices = 0, lat_stages = 0;
    const bool lat_fits = R <= kLatMaxR && lat_pick_layout(e4m3, R, c->d, k, c->max_smem, &lat_npad, &lat_slices,
                                                            &lat_stages);
    if (lat_fits && (c->path == SKIP_PATH_LATENCY || (c->path == SKIP_PATH_AUTO && tensor))) {
        pl.tensor = true;
        pl.latency = true;
        pl.tiles = (c->N + 127) / 128;
        pl.G = pick_chunks(1, pl.tiles, ctas);
        pl.grid = std::min(pl.G, ctas);
        pl.R_pad = R;
        pl.stages = lat_stages;
        pl.list_in_smem = true;
        const size_t parts_bytes = e4m3 ? align_up((size_t)96 * c->d, 256) : 0;
        const size_t qs_bytes = e4m3 ? align_up((size_t)3 * R * sizeof(float), 256) : 0;
        const size_t lists_bytes = (size_t)pl.G * R * k * sizeof(uint64_t);
        skip_status_t st = ensure_ws(c, align_up(ws_extra, 256) + parts_bytes + qs_bytes + lists_bytes);
        if (st) return st;
        if (!c->lat_tau) {
            if (dev_alloc(reinterpret_cast<void **>(&c->lat_tau), 2 * kLatMaxR * sizeof(uint32_t), "workspace") !=
                cudaSuccess) {
                cudaGetLastError();
                c->lat_tau = nullptr;
                return SKIP_ENOMEM;
            }
            if (cudaMemsetAsync(c->lat_tau, 0, 2 * kLatMaxR * sizeof(uint32_t), s) != cudaSuccess) return SKIP_ECUDA;
        }
        char *w = (char *)c->ws + align_up(ws_extra, 256);
        uint32_t *tau = c->lat_tau + c->lat_parity * kLatMaxR;
        uint8_t *parts = reinterpret_cast<uint8_t *>(w);
        float *qscale = reinterpret_cast<float *>(w + parts_bytes);
        uint64_t *lists = reinterpret_cast<uint64_t *>(w + parts_bytes + qs_bytes);
        if (keys_out) *keys_out = reg_keys = reinterpret_cast<uint64_t *>(c->ws);
        CUtensorMap ta, tb;
        if (e4m3) {
            record(c, s, "split_queries");
            cudaError_t e = launch_split_queries(regions, R, c->d, parts, qscale, s);
            if (e != cudaSuccess) return cuda_status(e);
            ++pl.launches;
            if (!encode_e4m3_rows(&ta, c->rows, c->N, c->d, 128) || !encode_e4m3_rows(&tb, parts, 96, c->d, 96))
                return SKIP_ECUDA;
        } else {
            if (!encode_bf16_rows(&ta, c->rows, c->N, c->d, 128) || !encode_bf16_rows(&tb, regions, R, c->d, lat_npad))
                return SKIP_ECUDA;
        }
        LatParams p;
        p.N = c->N;
        p.d = c->d;
        p.R = R;
        p.k = k;
        p.Npad = lat_npad;
        p.slices = lat_slices;
        p.stages = lat_stages;
        p.tiles = pl.tiles;
        p.G = pl.G;
        p.corpus_scale = c->scale;
        p.qscale = qscale;
        p.lists = lists;
        p.tau = tau;
        p.tau_clear = c->lat_tau + (1 - c->lat_parity) * kLatMaxR;
        p.err = c->err;
        p.timeout_ns = c->timeout_ns;
        record(c, s, e4m3 ? "score_topk_latency_e4m3" : "score_topk_latency");
        cudaError_t e = launch_latency(e4m3, ta, tb, p, pl.grid, s);
        if (e != cudaSuccess) return cuda_status(e);
        c->lat_parity ^= 1;
        ++pl.launches;
        if (qm && qm->after_score) {
            const skip_status_t hs = qm->after_score();
            if (hs) return hs;
        }
        // One block per question merges all its region rows: only while the
        // questions average at most 8 regions (one question of 32 regions,
        // merged by one block, took 28 us against 23 us for the two launches).
        if (qm && qm->Q > 0 && R <= 8 * qm->Q && (int64_t)R * k <= question_merge_capacity() &&
            qm->K <= question_merge_capacity() && pl.G <= 512) {
            record(c, s, "merge_regions_questions");
            e = launch_merge_regions_questions(lists, pl.G, (int64_t)R * k, R, k, qm->offsets, qm->Q, qm->K,
                                               qm->out_ids, qm->out_scores, c->err, s, true);
            if (e != cudaSuccess) return cuda_status(e);
            ++pl.launches;
            qm->done = true;
            return SKIP_OK;
        }
        record(c, s, "merge_lists");
        e = launch_merge_lists(lists, pl.G, (int64_t)R * k, R, k, reg_keys, reg_ids, reg_scores, s, true);
        if (e != cudaSuccess) return cuda_status(e);
        ++pl.launches;
        return SKIP_OK;
    }
    pl.tensor = tensor;
    if (tensor && e4m3) {
        // e4m3 corpus: single-CTA MMA on bf16-widened corpus tiles.
        pl.MB = (R + kTcTileM - 1) / kTcTileM;
        pl.tiles = (c->N + kTcTileN - 1) / kTcTileN;
        pl.R_pad = pl.MB * kTcTileM;
        pl.CL = 1;
        pl.G = pick_chunks(pl.MB, pl.tiles, ctas);
        const int items = pl.MB * pl.G;
        pl.grid = std::min(items, ctas);
        bool in_smem = false;
        int stages = 0, raw_stages = 0;
        tc_fp8_pick_layout(k, c->max_smem, &stages, &raw_stages, &in_smem);
        const size_t lists_bytes = (size_t)pl.G * pl.R_pad * k * sizeof(uint64_t);
        const size_t tau_bytes = align_up((size_t)pl.R_pad * sizeof(uint32_t), 256);
        skip_status_t st = ensure_ws(c, align_up(ws_extra, 256) + tau_bytes + lists_bytes);
        if (st) return st;
        uint32_t *tau = reinterpret_cast<uint32_t *>((char *)c->ws + align_up(ws_extra, 256));
        uint64_t *lists = reinterpret_cast<uint64_t *>((char *)tau + tau_bytes);
        if (keys_out) *keys_out = reg_keys = reinterpret_cast<uint64_t *>(c->ws);
        if (cudaMemsetAsync(tau, 0, tau_bytes, s) != cudaSuccess) return SKIP_ECUDA;
        CUtensorMap tq, traw;
        if (!encode_bf16_rows(&tq, regions, R, c->d, kTcTileM)) return SKIP_ECUDA;
        if (!encode_e4m3_rows(&traw, c->rows, c->N, c->d)) return SKIP_ECUDA;
        TcParams p;
        p.tile_stride = 1;
        p.share = 1;
        p.dense = 0;
        p.N = c->N;
        p.d = c->d;
        p.R = R;
        p.R_pad = pl.R_pad;
        p.k = k;
        p.MB = pl.MB;
        p.CL = 1;
        p.QG = pl.MB;
        p.G = pl.G;
        p.tiles = pl.tiles;
        p.lists = lists;
        p.tau = tau;
        p.err = c->err;
        p.timeout_ns = c->timeout_ns;
        p.stages = stages;
        p.raw_stages = raw_stages;
        p.list_in_smem = in_smem;
        p.a_res = 0;
        p.sched = nullptr;
        p.scale = c->scale;
        pl.stages = stages;
        pl.list_in_smem = in_smem;
        record(c, s, "score_topk_tc_e4m3");
        cudaError_t e = launch_tc_fp8(tq, traw, p, pl.grid, s);
        if (e != cudaSuccess) return cuda_status(e);
        ++pl.launches;
        if (qm && qm->after_score) {
            const skip_status_t hs = qm->after_score();
            if (hs) return hs;
        }
        record(c, s, "merge_lists");
        e = launch_merge_lists(lists, pl.G, (int64_t)pl.R_pad * k, R, k, reg_keys, reg_ids, reg_scores, s, true);
        if (e != cudaSuccess) return cuda_status(e);
        ++pl.launches;
        return SKIP_OK;
    }
    if (tensor) {
        pl.MB = (R + kTcTileM - 1) / kTcTileM;
        pl.tiles = (c->N + kTcTileN - 1) / kTcTileN;
        // MMA shape: CTA pairs (M = 256) whenever there are two query blocks
        // to pair, unless set by option.
        const bool pair = c->mma == 2 || (c->mma == 0 && pl.MB >= 2);
        bool in_smem = false;
        int stages = 0;
        tc_pick_layout(pair, k, c->max_smem, &stages, &in_smem);
        auto max_clusters = [&](int CL, int st, bool sm, int slices) {
            const int key = (pair ? 100000 : 0) + slices * 10000 + CL * 100 + st * 10 + (sm ? 1 : 0);
            auto hit = c->cluster_cache.find(key);
            if (hit == c->cluster_cache.end())
                hit = c->cluster_cache.emplace(key, tc_max_clusters(pair, CL, st, k, sm, slices)).first;
            return hit->second;
        };
        // A pair is a cluster of two CTAs; single-CTA MMA runs without
        // clusters, each CTA loading its own corpus tiles.
        const int cl_best = pair ? 2 : 1;
        const int ncl_best = max_clusters(cl_best, stages, in_smem, 0);
        if (ncl_best == 0) return SKIP_ECUDA;
        pl.CL = cl_best;
        const int QG = (pl.MB + cl_best - 1) / cl_best;
        const int ncl = std::max(1, std::min(ncl_best, ctas / cl_best));
        pl.R_pad = QG * cl_best * kTcTileM;
        // Items of at most kTcChunkTiles corpus tiles: the query groups that
        // read a chunk at the same time then all find it in L2 (a long chunk
        // lets them drift apart, and each re-reads it from HBM).
        pl.G = pick_chunks(QG, pl.tiles, ncl, (int)((pl.tiles + kTcChunkTiles - 1) / kTcChunkTiles));
        // the per-row thresholds, then the two launches' work-item counters
        const size_t tau_bytes = align_up((size_t)pl.R_pad * sizeof(uint32_t), 256) + 256;
        // Bounding pass: the same kernel over every kBoundStride-th corpus
        // tile first; the merged sample top-k of each row is k ids whose
        // scores (computed bit for bit as the full pass computes them) are at
        // least its k-th key, so that score bounds the row's k-th best over
        // the whole corpus from below and seeds the shared threshold.  The
        // full pass's epilogue then admits far fewer keys.
        // Each sample chunk keeps only its top k_s (about twice its share of
        // k) with no bound shared between chunks, so its epilogue stays cheap
        // on short streams; the k-th best of the union of the chunks' lists is
        // still k distinct rows' scores, hence still a bound.  The merge of
        // the short lists raises each row's threshold itself.
        // By default it runs where the full pass's epilogue would be busy: a
        // row's chunks admit about G k (1 + ln(N / (G k))) keys without a
        // bound (a running top-k over random order), and at one key per
        // thousand scores or more the inserts, not the MMA, set the pace
        // (clustered_1m: 3.4e-3, on; throughput_10m: 4e-4, off).
        const int64_t stiles = (pl.tiles + kBoundStride - 1) / kBoundStride;
        const double gk = (double)pl.G * k;
        const double ins_per_score = gk * (1.0 + std::log(std::max(1.0, (double)c->N / gk))) / (double)c->N;
        const bool bound = c->bound == 2 || (c->bound == 0 && pl.tiles >= kBoundMinTiles && ins_per_score >= 1e-3);
        // Sample chunks keep four keys per row in registers when there are at
        // least k / 2 of them (the k-th of the union of 2k keys or more);
        // with too few sample tiles for that, lists of about 2k / chunks.
        int chunks_s = bound ? pick_chunks(QG, stiles, ncl) : 0;
        if (bound && chunks_s * 4 < 2 * k && stiles >= (k + 1) / 2)
            chunks_s = pick_chunks(QG, stiles, ncl, (k + 1) / 2);
        const int k_s = bound ? std::min(k, std::max(4, (2 * k + chunks_s - 1) / chunks_s)) : 0;
        // Query blocks resident in shared memory (pairs, d <= 512): the sets
        // go to global memory, where the bounding pass keeps them short.
        int res_stages = (pair && bound && c->resident != 1) ? tc_pick_resident_stages(c->d, c->max_smem) : 0;
        const int res_slices = res_stages > 0 ? (c->d + kTcTileK - 1) / kTcTileK : 0;
        if (res_stages > 0 && max_clusters(cl_best, res_stages, false, res_slices) < ncl) res_stages = 0;
        if (res_stages > 0) {
            // The sets then live in global memory, where a full set costs a
            // rescan from L2 and a long one a slow sort; keep the keys an
            // item admits few: the sample's k-th score is about the
            // (kBoundStride k)-th best of the corpus, so an item of T tiles
            // holds about kBoundStride k T / tiles keys above it.  Items of
            // at most 16 such keys, and of at least 64 tiles (else the
            // per-item cost of loading the query block shows).
            const int64_t t_keys = (int64_t)(16.0 * (double)pl.tiles / ((double)kBoundStride * k));
            int64_t gmin = (pl.tiles + std::max<int64_t>(1, std::min<int64_t>(kTcChunkTiles, t_keys)) - 1) /
                           std::max<int64_t>(1, std::min<int64_t>(kTcChunkTiles, t_keys));
            gmin = std::min<int64_t>(gmin, 512);
            if (c->resident == 2) {  // forced: items as for shared-memory sets
                stages = res_stages;
                in_smem = false;
            } else if ((pl.tiles + gmin - 1) / gmin < 64 || t_keys < 1) {
                res_stages = 0;
            } else {
                pl.G = pick_chunks(QG, pl.tiles, ncl, (int)gmin);
                stages = res_stages;
                in_smem = false;
            }
        }
        const int items = QG * pl.G;
        pl.grid = std::min(items, ncl) * cl_best;
        const size_t lists_bytes = (size_t)pl.G * pl.R_pad * k * sizeof(uint64_t);
        const size_t lists_s_bytes = align_up((size_t)chunks_s * pl.R_pad * k_s * sizeof(uint64_t), 256);
        skip_status_t st = ensure_ws(c, align_up(ws_extra, 256) + tau_bytes + align_up(lists_bytes, 256) +
                                            lists_s_bytes);
        if (st) return st;
        uint32_t *tau = reinterpret_cast<uint32_t *>((char *)c->ws + align_up(ws_extra, 256));
        uint64_t *lists = reinterpret_cast<uint64_t *>((char *)tau + tau_bytes);
        uint64_t *lists_s = reinterpret_cast<uint64_t *>((char *)lists + align_up(lists_bytes, 256));
        if (keys_out) *keys_out = reg_keys = reinterpret_cast<uint64_t *>(c->ws);
        if (cudaMemsetAsync(tau, 0, tau_bytes, s) != cudaSuccess) return SKIP_ECUDA;
        CUtensorMap tq, tx;
        if (!encode_bf16_rows(&tq, regions, R, c->d, kTcTileM)) return SKIP_ECUDA;
        if (!encode_bf16_rows(&tx, c->rows, c->N, c->d, pair ? kTcTileN / 2 : kTcTileN / cl_best))
            return SKIP_ECUDA;
        TcParams p;
        p.tile_stride = 1;
        p.share = 1;
        p.dense = 0;
        p.N = c->N;
        p.d = c->d;
        p.R = R;
        p.R_pad = pl.R_pad;
        p.k = k;
        p.MB = pl.MB;
        p.CL = pl.CL;
        p.QG = QG;
        p.G = pl.G;
        p.tiles = pl.tiles;
        p.lists = lists;
        p.tau = tau;
        p.err = c->err;
        p.timeout_ns = c->timeout_ns;
        p.stages = stages;
        p.list_in_smem = in_smem;
        p.scale = nullptr;
        p.raw_stages = 0;
        p.tile_stride = 1;
        p.a_res = res_stages > 0 ? 1 : 0;
        int *counters = reinterpret_cast<int *>((char *)tau + tau_bytes - 256);
        p.sched = counters;
        pl.stages = p.stages;
        pl.list_in_smem = in_smem;
        pl.pair = pair;
        pl.bound = bound;
        pl.resident = res_stages > 0;
        cudaError_t e;
        if (bound) {
            TcParams ps = p;
            ps.sched = counters + 1;
            ps.tiles = stiles;
            ps.tile_stride = kBoundStride;
            ps.G = chunks_s;
            ps.lists = lists_s;
            ps.k = k_s;
            ps.share = 0;
            ps.dense = k_s == 4;
            int st_s = 0;
            bool smem_s = false;
            tc_pick_layout(pair, k_s, c->max_smem, &st_s, &smem_s);
            if (res_stages > 0 && ps.dense) {
                st_s = res_stages;  // the four keys live in registers: no sets at all
                smem_s = false;
            } else {
                ps.a_res = 0;
            }
            ps.stages = st_s;
            ps.list_in_smem = smem_s;
            record(c, s, "score_topk_tc_bound");
            e = launch_tc(pair, tq, tx, ps, std::min(QG * chunks_s, ncl) * cl_best, s);
            if (e != cudaSuccess) return cuda_status(e);
            record(c, s, "merge_bound");
            e = launch_merge_lists_len(lists_s, chunks_s, (int64_t)pl.R_pad * k_s, k_s, R, k, nullptr, nullptr,
                                       nullptr, tau, s, true);
            if (e != cudaSuccess) return cuda_status(e);
            pl.launches += 2;
        }
        record(c, s, "score_topk_tc");
        e = launch_tc(pair, tq, tx, p, pl.grid, s, bound);
        if (e != cudaSuccess) return cuda_status(e);
        ++pl.launches;
        if (qm && qm->after_score) {
            const skip_status_t hs = qm->after_score();
            if (hs) return hs;
        }
        record(c, s, "merge_lists");
        e = launch_merge_lists(lists, pl.G, (int64_t)pl.R_pad * k, R, k, reg_keys, reg_ids, reg_scores, s, true);
        if (e != cudaSuccess) return cuda_status(e);
        ++pl.launches;
        return SKIP_OK;
    }
    // Warp-dot path: groups of up to 8 queries per launch.
    pl.grid = (int)std::min<int64_t>(std::min<int64_t>((int64_t)ctas * 2, 512),
                                     std::max<int64_t>(1, (c->N + 255) / 256));
    pl.G = pl.grid;
    pl.R_pad = R;
    const size_t lists_bytes = (size_t)pl.grid * R * k * sizeof(uint64_t);
    const size_t wl_bytes = (size_t)pl.grid * kWarpDotWarps * 8 * k * sizeof(uint64_t);
    skip_status_t st = ensure_ws(c, align_up(ws_extra, 256) + align_up(lists_bytes, 256) + wl_bytes);
    if (st) return st;
    uint64_t *lists = reinterpret_cast<uint64_t *>((char *)c->ws + align_up(ws_extra, 256));
    uint64_t *wl = reinterpret_cast<uint64_t *>((char *)lists + align_up(lists_bytes, 256));
    if (keys_out) *keys_out = reg_keys = reinterpret_cast<uint64_t *>(c->ws);
    record(c, s, "score_topk_warpdot");
    for (int q0 = 0; q0 < R; q0 += 8) {
        WarpDotParams p;
        p.corpus = reinterpret_cast<const uint8_t *>(c->rows);
        p.scale = c->scale;
        p.N = c->N;
        p.d = c->d;
        p.regions = regions + (size_t)q0 * c->d;
        p.nq = std::min(8, R - q0);
        p.k = k;
        p.warp_lists = wl;
        p.lists = lists;
        p.list_g_stride = (int64_t)R * k;
        p.q0 = q0;
        cudaError_t e = launch_warpdot(p, e4m3, pl.grid, s);
        if (e != cudaSuccess) return cuda_status(e);
        ++pl.launches;
    }
    if (qm && qm->after_score) {
        const skip_status_t hs = qm->after_score();
        if (hs) return hs;
    }
    record(c, s, "merge_lists");
    cudaError_t e = launch_merge_lists(lists, pl.G, (int64_t)R * k, R, k, reg_keys, reg_ids, reg_scores, s, true);
    if (e != cudaSuccess) return cuda_status(e);
    ++pl.launches;
    return SKIP_OK;
}

void write_plan(skip_corpus *c, const Plan &pl, int R, int Q, int k, int K) {
    snprintf(c->plan, sizeof c->plan,
             "{\"path\": \"%s\", \"grid\": %d, \"lists_per_row\": %d, \"query_blocks\": %d, "
             "\"R_total\": %d, \"Q\": %d, \"k_region\": %d, \"K\": %d, \"launches\": %d, "
             "\"stages\": %d, \"cluster\": %d, \"mma\": \"%s\", \"lists\": \"%s\", \"bound\": %d, "
             "\"resident_queries\": %d}",
             pl.latency ? "latency" : pl.tensor ? "tensor" : "warpdot", pl.grid, pl.G, pl.MB, R, Q, k, K, pl.launches,
             pl.stages, pl.CL,
             pl.pair ? "pair" : "single",
             pl.tensor ? (pl.list_in_smem ? "shared" : "global") : "global", pl.bound ? 1 : 0, pl.resident ? 1 : 0);
}

// Argument rules of skip_retrieve.
skip_status_t check_retrieve(skip_corpus *c, const void *regions, const int32_t *region_offsets, int32_t Q,
                             int32_t R_total, int32_t k_region, int32_t K) {
    skip_status_t st = check_common(c, regions, R_total, k_region);
    if (st) return st;
    if (Q < 0 || K < 1 || K > SKIP_MAX_K || (Q > 0 && !region_offsets)) return SKIP_EINVAL;
    if (Q == 0 && R_total != 0) return SKIP_EINVAL;
    return SKIP_OK;
}

// Per-region step, then the per-question merge into out_ids / out_scores.
skip_status_t retrieve_impl(skip_corpus *c, const void *regions, const int32_t *region_offsets, int32_t Q,
                            int32_t R_total, int32_t k_region, int32_t K, int64_t *out_ids, float *out_scores,
                            cudaStream_t s, Plan &pl, std::function<skip_status_t()> after_score = nullptr) {
    const size_t keys_bytes = align_up((size_t)std::max(R_total, 1) * k_region * sizeof(uint64_t), 256);
    uint64_t *reg_keys = nullptr;
    skip_status_t st;
    QuestionMerge qm;
    qm.offsets = region_offsets;
    qm.Q = Q;
    qm.K = K;
    qm.out_ids = out_ids;
    qm.out_scores = out_scores;
    qm.after_score = std::move(after_score);
    if (R_total > 0) {
        st = run_regions(c, reinterpret_cast<const uint16_t *>(regions), R_total, k_region, &reg_keys,
                         nullptr, nullptr, s, pl, keys_bytes, &qm);
        if (st) return st;
    } else {
        st = ensure_ws(c, keys_bytes);
        if (st) return st;
        reg_keys = reinterpret_cast<uint64_t *>(c->ws);
    }
    if (Q > 0 && !qm.done) {
        record(c, s, "question_merge");
        cudaError_t e = launch_question_merge(reg_keys, k_region, region_offsets, Q, R_total, K, out_ids,
                                              out_scores, c->err, s, R_total > 0);
        if (e != cudaSuccess) return cuda_status(e);
        ++pl.launches;
    }
    return SKIP_OK;
}

// Argument rules of the SKV gate (the corpus handle is already checked).
skip_status_t check_skv(skip_corpus *c, int32_t Q, int32_t K, const uint16_t *qbar, const uint16_t *vbar,
                        const skip_skv_mlp_t *mlp, float tau, float rho, const void *out_ids, const void *out_nu,
                        const void *out_count) {
    if (Q < 0 || K < 1 || K > SKIP_MAX_K || !mlp) return SKIP_EINVAL;
    if (!(tau == tau) || !(rho >= 0.f && rho <= 1.f)) return SKIP_EINVAL;
    if (mlp->hidden < kSkvHidden || mlp->hidden % kSkvHidden != 0 || !mlp->w1 || !mlp->b1 || !mlp->w2)
        return SKIP_EINVAL;
    if (Q > 0 && (!qbar || !vbar || !out_ids || !out_nu || !out_count)) return SKIP_EINVAL;
    // qbar, vbar and W1 are read by TMA and as 16-byte vectors
    if ((((uintptr_t)qbar | (uintptr_t)vbar | (uintptr_t)mlp->w1) & 15) != 0) return SKIP_EINVAL;
    if (c->dtype != SKIP_BF16 || c->d % 64 != 0 || c->d > 1024) return SKIP_EUNSUPPORTED;
    return SKIP_OK;
}

// Partial-logit slabs of the MLP: at most H / 32 (128 units a pair, two K
// parts, two column halves).
size_t skv_ws_bytes(int Q, int K, int H, int d) {
    const size_t P = (size_t)Q * K;
    return align_up((size_t)kSkvCqSplits * Q * H * 4, 256) + align_up((size_t)(H / 32) * P * 4, 256) +
           align_up(P * 3 * (size_t)d * 2, 256);
}

// The per-question bias c_q = b1 + W1[:, 0:d] qbar + W1[:, d:2d] vbar of every
// question: one GEMM over the two column blocks of W1, K split over up to
// kSkvCqSplits CTAs per tile (k_skv_mlp sums the slabs), into the head of
// gws.  It needs no retrieval result: in skip_retrieve_skv it runs on the
// handle's second stream, forked from s once the score kernel is queued (so
// that it overlaps the merge kernels, which leave most SMs idle); a flag it
// raises afterwards (a per-call epoch) tells the MLP kernel that c_q is
// complete, and the second stream is joined back into s after the gate's
// last kernel, so that no event wait sits between the retrieval and the
// gate.  Otherwise (no retrieval, or per-kernel timing on) it runs on s
// before the gate.
struct CqLaunch {
    CUtensorMap ta, tb, ta2, tb2;
    int tn = 0, Q = 0, H = 0, splits = 1;
    const float *b1 = nullptr;
    bool launched = false, forked = false;
    int epoch = 0;
};
skip_status_t skv_prepare_cq(skip_corpus *c, int32_t Q, const uint16_t *qbar, const uint16_t *vbar,
                             const skip_skv_mlp_t *mlp, CqLaunch &cl) {
    if (Q == 0) return SKIP_OK;
    cl.Q = Q;
    cl.H = mlp->hidden;
    cl.b1 = mlp->b1;
    cl.tn = gemm_tile_n(Q, cl.H, c->sm_count);
    cl.splits = std::min(kSkvCqSplits, gemm_splits(Q, cl.H, 2 * c->d, cl.tn, c->sm_count));
    if (!encode_bf16_rows(&cl.ta, qbar, Q, c->d, 128) || !encode_bf16_rows(&cl.ta2, vbar, Q, c->d, 128) ||
        !encode_bf16_block(&cl.tb, mlp->w1, cl.H, c->d, 5 * (int64_t)c->d, cl.tn) ||
        !encode_bf16_block(&cl.tb2, mlp->w1 + c->d, cl.H, c->d, 5 * (int64_t)c->d, cl.tn))
        return SKIP_ECUDA;
    return SKIP_OK;
}

// Launches the c_q GEMM: forked onto the handle's second stream after the
// work queued on s so far, or on s itself.
skip_status_t skv_launch_cq(skip_corpus *c, CqLaunch &cl, cudaStream_t s, bool fork) {
    if (cl.Q == 0 || cl.launched) return SKIP_OK;
    cudaStream_t g = s;
    if (fork) {
        if (!c->aux) {
            if (cudaStreamCreateWithFlags(&c->aux, cudaStreamNonBlocking) != cudaSuccess ||
                cudaEventCreateWithFlags(&c->ev_fork, cudaEventDisableTiming) != cudaSuccess ||
                cudaEventCreateWithFlags(&c->ev_join, cudaEventDisableTiming) != cudaSuccess) {
                cudaGetLastError();
                return SKIP_ECUDA;
            }
        }
        if (!c->cq_flag) {
            if (dev_alloc(reinterpret_cast<void **>(&c->cq_flag), 16, "gate") != cudaSuccess) {
                cudaGetLastError();
                c->cq_flag = nullptr;
                return SKIP_ENOMEM;
            }
            if (cudaMemsetAsync(c->cq_flag, 0, 16, s) != cudaSuccess) return SKIP_ECUDA;
        }
        if (cudaEventRecord(c->ev_fork, s) != cudaSuccess || cudaStreamWaitEvent(c->aux, c->ev_fork, 0) != cudaSuccess)
            return SKIP_ECUDA;
        g = c->aux;
    } else {
        record(c, s, "skv_qbias");
    }
    cudaError_t e = launch_gemm2_bf16_f32(cl.ta, cl.tb, &cl.ta2, &cl.tb2, cl.tn, cl.Q, cl.H, c->d, c->d, 1.f, cl.b1,
                                          reinterpret_cast<float *>(c->gws), cl.H, c->err, c->timeout_ns, g,
                                          cl.splits, (int64_t)cl.Q * cl.H);
    if (e != cudaSuccess) return cuda_status(e);
    if (fork) {
        c->cq_epoch = c->cq_epoch == 0x7fffffff ? 1 : c->cq_epoch + 1;
        cl.epoch = c->cq_epoch;
        if ((e = launch_skv_cq_ready(c->cq_flag, cl.epoch, c->aux)) != cudaSuccess) return cuda_status(e);
        if (cudaEventRecord(c->ev_join, c->aux) != cudaSuccess) return SKIP_ECUDA;
    }
    cl.launched = true;
    cl.forked = fork;
    return SKIP_OK;
}

// The gate on cand_ids (c_q prepared by skv_prepare_cq, launched here if it
// has not been); its workspace is the head of gws (skv_ws_bytes).
skip_status_t skv_impl(skip_corpus *c, const int64_t *cand_ids, int32_t Q, int32_t K, const uint16_t *qbar,
                       const uint16_t *vbar, const skip_skv_mlp_t *mlp, float tau, float rho, int64_t *out_ids,
                       float *out_nu, int32_t *out_count, float *nu_all, CqLaunch &cl, cudaStream_t s,
                       Plan &pl) {
    if (Q == 0) return SKIP_OK;
    skip_status_t st = skv_launch_cq(c, cl, s, false);
    if (st) return st;
    const int H = mlp->hidden;
    SkvParams p;
    p.rows = reinterpret_cast<const uint16_t *>(c->rows);
    p.N = c->N;
    p.d = c->d;
    p.ids = cand_ids;
    p.P = (int64_t)Q * K;
    p.K = K;
    p.Q = Q;
    p.qbar = qbar;
    p.vbar = vbar;
    p.w1 = mlp->w1;
    p.b1 = mlp->b1;
    p.w2 = mlp->w2;
    p.b2 = mlp->b2;
    p.H = H;
    p.tau = tau;
    p.rho = rho;
    p.cq = reinterpret_cast<float *>(c->gws);
    p.cq_splits = cl.splits;
    p.cq_flag = cl.forked ? c->cq_flag : nullptr;
    p.cq_epoch = cl.epoch;
    p.partial = reinterpret_cast<float *>((char *)c->gws + align_up((size_t)kSkvCqSplits * Q * H * 4, 256));
    uint16_t *F = reinterpret_cast<uint16_t *>((char *)p.partial + align_up((size_t)(H / 32) * p.P * 4, 256));
    p.out_ids = out_ids;
    p.out_nu = out_nu;
    p.out_count = out_count;
    p.nu_all = nu_all;
    p.err = c->err;
    p.timeout_ns = c->timeout_ns;
    int BN = 0, S = 0;
    skv_mlp_shape(p.P, H, &BN, &S);
    p.nparts = H / BN * S * 2;
    CUtensorMap tf, tw;
    if (!encode_bf16_rows(&tf, F, p.P, 3 * c->d, 128) || !encode_bf16_rows(&tw, mlp->w1, H, 5 * c->d, BN / 2))
        return SKIP_ECUDA;
    record(c, s, "skv_features");
    cudaError_t e = launch_skv_features(p, F, s);
    if (e != cudaSuccess) return cuda_status(e);
    record(c, s, "skv_mlp");
    e = launch_skv_mlp(tf, tw, p, BN, S, s);
    if (e != cudaSuccess) return cuda_status(e);
    record(c, s, "skv_select");
    e = launch_skv_select(p, s);
    if (e != cudaSuccess) return cuda_status(e);
    pl.launches += cl.forked ? 5 : 4;  // the GEMM (and its ready flag), features, MLP, selection
    // the second stream joins s again (its GEMM is long done by now)
    if (cl.forked && cudaStreamWaitEvent(s, c->ev_join, 0) != cudaSuccess) return SKIP_ECUDA;
    return SKIP_OK;
}

}  // namespace

extern "C" {

const char *skip_status_string(skip_status_t s) {
    switch (s) {
        case SKIP_OK: return "ok";
        case SKIP_EINVAL: return "invalid argument";
        case SKIP_ENOMEM: return "out of device memory";
        case SKIP_EUNSUPPORTED: return "unsupported device or size";
        case SKIP_ETIMEOUT: return "a kernel wait timed out";
        case SKIP_ECUDA: return "CUDA error";
        case SKIP_ECANARY: return "guard bytes after a library buffer were overwritten";
    }
    return "unknown status";
}

skip_status_t skip_corpus_load(const void *rows, int rows_on_device, int64_t N, int32_t d,
                               skip_dtype_t dtype, const float *row_scale, void *stream,
                               skip_corpus_t *out) {
    if (!out || !rows || N < 1 || N >= (1LL << 31) || d < 16 || d % 16 != 0 || d > kMaxD)
        return SKIP_EINVAL;
    if (dtype != SKIP_BF16 && dtype != SKIP_E4M3) return SKIP_EINVAL;
    if ((dtype == SKIP_E4M3) != (row_scale != nullptr)) return SKIP_EINVAL;
    *out = nullptr;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) {
        cudaGetLastError();
        return SKIP_EUNSUPPORTED;
    }
    int major = 0, minor = 0, sms = 0;
    cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
    cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    int max_smem = 0;
    cudaDeviceGetAttribute(&max_smem, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
    if (major != 10 || minor != 3) return SKIP_EUNSUPPORTED;

    skip_corpus *c = new (std::nothrow) skip_corpus();
    if (!c) return SKIP_ENOMEM;
    c->device = dev;
    c->sm_count = sms;
    c->max_smem = max_smem;
    c->N = N;
    c->d = d;
    c->dtype = dtype;
    const size_t elem = dtype == SKIP_BF16 ? 2 : 1;
    const size_t bytes = (size_t)N * d * elem;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    skip_status_t st = SKIP_OK;
    if (dev_alloc(&c->rows, bytes, "corpus") != cudaSuccess ||
        dev_alloc((void **)&c->err, sizeof(int), "corpus") != cudaSuccess ||
        (dtype == SKIP_E4M3 && dev_alloc((void **)&c->scale, N * sizeof(float), "corpus") != cudaSuccess)) {
        cudaGetLastError();
        st = SKIP_ENOMEM;
    }
    const cudaMemcpyKind kind = rows_on_device ? cudaMemcpyDeviceToDevice : cudaMemcpyHostToDevice;
    if (!st) st = cuda_status(cudaMemcpyAsync(c->rows, rows, bytes, kind, s));
    if (!st && c->scale) st = cuda_status(cudaMemcpyAsync(c->scale, row_scale, N * sizeof(float), kind, s));
    if (!st) st = cuda_status(cudaMemsetAsync(c->err, 0, sizeof(int), s));
    if (!st) st = cuda_status(cudaStreamSynchronize(s));
    if (!st && dtype == SKIP_BF16) c->tmap_ok = encode_bf16_rows(&c->tmap_x, c->rows, N, d, kTcTileN);
    if (st) {
        skip_corpus_free(c);
        return st;
    }
    *out = c;
    return SKIP_OK;
}

skip_status_t skip_corpus_free(skip_corpus_t c) {
    if (!c) return SKIP_OK;
    cudaDeviceSynchronize();
    cudaFree(c->rows);
    cudaFree(c->scale);
    cudaFree(c->err);
    cudaFree(c->ws);
    cudaFree(c->io);
    cudaFree(c->gws);
    for (cudaEvent_t e : c->ev_pool) cudaEventDestroy(e);
    if (c->ev_fork) cudaEventDestroy(c->ev_fork);
    if (c->ev_join) cudaEventDestroy(c->ev_join);
    if (c->aux) cudaStreamDestroy(c->aux);
    cudaFree(c->cq_flag);
    cudaFree(c->lat_tau);
    delete c;
    return SKIP_OK;
}

skip_status_t skip_corpus_set_option(skip_corpus_t c, int option, int64_t value) {
    if (!c) return SKIP_EINVAL;
    switch (option) {
        case SKIP_OPT_PATH:
            if (value < SKIP_PATH_AUTO || value > SKIP_PATH_LATENCY) return SKIP_EINVAL;
            c->path = (int)value;
            return SKIP_OK;
        case SKIP_OPT_WAIT_TIMEOUT_NS:
            if (value < 0) return SKIP_EINVAL;
            c->timeout_ns = (uint64_t)value;
            return SKIP_OK;
        case SKIP_OPT_GRID:
            if (value < 0 || value > 65535) return SKIP_EINVAL;
            c->grid = (int)value;
            return SKIP_OK;
        case SKIP_OPT_TIMING:
            c->timing = value != 0;
            return SKIP_OK;
        case SKIP_OPT_MMA:
            if (value < 0 || value > 2) return SKIP_EINVAL;
            c->mma = (int)value;
            return SKIP_OK;
        case SKIP_OPT_CLUSTER:
            // Kept for the ABI: single-CTA tensor launches use no clusters.
            if (value != 0 && value != 1) return SKIP_EINVAL;
            return SKIP_OK;
        case SKIP_OPT_BOUND:
            if (value < 0 || value > 2) return SKIP_EINVAL;
            c->bound = (int)value;
            return SKIP_OK;
        case SKIP_OPT_RESIDENT:
            if (value < 0 || value > 2) return SKIP_EINVAL;
            c->resident = (int)value;
            return SKIP_OK;
        case SKIP_OPT_CANARY:
            if (value != 0 && value != 1) return SKIP_EINVAL;
            if ((value != 0) != c->canary) {
                // The growable buffers are allocated again in the new mode.
                if (cudaDeviceSynchronize() != cudaSuccess) return SKIP_ECUDA;
                cudaFree(c->ws);
                cudaFree(c->io);
                cudaFree(c->gws);
                c->ws = c->io = c->gws = nullptr;
                c->ws_bytes = c->io_bytes = c->gws_bytes = 0;
                c->canary = value != 0;
            }
            return SKIP_OK;
    }
    return SKIP_EINVAL;
}

skip_status_t skip_retrieve(skip_corpus_t c, const void *regions, const int32_t *region_offsets,
                            int32_t Q, int32_t R_total, int32_t k_region, int32_t K, int64_t *out_ids,
                            float *out_scores, void *stream) {
    skip_status_t st = check_retrieve(c, regions, region_offsets, Q, R_total, k_region, K);
    if (st) return st;
    if (Q > 0 && (!out_ids || !out_scores)) return SKIP_EINVAL;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    ++c->call_id;
    Plan pl;
    st = retrieve_impl(c, regions, region_offsets, Q, R_total, k_region, K, out_ids, out_scores, s, pl);
    if (st) return st;
    record(c, s, "end");
    write_plan(c, pl, R_total, Q, k_region, K);
    return SKIP_OK;
}

skip_status_t skip_retrieve_regions(skip_corpus_t c, const void *regions, int32_t R_total,
                                    int32_t k_region, int64_t *reg_ids, float *reg_scores,
                                    void *stream) {
    skip_status_t st = check_common(c, regions, R_total, k_region);
    if (st) return st;
    if (R_total > 0 && (!reg_ids || !reg_scores)) return SKIP_EINVAL;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    ++c->call_id;
    Plan pl;
    if (R_total > 0) {
        st = run_regions(c, reinterpret_cast<const uint16_t *>(regions), R_total, k_region, nullptr, reg_ids,
                         reg_scores, s, pl, 0);
        if (st) return st;
    }
    record(c, s, "end");
    write_plan(c, pl, R_total, 0, k_region, 0);
    return SKIP_OK;
}

skip_status_t skip_sync_status(skip_corpus_t c, void *stream) {
    if (!c) return SKIP_EINVAL;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    if (cudaStreamSynchronize(s) != cudaSuccess) return SKIP_ECUDA;
    int err = 0;
    if (cudaMemcpy(&err, c->err, sizeof(int), cudaMemcpyDeviceToHost) != cudaSuccess) return SKIP_ECUDA;
    if (err) {
        if (cudaMemset(c->err, 0, sizeof(int)) != cudaSuccess) return SKIP_ECUDA;
        return (err & kErrTimeout) ? SKIP_ETIMEOUT : SKIP_EINVAL;
    }
    if (c->canary) {
        bool ok = true;
        if (!canaries_intact(c, &ok)) return SKIP_ECUDA;
        if (!ok) return SKIP_ECANARY;
    }
    return SKIP_OK;
}

skip_status_t skip_retrieve_host(skip_corpus_t c, const uint16_t *regions, const int32_t *region_offsets,
                                 int32_t Q, int32_t R_total, int32_t k_region, int32_t K, int64_t *out_ids,
                                 float *out_scores, void *stream) {
    skip_status_t st = check_common(c, regions, R_total, k_region);
    if (st) return st;
    if (Q < 0 || K < 1 || K > SKIP_MAX_K || (Q > 0 && (!region_offsets || !out_ids || !out_scores)))
        return SKIP_EINVAL;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    const size_t rb = align_up((size_t)R_total * c->d * 2, 256);
    const size_t ob = align_up((size_t)(Q + 1) * sizeof(int32_t), 256);
    const size_t ib = align_up((size_t)Q * K * sizeof(int64_t), 256);
    const size_t sb = align_up((size_t)Q * K * sizeof(float), 256);
    const size_t need = rb + ob + ib + sb;
    st = ensure_buf(c->io, c->io_bytes, need, "staging", c->canary);
    if (st) return st;
    char *io = reinterpret_cast<char *>(c->io);
    void *d_reg = io;
    int32_t *d_off = reinterpret_cast<int32_t *>(io + rb);
    int64_t *d_ids = reinterpret_cast<int64_t *>(io + rb + ob);
    float *d_sc = reinterpret_cast<float *>(io + rb + ob + ib);
    if (R_total > 0) {
        st = cuda_status(cudaMemcpyAsync(d_reg, regions, (size_t)R_total * c->d * 2, cudaMemcpyHostToDevice, s));
        if (st) return st;
    }
    if (Q > 0) {
        st = cuda_status(cudaMemcpyAsync(d_off, region_offsets, (size_t)(Q + 1) * sizeof(int32_t),
                                         cudaMemcpyHostToDevice, s));
        if (st) return st;
    }
    st = skip_retrieve(c, R_total > 0 ? d_reg : nullptr, d_off, Q, R_total, k_region, K, d_ids, d_sc, stream);
    if (st) return st;
    if (Q > 0) {
        st = cuda_status(cudaMemcpyAsync(out_ids, d_ids, (size_t)Q * K * sizeof(int64_t), cudaMemcpyDeviceToHost, s));
        if (!st)
            st = cuda_status(cudaMemcpyAsync(out_scores, d_sc, (size_t)Q * K * sizeof(float), cudaMemcpyDeviceToHost, s));
        if (st) return st;
    }
    return skip_sync_status(c, stream);
}

skip_status_t skip_last_plan(skip_corpus_t c, char *buf, int32_t len) {
    if (!c || !buf || len < 1) return SKIP_EINVAL;
    std::string times;
    if (c->timing && c->ev_used > 1) {
        bool first = true;
        for (size_t i = 0; i + 1 < c->ev_used; ++i) {
            if (c->ev_call[i] != c->call_id || c->ev_call[i + 1] != c->call_id) continue;
            float ms = 0.0f;
            if (cudaEventSynchronize(c->ev_pool[i + 1]) != cudaSuccess ||
                cudaEventElapsedTime(&ms, c->ev_pool[i], c->ev_pool[i + 1]) != cudaSuccess)
                return SKIP_ECUDA;
            char item[96];
            snprintf(item, sizeof item, "%s\"%s\": %.6f", first ? "" : ", ", c->ev_name[i], ms);
            times += item;
            first = false;
        }
        times = ", \"ms\": {" + times + "}";
    }
    const int plen = (int)strlen(c->plan);
    snprintf(buf, len, "%.*s%s}", plen > 0 ? plen - 1 : 0, c->plan, times.c_str());
    return SKIP_OK;
}

skip_status_t skip_timing_report(skip_corpus_t c, char *buf, int32_t len) {
    if (!c || !buf || len < 1) return SKIP_EINVAL;
    std::map<std::string, std::pair<int64_t, double>> acc;
    if (c->ev_used > 0 && cudaEventSynchronize(c->ev_pool[c->ev_used - 1]) != cudaSuccess) return SKIP_ECUDA;
    for (size_t i = 0; i + 1 < c->ev_used; ++i) {
        if (c->ev_call[i] != c->ev_call[i + 1]) continue;
        float ms = 0.0f;
        if (cudaEventElapsedTime(&ms, c->ev_pool[i], c->ev_pool[i + 1]) != cudaSuccess) return SKIP_ECUDA;
        auto &a = acc[c->ev_name[i]];
        a.first += 1;
        a.second += ms;
    }
    c->ev_used = 0;
    std::string out = "{";
    bool first = true;
    for (auto &kv : acc) {
        char item[160];
        snprintf(item, sizeof item, "%s\"%s\": {\"launches\": %lld, \"ms\": %.6f}", first ? "" : ", ",
                 kv.first.c_str(), (long long)kv.second.first, kv.second.second);
        out += item;
        first = false;
    }
    out += "}";
    if ((int)out.size() + 1 > len) return SKIP_EINVAL;
    memcpy(buf, out.c_str(), out.size() + 1);
    return SKIP_OK;
}

}  // extern "C"

extern "C" {

skip_status_t skip_skv_gate(skip_corpus_t c, const int64_t *cand_ids, int32_t Q, int32_t K, const uint16_t *qbar,
                            const uint16_t *vbar, const skip_skv_mlp_t *mlp, float tau_nu, float rho_r,
                            int64_t *out_ids, float *out_nu, int32_t *out_count, float *nu_all, void *stream) {
    if (!c) return SKIP_EINVAL;
    skip_status_t st = check_skv(c, Q, K, qbar, vbar, mlp, tau_nu, rho_r, out_ids, out_nu, out_count);
    if (st) return st;
    if (Q > 0 && !cand_ids) return SKIP_EINVAL;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    st = ensure_buf(c->gws, c->gws_bytes, skv_ws_bytes(Q, K, mlp->hidden, c->d), "gate", c->canary);
    if (st) return st;
    ++c->call_id;
    Plan pl;
    CqLaunch cl;
    st = skv_prepare_cq(c, Q, qbar, vbar, mlp, cl);
    if (st) return st;
    st = skv_impl(c, cand_ids, Q, K, qbar, vbar, mlp, tau_nu, rho_r, out_ids, out_nu, out_count, nu_all, cl, s,
                  pl);
    if (st) return st;
    record(c, s, "end");
    return SKIP_OK;
}

skip_status_t skip_retrieve_skv(skip_corpus_t c, const void *regions, const int32_t *region_offsets, int32_t Q,
                                int32_t R_total, int32_t k_region, int32_t K, const uint16_t *qbar,
                                const uint16_t *vbar, const skip_skv_mlp_t *mlp, float tau_nu, float rho_r,
                                int64_t *out_ids, float *out_nu, int32_t *out_count, int64_t *merged_ids,
                                float *merged_scores, void *stream) {
    skip_status_t st = check_retrieve(c, regions, region_offsets, Q, R_total, k_region, K);
    if (st) return st;
    st = check_skv(c, Q, K, qbar, vbar, mlp, tau_nu, rho_r, out_ids, out_nu, out_count);
    if (st) return st;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    // gate workspace first, then the merged lists (unless the caller keeps them)
    const size_t gate = skv_ws_bytes(Q, K, mlp->hidden, c->d);
    const size_t mid = align_up((size_t)Q * K * 8, 256), msc = align_up((size_t)Q * K * 4, 256);
    st = ensure_buf(c->gws, c->gws_bytes, gate + mid + msc, "gate", c->canary);
    if (st) return st;
    int64_t *mids = merged_ids ? merged_ids : reinterpret_cast<int64_t *>((char *)c->gws + gate);
    float *mscs = merged_scores ? merged_scores : reinterpret_cast<float *>((char *)c->gws + gate + mid);
    ++c->call_id;
    Plan pl;
    CqLaunch cl;
    st = skv_prepare_cq(c, Q, qbar, vbar, mlp, cl);
    if (st) return st;
    const bool fork = !c->timing;
    st = retrieve_impl(c, regions, region_offsets, Q, R_total, k_region, K, mids, mscs, s, pl,
                       [&]() { return fork ? skv_launch_cq(c, cl, s, true) : SKIP_OK; });
    if (st) return st;
    st = skv_impl(c, mids, Q, K, qbar, vbar, mlp, tau_nu, rho_r, out_ids, out_nu, out_count, nullptr, cl, s, pl);
    if (st) return st;
    record(c, s, "end");
    write_plan(c, pl, R_total, Q, k_region, K);
    return SKIP_OK;
}

}  // extern "C"

// ---------------------------------------------------------------- IVF-PQ

struct skip_ivfpq {
    skip_corpus *cent = nullptr;  // the centroids as a searchable set (coarse step)
    int64_t N = 0;
    int d = 0, C = 0, M = 0, ds = 0;
    float *codebook = nullptr;    // [M x 256 x ds]
    float *cbT = nullptr;         // [256 x ds x Mp] (Mp = M rounded up to 32)
    int64_t *offsets = nullptr;   // [C + 1] list starts (entries)
    int64_t *boff = nullptr;      // [C + 1] list starts (blocks of 32 entries)
    int32_t *ids = nullptr;       // [N] list order
    uint8_t *codes = nullptr;     // [boff[C] x M * 32] blocks of 32 entries (layout: k_ivfpq.cu il_offset)
    void *ws = nullptr;           // search workspace
    size_t ws_bytes = 0;
    int split = 0;                // parts per region of the list scan (0: pick)
    bool gemm_probe = false;      // coarse probe: one GEMM + per-region sort (C <= kIvfCoarseMaxC)
    const skip_corpus *src = nullptr;  // corpus the index was built from (exact re-rank), or null
    int refine = 0;               // SKIP_OPT_IVF_REFINE: shortlist refine * k by s^, re-ranked exactly
};

namespace {

void ivf_release(skip_ivfpq *ix) {
    if (!ix) return;
    cudaDeviceSynchronize();
    if (ix->cent) skip_corpus_free(ix->cent);
    cudaFree(ix->codebook);
    cudaFree(ix->cbT);
    cudaFree(ix->offsets);
    cudaFree(ix->boff);
    cudaFree(ix->ids);
    cudaFree(ix->codes);
    cudaFree(ix->ws);
    delete ix;
}

// Allocates the index arrays and the centroid set; fills sizes.
skip_status_t ivf_create(const void *centroids, int C, int d, const float *codebook, int M, int64_t N,
                         cudaStream_t s, skip_ivfpq **out) {
    auto *ix = new skip_ivfpq();
    ix->N = N, ix->d = d, ix->C = C, ix->M = M, ix->ds = d / M;
    skip_status_t st = skip_corpus_load(centroids, 1, C, d, SKIP_BF16, nullptr, s, &ix->cent);
    if (st) {
        ivf_release(ix);
        return st;
    }
    const size_t cb = (size_t)M * 256 * ix->ds * sizeof(float);
    ix->gemm_probe = C <= kIvfCoarseMaxC;
    const size_t cbt = (size_t)256 * ix->ds * ivf_padded_m(M) * sizeof(float);
    if (dev_alloc((void **)&ix->codebook, cb, "ivfpq") != cudaSuccess || dev_alloc((void **)&ix->cbT, cbt, "ivfpq") != cudaSuccess ||
        dev_alloc((void **)&ix->offsets, (size_t)(C + 1) * 8, "ivfpq") != cudaSuccess ||
        dev_alloc((void **)&ix->boff, (size_t)(C + 1) * 8, "ivfpq") != cudaSuccess ||
        dev_alloc((void **)&ix->ids, (size_t)std::max<int64_t>(N, 1) * 4, "ivfpq") != cudaSuccess) {
        cudaGetLastError();
        ivf_release(ix);
        return SKIP_ENOMEM;
    }
    if (cudaMemcpyAsync(ix->codebook, codebook, cb, cudaMemcpyDeviceToDevice, s) != cudaSuccess ||
        launch_pq_codebook_t(ix->codebook, M, ix->ds, ix->cbT, s) != cudaSuccess) {
        ivf_release(ix);
        return SKIP_ECUDA;
    }
    *out = ix;
    return SKIP_OK;
}

skip_status_t ivf_check_shape(int C, int d, int M) {
    if (C < 1 || d < 1 || M < 1) return SKIP_EINVAL;
    if (C > (1 << 20) || M % 16 != 0 || M > kIvfMaxM || d % M != 0 || d / M > kIvfMaxDs) return SKIP_EUNSUPPORTED;
    return SKIP_OK;
}

IvfParams ivf_params(const skip_ivfpq *ix) {
    IvfParams p;
    p.rows = nullptr;
    p.N = ix->N;
    p.d = ix->d;
    p.centroids = ix->cent->rows;
    p.C = ix->C;
    p.codebook = ix->codebook;
    p.cbT = ix->cbT;
    p.M = ix->M;
    p.ds = ix->ds;
    p.offsets = ix->offsets;
    p.boff = ix->boff;
    p.ids = ix->ids;
    p.codes = ix->codes;
    return p;
}

// Checks the list offsets (0 = off[0] <= ... <= off[C] = N), derives the
// block offsets and stores `rows` (codes in list order, one row of M bytes
// per entry; device) in blocks of 32 entries.  Returns after the copy.
skip_status_t ivf_layout(skip_ivfpq *ix, const uint8_t *rows, cudaStream_t s) {
    const int C = ix->C;
    std::vector<int64_t> off((size_t)C + 1), boff((size_t)C + 1);
    if (cudaMemcpyAsync(off.data(), ix->offsets, (size_t)(C + 1) * 8, cudaMemcpyDeviceToHost, s) != cudaSuccess ||
        cudaStreamSynchronize(s) != cudaSuccess)
        return SKIP_ECUDA;
    if (off[0] != 0 || off[C] != ix->N) return SKIP_EINVAL;
    boff[0] = 0;
    for (int l = 0; l < C; ++l) {
        if (off[l + 1] < off[l]) return SKIP_EINVAL;
        boff[l + 1] = boff[l] + (off[l + 1] - off[l] + 31) / 32;
    }
    const size_t bytes = (size_t)std::max<int64_t>(boff[C], 1) * 32 * ix->M;
    if (dev_alloc((void **)&ix->codes, bytes, "ivfpq") != cudaSuccess) {
        cudaGetLastError();
        return SKIP_ENOMEM;
    }
    if (cudaMemcpyAsync(ix->boff, boff.data(), (size_t)(C + 1) * 8, cudaMemcpyHostToDevice, s) != cudaSuccess ||
        cudaMemsetAsync(ix->codes, 0, bytes, s) != cudaSuccess ||
        launch_ivf_interleave(ivf_params(ix), rows, ix->codes, ix->cent->sm_count, s) != cudaSuccess ||
        cudaStreamSynchronize(s) != cudaSuccess)
        return SKIP_ECUDA;
    return SKIP_OK;
}

// Coarse probes then the list scan: top-k keys of each of the G parts of
// each region ([G x R x k], the head of the index workspace), and room for
// R x k merged keys after them (*merged).
skip_status_t ivf_regions(skip_ivfpq *ix, const void *regions, int R, int nprobe, int k, cudaStream_t s,
                          uint64_t **keys_out, uint64_t **merged, int *G_out) {
    int G = 1;
    if (R > 0) {
        skip_status_t st = cuda_status(ivfpq_scan_split(ix->M, nprobe, R, ix->cent->sm_count, ix->split, &G));
        if (st) return st;
    }
    const size_t pid = align_up((size_t)R * nprobe * 8, 256), psc = align_up((size_t)R * nprobe * 4, 256);
    const size_t kb = align_up((size_t)std::max(R, 1) * k * 8, 256);
    const size_t scb = ix->gemm_probe ? align_up((size_t)R * ix->C * 4, 256) : 0;  // coarse GEMM scores
    skip_status_t st = ensure_buf(ix->ws, ix->ws_bytes, (G + 1) * kb + pid + psc + scb, "ivfpq", false);
    if (st) return st;
    uint64_t *keys = reinterpret_cast<uint64_t *>(ix->ws);
    int64_t *probe_ids = reinterpret_cast<int64_t *>((char *)ix->ws + (G + 1) * kb);
    float *probe_sc = reinterpret_cast<float *>((char *)ix->ws + (G + 1) * kb + pid);
    *keys_out = keys;
    *merged = reinterpret_cast<uint64_t *>((char *)ix->ws + G * kb);
    *G_out = G;
    if (R == 0) return SKIP_OK;
    if (ix->gemm_probe) {
        // coarse scores [R x C] = regions [R x d] . centroids [C x d]^T on the
        // tensor cores, then the nprobe best per region
        float *scores = reinterpret_cast<float *>((char *)ix->ws + (G + 1) * kb + pid + psc);
        CUtensorMap ta, tb;
        const int tn = gemm_tile_n(R, ix->C, ix->cent->sm_count);
        if (!encode_bf16_rows(&ta, regions, R, ix->d, 128) ||
            !encode_bf16_rows(&tb, ix->cent->rows, ix->C, ix->d, tn))
            return SKIP_ECUDA;
        record(ix->cent, s, "ivf_probe");
        st = cuda_status(launch_gemm_bf16_f32(ta, tb, tn, R, ix->C, ix->d, 1.f, scores, ix->C, ix->cent->err,
                                              ix->cent->timeout_ns, s));
        if (st) return st;
        st = cuda_status(launch_ivf_probe_select(scores, R, ix->C, nprobe, probe_ids, probe_sc, s));
    } else {
        Plan pl;
        st = run_regions(ix->cent, reinterpret_cast<const uint16_t *>(regions), R, nprobe, nullptr, probe_ids,
                         probe_sc, s, pl, 0);
    }
    if (st) return st;
    record(ix->cent, s, "ivfpq_scan");
    cudaError_t e = launch_ivfpq_scan(ivf_params(ix), reinterpret_cast<const uint16_t *>(regions), R, probe_ids,
                                      probe_sc, nprobe, k, G, keys, ix->cent->sm_count, s);
    return cuda_status(e);
}

skip_status_t ivf_check_search(skip_ivfpq *ix, const void *regions, int R, int nprobe, int k) {
    if (!ix || R < 0 || (R > 0 && !regions)) return SKIP_EINVAL;
    if (nprobe < 1 || nprobe > std::min(ix->C, SKIP_MAX_K_REGION)) return SKIP_EINVAL;
    if (k < 1 || k > SKIP_MAX_K_REGION) return SKIP_EINVAL;
    return SKIP_OK;
}

// Each region's k keys [R x k] (sorted), in the index workspace: the scan's
// top k by s^, or with a refine factor its top min(refine k, 1024) re-ranked
// by exact scores against the corpus the index was built from.
skip_status_t ivf_region_keys(skip_ivfpq *ix, const void *regions, int R, int nprobe, int k, cudaStream_t s,
                              uint64_t **out) {
    const int ks = ix->refine > 1 ? (int)std::min<int64_t>(std::min<int64_t>((int64_t)ix->refine * k, kIvfMaxRefine),
                                                           ix->N)
                                  : k;
    uint64_t *keys = nullptr, *merged = nullptr;
    int G = 1;
    skip_status_t st = ivf_regions(ix, regions, R, nprobe, std::max(ks, k), s, &keys, &merged, &G);
    if (st || R == 0) {
        *out = keys;
        return st;
    }
    const int kk = std::max(ks, k);
    if (G > 1) {
        record(ix->cent, s, "merge_lists");
        st = cuda_status(launch_merge_lists(keys, G, (int64_t)R * kk, R, kk, merged, nullptr, nullptr, s));
        if (st) return st;
    } else {
        merged = keys;
    }
    if (ks > k) {
        // the shortlist (merged) is re-ranked into the head of the workspace
        uint64_t *dst = merged == keys ? keys + (size_t)R * kk : keys;
        record(ix->cent, s, "ivf_refine");
        st = cuda_status(launch_ivf_refine(reinterpret_cast<const uint16_t *>(ix->src->rows), ix->src->N,
                                           ix->src->d, reinterpret_cast<const uint16_t *>(regions), R, merged, ks,
                                           k, dst, s));
        *out = dst;
        return st;
    }
    *out = merged;
    return SKIP_OK;
}

}  // namespace

extern "C" {

skip_status_t skip_ivfpq_build(skip_corpus_t c, const void *centroids, int32_t C, const float *codebook, int32_t M,
                               void *stream, skip_ivfpq_t *out) {
    if (!c || !centroids || !codebook || !out) return SKIP_EINVAL;
    skip_status_t st = ivf_check_shape(C, c->d, M);
    if (st) return st;
    if (c->dtype != SKIP_BF16) return SKIP_EUNSUPPORTED;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    skip_ivfpq *ix = nullptr;
    st = ivf_create(centroids, C, c->d, codebook, M, c->N, s, &ix);
    if (st) return st;
    ix->src = c;
    const int64_t N = c->N;
    void *tmp = nullptr;
    const size_t rl = align_up((size_t)N * 8, 256), rs = align_up((size_t)N * 4, 256);
    const size_t cr = align_up((size_t)N * M, 256), cc = align_up((size_t)C * 8, 256);
    if (dev_alloc((void **)&tmp, rl + rs + 2 * cr + 2 * cc, "ivfpq") != cudaSuccess) {
        cudaGetLastError();
        ivf_release(ix);
        return SKIP_ENOMEM;
    }
    int64_t *row_list = reinterpret_cast<int64_t *>(tmp);
    float *row_score = reinterpret_cast<float *>((char *)tmp + rl);
    uint8_t *codes_rows = reinterpret_cast<uint8_t *>((char *)tmp + rl + rs);
    int64_t *counts = reinterpret_cast<int64_t *>((char *)tmp + rl + rs + cr);
    int64_t *cursor = reinterpret_cast<int64_t *>((char *)tmp + rl + rs + cr + cc);
    uint8_t *codes_list = reinterpret_cast<uint8_t *>((char *)tmp + rl + rs + cr + 2 * cc);
    Plan pl;
    st = run_regions(ix->cent, reinterpret_cast<const uint16_t *>(c->rows), (int)N, 1, nullptr, row_list, row_score,
                     s, pl, 0);
    IvfParams p = ivf_params(ix);
    p.rows = c->rows;
    if (!st) st = cuda_status(launch_pq_encode(p, row_list, codes_rows, s));
    if (!st)
        st = cuda_status(launch_ivf_lists(p, row_list, codes_rows, counts, cursor, ix->offsets, ix->ids, codes_list,
                                          ix->cent->err, ix->cent->sm_count, s));
    if (!st) st = skip_sync_status(ix->cent, stream);
    if (!st) st = ivf_layout(ix, codes_list, s);
    cudaFree(tmp);
    if (st) {
        ivf_release(ix);
        return st;
    }
    *out = ix;
    return SKIP_OK;
}

skip_status_t skip_ivfpq_load(const void *centroids, int32_t C, int32_t d, const float *codebook, int32_t M,
                              const int64_t *list_offsets, const int32_t *ids, const uint8_t *codes, int64_t N,
                              void *stream, skip_ivfpq_t *out) {
    if (!centroids || !codebook || !list_offsets || !out || N < 0 || N >= ((int64_t)1 << 31)) return SKIP_EINVAL;
    if (N > 0 && (!ids || !codes)) return SKIP_EINVAL;
    if (d % 16 != 0) return SKIP_EINVAL;
    skip_status_t st = ivf_check_shape(C, d, M);
    if (st) return st;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    skip_ivfpq *ix = nullptr;
    st = ivf_create(centroids, C, d, codebook, M, N, s, &ix);
    if (st) return st;
    if (cudaMemcpyAsync(ix->offsets, list_offsets, (size_t)(C + 1) * 8, cudaMemcpyDeviceToDevice, s) != cudaSuccess ||
        (N > 0 && cudaMemcpyAsync(ix->ids, ids, (size_t)N * 4, cudaMemcpyDeviceToDevice, s) != cudaSuccess)) {
        ivf_release(ix);
        return SKIP_ECUDA;
    }
    st = ivf_layout(ix, codes, s);
    if (st) {
        ivf_release(ix);
        return st;
    }
    *out = ix;
    return SKIP_OK;
}

skip_status_t skip_ivfpq_lists(skip_ivfpq_t ix, int64_t *list_offsets, int32_t *ids, uint8_t *codes, void *stream) {
    if (!ix) return SKIP_EINVAL;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    if ((list_offsets && cudaMemcpyAsync(list_offsets, ix->offsets, (size_t)(ix->C + 1) * 8, cudaMemcpyDeviceToDevice,
                                         s) != cudaSuccess) ||
        (ids && ix->N > 0 && cudaMemcpyAsync(ids, ix->ids, (size_t)ix->N * 4, cudaMemcpyDeviceToDevice, s) != cudaSuccess) ||
        (codes && launch_ivf_deinterleave(ivf_params(ix), codes, ix->cent->sm_count, s) != cudaSuccess) ||
        cudaStreamSynchronize(s) != cudaSuccess)
        return SKIP_ECUDA;
    return SKIP_OK;
}

skip_status_t skip_ivfpq_info(skip_ivfpq_t ix, int64_t *N, int32_t *d, int32_t *C, int32_t *M) {
    if (!ix) return SKIP_EINVAL;
    if (N) *N = ix->N;
    if (d) *d = ix->d;
    if (C) *C = ix->C;
    if (M) *M = ix->M;
    return SKIP_OK;
}

skip_status_t skip_ivfpq_free(skip_ivfpq_t ix) {
    ivf_release(ix);
    return SKIP_OK;
}

skip_status_t skip_ivfpq_search_regions(skip_ivfpq_t ix, const void *regions, int32_t R_total, int32_t nprobe,
                                        int32_t k_region, int64_t *reg_ids, float *reg_scores, void *stream) {
    skip_status_t st = ivf_check_search(ix, regions, R_total, nprobe, k_region);
    if (st) return st;
    if (R_total > 0 && (!reg_ids || !reg_scores)) return SKIP_EINVAL;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    ++ix->cent->call_id;
    uint64_t *keys = nullptr;
    st = ivf_region_keys(ix, regions, R_total, nprobe, k_region, s, &keys);
    if (st || R_total == 0) return st;
    record(ix->cent, s, "merge_lists");
    st = cuda_status(launch_merge_lists(keys, 1, (int64_t)R_total * k_region, R_total, k_region, nullptr, reg_ids,
                                        reg_scores, s));
    record(ix->cent, s, "end");
    return st;
}

skip_status_t skip_ivfpq_search(skip_ivfpq_t ix, const void *regions, const int32_t *region_offsets, int32_t Q,
                                int32_t R_total, int32_t nprobe, int32_t k_region, int32_t K, int64_t *out_ids,
                                float *out_scores, void *stream) {
    skip_status_t st = ivf_check_search(ix, regions, R_total, nprobe, k_region);
    if (st) return st;
    if (Q < 0 || K < 1 || K > SKIP_MAX_K || (Q > 0 && (!region_offsets || !out_ids || !out_scores))) return SKIP_EINVAL;
    if (Q == 0 && R_total != 0) return SKIP_EINVAL;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    ++ix->cent->call_id;
    uint64_t *keys = nullptr;
    st = ivf_region_keys(ix, regions, R_total, nprobe, k_region, s, &keys);
    if (st) return st;
    if (Q > 0) {
        record(ix->cent, s, "question_merge");
        st = cuda_status(launch_question_merge(keys, k_region, region_offsets, Q, R_total, K, out_ids, out_scores,
                                               ix->cent->err, s));
    }
    record(ix->cent, s, "end");
    return st;
}

skip_status_t skip_ivfpq_sync_status(skip_ivfpq_t ix, void *stream) {
    if (!ix) return SKIP_EINVAL;
    return skip_sync_status(ix->cent, stream);
}

skip_status_t skip_ivfpq_set_option(skip_ivfpq_t ix, int option, int64_t value) {
    if (!ix) return SKIP_EINVAL;
    if (option == SKIP_OPT_IVF_SPLIT) {
        if (value < 0 || value > kIvfMaxSplit) return SKIP_EINVAL;
        ix->split = (int)value;
        return SKIP_OK;
    }
    if (option == SKIP_OPT_IVF_REFINE) {
        if (value < 0 || value > kIvfMaxRefine) return SKIP_EINVAL;
        if (value > 1 && !ix->src) return SKIP_EUNSUPPORTED;
        ix->refine = value > 1 ? (int)value : 0;
        return SKIP_OK;
    }
    return skip_corpus_set_option(ix->cent, option, value);
}

skip_status_t skip_ivfpq_timing_report(skip_ivfpq_t ix, char *buf, int32_t len) {
    if (!ix) return SKIP_EINVAL;
    return skip_timing_report(ix->cent, buf, len);
}

}  // extern "C"

// ---------------------------------------------------------------- QVS

struct skip_qvs {
    int device = 0, sms = 0;
    int d = 0, dk = 0, max_b = 0, max_l = 0;
    int dkp = 0;                            // d_k rounded up to 8 (zero columns past d_k)
    uint16_t *wvt = nullptr;                // W_v^T [d x dkp] bf16
    uint16_t *fqp = nullptr;                // [max_b x dkp] staging for f_q when d_k % 8 != 0
    float *bv = nullptr, *wb = nullptr;
    float *u = nullptr, *logits = nullptr;  // workspace
    int *err = nullptr;                     // device error word of the GEMM's bounded waits
    uint64_t timeout_ns = kDefaultTimeoutNs;
};

namespace {

void qvs_release(skip_qvs *q) {
    if (!q) return;
    cudaDeviceSynchronize();
    cudaFree(q->wvt);
    cudaFree(q->fqp);
    cudaFree(q->bv);
    cudaFree(q->wb);
    cudaFree(q->u);
    cudaFree(q->logits);
    cudaFree(q->err);
    delete q;
}

}  // namespace

extern "C" {

int32_t skip_qvs_count(int32_t L, float rho_v) {
    const double v = ceil((double)rho_v * (double)L - 1e-3);
    return (int32_t)std::max(0.0, std::min((double)L, v));
}

skip_status_t skip_qvs_create(const uint16_t *wv, const float *bv, const float *wb, int32_t d, int32_t dk,
                              int32_t max_images, int32_t max_tokens, void *stream, skip_qvs_t *out) {
    if (!wv || !wb || !out || d < 8 || dk < 1 || max_images < 1 || max_tokens < 1) return SKIP_EINVAL;
    if (d % 8 != 0 || d > 8192 || dk > kQvsMaxDk || max_tokens > kQvsMaxL) return SKIP_EUNSUPPORTED;
    int dev = 0;
    cudaDeviceProp prop;
    if (cudaGetDevice(&dev) != cudaSuccess || cudaGetDeviceProperties(&prop, dev) != cudaSuccess) {
        cudaGetLastError();
        return SKIP_EUNSUPPORTED;
    }
    if (prop.major != 10 || prop.minor != 3) return SKIP_EUNSUPPORTED;
    auto *q = new skip_qvs();
    q->device = dev, q->sms = prop.multiProcessorCount;
    q->d = d, q->dk = dk, q->max_b = max_images, q->max_l = max_tokens;
    q->dkp = (dk + 7) / 8 * 8;
    if (dev_alloc((void **)&q->wvt, (size_t)q->dkp * d * 2, "qvs") != cudaSuccess ||
        (q->dkp != dk && dev_alloc((void **)&q->fqp, (size_t)max_images * q->dkp * 2, "qvs") != cudaSuccess) ||
        dev_alloc((void **)&q->bv, (size_t)dk * 4, "qvs") != cudaSuccess ||
        dev_alloc((void **)&q->wb, (size_t)d * 4, "qvs") != cudaSuccess ||
        dev_alloc((void **)&q->u, (size_t)kQvsUSplits * max_images * d * 4, "qvs") != cudaSuccess ||
        dev_alloc((void **)&q->logits, (size_t)max_images * max_tokens * 4, "qvs") != cudaSuccess ||
        dev_alloc((void **)&q->err, sizeof(int), "qvs") != cudaSuccess) {
        cudaGetLastError();
        qvs_release(q);
        return SKIP_ENOMEM;
    }
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    // W_v^T is kept so that both operands of the projection GEMM are K-major;
    // with d_k % 8 != 0 both operands carry zero columns up to dkp (the row
    // pitch a TMA copy needs), which add nothing to the sums.
    if ((q->dkp != dk && (cudaMemsetAsync(q->wvt, 0, (size_t)q->dkp * d * 2, s) != cudaSuccess ||
                          cudaMemsetAsync(q->fqp, 0, (size_t)max_images * q->dkp * 2, s) != cudaSuccess)) ||
        launch_transpose_bf16(wv, dk, d, q->wvt, q->dkp, s) != cudaSuccess ||
        cudaMemsetAsync(q->err, 0, sizeof(int), s) != cudaSuccess ||
        (bv ? cudaMemcpyAsync(q->bv, bv, (size_t)dk * 4, cudaMemcpyDeviceToDevice, s)
            : cudaMemsetAsync(q->bv, 0, (size_t)dk * 4, s)) != cudaSuccess ||
        cudaMemcpyAsync(q->wb, wb, (size_t)d * 4, cudaMemcpyDeviceToDevice, s) != cudaSuccess ||
        cudaStreamSynchronize(s) != cudaSuccess) {
        qvs_release(q);
        return SKIP_ECUDA;
    }
    *out = q;
    return SKIP_OK;
}

skip_status_t skip_qvs_free(skip_qvs_t q) {
    qvs_release(q);
    return SKIP_OK;
}

skip_status_t skip_qvs_prune(skip_qvs_t q, const uint16_t *tokens, int32_t B, int32_t L, const uint16_t *fq,
                             float rho_v, int32_t *out_idx, float *out_score, uint16_t *out_tokens, float *logits,
                             void *stream) {
    if (!q || B < 0 || B > q->max_b || L < 1 || L > q->max_l) return SKIP_EINVAL;
    if (!(rho_v >= 0.f && rho_v <= 1.f)) return SKIP_EINVAL;
    const int n = skip_qvs_count(L, rho_v);
    if (B > 0 && (!tokens || !fq || (n > 0 && (!out_idx || !out_score)))) return SKIP_EINVAL;
    if (B > 0 && ((uintptr_t)tokens & 15) != 0) return SKIP_EINVAL;
    if (B == 0) return SKIP_OK;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    QvsParams p;
    p.tokens = tokens;
    p.fq = fq;
    p.wvt = q->wvt;
    p.bv = q->bv;
    p.wb = q->wb;
    p.B = B, p.L = L, p.d = q->d, p.dk = q->dk, p.n = n;
    p.u = q->u;
    p.logits = logits ? logits : q->logits;
    p.out_idx = out_idx;
    p.out_score = out_score;
    p.out_tokens = out_tokens;
    // U [B x d] = F_q [B x d_k] (W_v^T [d x d_k])^T / sqrt(d_k) on the tensor cores.
    const uint16_t *fa = fq;
    if (q->dkp != q->dk || ((uintptr_t)fq & 15) != 0) {
        if (!q->fqp && dev_alloc((void **)&q->fqp, (size_t)q->max_b * q->dkp * 2, "qvs") != cudaSuccess) {
            cudaGetLastError();
            return SKIP_ENOMEM;
        }
        if (cudaMemcpy2DAsync(q->fqp, (size_t)q->dkp * 2, fq, (size_t)q->dk * 2, (size_t)q->dk * 2, B,
                              cudaMemcpyDeviceToDevice, s) != cudaSuccess)
            return SKIP_ECUDA;
        fa = q->fqp;
    }
    CUtensorMap ta, tb;
    const int tn = gemm_tile_n(B, q->d, q->sms);
    if (!encode_bf16_rows(&ta, fa, B, q->dkp, 128) || !encode_bf16_rows(&tb, q->wvt, q->d, q->dkp, tn))
        return SKIP_ECUDA;
    // K split over up to kQvsUSplits CTAs per tile (a [B x d] product has few
    // tiles); the logits kernel sums the partial slabs.
    p.u_splits = std::min(kQvsUSplits, gemm_splits(B, q->d, q->dkp, tn, q->sms));
    cudaError_t e = launch_gemm_bf16_f32(ta, tb, tn, B, q->d, q->dkp, 1.f / std::sqrt((float)q->dk), q->u, q->d,
                                         q->err, q->timeout_ns, s, p.u_splits, (int64_t)B * q->d);
    if (e == cudaSuccess) e = launch_qvs_logits(p, q->sms, s);
    if (e == cudaSuccess) e = launch_qvs_select(p, s);
    return cuda_status(e);
}

skip_status_t skip_qvs_sync_status(skip_qvs_t q, void *stream) {
    if (!q) return SKIP_EINVAL;
    if (cudaStreamSynchronize(reinterpret_cast<cudaStream_t>(stream)) != cudaSuccess) return SKIP_ECUDA;
    int err = 0;
    if (cudaMemcpy(&err, q->err, sizeof(int), cudaMemcpyDeviceToHost) != cudaSuccess) return SKIP_ECUDA;
    if (err) {
        if (cudaMemset(q->err, 0, sizeof(int)) != cudaSuccess) return SKIP_ECUDA;
        return SKIP_ETIMEOUT;
    }
    return SKIP_OK;
}

}  // extern "C"

// ---------------------------------------------------------------- BSCA

struct skip_bsca {
    int dp = 0, dh = 0, dout = 0, max_q = 0, max_t = 0;
    float *cos = nullptr, *tau = nullptr;
    uint32_t *hist = nullptr;  // per-question cosine histograms, zero between calls
    int *err = nullptr;
};

namespace {

void bsca_release(skip_bsca *b) {
    if (!b) return;
    cudaDeviceSynchronize();
    cudaFree(b->cos);
    cudaFree(b->hist);
    cudaFree(b->tau);
    cudaFree(b->err);
    delete b;
}

}  // namespace

extern "C" {

skip_status_t skip_bsca_create(int32_t d_p, int32_t d_h, int32_t d_o, int32_t max_questions, int32_t max_tokens,
                               skip_bsca_t *out) {
    if (!out || d_p < 1 || d_h < 1 || d_o < 2 || max_questions < 1 || max_tokens < 1) return SKIP_EINVAL;
    if (d_p > kBscaMaxDp || d_h > kBscaMaxDh || d_o > kBscaMaxDo || d_o % 2 != 0) return SKIP_EUNSUPPORTED;
    int dev = 0, major = 0, minor = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) {
        cudaGetLastError();
        return SKIP_EUNSUPPORTED;
    }
    cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
    cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
    if (major != 10 || minor != 3) return SKIP_EUNSUPPORTED;
    auto *b = new skip_bsca();
    b->dp = d_p, b->dh = d_h, b->dout = d_o, b->max_q = max_questions, b->max_t = max_tokens;
    if (dev_alloc((void **)&b->cos, (size_t)max_tokens * kBscaMaxR * 4, "bsca") != cudaSuccess ||
        dev_alloc((void **)&b->tau, (size_t)max_questions * 4, "bsca") != cudaSuccess ||
        dev_alloc((void **)&b->hist, (size_t)max_questions * kBscaBins * 4, "bsca") != cudaSuccess ||
        cudaMemset(b->hist, 0, (size_t)max_questions * kBscaBins * 4) != cudaSuccess ||
        dev_alloc((void **)&b->err, sizeof(int), "bsca") != cudaSuccess || cudaMemset(b->err, 0, sizeof(int)) != cudaSuccess) {
        cudaGetLastError();
        bsca_release(b);
        return SKIP_ENOMEM;
    }
    *out = b;
    return SKIP_OK;
}

skip_status_t skip_bsca_free(skip_bsca_t b) {
    bsca_release(b);
    return SKIP_OK;
}

skip_status_t skip_bsca_run(skip_bsca_t b, int32_t Q, const int32_t *vis_offsets, const int32_t *chunk_offsets,
                            int32_t total_tokens, const uint16_t *hv, const uint16_t *qh, const uint16_t *hk,
                            const uint16_t *kh, const uint16_t *vh, float dbar, float *out, int32_t *degree,
                            uint64_t *edges, float *tau_e, void *stream) {
    if (!b || Q < 0 || Q > b->max_q || total_tokens < 0 || total_tokens > b->max_t) return SKIP_EINVAL;
    if (!(dbar >= 0.f)) return SKIP_EINVAL;
    if (Q > 0 && (!vis_offsets || !chunk_offsets || !hk || !kh || !vh)) return SKIP_EINVAL;
    if (total_tokens > 0 && (!hv || !qh || !out)) return SKIP_EINVAL;
    if (Q == 0) return SKIP_OK;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    BscaParams p;
    p.Q = Q;
    p.vis_offsets = vis_offsets;
    p.chunk_offsets = chunk_offsets;
    p.Nv = total_tokens;
    p.hv = hv, p.qh = qh, p.hk = hk, p.kh = kh, p.vh = vh;
    p.dp = b->dp, p.dh = b->dh, p.dout = b->dout;
    p.dbar = dbar;
    p.cos = b->cos;
    p.hist = b->hist;
    p.tau = tau_e ? tau_e : b->tau;
    p.degree = degree;
    p.edges = edges;
    p.out = out;
    p.err = b->err;
    return cuda_status(launch_bsca(p, s));
}

skip_status_t skip_bsca_sync_status(skip_bsca_t b, void *stream) {
    if (!b) return SKIP_EINVAL;
    if (cudaStreamSynchronize(reinterpret_cast<cudaStream_t>(stream)) != cudaSuccess) return SKIP_ECUDA;
    int err = 0;
    if (cudaMemcpy(&err, b->err, sizeof(int), cudaMemcpyDeviceToHost) != cudaSuccess) return SKIP_ECUDA;
    if (err && cudaMemset(b->err, 0, sizeof(int)) != cudaSuccess) return SKIP_ECUDA;
    if (err & kErrConfig) return SKIP_EINVAL;
    return SKIP_OK;
}

}  // extern "C"
