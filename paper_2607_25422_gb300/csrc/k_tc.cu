// Tensor-core score + fused top-k (tcgen05 / TMEM / TMA, sm_103a).
//
// Step: per-region MIPS top-k over the corpus (paper App. B.2 Def. B.2,
// MIPS(q_r, D; k_r); §3.3 Eq. rcsr).  For a batch of region queries the
// scores S = Q X^T are a dense bf16 contraction with fp32 accumulation; this
// kernel computes them on the 5th-generation tensor cores and never writes
// them to HBM: the epilogue reads each accumulator tile out of tensor memory
// and keeps, per region row, a sorted top-k list and its k-th score.
//
// Tile: A = 128 region rows (TMEM lanes), B = 256 corpus rows (TMEM
// columns), K streamed in 64-element (128-byte) slices.  One thread of the
// epilogue owns one region row, so its threshold lives in a register and the
// common case -- no score of a 32-column chunk beats it -- costs a max and a
// compare per chunk.  Corpus rows of a tile are visited in increasing id
// order, so "beats" is a strict score comparison and ties keep the lower id.
//
// Work: items (query block, corpus chunk); a persistent CTA walks items
// blockIdx.x, blockIdx.x + gridDim.x, ...  Items are numbered chunk-major, so
// the CTAs running at the same time read the same corpus chunk and every
// corpus tile comes from HBM about once and is re-read by the other query
// blocks from L2.  Each item leaves one sorted list per region row; the merge
// kernel combines the chunks.
//
// Warp roles (192 threads): warp 0 issues TMA loads into a 4-stage
// shared-memory ring; warp 1 owns TMEM (two 256-column fp32 accumulators)
// and issues tcgen05.mma from one thread; warps 2..5 are the epilogue, warp w
// reading TMEM lanes 32 * (w % 4) .. + 31.  Every wait is bounded; a wait
// that gives up sets the error word, the other roles then give up too, and
// before exit the producer waits for its copies in flight and the MMA thread
// for its MMAs, so that TMEM is freed by its owner with nothing outstanding.
#include "skip_device.cuh"
#include "skip_internal.h"

namespace skipk {
namespace {

constexpr int kABytes = kTcTileM * kTcTileK * 2;  // 16 KB
constexpr int kBBytes = kTcTileN * kTcTileK * 2;  // 32 KB
constexpr int kStageBytes = kABytes + kBBytes;
constexpr uint32_t kTmemCols = 512;                 // two 256-column accumulators
constexpr uint64_t kDrainTimeoutNs = 1000000000ull;  // 1 s for copies/MMAs in flight
constexpr uint32_t kIdesc = idesc_bf16_f32(kTcTileM, kTcTileN);

struct __align__(8) TcShared {
    uint64_t full[kTcStages];   // stage loaded (TMA transaction bytes)
    uint64_t empty[kTcStages];  // stage consumed (tcgen05.commit)
    uint64_t tfull[2];          // accumulator ready (tcgen05.commit)
    uint64_t tempty[2];         // accumulator drained (4 epilogue warps)
    uint64_t drain;             // MMA completion at exit
    uint32_t tmem_base;
};

struct Item {
    int mb;
    int g;
    int64_t t0, t1;
};

__device__ __forceinline__ Item item_of(const TcParams &p, int u) {
    Item it;
    it.g = u / p.MB;
    it.mb = u - it.g * p.MB;
    it.t0 = (int64_t)it.g * p.tiles / p.G;
    it.t1 = (int64_t)(it.g + 1) * p.tiles / p.G;
    return it;
}

__device__ __noinline__ uint64_t insert_key(uint64_t *list, int nfill, int k, uint64_t key) {
    return sorted_insert(list, nfill, k, key);
}

__device__ __forceinline__ float fmax32(const uint32_t (&v)[32]) {
    float m[16];
#pragma unroll
    for (int j = 0; j < 16; ++j) m[j] = fmaxf(__uint_as_float(v[j]), __uint_as_float(v[j + 16]));
#pragma unroll
    for (int w = 8; w; w >>= 1)
#pragma unroll
        for (int j = 0; j < w; ++j) m[j] = fmaxf(m[j], m[j + w]);
    return m[0];
}

__global__ void __launch_bounds__(kTcThreads, 1)
    k_tc_score_topk(const __grid_constant__ CUtensorMap tq, const __grid_constant__ CUtensorMap tx,
                    const TcParams p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    uint8_t *sA = smem;
    uint8_t *sB = smem + kTcStages * kABytes;
    TcShared *sh = reinterpret_cast<TcShared *>(smem + kTcStages * kStageBytes);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int items = p.MB * p.G;
    const int KB = (p.d + kTcTileK - 1) / kTcTileK;

    if (threadIdx.x == 0) {
        for (int s = 0; s < kTcStages; ++s) {
            mbar_init(smem_addr(&sh->full[s]), 1);
            mbar_init(smem_addr(&sh->empty[s]), 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(smem_addr(&sh->tfull[b]), 1);
            mbar_init(smem_addr(&sh->tempty[b]), 4);
        }
        mbar_init(smem_addr(&sh->drain), 1);
        mbar_fence_init();
    }
    if (warp == 0 && lane == 0) {
        tma_prefetch_desc(&tq);
        tma_prefetch_desc(&tx);
    }
    if (warp == 1) {
        tmem_alloc(smem_addr(&sh->tmem_base), kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = sh->tmem_base;

    if (warp == 0) {
        // ------------------------------------------------ TMA producer
        if (lane == 0) {
            int s = 0;
            uint32_t ph = 0;
            int64_t issued = 0;
            bool ok = true;
            for (int u = blockIdx.x; u < items && ok; u += gridDim.x) {
                const Item it = item_of(p, u);
                for (int64_t t = it.t0; t < it.t1 && ok; ++t) {
                    for (int kb = 0; kb < KB; ++kb) {
                        if (!mbar_wait(smem_addr(&sh->empty[s]), ph ^ 1u, p.timeout_ns)) {
                            ok = false;
                            break;
                        }
                        const uint32_t fb = smem_addr(&sh->full[s]);
                        mbar_arrive_expect_tx(fb, kStageBytes);
                        tma_load_2d(smem_addr(sA + s * kABytes), &tq, fb, kb * kTcTileK, it.mb * kTcTileM);
                        tma_load_2d(smem_addr(sB + s * kBBytes), &tx, fb, kb * kTcTileK, (int)(t * kTcTileN));
                        ++issued;
                        if (++s == kTcStages) {
                            s = 0;
                            ph ^= 1u;
                        }
                    }
                }
            }
            if (!ok) atomicOr(p.err, kErrTimeout);
            // Copies in flight: wait for the last load issued on every stage.
            for (int st = 0; st < kTcStages; ++st) {
                const int64_t uses = issued / kTcStages + (st < issued % kTcStages ? 1 : 0);
                if (uses == 0) continue;
                if (!mbar_wait(smem_addr(&sh->full[st]), (uint32_t)((uses - 1) & 1), kDrainTimeoutNs))
                    atomicOr(p.err, kErrTimeout);
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------ MMA issuer
        if (lane == 0) {
            int s = 0;
            uint32_t ph = 0;
            uint32_t lt = 0;
            bool ok = true;
            for (int u = blockIdx.x; u < items && ok; u += gridDim.x) {
                const Item it = item_of(p, u);
                for (int64_t t = it.t0; t < it.t1 && ok; ++t, ++lt) {
                    const uint32_t buf = lt & 1u, use = lt >> 1;
                    if (!mbar_wait(smem_addr(&sh->tempty[buf]), (use & 1u) ^ 1u, p.timeout_ns)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t dt = tmem + buf * kTcTileN;
                    for (int kb = 0; kb < KB; ++kb) {
                        if (!mbar_wait(smem_addr(&sh->full[s]), ph, p.timeout_ns)) {
                            ok = false;
                            break;
                        }
                        tc_fence_after();
                        const uint64_t ad = smem_desc_k128(smem_addr(sA + s * kABytes));
                        const uint64_t bd = smem_desc_k128(smem_addr(sB + s * kBBytes));
#pragma unroll
                        for (int kk = 0; kk < kTcTileK / 16; ++kk)
                            tc_mma_f16(dt, ad + (uint64_t)(kk * 2), bd + (uint64_t)(kk * 2), kIdesc,
                                       (kb | kk) != 0);
                        tc_commit(smem_addr(&sh->empty[s]));
                        if (++s == kTcStages) {
                            s = 0;
                            ph ^= 1u;
                        }
                    }
                    if (!ok) break;
                    tc_commit(smem_addr(&sh->tfull[buf]));
                }
            }
            if (!ok) atomicOr(p.err, kErrTimeout);
            // MMAs in flight: a commit arrives once all earlier ones are done.
            tc_commit(smem_addr(&sh->drain));
            if (!mbar_wait(smem_addr(&sh->drain), 0, kDrainTimeoutNs)) atomicOr(p.err, kErrTimeout);
        }
    } else {
        // ------------------------------------------------ epilogue
        const int sub = warp & 3;
        const int rib = sub * 32 + lane;  // region row within the query block
        const uint32_t lane_addr = (uint32_t)(sub * 32) << 16;
        const float kNegInf = -__int_as_float(0x7f800000);
        uint32_t lt = 0;
        bool ok = true;
        for (int u = blockIdx.x; u < items && ok; u += gridDim.x) {
            const Item it = item_of(p, u);
            const int row = it.mb * kTcTileM + rib;
            const bool row_valid = row < p.R;
            uint64_t *list = p.lists + ((int64_t)it.g * p.R_pad + row) * p.k;
            int nfill = 0;
            float thr = kNegInf;
            for (int64_t t = it.t0; t < it.t1; ++t, ++lt) {
                const uint32_t buf = lt & 1u, use = lt >> 1;
                if (!mbar_wait(smem_addr(&sh->tfull[buf]), use & 1u, p.timeout_ns)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const int64_t n0 = t * kTcTileN;
                const bool tail = n0 + kTcTileN > p.N;
#pragma unroll 1
                for (int c = 0; c < kTcTileN / 32; ++c) {
                    uint32_t v[32];
                    tmem_ld_32x32b_x32(tmem + lane_addr + buf * kTcTileN + c * 32, v);
                    tmem_ld_wait(v);
                    const uint32_t id0 = (uint32_t)(n0 + c * 32);
                    if (tail) {
#pragma unroll
                        for (int j = 0; j < 32; ++j)
                            if ((int64_t)id0 + j >= p.N) v[j] = 0xFF800000u;
                    }
                    if (row_valid && fmax32(v) > thr) {
#pragma unroll
                        for (int j = 0; j < 32; ++j) {
                            const float sj = __uint_as_float(v[j]);
                            if (sj > thr) {
                                const uint64_t kth = insert_key(list, nfill, p.k, make_key(sj, id0 + j));
                                if (nfill < p.k) ++nfill;
                                thr = kth ? key_score(kth) : kNegInf;
                            }
                        }
                    }
                }
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(smem_addr(&sh->tempty[buf]));
            }
            if (row_valid)
                for (int t = nfill; t < p.k; ++t) list[t] = 0ull;
        }
        if (!ok && lane == 0) atomicOr(p.err, kErrTimeout);
    }

    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 1) {
        __syncwarp();
        tmem_dealloc(tmem, kTmemCols);
    }
}

}  // namespace

size_t tc_smem_bytes() { return 1024 + (size_t)kTcStages * kStageBytes + sizeof(TcShared); }

cudaError_t launch_tc(const CUtensorMap &tq, const CUtensorMap &tx, const TcParams &p, int grid,
                      cudaStream_t s) {
    const size_t smem = tc_smem_bytes();
    cudaError_t e = cudaFuncSetAttribute(k_tc_score_topk, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess) return e;
    k_tc_score_topk<<<grid, kTcThreads, smem, s>>>(tq, tx, p);
    return cudaGetLastError();
}

}  // namespace skipk
