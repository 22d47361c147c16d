// Tensor-core score + fused top-k (tcgen05 / TMEM / TMA, sm_103a).
//
// Step: per-region MIPS top-k over the corpus (paper App. B.2 Def. B.2,
// MIPS(q_r, D; k_r); §3.3 Eq. rcsr).  For a batch of region queries the
// scores S = Q X^T are a dense bf16 contraction with fp32 accumulation; this
// kernel computes them on the 5th-generation tensor cores and never writes
// them to HBM: the epilogue reads each accumulator tile out of tensor memory
// and keeps, per region row, a sorted top-k list and its k-th score.
//
// Tile: 128 region rows per CTA (TMEM lanes) x 256 corpus rows (TMEM
// columns), K streamed in 64-element (128-byte) slices.  One thread of the
// epilogue owns one region row, so its threshold lives in a register and the
// common case -- no score of a 32-column chunk beats it -- costs a max and a
// compare per chunk.  Corpus rows of a tile are visited in increasing id
// order, so "beats" is a strict score comparison and ties keep the lower id.
//
// Two MMA shapes:
//  * single CTA (cta_group::1, M = 128): the CTA stages its 128 region rows
//    and the whole 256-row corpus tile itself (CTAs of other query blocks
//    that read the same tile find it in L2);
//  * CTA pair (cta_group::2, M = 256): a cluster of two CTAs on two SMs
//    computes 256 region rows (two query blocks) against a 256-row corpus
//    tile, each CTA staging its own 128 region rows and half of the corpus
//    tile (32 KB per 64-wide slice instead of 48 KB), which buys a deeper
//    pipeline for the same shared memory.  One thread of the even CTA
//    issues the MMAs; both CTAs' copies complete on the even CTA's barrier,
//    its commits are multicast to both CTAs, and both CTAs' epilogues hand
//    the accumulator back to it.
//
// Work: persistent clusters take items (query group, corpus chunk) from a
// counter shared by the grid, one at a time; items are numbered
// chunk-major, so the clusters at work hold the query groups of one or two
// chunks and each corpus tile, read once from HBM, serves the others from
// L2.  Each item leaves one sorted list per region row; the merge kernel
// combines the chunks.
//
// The k-th best score of any chunk of a row bounds the row's global top-k
// from below, so the chunks of a row share one threshold: each CTA publishes
// its chunk's k-th score with an atomic max on the order-preserving integer
// and re-reads the row's best once per tile; a score is kept only if it
// beats its own chunk's k-th score and is not below the shared one (equal
// scores from another chunk may still win on id).
//
// Per-row top-k sets live in shared memory ([slot][row], k slots) when they
// fit next to a pipeline of at least two stages, else in global memory; a
// set is unsorted with its smallest key tracked, and sorted at chunk end
// (in registers when it holds at most 32 keys); a list shorter than k ends
// with an empty key, which is as far as the merge reads.
//
// Resident query block (CTA pair, d <= 512, sets in global memory): each CTA
// keeps its 128 region rows x d for the whole item in shared memory (loaded
// once per item, released by an MMA commit when the item's last MMA is
// done) and the ring carries only corpus slices, which halves the bytes
// moved from L2 per tile.  Used with the bounding pass, which keeps the sets
// short enough that they rarely fill (so rarely need a rescan from L2).
//
// Warp roles (192 threads): warp 0 issues TMA loads into the shared-memory
// ring; warp 1 owns TMEM (two 256-column fp32 accumulators) and issues
// tcgen05.mma from one thread; warps 2..5 are the epilogue, warp w reading
// TMEM lanes 32 * (w % 4) .. + 31.  Every wait is bounded; a wait that gives
// up sets the error word, the other roles then give up too, and before exit
// the producer waits for its copies in flight and the MMA thread for its
// MMAs, and the cluster synchronises, so that TMEM is freed with nothing
// outstanding.
#include "skip_device.cuh"
#include "skip_internal.h"
#include "tc_common.cuh"

namespace skipk {
namespace {

using namespace tc;

constexpr int kABytes = kTcTileM * kTcTileK * 2;  // 16 KB: 128 region rows x 64
constexpr int kBFull = kTcTileN * kTcTileK * 2;   // 32 KB: 256 corpus rows x 64
constexpr uint32_t kTmemCols = 512;               // two 256-column accumulators
constexpr uint64_t kDrainTimeoutNs = 1000000000ull;  // 1 s for copies/MMAs in flight
constexpr int kMaxStages = 8;
constexpr int kSchedQ = 4;  // work items published ahead of the slowest role

template <bool PAIR>
struct Geom {
    static constexpr int kBBytes = PAIR ? kBFull / 2 : kBFull;  // corpus rows staged by one CTA
    static constexpr int kStageBytes = kABytes + kBBytes;       // per CTA and stage
    static constexpr uint32_t kTxBytes = PAIR ? 2 * kStageBytes : kStageBytes;  // on the MMA CTA's barrier
    static constexpr uint32_t kIdesc = idesc_bf16_f32(PAIR ? 2 * kTcTileM : kTcTileM, kTcTileN);
    static constexpr int kMaxSt = PAIR ? 6 : 4;
};

struct __align__(8) TcShared {
    uint64_t full[kMaxStages];   // stage loaded (TMA transaction bytes)
    uint64_t empty[kMaxStages];  // stage consumed (tcgen05.commit)
    uint64_t tfull[2];           // accumulator ready (tcgen05.commit)
    uint64_t tempty[2];          // accumulator drained (epilogue warps)
    uint64_t drain;              // MMA completion at exit
    uint64_t afull, aempty;      // resident query block loaded / released
    uint64_t sfull[kSchedQ];     // work item published (the pair's MMA CTA publishes to both CTAs)
    uint64_t sempty[kSchedQ];    // ... taken by every role of the pair
    int sched[kSchedQ];          // item index, -1 = no more work
    uint32_t tmem_base;
};

template <bool PAIR>
__global__ void __launch_bounds__(kTcThreads, 1)
    k_tc_score_topk(const __grid_constant__ CUtensorMap tq, const __grid_constant__ CUtensorMap tx,
                    const TcParams p) {
    using Gm = Geom<PAIR>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    const int S = p.stages;
    const int KB = (p.d + kTcTileK - 1) / kTcTileK;
    const bool ar = PAIR && p.a_res;  // query block resident for the item; ring = corpus slices only
    uint8_t *sA = smem;
    uint8_t *sB = ar ? smem + KB * kABytes : smem + S * kABytes;
    const size_t ring_bytes = ar ? (size_t)KB * kABytes + (size_t)S * Gm::kBBytes : (size_t)S * Gm::kStageBytes;
    uint64_t *slists = reinterpret_cast<uint64_t *>(smem + ring_bytes);
    const size_t list_bytes = p.list_in_smem ? (size_t)kTcTileM * p.k * 8 : 0;
    TcShared *sh = reinterpret_cast<TcShared *>(smem + ring_bytes + list_bytes);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int items = p.QG * p.G;
    // A pair is a cluster of two CTAs; a single-CTA launch has no clusters.
    const int rank = PAIR ? (int)cluster_rank() : 0;
    const bool mma_cta = !PAIR || rank == 0;

    // Work items are handed out dynamically: the MMA CTA's producer takes the
    // next index from a counter shared by the grid and publishes it to every
    // role of the pair through a small ring in shared memory, so that the
    // CTAs at work always hold nearly consecutive items (the query groups of
    // one corpus chunk, which then find its tiles in L2).
    auto sched_take = [&](uint32_t n, int &v) -> bool {
        const int j = (int)(n % kSchedQ);
        if (!mbar_wait_cluster(smem_addr(&sh->sfull[j]), (n / kSchedQ) & 1u, p.timeout_ns)) return false;
        v = *reinterpret_cast<volatile int *>(&sh->sched[j]);
        return true;
    };
    auto sched_release = [&](uint32_t n) {
        const uint32_t e = smem_addr(&sh->sempty[n % kSchedQ]);
        if (PAIR && rank != 0)
            mbar_arrive_cluster(mapa_shared(e, 0));
        else
            mbar_arrive(e);
    };
    auto sched_publish = [&](uint32_t n, int &v) -> bool {
        const int j = (int)(n % kSchedQ);
        if (!mbar_wait_cluster(smem_addr(&sh->sempty[j]), ((n / kSchedQ) & 1u) ^ 1u, p.timeout_ns)) return false;
        const int x = atomicAdd(p.sched, 1);
        v = x < items ? x : -1;
        sh->sched[j] = v;
        mbar_arrive(smem_addr(&sh->sfull[j]));
        if constexpr (PAIR) {
            st_shared_cluster_u32(mapa_shared(smem_addr(&sh->sched[j]), 1), (uint32_t)v);
            mbar_arrive_cluster(mapa_shared(smem_addr(&sh->sfull[j]), 1));
        }
        return true;
    };

    if (threadIdx.x == 0) {
        for (int s = 0; s < S; ++s) {
            mbar_init(smem_addr(&sh->full[s]), 1);
            mbar_init(smem_addr(&sh->empty[s]), 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(smem_addr(&sh->tfull[b]), 1);
            mbar_init(smem_addr(&sh->tempty[b]), PAIR ? 8 : 4);
        }
        mbar_init(smem_addr(&sh->drain), 1);
        mbar_init(smem_addr(&sh->afull), 1);
        mbar_init(smem_addr(&sh->aempty), 1);
        for (int j = 0; j < kSchedQ; ++j) {
            mbar_init(smem_addr(&sh->sfull[j]), 1);
            // takers: the MMA thread and the epilogue warps (and, in a pair,
            // the other CTA's epilogue warps and producer)
            mbar_init(smem_addr(&sh->sempty[j]), PAIR ? 10 : 5);
        }
        mbar_fence_init();
    }
    if (warp == 0 && lane == 0) {
        tma_prefetch_desc(&tq);
        tma_prefetch_desc(&tx);
    }
    if (warp == 1) {
        if constexpr (PAIR) {
            tmem_alloc_pair(smem_addr(&sh->tmem_base), kTmemCols);
            tmem_relinquish_pair();
        } else {
            tmem_alloc(smem_addr(&sh->tmem_base), kTmemCols);
            tmem_relinquish();
        }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    // Every CTA's barriers are initialised before any peer copy or arrive.
    if constexpr (PAIR) cluster_sync_all();
    const uint32_t tmem = sh->tmem_base;

    if (warp == 0) {
        // ------------------------------------------------ TMA producer
        if (lane == 0) {
            int s = 0;
            uint32_t ph = 0;
            int64_t issued = 0;
            bool ok = true;
            uint32_t na = 0;  // query blocks loaded (resident mode)
            for (uint32_t n = 0; ok; ++n) {
                int v = -1;
                if (mma_cta) {
                    if (!sched_publish(n, v)) {
                        ok = false;
                        break;
                    }
                } else {
                    if (!sched_take(n, v)) {
                        ok = false;
                        break;
                    }
                    sched_release(n);
                }
                if (v < 0) break;
                const Item it = item_of(p, v, rank);
                if (ar) {
                    // The previous item's MMAs have released the block: load
                    // this item's, both CTAs' copies counted on the MMA CTA.
                    if (!mbar_wait(smem_addr(&sh->aempty), (na & 1u) ^ 1u, p.timeout_ns)) {
                        ok = false;
                        break;
                    }
                    const uint32_t fa = smem_addr(&sh->afull);
                    if (mma_cta) mbar_arrive_expect_tx(fa, (uint32_t)(2 * KB * kABytes));
                    for (int kb = 0; kb < KB; ++kb)
                        tma_load_2d_pair(smem_addr(sA + kb * kABytes), &tq, mapa_shared(fa, 0), kb * kTcTileK,
                                         it.mb * kTcTileM);
                    ++na;
                }
                for (int64_t t = it.t0; t < it.t1 && ok; ++t) {
                    for (int kb = 0; kb < KB; ++kb) {
                        if (!mbar_wait(smem_addr(&sh->empty[s]), ph ^ 1u, p.timeout_ns)) {
                            ok = false;
                            break;
                        }
                        const uint32_t fb = smem_addr(&sh->full[s]);
                        if (mma_cta) mbar_arrive_expect_tx(fb, ar ? 2u * Gm::kBBytes : Gm::kTxBytes);
                        const int x = kb * kTcTileK;
                        if constexpr (PAIR) {
                            // Both CTAs' copies complete on the MMA CTA's barrier.
                            const uint32_t fl = mapa_shared(fb, 0);
                            if (!ar) tma_load_2d_pair(smem_addr(sA + s * kABytes), &tq, fl, x, it.mb * kTcTileM);
                            tma_load_2d_pair(smem_addr(sB + s * Gm::kBBytes), &tx, fl, x,
                                             (int)(t * p.tile_stride * kTcTileN) + rank * (kTcTileN / 2));
                        } else {
                            tma_load_2d(smem_addr(sA + s * kABytes), &tq, fb, x, it.mb * kTcTileM);
                            tma_load_2d(smem_addr(sB + s * Gm::kBBytes), &tx, fb, x,
                                        (int)(t * p.tile_stride * kTcTileN));
                        }
                        ++issued;
                        if (++s == S) {
                            s = 0;
                            ph ^= 1u;
                        }
                    }
                }
            }
            if (!ok) atomicOr(p.err, kErrTimeout);
            // Copies in flight: wait for the last load issued on every stage.
            // In a pair both CTAs' copies complete on the MMA CTA's barrier, so
            // the other CTA waits instead for the release of its last stages
            // (which follows their arrival); a release that never comes ends
            // the wait after the bound, long after any copy has landed.
            for (int st = 0; st < S; ++st) {
                const int64_t uses = issued / S + (st < issued % S ? 1 : 0);
                if (uses == 0) continue;
                const uint32_t bar = mma_cta ? smem_addr(&sh->full[st]) : smem_addr(&sh->empty[st]);
                if (!mbar_wait(bar, (uint32_t)((uses - 1) & 1), kDrainTimeoutNs)) atomicOr(p.err, kErrTimeout);
            }
            if (ar && na > 0) {
                // the last query block: its arrival (MMA CTA) or its release
                const uint32_t bar = mma_cta ? smem_addr(&sh->afull) : smem_addr(&sh->aempty);
                if (!mbar_wait(bar, (na - 1) & 1u, kDrainTimeoutNs)) atomicOr(p.err, kErrTimeout);
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------ MMA issuer
        if (lane == 0 && mma_cta) {
            int s = 0;
            uint32_t ph = 0;
            uint32_t lt = 0;
            bool ok = true;
            uint32_t na = 0;  // query blocks used (resident mode)
            for (uint32_t n = 0; ok; ++n) {
                int v = -1;
                if (!sched_take(n, v)) {
                    ok = false;
                    break;
                }
                sched_release(n);
                if (v < 0) break;
                const Item it = item_of(p, v, rank);
                if (ar) {
                    if (!mbar_wait(smem_addr(&sh->afull), na & 1u, p.timeout_ns)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                }
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
                        const uint64_t ad = smem_desc_k128(smem_addr(sA + (ar ? kb : s) * kABytes));
                        const uint64_t bd = smem_desc_k128(smem_addr(sB + s * Gm::kBBytes));
#pragma unroll
                        for (int kk = 0; kk < kTcTileK / 16; ++kk) {
                            if constexpr (PAIR)
                                tc_mma_f16_pair(dt, ad + (uint64_t)(kk * 2), bd + (uint64_t)(kk * 2), Gm::kIdesc,
                                                (kb | kk) != 0);
                            else
                                tc_mma_f16(dt, ad + (uint64_t)(kk * 2), bd + (uint64_t)(kk * 2), Gm::kIdesc,
                                           (kb | kk) != 0);
                        }
                        if constexpr (PAIR)
                            tc_commit_pair_mc(smem_addr(&sh->empty[s]), 3);
                        else
                            tc_commit(smem_addr(&sh->empty[s]));
                        if (++s == S) {
                            s = 0;
                            ph ^= 1u;
                        }
                    }
                    if (!ok) break;
                    if constexpr (PAIR)
                        tc_commit_pair_mc(smem_addr(&sh->tfull[buf]), 3);
                    else
                        tc_commit(smem_addr(&sh->tfull[buf]));
                }
                if (ar && ok) {
                    // the block is free once this item's MMAs are done
                    if constexpr (PAIR) tc_commit_pair_mc(smem_addr(&sh->aempty), 3);
                    ++na;
                }
            }
            if (!ok) atomicOr(p.err, kErrTimeout);
            // MMAs in flight: a commit arrives once all earlier ones are done.
            if constexpr (PAIR)
                tc_commit_pair_mc(smem_addr(&sh->drain), 3);
            else
                tc_commit(smem_addr(&sh->drain));
            if (!mbar_wait(smem_addr(&sh->drain), 0, kDrainTimeoutNs)) atomicOr(p.err, kErrTimeout);
        } else if (lane == 0 && PAIR) {
            // The other CTA of the pair: its TMEM is written by the MMA CTA.
            if (!mbar_wait(smem_addr(&sh->drain), 0, kDrainTimeoutNs)) atomicOr(p.err, kErrTimeout);
        }
    } else {
        // ------------------------------------------------ epilogue
        // The shared thresholds may come from the grid before this one (the
        // bounding pass's merge, launched as its programmatic dependent):
        // the TMA and MMA roles start at once, the epilogue waits for it.
        grid_dep_wait();
        const int sub = warp & 3;
        const int rib = sub * 32 + lane;  // region row within the query block
        const uint32_t lane_addr = (uint32_t)(sub * 32) << 16;
        const float kNegInf = -__int_as_float(0x7f800000);
        uint32_t lt = 0;
        bool ok = true;
        for (uint32_t n = 0; ok; ++n) {
            int v = -1;
            const bool got_item = sched_take(n, v);
            if (!__all_sync(0xffffffffu, got_item)) {
                ok = false;
                break;
            }
            __syncwarp();
            if (lane == 0) sched_release(n);
            if (v < 0) break;
            const Item it = item_of(p, v, rank);
            const int row = it.mb * kTcTileM + rib;
            const bool row_valid = it.mb < p.MB && row < p.R;
            uint64_t *glist = p.lists + ((int64_t)it.g * p.R_pad + row) * p.k;
            uint64_t *L = p.list_in_smem ? slists + rib : glist;
            const int ls = p.list_in_smem ? kTcTileM : 1;
            RowTopK top;
            float thr = kNegInf;   // this chunk's k-th score (strict: later ids lose ties)
            float gthr = kNegInf;  // best k-th score any chunk of this row has found
            uint32_t published = 0;
            uint32_t *tau = p.tau + row;
            // The shared threshold is read one tile ahead, off the critical path.
            uint32_t tau_next = row_valid && p.share ? *reinterpret_cast<volatile uint32_t *>(tau) : 0u;
            // Common case: no score of 64 columns beats the threshold of any
            // row of the warp (a max and a warp vote).  Otherwise, per 32
            // columns, a branch-free bit mask of the survivors is walked in
            // increasing column (= id) order, so that lanes without
            // survivors idle for a few instructions only.
            // One compare per score: s > thr and s >= gthr is s > cthr
            // (padding columns hold -inf and never pass).
            float gbelow = kNegInf, cthr = kNegInf;
            // dense (a bounding pass with four-slot lists): the row's four
            // largest scores of the chunk, kept sorted in registers
            // (d4[0] >= .. >= d4[3]); each score that beats d4[3] is bubbled in
            float d4[4] = {kNegInf, kNegInf, kNegInf, kNegInf};
            auto dense32 = [&](const uint32_t (&vv)[32]) {
#pragma unroll
                for (int j = 0; j < 32; ++j) {
                    const float x = __uint_as_float(vv[j]);
                    const float m1 = fminf(d4[0], x);
                    d4[0] = fmaxf(d4[0], x);
                    const float m2 = fminf(d4[1], m1);
                    d4[1] = fmaxf(d4[1], m1);
                    const float m3 = fminf(d4[2], m2);
                    d4[2] = fmaxf(d4[2], m2);
                    d4[3] = fmaxf(d4[3], m3);
                }
            };
            auto scan32 = [&](uint32_t (&vv)[32], uint32_t id0) {
                if (!row_valid) return;
                const float mx = fmax32(vv);
                if (!(mx > cthr)) return;
                uint32_t m = 0;
#pragma unroll
                for (int j = 0; j < 32; ++j) m |= (__uint_as_float(vv[j]) > cthr ? 1u : 0u) << j;
                while (m) {
                    const int j = __ffs(m) - 1;
                    m &= m - 1;
                    const float sj = __uint_as_float(select32(vv, j));
                    if (sj > thr) {
                        topk_add(L, ls, p.k, top, make_key(sj, id0 + j));
                        if (top.n == p.k) {
                            thr = key_score(top.min_key);
                            cthr = fmaxf(thr, gbelow);
                        }
                    }
                }
            };
            for (int64_t t = it.t0; t < it.t1; ++t, ++lt) {
                const uint32_t buf = lt & 1u, use = lt >> 1;
                // The warp gives up together, so that its vote below stays
                // convergent.
                const bool got = mbar_wait(smem_addr(&sh->tfull[buf]), use & 1u, p.timeout_ns);
                if (!__all_sync(0xffffffffu, got)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                if (row_valid && p.share) {
                    // Publish this chunk's k-th score, then adopt the row's best.
                    const uint32_t mine = top.n == p.k ? ord_of_score(thr) : 0u;
                    if (mine > published) {
                        atomicMax(tau, mine);
                        published = mine;
                    }
                    if (tau_next > published) {
                        gthr = score_of_ord(tau_next);
                        gbelow = float_below(gthr);
                        cthr = fmaxf(thr, gbelow);
                    }
                    tau_next = *reinterpret_cast<volatile uint32_t *>(tau);
                }
                const int64_t n0 = t * p.tile_stride * kTcTileN;
                const bool tail = n0 + kTcTileN > p.N;
#pragma unroll 1
                for (int c = 0; c < kTcTileN / 64; ++c) {
                    uint32_t v0[32], v1[32];
                    const uint32_t taddr = tmem + lane_addr + buf * kTcTileN + c * 64;
                    tmem_ld_32x32b_x32(taddr, v0);
                    tmem_ld_32x32b_x32(taddr + 32, v1);
                    tmem_ld_wait(v0);
                    regs_after_wait(v1);
                    const uint32_t id0 = (uint32_t)(n0 + c * 64);
                    if (tail) {
#pragma unroll
                        for (int j = 0; j < 32; ++j) {
                            if ((int64_t)id0 + j >= p.N) v0[j] = 0xFF800000u;
                            if ((int64_t)id0 + 32 + j >= p.N) v1[j] = 0xFF800000u;
                        }
                    }
                    if (c == kTcTileN / 64 - 1) {
                        // Last read of this accumulator: hand it back before scanning.
                        tc_fence_before();
                        __syncwarp();
                        if (lane == 0) {
                            const uint32_t te = smem_addr(&sh->tempty[buf]);
                            if (PAIR && rank != 0)
                                mbar_arrive_cluster(mapa_shared(te, 0));
                            else
                                mbar_arrive(te);
                        }
                    }
                    const float mx = fmaxf(fmax32(v0), fmax32(v1));
                    if (p.dense) {
                        if (__any_sync(0xffffffffu, row_valid && mx > d4[3])) {
                            dense32(v0);
                            dense32(v1);
                        }
                    } else if (__any_sync(0xffffffffu, row_valid && mx > cthr)) {
                        scan32(v0, id0);
                        scan32(v1, id0 + 32);
                    }
                }
            }
            if (row_valid && p.dense) {
                // scores only: the ids stand for four distinct rows of this chunk
#pragma unroll
                for (int t = 0; t < 4; ++t)
                    glist[t] = d4[t] > kNegInf ? make_key(d4[t], (uint32_t)(it.g * 4 + t)) : 0ull;
            } else if (row_valid) {
                if (!p.list_in_smem && top.n <= 16) {
                    sortw_desc_in_place<16>(glist, top.n);
                } else if (!p.list_in_smem && top.n <= 32) {
                    sortw_desc_in_place<32>(glist, top.n);
                } else {
                    topk_sort(L, ls, top.n);
                    if (p.list_in_smem)
                        for (int t = 0; t < top.n; ++t) glist[t] = L[t * ls];
                }
                if (top.n < p.k) glist[top.n] = 0ull;  // end of a short list
            }
        }
        if (!ok && lane == 0) atomicOr(p.err, kErrTimeout);
    }

    tc_fence_before();
    __syncthreads();
    // No peer may still copy into, arrive on, or (pair) write the TMEM of
    // this CTA when it frees TMEM and exits.
    if constexpr (PAIR) cluster_sync_all();
    tc_fence_after();
    if (warp == 1) {
        __syncwarp();
        if constexpr (PAIR)
            tmem_dealloc_pair(tmem, kTmemCols);
        else
            tmem_dealloc(tmem, kTmemCols);
    }
}

template <bool PAIR>
size_t smem_bytes(int stages, int k, bool list_in_smem, int a_res_slices) {
    const size_t ring = a_res_slices > 0 ? (size_t)a_res_slices * kABytes + (size_t)stages * Geom<PAIR>::kBBytes
                                         : (size_t)stages * Geom<PAIR>::kStageBytes;
    return 1024 + ring + (list_in_smem ? (size_t)kTcTileM * k * 8 : 0) + sizeof(TcShared);
}

cudaLaunchConfig_t tc_config(int grid, int CL, size_t smem, cudaStream_t s, cudaLaunchAttribute *attr,
                             bool pdl = false) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid, 1, 1);
    cfg.blockDim = dim3(kTcThreads, 1, 1);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = CL;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl ? 2 : 1;
    return cfg;
}

}  // namespace

size_t tc_smem_bytes(bool pair, int stages, int k, bool list_in_smem, int a_res_slices) {
    return pair ? smem_bytes<true>(stages, k, list_in_smem, a_res_slices)
                : smem_bytes<false>(stages, k, list_in_smem, 0);
}

void tc_pick_layout(bool pair, int k, int max_smem, int *stages, bool *list_in_smem) {
    const int top = pair ? Geom<true>::kMaxSt : Geom<false>::kMaxSt;
    for (int st = top; st >= 2; --st)
        if (tc_smem_bytes(pair, st, k, true, 0) <= (size_t)max_smem) {
            *stages = st;
            *list_in_smem = true;
            return;
        }
    *stages = 4;
    *list_in_smem = false;
}

int tc_pick_resident_stages(int d, int max_smem) {
    const int KB = (d + kTcTileK - 1) / kTcTileK;
    if (KB > kMaxResidentSlices) return 0;
    for (int st = Geom<true>::kMaxSt; st >= 3; --st)
        if (tc_smem_bytes(true, st, 0, false, KB) <= (size_t)max_smem) return st;
    return 0;
}

int tc_max_clusters(bool pair, int CL, int stages, int k, bool list_in_smem, int a_res_slices) {
    const size_t smem = tc_smem_bytes(pair, stages, k, list_in_smem, a_res_slices);
    auto kern = pair ? k_tc_score_topk<true> : k_tc_score_topk<false>;
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess) {
        cudaGetLastError();
        return 0;
    }
    cudaLaunchAttribute attr[2];
    cudaLaunchConfig_t cfg = tc_config(CL * 64, CL, smem, 0, attr);
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, kern, &cfg) != cudaSuccess) {
        cudaGetLastError();
        return 0;
    }
    return n;
}

cudaError_t launch_tc(bool pair, const CUtensorMap &tq, const CUtensorMap &tx, const TcParams &p, int grid,
                      cudaStream_t s, bool pdl) {
    if (p.CL != (pair ? 2 : 1)) return cudaErrorInvalidValue;
    if (p.a_res && (!pair || p.list_in_smem)) return cudaErrorInvalidValue;
    const int slices = p.a_res ? (p.d + kTcTileK - 1) / kTcTileK : 0;
    if (slices > kMaxResidentSlices) return cudaErrorInvalidValue;
    const size_t smem = tc_smem_bytes(pair, p.stages, p.k, p.list_in_smem != 0, slices);
    auto kern = pair ? k_tc_score_topk<true> : k_tc_score_topk<false>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    cudaLaunchAttribute attr[2];
    cudaLaunchConfig_t cfg = tc_config(grid, p.CL, smem, s, attr, pdl);
    return cudaLaunchKernelEx(&cfg, kern, tq, tx, p);
}

}  // namespace skipk
