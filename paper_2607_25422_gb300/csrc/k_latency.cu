// Tensor-core score + fused top-k for small region batches (latency mode).
//
// Step: per-region MIPS top-k (paper App. B.2 Def. B.2, MIPS(q_r, D; k_r);
// §3.3 Eq. rcsr) when a batch holds at most 32 region rows -- one question
// with its regions, the paper's serving case.  Such a scan is bound by
// streaming the corpus from HBM, so the corpus tile is the streamed MMA
// operand A (128 corpus rows = 128 TMEM lanes) and the region queries are a
// small operand B that stays in shared memory for the whole launch: the MMA
// D = X_tile Q^T leaves, in each TMEM lane, one corpus row's scores against
// every query.
//
// e4m3 corpus: the tensor cores take e4m3 directly (kind::f8f6f4), so the
// corpus tile is never widened; instead each bf16 query q is split once per
// call into three e4m3 parts with power-of-two scales,
//     q ~= s0 a + s1 b + s2 c,   a = e4m3(q / s0), b = e4m3((q - s0 a) / s1), ...
// each part capturing the previous residual to 4 significant bits, so the
// remainder is below 2^-12 |q| per element and the score differs from the
// exact one by less than 2^-12 |q| |x| (unit vectors: 2.5e-4).  Part p of
// query r is row 32 p + r of B (96 rows); the epilogue combines the three
// 32-column groups, times the corpus row's scale.  Products of e4m3 values
// are exact in the fp32 accumulator.
// bf16 corpus: B is the bf16 queries themselves (kind::f16).
//
// Epilogue: lane = corpus row, so for each query the 32 rows of a warp are
// compared with the query's filter at once (a ballot); lane q owns the
// running top-k set of query q for its warp's rows (bf16 with k <= 16: a
// sorted array in registers; else an unsorted set with its minimum tracked,
// in shared memory) and inserts the ballot's survivors in increasing row
// (= id) order.  Eight epilogue warps in two sets of four
// drain the two TMEM accumulators in turn (set j takes the tiles that land
// in accumulator j), so that the survivor work of one tile overlaps the
// ballots of the next.  A query's filter is the largest of its own set's
// k-th score, the k-th scores of the CTA's other warps' sets (each is k
// distinct rows' scores, so a score below it cannot reach the CTA's top k)
// and a threshold shared by all CTAs (atomic max of the sets' k-th scores).
// At the end of a chunk the eight warps' sets of each query are merged into
// the chunk's list.
//
// Warps (320 threads): 0 TMA producer, 1 TMEM owner and MMA issuer, 2..9
// epilogue.  Bounded waits and drains as in the other tensor kernels.
#include "skip_device.cuh"
#include "skip_internal.h"
#include "tc_common.cuh"

namespace skipk {
namespace {

using namespace tc;

constexpr int kRows = 128;                      // corpus rows per tile
constexpr int kSlice = 128;                     // bytes of a row per K slice
constexpr int kAStage = kRows * kSlice;         // 16 KB
constexpr int kMaxStages = 12;
constexpr int kEpiWarps = 8;                    // two sets of four
constexpr int kThreads = 64 + 32 * kEpiWarps;
constexpr uint32_t kTmemCols = 256;             // two 128-column accumulators
constexpr uint64_t kDrainTimeoutNs = 1000000000ull;

struct __align__(8) LatShared {
    uint64_t full[kMaxStages];
    uint64_t empty[kMaxStages];
    uint64_t bfull;  // resident query operand loaded
    uint64_t tfull[2];
    uint64_t tempty[2];
    uint64_t drain;
    uint64_t sorted;  // the epilogue threads have sorted their sets
    uint64_t halved;  // register-set path: eight sets merged pairwise into four ...
    uint64_t quartered;  // ... and into two
    uint64_t merged;  // ... and merged them into the chunk's lists
    uint32_t tmem_base;
    float qscale[3][kLatMaxR];
    float thr[kEpiWarps][32];   // per epilogue warp: each query's set threshold (k-th score)
    float filt[kEpiWarps][32];  // ... and the filter its next ballots use (strict compare)
};

// Running top-k of one query in registers (k <= KM): ascending, a[0] the
// k-th best key (0 while fewer than k keys are held), a[i] = ~0 for i >= k.
// Inserting x drops a[0]: a[i] <- max(a[i], min(x, a[i + 1])) (a[KM] = ~0)
// shifts the keys below x down one place and puts x in its slot; with
// x <= a[0] every a[i] stays as it is, so the network runs unconditionally
// on max(x, a[0]).  Straight-line code on registers: no shared-memory
// round trips per key.
template <int KM>
__device__ __forceinline__ void regset_insert(uint64_t (&a)[KM], uint64_t x) {
    x = x > a[0] ? x : a[0];
#pragma unroll
    for (int i = 0; i < KM - 1; ++i) {
        const uint64_t t = x < a[i + 1] ? x : a[i + 1];
        a[i] = a[i] > t ? a[i] : t;
    }
    a[KM - 1] = a[KM - 1] > x ? a[KM - 1] : x;
}

// The k-th largest (k <= 16) of the 16 pair maxima max(s_j, s_{j+16}) over
// the rows j of mask m (others -inf); s_j = col[33 j].  The pair maxima are
// sorted descending by a bitonic network on sixteen named registers (an
// array here was placed in local memory).
#define CED(a, b) { const float x_ = a, y_ = b; a = fmaxf(x_, y_); b = fminf(x_, y_); }
#define CEA(a, b) { const float x_ = a, y_ = b; a = fminf(x_, y_); b = fmaxf(x_, y_); }
__device__ __forceinline__ float pair_max_bound(const float *col, uint32_t m, int k) {
    const float ninf = -__int_as_float(0x7f800000);
#define PM(j) const float a##j = (m >> j) & 1u ? col[j * 33] : ninf, b##j = (m >> (j + 16)) & 1u ? col[(j + 16) * 33] : ninf; \
    float g##j = fmaxf(a##j, b##j);
    PM(0) PM(1) PM(2) PM(3) PM(4) PM(5) PM(6) PM(7)
    PM(8) PM(9) PM(10) PM(11) PM(12) PM(13) PM(14) PM(15)
#undef PM
    CED(g0, g1); CEA(g2, g3); CED(g4, g5); CEA(g6, g7);
    CED(g8, g9); CEA(g10, g11); CED(g12, g13); CEA(g14, g15);
    CED(g0, g2); CED(g1, g3); CEA(g4, g6); CEA(g5, g7);
    CED(g8, g10); CED(g9, g11); CEA(g12, g14); CEA(g13, g15);
    CED(g0, g1); CED(g2, g3); CEA(g4, g5); CEA(g6, g7);
    CED(g8, g9); CED(g10, g11); CEA(g12, g13); CEA(g14, g15);
    CED(g0, g4); CED(g1, g5); CED(g2, g6); CED(g3, g7);
    CEA(g8, g12); CEA(g9, g13); CEA(g10, g14); CEA(g11, g15);
    CED(g0, g2); CED(g1, g3); CED(g4, g6); CED(g5, g7);
    CEA(g8, g10); CEA(g9, g11); CEA(g12, g14); CEA(g13, g15);
    CED(g0, g1); CED(g2, g3); CED(g4, g5); CED(g6, g7);
    CEA(g8, g9); CEA(g10, g11); CEA(g12, g13); CEA(g14, g15);
    CED(g0, g8); CED(g1, g9); CED(g2, g10); CED(g3, g11);
    CED(g4, g12); CED(g5, g13); CED(g6, g14); CED(g7, g15);
    CED(g0, g4); CED(g1, g5); CED(g2, g6); CED(g3, g7);
    CED(g8, g12); CED(g9, g13); CED(g10, g14); CED(g11, g15);
    CED(g0, g2); CED(g1, g3); CED(g4, g6); CED(g5, g7);
    CED(g8, g10); CED(g9, g11); CED(g12, g14); CED(g13, g15);
    CED(g0, g1); CED(g2, g3); CED(g4, g5); CED(g6, g7);
    CED(g8, g9); CED(g10, g11); CED(g12, g13); CED(g14, g15);
    float T = g0;
#define PICK(j) T = (j == k - 1) ? g##j : T;
    PICK(1) PICK(2) PICK(3) PICK(4) PICK(5) PICK(6) PICK(7) PICK(8)
    PICK(9) PICK(10) PICK(11) PICK(12) PICK(13) PICK(14) PICK(15)
#undef PICK
    return T;
}
#undef CED
#undef CEA

// KM > 0: the epilogue keeps each query's set in registers (k <= KM);
// KM == 0: in shared memory (any k).
template <bool FP8, int KM>
__global__ void __launch_bounds__(kThreads, 1)
    k_latency_score_topk(const __grid_constant__ CUtensorMap ta, const __grid_constant__ CUtensorMap tb,
                         const LatParams p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    const int S = p.stages;
    const int KS = p.slices;                 // K slices per corpus row
    const int bslice = p.Npad * kSlice;      // bytes of one resident B slice
    uint8_t *sB = smem;
    uint8_t *sA = sB + KS * bslice;
    uint64_t *slists = reinterpret_cast<uint64_t *>(sA + S * kAStage);
    float *strans = reinterpret_cast<float *>(slists + (size_t)kEpiWarps * p.R * p.k);  // [8][32][33]
    LatShared *sh = reinterpret_cast<LatShared *>(strans + kEpiWarps * 32 * 33);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    constexpr int kElemsPerSlice = FP8 ? 128 : 64;
    constexpr uint32_t kIdescBase = FP8 ? idesc_e4m3_f32(kRows, 16) : idesc_bf16_f32(kRows, 16);
    const uint32_t idesc = (kIdescBase & ~(0x3Fu << 17)) | ((uint32_t)(p.Npad >> 3) << 17);

    if (threadIdx.x == 0) {
        for (int s = 0; s < S; ++s) {
            mbar_init(smem_addr(&sh->full[s]), 1);
            mbar_init(smem_addr(&sh->empty[s]), 1);
        }
        mbar_init(smem_addr(&sh->bfull), 1);
        for (int b = 0; b < 2; ++b) {
            mbar_init(smem_addr(&sh->tfull[b]), 1);
            mbar_init(smem_addr(&sh->tempty[b]), 4);
        }
        mbar_init(smem_addr(&sh->drain), 1);
        mbar_init(smem_addr(&sh->sorted), 32 * kEpiWarps);
        mbar_init(smem_addr(&sh->halved), 32 * kEpiWarps);
        mbar_init(smem_addr(&sh->quartered), 32 * kEpiWarps);
        mbar_init(smem_addr(&sh->merged), 32 * kEpiWarps);
        mbar_fence_init();
    }
    for (int i = threadIdx.x; i < kEpiWarps * 32; i += blockDim.x) {
        sh->thr[i / 32][i % 32] = -__int_as_float(0x7f800000);
        sh->filt[i / 32][i % 32] = -__int_as_float(0x7f800000);
    }
    if (FP8)
        for (int i = threadIdx.x; i < 3 * kLatMaxR; i += blockDim.x) {
            const int part = i / kLatMaxR, q = i % kLatMaxR;
            sh->qscale[part][q] = q < p.R ? p.qscale[part * p.R + q] : 0.0f;
        }
    if (warp == 0 && lane == 0) {
        tma_prefetch_desc(&ta);
        tma_prefetch_desc(&tb);
    }
    if (warp == 1) {
        tmem_alloc(smem_addr(&sh->tmem_base), kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = sh->tmem_base;
    const int items = p.G;
    // The merge after this kernel may launch now (it waits for the lists
    // itself), and the next call's thresholds start from zero: this kernel
    // clears them (the next call's kernel starts after this one completes).
    grid_dep_launch();
    if (blockIdx.x == 0 && threadIdx.x < kLatMaxR) p.tau_clear[threadIdx.x] = 0u;

    if (warp == 0) {
        // ------------------------------------------------ TMA producer
        if (lane == 0) {
            const uint32_t bb = smem_addr(&sh->bfull);
            mbar_arrive_expect_tx(bb, (uint32_t)(KS * bslice));
            for (int ks = 0; ks < KS; ++ks)
                tma_load_2d(smem_addr(sB + ks * bslice), &tb, bb, ks * kElemsPerSlice, 0);
            int s = 0;
            uint32_t ph = 0;
            int64_t issued = 0;
            bool ok = true;
            for (int v = blockIdx.x; v < items && ok; v += gridDim.x) {
                const int64_t t0 = (int64_t)v * p.tiles / p.G, t1 = (int64_t)(v + 1) * p.tiles / p.G;
                for (int64_t t = t0; t < t1 && ok; ++t)
                    for (int ks = 0; ks < KS; ++ks) {
                        if (!mbar_wait(smem_addr(&sh->empty[s]), ph ^ 1u, p.timeout_ns)) {
                            ok = false;
                            break;
                        }
                        const uint32_t fb = smem_addr(&sh->full[s]);
                        mbar_arrive_expect_tx(fb, kAStage);
                        tma_load_2d(smem_addr(sA + s * kAStage), &ta, fb, ks * kElemsPerSlice, (int)(t * kRows));
                        ++issued;
                        if (++s == S) {
                            s = 0;
                            ph ^= 1u;
                        }
                    }
            }
            if (!ok) atomicOr(p.err, kErrTimeout);
            for (int st = 0; st < S; ++st) {
                const int64_t uses = issued / S + (st < issued % S ? 1 : 0);
                if (uses && !mbar_wait(smem_addr(&sh->full[st]), (uint32_t)((uses - 1) & 1), kDrainTimeoutNs))
                    atomicOr(p.err, kErrTimeout);
            }
            if (!mbar_wait(bb, 0, kDrainTimeoutNs)) atomicOr(p.err, kErrTimeout);
        }
    } else if (warp == 1) {
        // ------------------------------------------------ MMA issuer
        if (lane == 0) {
            int s = 0;
            uint32_t ph = 0, lt = 0;
            bool ok = mbar_wait(smem_addr(&sh->bfull), 0, p.timeout_ns);
            for (int v = blockIdx.x; v < items && ok; v += gridDim.x) {
                const int64_t t0 = (int64_t)v * p.tiles / p.G, t1 = (int64_t)(v + 1) * p.tiles / p.G;
                for (int64_t t = t0; t < t1 && ok; ++t, ++lt) {
                    const uint32_t buf = lt & 1u, use = lt >> 1;
                    if (!mbar_wait(smem_addr(&sh->tempty[buf]), (use & 1u) ^ 1u, p.timeout_ns)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t dt = tmem + buf * 128;
                    for (int ks = 0; ks < KS; ++ks) {
                        if (!mbar_wait(smem_addr(&sh->full[s]), ph, p.timeout_ns)) {
                            ok = false;
                            break;
                        }
                        tc_fence_after();
                        const uint64_t ad = smem_desc_k128(smem_addr(sA + s * kAStage));
                        const uint64_t bd = smem_desc_k128(smem_addr(sB + ks * bslice));
#pragma unroll
                        for (int kk = 0; kk < 4; ++kk) {
                            if constexpr (FP8)
                                tc_mma_f8(dt, ad + (uint64_t)(kk * 2), bd + (uint64_t)(kk * 2), idesc, (ks | kk) != 0);
                            else
                                tc_mma_f16(dt, ad + (uint64_t)(kk * 2), bd + (uint64_t)(kk * 2), idesc, (ks | kk) != 0);
                        }
                        tc_commit(smem_addr(&sh->empty[s]));
                        if (++s == S) {
                            s = 0;
                            ph ^= 1u;
                        }
                    }
                    if (!ok) break;
                    tc_commit(smem_addr(&sh->tfull[buf]));
                }
            }
            if (!ok) atomicOr(p.err, kErrTimeout);
            tc_commit(smem_addr(&sh->drain));
            if (!mbar_wait(smem_addr(&sh->drain), 0, kDrainTimeoutNs)) atomicOr(p.err, kErrTimeout);
        }
    } else {
        // ------------------------------------------------ epilogue (warps 2..9)
        const int ew = warp - 2;        // epilogue warp 0..7
        const uint32_t set = ew >> 2;   // drains accumulator `set`: the tiles with lt % 2 == set
        const int sub = warp & 3;       // TMEM lane quadrant this warp may read
        const uint32_t lane_addr = (uint32_t)(sub * 32) << 16;
        const float kNegInf = -__int_as_float(0x7f800000);
        const int R = p.R, k = p.k;
        uint64_t *Lw = slists + (size_t)ew * R * k;  // this warp's set of query q at Lw + q * k
        float *thr_w = sh->thr[ew], *filt_w = sh->filt[ew];
        float *Sw = strans + ew * 32 * 33;  // [32 rows][33]: one row's scores per lane
        uint32_t lt = 0, chunk = 0;
        bool ok = true;
        for (int v = blockIdx.x; v < items && ok; v += gridDim.x) {
            const int64_t t0 = (int64_t)v * p.tiles / p.G, t1 = (int64_t)(v + 1) * p.tiles / p.G;
            // Lane q keeps query q's set for this warp's rows of the chunk; its
            // k-th score and its filter are mirrored in shared memory.
            // A mirror in thr[][] only ever rises: it is the k-th score of k
            // distinct corpus rows (of this chunk or an earlier one), so it
            // bounds the k-th best score over the whole corpus from below.
            RowTopK top;
            uint64_t ra[KM > 0 ? KM : 1];
#pragma unroll
            for (int i = 0; i < (KM > 0 ? KM : 1); ++i) ra[i] = i < k ? 0ull : ~0ull;
            float thr = kNegInf;  // own set's k-th score (strict: later rows lose ties)
            float cthr = kNegInf; // filter: s > cthr  <=>  s > thr and s >= every bound from elsewhere
            uint32_t published = 0;
            // The shared threshold is read one tile ahead, off the critical path.
            uint32_t tau_next = lane < R ? *reinterpret_cast<volatile uint32_t *>(p.tau + lane) : 0u;
            for (int64_t t = t0; t < t1; ++t, ++lt) {
                const uint32_t buf = lt & 1u, use = lt >> 1;
                if (buf != set) continue;
                if (!mbar_wait(smem_addr(&sh->tfull[buf]), use & 1u, p.timeout_ns)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                if (lane < R) {
                    const bool full = KM > 0 ? ra[0] != 0ull : top.n == k;
                    const uint32_t mine = full ? ord_of_score(thr) : 0u;
                    if (mine > published) {
                        atomicMax(p.tau + lane, mine);
                        published = mine;
                    }
                    // Bound from elsewhere: the shared threshold and the
                    // mirrors of the CTA's warps (possibly stale, hence lower:
                    // still bounds).
                    float other = tau_next ? score_of_ord(tau_next) : kNegInf;
                    tau_next = *reinterpret_cast<volatile uint32_t *>(p.tau + lane);
                    const volatile float *vt = &sh->thr[0][0];
#pragma unroll
                    for (int w = 0; w < kEpiWarps; ++w) other = fmaxf(other, vt[w * 32 + lane]);
                    cthr = fmaxf(thr, float_below(other));
                    filt_w[lane] = cthr;
                }
                __syncwarp();
                const int64_t rowbase = t * kRows + sub * 32;
                const int64_t i = rowbase + lane;
                const bool valid = i < p.N;
                uint32_t d0[32], d1[32], d2[32];
                const uint32_t taddr = tmem + lane_addr + buf * 128;
                tmem_ld_32x32b_x32(taddr, d0);
                if constexpr (FP8) {
                    tmem_ld_32x32b_x32(taddr + 32, d1);
                    tmem_ld_32x32b_x32(taddr + 64, d2);
                }
                tmem_ld_wait(d0);
                if constexpr (FP8) {
                    regs_after_wait(d1);
                    regs_after_wait(d2);
                }
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(smem_addr(&sh->tempty[buf]));
                const float cs = FP8 ? (valid ? __ldg(p.corpus_scale + i) : 0.0f) : 1.0f;
                // All queries' scores of this lane's row.
                float sc[kLatMaxR];
#pragma unroll
                for (int q = 0; q < kLatMaxR; ++q) {
                    if constexpr (FP8)
                        sc[q] = (sh->qscale[0][q] * __uint_as_float(d0[q]) + sh->qscale[1][q] * __uint_as_float(d1[q]) +
                                 sh->qscale[2][q] * __uint_as_float(d2[q])) * cs;
                    else
                        sc[q] = __uint_as_float(d0[q]);
                }
                // One ballot per query against that query's filter (branch-free).
                uint32_t m[kLatMaxR];
                uint32_t anym = 0;
#pragma unroll
                for (int q = 0; q < kLatMaxR; ++q) {
                    m[q] = __ballot_sync(0xffffffffu, valid && q < R && sc[q] > filt_w[q]);
                    anym |= m[q];
                }
                if (anym) {
                    // Survivors: transpose the warp's 32 x 32 scores through
                    // shared memory, then lane q inserts query q's survivors
                    // in increasing row (= id) order, all queries in parallel.
#pragma unroll
                    for (int q = 0; q < kLatMaxR; ++q) Sw[lane * 33 + q] = sc[q];
                    __syncwarp();
                    uint32_t mine_m = select32(m, lane);
                    if (lane < R) {
                        float below_other = cthr > thr ? cthr : kNegInf;  // the part of cthr from elsewhere
                        if constexpr (KM > 0) {
                            if (__popc(mine_m) > KM) {
                                // Many survivors (a warp's first tile of a chunk): a bound
                                // from the tile itself.  The k-th largest of the 16 pair
                                // maxima max(s_j, s_{j+16}) is met or beaten by k distinct
                                // rows, so a score below it cannot reach the warp's top k;
                                // about k + 2 rows of 32 pass it instead of all 32.  (The
                                // lanes insert in step, so a round costs the same whether
                                // one lane or all insert: it is the rounds that count.)
                                const float T = pair_max_bound(Sw + lane, mine_m, k);
                                if (T > kNegInf) {
                                    below_other = fmaxf(below_other, float_below(T));
                                    cthr = fmaxf(cthr, below_other);
                                    // Drop the rows below the bound from the mask: the
                                    // insert loop below runs as many rounds as the lane
                                    // with the most rows left, all lanes in step.
                                    uint32_t keep = 0;
#pragma unroll
                                    for (int j = 0; j < 32; ++j) keep |= (Sw[j * 33 + lane] > cthr ? 1u : 0u) << j;
                                    mine_m &= keep;
                                }
                            }
                        }
                        while (mine_m) {
                            const int l = __ffs(mine_m) - 1;
                            mine_m &= mine_m - 1;
                            const float sl = Sw[l * 33 + lane];
                            if (sl > cthr) {
                                const uint64_t key = make_key(sl, (uint32_t)(rowbase + l));
                                if constexpr (KM > 0) {
                                    regset_insert<KM>(ra, key);
                                    if (ra[0] != 0ull) {
                                        thr = key_score(ra[0]);
                                        cthr = fmaxf(thr, below_other);
                                    }
                                } else {
                                    topk_add(Lw + (size_t)lane * k, 1, k, top, key);
                                    if (top.n == k) {
                                        thr = key_score(top.min_key);
                                        cthr = fmaxf(thr, below_other);
                                    }
                                }
                            }
                        }
                        if (thr > thr_w[lane]) thr_w[lane] = thr;
                        filt_w[lane] = cthr;
                    }
                    __syncwarp();
                }
            }
            // Chunk done: each warp writes its sets sorted (lane q: query q),
            // then the eight sorted sets of every query are merged into the
            // chunk's list: pairwise in three rounds on the register-set path
            // (tiny_100k: 2.9 us against 3.8 us for one lane per query taking
            // the largest of eight heads k times), else lane q of warp q mod 8
            // merging the eight sets of query q.  (Ranking every key by binary
            // searches in the other sets, all 256 threads at once, measured
            // six times slower.)  The hand-offs between the epilogue warps are
            // bounded waits, like every other wait.
            if (KM > 0 && lane < R) {
                // descending into the warp's slot of query `lane`
                uint64_t *Lq = Lw + (size_t)lane * k;
#pragma unroll
                for (int i = 0; i < (KM > 0 ? KM : 1); ++i)
                    if (i < k) Lq[k - 1 - i] = ra[i];
            } else if (lane < R) {
                uint64_t *Lq = Lw + (size_t)lane * k;
                for (int t = top.n; t < k; ++t) Lq[t] = 0ull;
                if (k <= 16)
                    sortw_desc_in_place<16>(Lq, top.n);
                else if (k <= 32)
                    sortw_desc_in_place<32>(Lq, top.n);
                else
                    topk_sort(Lq, 1, top.n);
            }
            const uint32_t par = (uint32_t)(chunk & 1);
            mbar_arrive(smem_addr(&sh->sorted));
            if (!mbar_wait(smem_addr(&sh->sorted), par, p.timeout_ns)) ok = false;
            if constexpr (KM > 0) {
                // Pairwise, all queries at once (lane q: query q): sets w and
                // w + 4 of warps 0..3 into four, those into two (warps 0, 1),
                // those into the chunk's list (warp 0), each a two-way merge
                // of sorted lists; the merged sets go to the transposition
                // scratch, free now (48 R k bytes <= its 33 KB for k <= 16).
                uint64_t *t1 = reinterpret_cast<uint64_t *>(strans);  // [4][R][k]
                uint64_t *t2 = t1 + (size_t)4 * R * k;                // [2][R][k]
                auto merge2 = [&](const uint64_t *A, const uint64_t *B, uint64_t *O) {
                    int i = 0, j = 0;
                    uint64_t a = A[0], b = B[0];
                    for (int t = 0; t < k; ++t) {
                        const bool take_a = a >= b;  // distinct keys; two empties give an empty
                        O[t] = take_a ? a : b;
                        if (take_a) {
                            ++i;
                            a = i < k ? A[i] : 0ull;
                        } else {
                            ++j;
                            b = j < k ? B[j] : 0ull;
                        }
                    }
                };
                const size_t ws = (size_t)R * k;  // one warp's sets
                if (ok && ew < 4 && lane < R)
                    merge2(slists + ew * ws + lane * k, slists + (ew + 4) * ws + lane * k, t1 + ew * ws + lane * k);
                mbar_arrive(smem_addr(&sh->halved));
                if (!mbar_wait(smem_addr(&sh->halved), par, p.timeout_ns)) ok = false;
                if (ok && ew < 2 && lane < R)
                    merge2(t1 + ew * ws + lane * k, t1 + (ew + 2) * ws + lane * k, t2 + ew * ws + lane * k);
                mbar_arrive(smem_addr(&sh->quartered));
                if (!mbar_wait(smem_addr(&sh->quartered), par, p.timeout_ns)) ok = false;
                if (ok && ew == 0 && lane < R)
                    merge2(t2 + lane * k, t2 + ws + lane * k, p.lists + ((int64_t)v * R + lane) * k);
            } else {
                const int q = lane * kEpiWarps + ew;
                if (ok && q < R) {
                    uint64_t *out = p.lists + ((int64_t)v * R + q) * k;
                    // heads of the eight sorted sets of query q
                    const uint64_t *Lq0 = slists + (size_t)q * k;  // warp w's set at Lq0 + w * R * k
                    const size_t wstride = (size_t)R * k;
                    uint64_t h[kEpiWarps];
                    int at[kEpiWarps];
#pragma unroll
                    for (int w = 0; w < kEpiWarps; ++w) {
                        at[w] = 0;
                        h[w] = Lq0[w * wstride];
                    }
                    for (int t = 0; t < k; ++t) {
                        uint64_t best = h[0];
                        int bw = 0;
#pragma unroll
                        for (int w = 1; w < kEpiWarps; ++w)
                            if (h[w] > best) {
                                best = h[w];
                                bw = w;
                            }
                        out[t] = best;
#pragma unroll
                        for (int w = 0; w < kEpiWarps; ++w)
                            if (w == bw) {
                                ++at[w];
                                h[w] = (best != 0ull && at[w] < k) ? Lq0[w * wstride + at[w]] : 0ull;
                            }
                    }
                }
            }
            mbar_arrive(smem_addr(&sh->merged));
            if (!mbar_wait(smem_addr(&sh->merged), par, p.timeout_ns)) ok = false;
            ++chunk;
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

// Splits each bf16 query row into three e4m3 parts with power-of-two scales
// (rows r, 32 + r, 64 + r of the 96-row operand).  One block per row slot
// r < 32: the slots past the batch's R rows write zero parts, so that the
// operand needs no clearing.
__global__ void __launch_bounds__(256) k_split_queries(const uint16_t *__restrict__ regions, int R, int d,
                                                       uint8_t *__restrict__ parts, float *__restrict__ qscale) {
    __shared__ float red[8];
    const int r = blockIdx.x;
    if (r >= R) {
        for (int j = threadIdx.x; j < d; j += blockDim.x)
            for (int part = 0; part < 3; ++part) parts[(size_t)(part * 32 + r) * d + j] = 0;
        return;
    }
    const uint16_t *q = regions + (size_t)r * d;
    auto block_max = [&](float v) {
        for (int o = 16; o; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
        if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = v;
        __syncthreads();
        float m = 0.0f;
        for (int w = 0; w < (int)(blockDim.x >> 5); ++w) m = fmaxf(m, red[w]);
        __syncthreads();
        return m;
    };
    auto pow2_scale = [](float m) {
        if (!(m > 0.0f)) return 1.0f;
        int e;
        frexpf(m / 448.0f, &e);  // m / 448 = f 2^e, 0.5 <= f < 1
        return ldexpf(1.0f, e);  // >= m / 448, so |x| / scale <= 448
    };
    // Each thread handles elements j = threadIdx.x + 256 t of the row.
    float m0 = 0.0f;
    for (int j = threadIdx.x; j < d; j += blockDim.x)
        m0 = fmaxf(m0, fabsf(__uint_as_float((uint32_t)q[j] << 16)));
    float res_scale[3];
    res_scale[0] = pow2_scale(block_max(m0));
    // Three passes over the row; the residual is recomputed from the parts
    // already written so that no per-element state has to be kept.
    for (int part = 0; part < 3; ++part) {
        const float sc = res_scale[part];
        float mnext = 0.0f;
        for (int j = threadIdx.x; j < d; j += blockDim.x) {
            float x = __uint_as_float((uint32_t)q[j] << 16);
            for (int pp = 0; pp < part; ++pp) {
                const __half_raw h = __nv_cvt_fp8_to_halfraw(parts[(size_t)(pp * 32 + r) * d + j], __NV_E4M3);
                x -= __half2float(__half(h)) * res_scale[pp];
            }
            const __nv_fp8_storage_t e = __nv_cvt_float_to_fp8(x / sc, __NV_SATFINITE, __NV_E4M3);
            parts[(size_t)(part * 32 + r) * d + j] = e;
            const __half_raw h = __nv_cvt_fp8_to_halfraw(e, __NV_E4M3);
            mnext = fmaxf(mnext, fabsf(x - __half2float(__half(h)) * sc));
        }
        if (part < 2) res_scale[part + 1] = pow2_scale(block_max(mnext));
        __syncthreads();
    }
    if (threadIdx.x < 3) qscale[threadIdx.x * R + r] = res_scale[threadIdx.x];
}

size_t smem_bytes(int Npad, int slices, int stages, int R, int k) {
    return 1024 + (size_t)slices * Npad * kSlice + (size_t)stages * kAStage + (size_t)kEpiWarps * R * k * 8 +
           (size_t)kEpiWarps * 32 * 33 * 4 + sizeof(LatShared);
}

}  // namespace

bool lat_pick_layout(bool fp8, int R, int d, int k, int max_smem, int *Npad, int *slices, int *stages) {
    if (R < 1 || R > kLatMaxR) return false;
    *Npad = fp8 ? 96 : (R + 15) / 16 * 16;
    *slices = fp8 ? (d + 127) / 128 : (d + 63) / 64;
    for (int st = kMaxStages; st >= 3; --st)
        if (smem_bytes(*Npad, *slices, st, R, k) <= (size_t)max_smem) {
            *stages = st;
            return true;
        }
    return false;
}

cudaError_t launch_split_queries(const uint16_t *regions, int R, int d, uint8_t *parts, float *qscale,
                                 cudaStream_t s) {
    k_split_queries<<<kLatMaxR, 256, 0, s>>>(regions, R, d, parts, qscale);
    return cudaGetLastError();
}

cudaError_t launch_latency(bool fp8, const CUtensorMap &ta, const CUtensorMap &tb, const LatParams &p, int grid,
                           cudaStream_t s) {
    const size_t smem = smem_bytes(p.Npad, p.slices, p.stages, p.R, p.k);
    // e4m3: the sets stay in shared memory (the three accumulator groups
    // leave no registers for them: a register set spilled and ran slower).
    auto kern = fp8 ? k_latency_score_topk<true, 0>
                    : (p.k <= 4    ? k_latency_score_topk<false, 4>
                       : p.k <= 8  ? k_latency_score_topk<false, 8>
                       : p.k <= 12 ? k_latency_score_topk<false, 12>
                       : p.k <= 16 ? k_latency_score_topk<false, 16>
                                   : k_latency_score_topk<false, 0>);
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    kern<<<grid, kThreads, smem, s>>>(ta, tb, p);
    return cudaGetLastError();
}

}  // namespace skipk
