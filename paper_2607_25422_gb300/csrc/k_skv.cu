// SKV passage gate (App. B.4 Def. B.4, Eq. skv_score; Alg. 1 "SKV: verify"
// and the TopK after it) on the merged retrieval lists.
//
//  (k_gemm)      per question: c_q = b1 + W1[:, qbar] qbar + W1[:, vbar] vbar
//                for all questions at once, on the tensor cores (k_gemm.cu);
//                it needs no retrieval result and runs beside it on a second
//                stream, after which k_skv_cq_ready raises a per-call flag
//                that the MLP kernel waits for before it reads c_q.
//  k_skv_features per passage slot: F = [e | bf16(e * qbar) | bf16(|e - qbar|)]
//                (3d bf16 in the column order of W1's passage blocks), from
//                the gathered corpus row and qbar; zeros for an empty slot.
//  k_skv_mlp     per 256 passage slots x BN hidden units: the passage part
//                of layer 1 on the tensor cores as a CTA pair (tcgen05
//                cta_group::2, M = 256, N = BN), both operands by TMA (the
//                feature rows and the matching W1 rows) into a ring of
//                stages; with few slots the feature columns are split over
//                two pairs of a cluster of four and the two sums added
//                through distributed shared memory (bulk copies of 32-column
//                chunks into a receive area); the epilogue adds c_q,
//                applies ReLU and the w2 dot over its units and writes one
//                partial logit per slot.  (Building the features in shared
//                memory inside this kernel instead, once per hidden block,
//                made the builders and their hand-offs set the pace.)
//  k_skv_select  per question: logit = b2 + sum of the partial logits,
//                nu = sigmoid(logit), gate nu >= tau, then the first
//                ceil(rho |K| - 1e-3) by (nu desc, id asc): each key placed
//                at its rank (K <= 256), else a bitonic sort.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <type_traits>

#include "skip_device.cuh"
#include "skip_internal.h"

namespace skipk {
namespace {

constexpr int kSkvRows = 128;                // passage slots per CTA (TMEM lanes); a pair has 256
constexpr int kSkvSliceA = kSkvRows * 128;   // one [128 x 64] bf16 K-slice of the features, bytes
constexpr int kSkvSmemMax = 227 * 1024;      // opt-in shared memory of a CTA, bytes
constexpr int kSkvMaxStages = 8;
constexpr int kSkvEpiWarps = 8;             // two per TMEM lane quarter, each on half the columns
constexpr int kSkvThreads = 64 + 32 * kSkvEpiWarps;  // TMA warp, MMA warp, epilogue warps
constexpr uint64_t kDrainTimeoutNs = 1000000000ull;  // 1 s for copies in flight
constexpr int kFeatWarps = 8;                // slots per feature block

// Epilogue operands staged during the main loop, after the ring: w2 of this
// CTA's columns, then c_q of its questions and columns (when they fit).
constexpr int kSkvEpiBytes = 17 * 1024;
constexpr int kSkvCqCap = (kSkvEpiBytes - 256 * 4) / 4;  // c_q floats
constexpr int kSkvChunk = kSkvRows * 128;                // 32 fp32 sums of 128 rows, bytes

// A CTA pair computes 256 slots x BN hidden units (tcgen05 cta_group::2,
// M = 256, N = BN): each CTA stages its own 128 feature rows and half of the
// W1 block (BN / 2 rows) per K-slice, and its TMEM holds its 128 rows x BN.
// With the K split (S = 2) a receive area after the epilogue operands holds
// the partner's sums for this CTA's column half, in chunks of 32 columns.
// Shared memory: ring | barriers (1 KB) | w2, c_q | receive area.
template <int BN, int S>
struct SkvGeom {
    static constexpr int kB = (BN / 2) * 128;              // this CTA's W1 rows of one K-slice, bytes
    static constexpr int kStage = kSkvSliceA + kB;
    static constexpr int kChunks = BN / 64;                // chunks of 32 columns in a column half
    static constexpr int kRecv = S == 2 ? kChunks * kSkvChunk : 0;
    static constexpr int kRingMax = kSkvSmemMax - 2 * 1024 - kSkvEpiBytes - kRecv;
    static constexpr int kStages = kRingMax / kStage < kSkvMaxStages ? kRingMax / kStage : kSkvMaxStages;
    static constexpr int kRing = kStages * kStage;
    static constexpr int kSmem = 1024 + kRing + 1024 + kSkvEpiBytes + kRecv;
    static constexpr uint32_t kIdesc = idesc_bf16_f32(2 * kSkvRows, BN);
    static_assert(kStages >= 4 && kSmem <= kSkvSmemMax, "ring of at least four stages");
    static_assert(kChunks * kSkvChunk <= kRing, "the outgoing half is staged in the ring");
};

struct SkvShared {
    uint64_t full[kSkvMaxStages];   // A and B slices of both CTAs landed (MMA CTA; tx bytes)
    uint64_t empty[kSkvMaxStages];  // stage consumed (commit, to both CTAs of the pair)
    uint64_t tfull;                 // accumulator complete (commit, to both CTAs)
    uint64_t recv[4];               // chunk c of the partner's sums landed (K split; tx bytes)
    uint32_t tmem_base;
};
static_assert(sizeof(SkvShared) <= 1024, "barriers fit their 1 KB");

// Byte offset of sum (row r, 16-byte group j of 8) within a chunk: rows 128
// bytes apart, the groups of a row permuted by r mod 8 so that a warp's 32
// rows hit distinct banks.
__device__ __forceinline__ int chunk_off(int r, int j) { return r * 128 + ((j ^ (r & 7)) << 4); }

// Bulk copy of `bytes` (a multiple of 16) from this CTA's shared memory to
// that of a CTA of the cluster, counted in bytes on its barrier `bar`.
__device__ __forceinline__ void bulk_copy_to_peer(uint32_t dst, uint32_t src, uint32_t bytes, uint32_t bar) {
    asm volatile("cp.async.bulk.shared::cluster.shared::cta.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                     dst),
                 "r"(src), "r"(bytes), "r"(bar)
                 : "memory");
}

__device__ __forceinline__ int ld_acquire_gpu(const int *p) {
    int v;
    asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

__device__ __forceinline__ void st_release_gpu(int *p, int v) {
    asm volatile("st.release.gpu.global.b32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

// Generic-proxy writes to shared memory before an async-proxy read of them.
__device__ __forceinline__ void fence_proxy_async_smem() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// Two bf16 lanes of a 32-bit word -> the two interaction features, rounded
// to bf16 (ties to even).
__device__ __forceinline__ void features2(uint32_t e2, uint32_t q2, uint32_t &eq2, uint32_t &ad2) {
    const __nv_bfloat162 e = *reinterpret_cast<const __nv_bfloat162 *>(&e2);
    const __nv_bfloat162 q = *reinterpret_cast<const __nv_bfloat162 *>(&q2);
    const float2 ef = __bfloat1622float2(e), qf = __bfloat1622float2(q);
    // e * qbar is exact in fp32 (two 8-bit significands); |e - qbar| is exact
    // in fp32 unless the exponents are more than 16 apart, where the bf16
    // result is the larger operand's magnitude either way.
    const __nv_bfloat162 m = __floats2bfloat162_rn(ef.x * qf.x, ef.y * qf.y);
    const __nv_bfloat162 a = __floats2bfloat162_rn(fabsf(ef.x - qf.x), fabsf(ef.y - qf.y));
    eq2 = *reinterpret_cast<const uint32_t *>(&m);
    ad2 = *reinterpret_cast<const uint32_t *>(&a);
}

// F[slot] = [e | bf16(e * qbar) | bf16(|e - qbar|)] (3d bf16, the column
// order of W1's passage blocks), zeros for an empty slot; a warp per slot,
// 16-byte loads and stores.  Launched as the programmatic dependent of the
// kernel that wrote the candidate ids (the question merge), for which it
// waits before it reads them.
__global__ void __launch_bounds__(32 * kFeatWarps) k_skv_features(const SkvParams p, uint16_t *__restrict__ F) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t slot = (int64_t)blockIdx.x * kFeatWarps + warp;
    grid_dep_wait();
    // the MLP kernel may set up now; it waits for these features itself
    grid_dep_launch();
    if (slot < p.P) {
        int64_t id = p.ids[slot];
        if (id >= p.N) {
            if (lane == 0) atomicOr(p.err, kErrConfig);
            id = -1;
        }
        const int q = (int)(slot / p.K);
        const int nw = p.d / 8;  // 16-byte words of a row
        const uint4 *erow = reinterpret_cast<const uint4 *>(p.rows + (id < 0 ? 0 : id) * (int64_t)p.d);
        const uint4 *qrow = reinterpret_cast<const uint4 *>(p.qbar + (int64_t)q * p.d);
        uint4 *f = reinterpret_cast<uint4 *>(F + slot * 3 * (int64_t)p.d);
        const uint4 zero = make_uint4(0, 0, 0, 0);
        // the whole row at once (d <= 1024: at most four 16-byte words a lane)
        uint4 e[4], qv[4];
#pragma unroll
        for (int h = 0; h < 4; ++h) {
            const int w = lane + 32 * h;
            e[h] = (id >= 0 && w < nw) ? __ldg(erow + w) : zero;
            qv[h] = (id >= 0 && w < nw) ? __ldg(qrow + w) : zero;
        }
#pragma unroll
        for (int h = 0; h < 4; ++h) {
            const int w = lane + 32 * h;
            if (w >= nw) continue;
            uint4 m, a;
            features2(e[h].x, qv[h].x, m.x, a.x);
            features2(e[h].y, qv[h].y, m.y, a.y);
            features2(e[h].z, qv[h].z, m.z, a.z);
            features2(e[h].w, qv[h].w, m.w, a.w);
            f[w] = e[h];
            f[nw + w] = m;
            f[2 * nw + w] = a;
        }
    }
}

// nu of slot `slot` (logit = b2 + the partial logits of the grid before)
// and its key (ordered nu bits << 32 | ~id; 0 when empty or below tau).
__device__ __forceinline__ uint64_t slot_key(const SkvParams &p, int64_t slot, float &nu, bool &nonempty) {
    // the id and the partial logits in one round of loads
    int64_t id = p.ids[slot];
    float logit = p.b2;
    for (int b = 0; b < p.nparts; ++b) logit += p.partial[(int64_t)b * p.P + slot];
    if (id >= p.N) id = -1;  // flagged by k_skv_features
    nu = -__int_as_float(0x7f800000);
    nonempty = id >= 0;
    if (id < 0) return 0ull;
    nu = 1.f / (1.f + expf(-logit));
    if (!(nu >= p.tau)) return 0ull;
    return ((uint64_t)(__float_as_uint(nu) | 0x80000000u) << 32) | (uint64_t)(0xFFFFFFFFu - (uint32_t)id);
}

// Output count: ceil(rho |K| - 1e-3) of the non-empty slots, at most the gated ones.
__device__ __forceinline__ int kept_count(const SkvParams &p, int nonempty, int ngated) {
    const double nd = ceil((double)p.rho * (double)nonempty - 1e-3);
    int n = nd < 0.0 ? 0 : (int)nd;
    if (n > nonempty) n = nonempty;
    if (n > ngated) n = ngated;
    return n;
}

// One block per question: nu for every slot, the gate, and the first n by
// (nu desc, id asc): for K <= 256 each gated key is written at its rank (the
// keys above it, and equal ones in earlier slots), else the keys are sorted
// (bitonic, descending).
constexpr int kSelThreads = 256;
__global__ void __launch_bounds__(kSelThreads) k_skv_select(const SkvParams p) {
    __shared__ uint64_t keys[kSkvMaxK];
    __shared__ int nonempty, ngated;
    const int q = blockIdx.x;
    const int K = p.K;
    int Kp = 1;
    while (Kp < K) Kp <<= 1;
    grid_dep_wait();  // the partial logits of the MLP kernel before this one
    if (threadIdx.x == 0) nonempty = 0, ngated = 0;
    __syncthreads();
    int my_ne = 0, my_g = 0;
    for (int j = threadIdx.x; j < Kp; j += kSelThreads) {
        uint64_t key = 0ull;
        if (j < K) {
            const int64_t slot = (int64_t)q * K + j;
            float nu;
            bool ne;
            key = slot_key(p, slot, nu, ne);
            my_ne += ne;
            my_g += key != 0ull;
            if (p.nu_all) p.nu_all[slot] = nu;
        }
        keys[j] = key;
    }
    if (my_ne) atomicAdd(&nonempty, my_ne);
    if (my_g) atomicAdd(&ngated, my_g);
    __syncthreads();
    const int n = kept_count(p, nonempty, ngated);
    if (K <= kSelThreads) {
        const int j = threadIdx.x;
        const uint64_t key = j < K ? keys[j] : 0ull;
        if (key != 0ull) {
            int rank = 0;
            for (int i = 0; i < K; ++i) {
                const uint64_t o = keys[i];
                rank += (o > key) || (o == key && i < j);
            }
            if (rank < n) {
                const int64_t o = (int64_t)q * K + rank;
                p.out_ids[o] = (int64_t)(0xFFFFFFFFu - (uint32_t)key);
                p.out_nu[o] = __uint_as_float((uint32_t)(key >> 32) & 0x7FFFFFFFu);
            }
        }
        if (j < K && j >= n) {
            p.out_ids[(int64_t)q * K + j] = -1;
            p.out_nu[(int64_t)q * K + j] = -__int_as_float(0x7f800000);
        }
    } else {
        for (int size = 2; size <= Kp; size <<= 1)
            for (int stride = size >> 1; stride > 0; stride >>= 1) {
                for (int t = threadIdx.x; t < Kp / 2; t += kSelThreads) {
                    const int lo = 2 * t - (t & (stride - 1));
                    const int hi = lo + stride;
                    const bool desc = (lo & size) == 0;
                    const uint64_t a = keys[lo], b = keys[hi];
                    if ((a < b) == desc) {
                        keys[lo] = b;
                        keys[hi] = a;
                    }
                }
                __syncthreads();
            }
        for (int j = threadIdx.x; j < K; j += kSelThreads) {
            const int64_t o = (int64_t)q * K + j;
            if (j < n) {
                const uint64_t key = keys[j];
                p.out_ids[o] = (int64_t)(0xFFFFFFFFu - (uint32_t)key);
                p.out_nu[o] = __uint_as_float((uint32_t)(key >> 32) & 0x7FFFFFFFu);
            } else {
                p.out_ids[o] = -1;
                p.out_nu[o] = -__int_as_float(0x7f800000);
            }
        }
    }
    if (threadIdx.x == 0) p.out_count[q] = n;
}

// Layer 1 of the verifier over the passage features, ReLU and the w2 dot.
// A cluster of 2 S CTAs computes 256 slots x BN hidden units: CTA rank r is
// half r & 1 of a CTA pair (its 128 slots, and half of the W1 rows it
// stages) over the K part r >> 1 of the 3d feature columns (S = 1 or 2).
// With S = 2 the two K parts' sums are added through distributed shared
// memory: each CTA stages the column half its partner finishes, 32 columns
// at a time, and sends each chunk by a bulk copy into the partner's receive
// area as soon as it is staged; it finishes the other half itself, chunk by
// chunk as the partner's copies land.  Each epilogue
// warp writes one partial logit per slot over its columns: slab
// ((hidden block * S + part) * 2 + half of the columns).
template <int BN, int S>
__global__ void __launch_bounds__(kSkvThreads, 1)
    k_skv_mlp(const __grid_constant__ CUtensorMap tf, const __grid_constant__ CUtensorMap tw, const SkvParams p) {
    using G = SkvGeom<BN, S>;
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t *sA = smem;
    uint8_t *sB = smem + G::kStages * kSkvSliceA;
    SkvShared *sh = reinterpret_cast<SkvShared *>(smem + G::kRing);
    uint8_t *recv = smem + G::kRing + 1024 + kSkvEpiBytes;  // the partner's sums (S = 2)
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t rank = cluster_rank();
    const int half = (int)(rank & 1u), part = (int)(rank >> 1);
    const uint32_t lead = rank & ~1u;  // the pair's MMA CTA
    const bool mma_cta = half == 0;
    const uint16_t pair_mask = (uint16_t)(3u << lead);
    const int ntc = p.H / BN;
    const int cl = (int)cluster_index();
    const int ct = cl % ntc;
    const int64_t m0 = (int64_t)(cl / ntc) * (2 * kSkvRows) + half * kSkvRows;
    const int n0 = ct * BN;
    const int nsl = 3 * (p.d / 64);  // K-slices over the 3d feature columns
    const int u0 = part * nsl / S;
    const int nk = (part + 1) * nsl / S - u0;
    // the selection kernel may launch now; it waits for this grid itself
    grid_dep_launch();

    if (threadIdx.x == 0) {
        for (int s = 0; s < G::kStages; ++s) {
            mbar_init(smem_addr(&sh->full[s]), 1);
            mbar_init(smem_addr(&sh->empty[s]), 1);
        }
        mbar_init(smem_addr(&sh->tfull), 1);
        for (int c = 0; c < G::kChunks; ++c) mbar_init(smem_addr(&sh->recv[c]), 1);
        mbar_fence_init();
        // the partner's half arrives as one bulk copy a chunk, counted in bytes
        if (S == 2)
            for (int c = 0; c < G::kChunks; ++c) mbar_arrive_expect_tx(smem_addr(&sh->recv[c]), (uint32_t)kSkvChunk);
    }
    if (warp == 0 && lane == 0) {
        tma_prefetch_desc(&tf);
        tma_prefetch_desc(&tw);
    }
    if (warp == 1) {
        tmem_alloc_pair(smem_addr(&sh->tmem_base), BN);
        tmem_relinquish_pair();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    // Every CTA's barriers are initialised before any peer copy or arrive.
    cluster_sync_all();
    const uint32_t tmem = sh->tmem_base;
    bool done = false;

    if (warp == 0) {
        // ------------------------------------------------ TMA: features and W1 rows
        if (lane == 0) {
            // the features come from the kernel before this one
            grid_dep_wait();
            bool ok = true;
            int issued = 0;
            for (int u = 0; u < nk && ok; ++u) {
                const int s = u % G::kStages;
                const uint32_t ph = (uint32_t)(u / G::kStages) & 1u;
                if (!mbar_wait(smem_addr(&sh->empty[s]), ph ^ 1u, p.timeout_ns)) {
                    ok = false;
                    break;
                }
                // both CTAs' copies complete on the MMA CTA's barrier
                const uint32_t fb = smem_addr(&sh->full[s]);
                if (mma_cta) mbar_arrive_expect_tx(fb, 2u * G::kStage);
                const uint32_t fl = mapa_shared(fb, lead);
                const int x = (u0 + u) * 64;
                tma_load_2d_pair(smem_addr(sA + s * kSkvSliceA), &tf, fl, x, (int)m0);
                tma_load_2d_pair(smem_addr(sB + s * G::kB), &tw, fl, 2 * p.d + x, n0 + half * (BN / 2));
                ++issued;
            }
            if (!ok) atomicOr(p.err, kErrTimeout);
            // Copies in flight: the MMA CTA waits for the last load of each
            // stage to land, the other CTA for the release of its last stages
            // (which follows their arrival; a release that never comes ends
            // the wait after the bound, long after any copy has landed).
            for (int s = 0; s < G::kStages; ++s) {
                const int uses = issued / G::kStages + (s < issued % G::kStages ? 1 : 0);
                if (uses == 0) continue;
                const uint32_t bar = mma_cta ? smem_addr(&sh->full[s]) : smem_addr(&sh->empty[s]);
                if (!mbar_wait(bar, (uint32_t)((uses - 1) & 1), kDrainTimeoutNs)) atomicOr(p.err, kErrTimeout);
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------ MMA issuer (MMA CTA of the pair)
        if (lane == 0 && mma_cta) {
            bool ok = true;
            for (int u = 0; u < nk && ok; ++u) {
                const int s = u % G::kStages;
                if (!mbar_wait(smem_addr(&sh->full[s]), (uint32_t)(u / G::kStages) & 1u, p.timeout_ns)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint64_t ad = smem_desc_k128(smem_addr(sA + s * kSkvSliceA));
                const uint64_t bd = smem_desc_k128(smem_addr(sB + s * G::kB));
#pragma unroll
                for (int kk = 0; kk < 4; ++kk)
                    tc_mma_f16_pair(tmem, ad + (uint64_t)(kk * 2), bd + (uint64_t)(kk * 2), G::kIdesc,
                                    (u | kk) != 0);
                tc_commit_pair_mc(smem_addr(&sh->empty[s]), pair_mask);
            }
            if (!ok) atomicOr(p.err, kErrTimeout);
            // Arrives on both CTAs once every MMA issued has completed (also
            // after a timeout).
            tc_commit_pair_mc(smem_addr(&sh->tfull), pair_mask);
        }
    }

    // ---------------------------------------------------- epilogue (warps 2..9)
    // Warp w reads TMEM lanes 32 (w % 4) .. (its slot rows) and handles half
    // of the columns (hal), so that two warps share each row.
    const int sub = warp & 3;
    const int r = sub * 32 + lane;  // TMEM lane = slot row of this CTA
    const uint32_t lane_addr = (uint32_t)(sub * 32) << 16;
    const bool epi = warp >= 2;
    const int hal = (warp - 2) >> 2;
    const int et = (warp - 2) * 32 + lane;  // 0 .. 255 for the epilogue
    // columns this CTA finishes, relative to n0
    const int c0 = S == 2 ? part * (BN / 2) : 0;
    const int ncol = S == 2 ? BN / 2 : BN;
    const int q0 = (int)(m0 < p.P ? m0 / p.K : 0);
    const int64_t last = (m0 + kSkvRows < p.P ? m0 + kSkvRows : p.P) - 1;
    const int nq = m0 < p.P ? (int)(last / p.K) - q0 + 1 : 0;  // <= 128
    float *w2s = reinterpret_cast<float *>(reinterpret_cast<uint8_t *>(sh) + 1024);
    float *cqs = w2s + 256;
    const bool cq_staged = nq * ncol <= kSkvCqCap;
    const int64_t slab = (int64_t)p.Q * p.H;
    if (epi) {
        // While the main loop runs: w2 and c_q (the GEMM's K-split slabs
        // summed once) of this CTA's columns into shared memory,
        // cqs[(q - q0) * ncol + c].  c_q comes from a kernel before this one
        // in the stream, or (cq_flag) from the GEMM on the other stream,
        // which raises the flag to cq_epoch once it has completed.
        grid_dep_wait();
        if (p.cq_flag) {
            if (et == 0) {
                const uint64_t t0 = globaltimer_ns();
                while (ld_acquire_gpu(p.cq_flag) != p.cq_epoch) {
                    if (globaltimer_ns() - t0 > p.timeout_ns) {
                        atomicOr(p.err, kErrTimeout);
                        break;
                    }
                    __nanosleep(256);
                }
            }
            asm volatile("bar.sync 1, %0;" ::"r"(32 * kSkvEpiWarps) : "memory");
            (void)ld_acquire_gpu(p.cq_flag);
        }
        for (int t = et; t < ncol; t += 32 * kSkvEpiWarps) w2s[t] = p.w2[n0 + c0 + t];
        if (cq_staged)
            for (int t = et; t < nq * ncol; t += 32 * kSkvEpiWarps) {
                const float *src = p.cq + (int64_t)(q0 + t / ncol) * p.H + n0 + c0 + t % ncol;
                float v = 0.f;
                for (int z = 0; z < p.cq_splits; ++z) v += src[z * slab];
                cqs[t] = v;
            }
        asm volatile("bar.sync 1, %0;" ::"r"(32 * kSkvEpiWarps) : "memory");  // the epilogue warps
        done = mbar_wait(smem_addr(&sh->tfull), 0, p.timeout_ns);
        if (!done) atomicOr(p.err, kErrTimeout);
        tc_fence_after();
    }
    // With the K split: the half of the sums the partner finishes, staged
    // chunk by chunk in this CTA's ring (free: its MMAs have completed) by
    // the four warps of the column half that owns the chunk, and pushed into
    // the partner's receive area as soon as those four warps are done with it.
    if (S == 2 && epi) {
        const int oc = (1 - part) * (BN / 2);
#pragma unroll 1
        for (int c = hal * (G::kChunks / 2); c < (hal + 1) * (G::kChunks / 2); ++c) {
            if (done) {
                uint32_t v[32];
                tmem_ld_32x32b_x32(tmem + lane_addr + (uint32_t)(oc + c * 32), v);
                tmem_ld_wait(v);
                uint8_t *ch = smem + c * kSkvChunk;
#pragma unroll
                for (int j = 0; j < 8; ++j)
                    *reinterpret_cast<uint4 *>(ch + chunk_off(r, j)) =
                        make_uint4(v[4 * j], v[4 * j + 1], v[4 * j + 2], v[4 * j + 3]);
                fence_proxy_async_smem();
            }
            asm volatile("bar.sync %0, %1;" ::"r"(2 + hal), "r"(kSkvRows) : "memory");  // this half's warps
            if (sub == 0 && lane == 0 && done) {
                const uint32_t peer = rank ^ 2u;
                bulk_copy_to_peer(mapa_shared(smem_addr(recv) + c * kSkvChunk, peer), smem_addr(smem) + c * kSkvChunk,
                                  (uint32_t)kSkvChunk, mapa_shared(smem_addr(&sh->recv[c]), peer));
            }
        }
    }
    if (epi && done) {
        const int64_t slot = m0 + r;
        // rows past the last slot read the first staged question and write nothing
        const int qq = slot < p.P ? (int)(slot / p.K) - q0 : 0;
        const int qc = qq < 0 ? 0 : qq >= nq ? (nq > 0 ? nq - 1 : 0) : qq;
        const float *cq = cqs + qc * ncol;
        const float *cqg = p.cq + (int64_t)(q0 + qc) * p.H + n0 + c0;
        bool got = true;
        // four partial sums of the w2 dot (any order is within the bound)
        float a0 = 0.f, a1 = 0.f, a2 = 0.f, a3 = 0.f;
        // the loop in two forms, so that no branch splits its body: c_q
        // staged in shared memory, or (more questions in the tile than the
        // staging holds, i.e. few slots each) summed from the GEMM's slabs
        auto run = [&](auto staged) {
            constexpr bool kStaged = decltype(staged)::value;
#pragma unroll 1
            for (int c = hal * (ncol / 64); c < (hal + 1) * (ncol / 64); ++c) {
                if (S == 2) {
                    // the partner's chunk c: a copy in flight writes into this
                    // CTA's shared memory, so wait for it at least as long as
                    // for any other copy before giving up
                    if (!mbar_wait(smem_addr(&sh->recv[c]), 0,
                                   p.timeout_ns > kDrainTimeoutNs ? p.timeout_ns : kDrainTimeoutNs)) {
                        got = false;
                        break;
                    }
                }
                uint32_t v[32];
                tmem_ld_32x32b_x32(tmem + lane_addr + (uint32_t)(c0 + c * 32), v);
                tmem_ld_wait(v);
                // four columns at a time: h = own sum (+ the partner's) + c_q,
                // ReLU, times w2
#pragma unroll
                for (int g = 0; g < 8; ++g) {
                    const int col = c * 32 + 4 * g;
                    float4 h = make_float4(__uint_as_float(v[4 * g]), __uint_as_float(v[4 * g + 1]),
                                           __uint_as_float(v[4 * g + 2]), __uint_as_float(v[4 * g + 3]));
                    if constexpr (S == 2) {
                        const float4 o = *reinterpret_cast<const float4 *>(recv + c * kSkvChunk + chunk_off(r, g));
                        h.x += o.x, h.y += o.y, h.z += o.z, h.w += o.w;
                    }
                    if constexpr (kStaged) {
                        const float4 b = *reinterpret_cast<const float4 *>(cq + col);
                        h.x += b.x, h.y += b.y, h.z += b.z, h.w += b.w;
                    } else {
                        for (int z = 0; z < p.cq_splits; ++z) {
                            const float4 b = __ldg(reinterpret_cast<const float4 *>(cqg + z * slab + col));
                            h.x += b.x, h.y += b.y, h.z += b.z, h.w += b.w;
                        }
                    }
                    const float4 w = *reinterpret_cast<const float4 *>(w2s + col);
                    a0 = fmaf(fmaxf(h.x, 0.f), w.x, a0);
                    a1 = fmaf(fmaxf(h.y, 0.f), w.y, a1);
                    a2 = fmaf(fmaxf(h.z, 0.f), w.z, a2);
                    a3 = fmaf(fmaxf(h.w, 0.f), w.w, a3);
                }
            }
        };
        if (cq_staged)
            run(std::true_type{});
        else
            run(std::false_type{});
        if (!got && lane == 0) atomicOr(p.err, kErrTimeout);
        const float acc = (a0 + a1) + (a2 + a3);
        if (got && slot < p.P) p.partial[(int64_t)((ct * S + part) * 2 + hal) * p.P + slot] = acc;
    }

    tc_fence_before();
    __syncthreads();
    // No peer may still copy into, arrive on, or write the TMEM of this CTA
    // when it frees TMEM and exits.
    cluster_sync_all();
    tc_fence_after();
    if (warp == 1) {
        __syncwarp();
        tmem_dealloc_pair(tmem, BN);
    }
}

}  // namespace

// Raises the c_q flag once the GEMM before this kernel in its stream has
// completed.
__global__ void k_skv_cq_ready(int *flag, int epoch) { st_release_gpu(flag, epoch); }

size_t skv_mlp_smem_bytes(int BN, int S) {
    return BN == 256 ? (S == 2 ? SkvGeom<256, 2>::kSmem : SkvGeom<256, 1>::kSmem)
                     : (S == 2 ? SkvGeom<128, 2>::kSmem : SkvGeom<128, 1>::kSmem);
}

template <int BN>
int skv_max_clusters(int CL) {
    auto kern = k_skv_mlp<BN, 2>;
    const size_t smem = skv_mlp_smem_bytes(BN, 2);
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess) {
        cudaGetLastError();
        return 0;
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)(CL * 64));
    cfg.blockDim = dim3((unsigned)kSkvThreads);
    cfg.dynamicSmemBytes = smem;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = (unsigned)CL;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, kern, &cfg) != cudaSuccess) {
        cudaGetLastError();
        return 0;
    }
    return n;
}

// The MLP's tile shape: hidden units per CTA pair (256 when H allows, else
// 128) and K parts (2 when the clusters of four CTAs that this takes all fit
// on the GPU at once, which puts more SMs to work on a small batch; else 1).
void skv_mlp_shape(int64_t P, int H, int *BN, int *S) {
    *BN = H % 256 == 0 ? 256 : 128;
    const int64_t clusters = (P + 2 * kSkvRows - 1) / (2 * kSkvRows) * (H / *BN);
    static int fit[2] = {-1, -1};  // clusters of four resident at once, per BN
    int &f = fit[*BN == 256 ? 1 : 0];
    if (f < 0) f = *BN == 256 ? skv_max_clusters<256>(4) : skv_max_clusters<128>(4);
    *S = clusters <= f ? 2 : 1;
}

// Launch as the programmatic dependent of the previous kernel in the stream.
template <typename... Args>
cudaError_t launch_dependent(void (*kern)(Args...), dim3 grid, int threads, size_t smem, cudaStream_t s,
                             Args... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = dim3((unsigned)threads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kern, args...);
}

cudaError_t launch_skv_features(const SkvParams &p, uint16_t *F, cudaStream_t s) {
    if (p.Q == 0) return cudaSuccess;
    const unsigned blocks = (unsigned)((p.P + kFeatWarps - 1) / kFeatWarps);
    return launch_dependent(k_skv_features, dim3(blocks), 32 * kFeatWarps, (size_t)0, s, p, F);
}

cudaError_t launch_skv_mlp(const CUtensorMap &tf, const CUtensorMap &tw, const SkvParams &p, int BN, int S,
                           cudaStream_t s) {
    if (p.Q == 0) return cudaSuccess;
    if ((BN != 128 && BN != 256) || (S != 1 && S != 2) || p.H % BN != 0 || p.nparts != p.H / BN * S * 2)
        return cudaErrorInvalidValue;
    const size_t smem = skv_mlp_smem_bytes(BN, S);
    auto kern = BN == 256 ? (S == 2 ? k_skv_mlp<256, 2> : k_skv_mlp<256, 1>)
                          : (S == 2 ? k_skv_mlp<128, 2> : k_skv_mlp<128, 1>);
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    const int64_t clusters = (p.P + 2 * kSkvRows - 1) / (2 * kSkvRows) * (p.H / BN);
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)(clusters * 2 * S));
    cfg.blockDim = dim3((unsigned)kSkvThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = (unsigned)(2 * S);
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    return cudaLaunchKernelEx(&cfg, kern, tf, tw, p);
}

cudaError_t launch_skv_cq_ready(int *flag, int epoch, cudaStream_t s) {
    k_skv_cq_ready<<<1, 1, 0, s>>>(flag, epoch);
    return cudaGetLastError();
}

cudaError_t launch_skv_select(const SkvParams &p, cudaStream_t s) {
    if (p.Q == 0) return cudaSuccess;
    return launch_dependent(k_skv_select, dim3((unsigned)p.Q), kSelThreads, 0, s, p);
}

}  // namespace skipk
