// SKV passage gate (App. B.4 Def. B.4, Eq. skv_score; Alg. 1 "SKV: verify"
// and the TopK after it) on the merged retrieval lists.
//
//  (k_gemm)      per question: c_q = b1 + W1[:, qbar] qbar + W1[:, vbar] vbar
//                for all questions at once, on the tensor cores (k_gemm.cu).
//  k_skv_mlp     per 128 passage slots x 128 hidden units: the passage part
//                of layer 1 on the tensor cores.  The A operand is built in
//                shared memory by sixteen warps (four threads per slot row,
//                each with three chunks of its row in flight) from the gathered corpus
//                rows and qbar: per 64-column chunk of d, three K-slices
//                e | bf16(e * qbar) | bf16(|e - qbar|) in the 128-byte
//                swizzled layout TMA would produce, one slice per stage of a
//                four-stage ring; the B operand is the matching W1 column
//                block, loaded by TMA into an eight-stage ring of its own.
//                Launched as the programmatic dependent of the c_q GEMM: it
//                gathers and multiplies while the GEMM runs and waits for c_q
//                only in its epilogue.  tcgen05.mma
//                (kind::f16, M = N = 128) accumulates in TMEM; the epilogue
//                adds c_q, applies ReLU and the w2 dot for its 128 units and
//                writes one partial logit per slot and hidden block.
//  k_skv_select  per question: logit = b2 + sum of the partial logits,
//                nu = sigmoid(logit), gate nu >= tau, then the first
//                ceil(rho |K| - 1e-3) by (nu desc, id asc) (bitonic sort).
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "skip_device.cuh"
#include "skip_internal.h"

namespace skipk {
namespace {

constexpr int kSkvRows = 128;                       // passage slots per CTA (TMEM lanes)
constexpr int kSkvSlice = kSkvRows * 128;           // one [128 x 64] bf16 K-slice, bytes
// A stage holds one K-slice of A (e, e*qbar or |e - qbar| of one 64-column
// chunk of d) or of B (the matching W1 column block for 128 units).  The two
// rings are separate: B, whose TMA copy from L2 takes microseconds, runs
// eight slices ahead; A, built from rows the builders already hold, four.
constexpr int kSkvStageA = kSkvSlice;
constexpr int kSkvStageB = kSkvSlice;
constexpr int kSkvStagesA = 4;
constexpr int kSkvStagesB = 8;
constexpr int kSkvBuilders = 16;                    // four builder warps per TMEM lane quadrant
constexpr int kSkvParts = kSkvBuilders / 4;          // builder threads per slot row
constexpr int kSkvWords = 8 / kSkvParts;             // 16-byte words of a 64-column chunk per thread
constexpr int kSkvThreads = 64 + 32 * kSkvBuilders;  // TMA warp, MMA warp, builders (4 of them: epilogue)
constexpr int kSkvAhead = 3;                         // chunks of corpus row in flight per builder thread
constexpr uint32_t kSkvIdesc = idesc_bf16_f32(128, kSkvHidden);
constexpr uint64_t kDrainTimeoutNs = 1000000000ull;  // 1 s for copies in flight

struct SkvShared {
    uint64_t fullA[kSkvStagesA];   // A built (one arrival per builder warp)
    uint64_t emptyA[kSkvStagesA];  // A stage consumed (tcgen05.commit)
    uint64_t fullB[kSkvStagesB];   // B landed (tx bytes)
    uint64_t emptyB[kSkvStagesB];  // B stage consumed (tcgen05.commit)
    uint64_t tfull;              // accumulator complete
    uint32_t tmem_base;
};

__device__ __forceinline__ void sts128(uint32_t addr, uint4 v) {
    asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(v.x), "r"(v.y), "r"(v.z),
                 "r"(v.w)
                 : "memory");
}

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

__global__ void __launch_bounds__(kSkvThreads, 1)
    k_skv_mlp(const __grid_constant__ CUtensorMap tw, const SkvParams p) {
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t *sA = smem;
    uint8_t *sB = smem + kSkvStagesA * kSkvStageA;
    SkvShared *sh = reinterpret_cast<SkvShared *>(sB + kSkvStagesB * kSkvStageB);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t m0 = (int64_t)blockIdx.x * kSkvRows;
    const int n0 = blockIdx.y * kSkvHidden;
    const int nc = p.d / 64;

    if (threadIdx.x == 0) {
        for (int s = 0; s < kSkvStagesA; ++s) {
            mbar_init(smem_addr(&sh->fullA[s]), kSkvBuilders);  // one arrival per builder warp
            mbar_init(smem_addr(&sh->emptyA[s]), 1);
        }
        for (int s = 0; s < kSkvStagesB; ++s) {
            mbar_init(smem_addr(&sh->fullB[s]), 1);
            mbar_init(smem_addr(&sh->emptyB[s]), 1);
        }
        mbar_init(smem_addr(&sh->tfull), 1);
        mbar_fence_init();
    }
    if (warp == 0 && lane == 0) tma_prefetch_desc(&tw);
    if (warp == 1) {
        tmem_alloc(smem_addr(&sh->tmem_base), kSkvHidden);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = sh->tmem_base;

    if (warp == 0) {
        // ------------------------------------------------ TMA: W1 column blocks
        if (lane == 0) {
            bool ok = true;
            int issued = 0;
            for (int u = 0; u < 3 * nc && ok; ++u) {
                const int s = u % kSkvStagesB, c = u / 3, b = u - 3 * c;
                const uint32_t ph = (uint32_t)(u / kSkvStagesB) & 1u;
                if (!mbar_wait(smem_addr(&sh->emptyB[s]), ph ^ 1u, p.timeout_ns)) {
                    ok = false;
                    break;
                }
                const uint32_t fb = smem_addr(&sh->fullB[s]);
                mbar_arrive_expect_tx(fb, kSkvStageB);
                tma_load_2d(smem_addr(sB + s * kSkvStageB), &tw, fb, (2 + b) * p.d + c * 64, n0);
                ++issued;
            }
            if (!ok) atomicOr(p.err, kErrTimeout);
            // Copies in flight: wait for the last use of each stage to complete.
            for (int s = 0; s < kSkvStagesB; ++s) {
                const int uses = issued / kSkvStagesB + (s < issued % kSkvStagesB ? 1 : 0);
                if (uses == 0) continue;
                if (!mbar_wait(smem_addr(&sh->fullB[s]), (uint32_t)((uses - 1) & 1), kDrainTimeoutNs))
                    atomicOr(p.err, kErrTimeout);
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------ MMA issuer
        if (lane == 0) {
            bool ok = true;
            for (int u = 0; u < 3 * nc && ok; ++u) {
                const int sa = u % kSkvStagesA, sb = u % kSkvStagesB;
                if (!mbar_wait(smem_addr(&sh->fullA[sa]), (uint32_t)(u / kSkvStagesA) & 1u, p.timeout_ns) ||
                    !mbar_wait(smem_addr(&sh->fullB[sb]), (uint32_t)(u / kSkvStagesB) & 1u, p.timeout_ns)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint64_t ad = smem_desc_k128(smem_addr(sA + sa * kSkvStageA));
                const uint64_t bd = smem_desc_k128(smem_addr(sB + sb * kSkvStageB));
#pragma unroll
                for (int kk = 0; kk < 4; ++kk)
                    tc_mma_f16(tmem, ad + (uint64_t)(kk * 2), bd + (uint64_t)(kk * 2), kSkvIdesc, (u | kk) != 0);
                tc_commit(smem_addr(&sh->emptyA[sa]));
                tc_commit(smem_addr(&sh->emptyB[sb]));
            }
            if (!ok) atomicOr(p.err, kErrTimeout);
            // Arrives once every MMA issued has completed (also after a timeout).
            tc_commit(smem_addr(&sh->tfull));
        }
    } else {
        // ------------------------------------------------ builders, then epilogue
        // Builder warps w, w + 4, w + 8 and w + 12 share a TMEM lane
        // quadrant: each thread owns one slot row and a quarter of every
        // 64-column chunk (16-byte words kSkvWords part ...), and keeps the
        // next kSkvAhead chunks of its corpus row and qbar in flight in
        // registers.  (Four threads a row instead of two: the builds set the
        // kernel's pace, the MMAs take a tenth of it.)
        const int bw = warp - 2, part = bw >> 2;
        const int r = (warp & 3) * 32 + lane;  // TMEM lane = slot row in the tile
        const int64_t slot = m0 + r;
        int64_t id = -1;
        int q = 0;
        if (slot < p.P) {
            id = p.ids[slot];
            q = (int)(slot / p.K);
            if (id >= p.N) {
                if (part == 0) atomicOr(p.err, kErrConfig);
                id = -1;
            }
        }
        const uint4 *erow =
            reinterpret_cast<const uint4 *>(p.rows + (id < 0 ? 0 : id) * (int64_t)p.d) + kSkvWords * part;
        const uint4 *qrow = reinterpret_cast<const uint4 *>(p.qbar + (int64_t)q * p.d) + kSkvWords * part;
        const uint4 zero = make_uint4(0, 0, 0, 0);
        uint4 eb[kSkvAhead][kSkvWords], qb[kSkvAhead][kSkvWords];
#pragma unroll
        for (int a = 0; a < kSkvAhead; ++a)
#pragma unroll
            for (int j = 0; j < kSkvWords; ++j) {
                const bool ld = id >= 0 && a < nc;
                eb[a][j] = ld ? __ldg(erow + a * 8 + j) : zero;
                qb[a][j] = ld ? __ldg(qrow + a * 8 + j) : zero;
            }
        bool ok = true;
        for (int c = 0; c < nc; ++c) {
            uint4 e[kSkvWords], qv[kSkvWords];
#pragma unroll
            for (int j = 0; j < kSkvWords; ++j) {
                e[j] = eb[0][j];
                qv[j] = qb[0][j];
            }
            // rotate the prefetch ring and issue chunk c + kSkvAhead
#pragma unroll
            for (int a = 0; a + 1 < kSkvAhead; ++a)
#pragma unroll
                for (int j = 0; j < kSkvWords; ++j) {
                    eb[a][j] = eb[a + 1][j];
                    qb[a][j] = qb[a + 1][j];
                }
            {
                const int cn = c + kSkvAhead;
                const bool ld = id >= 0 && cn < nc;
#pragma unroll
                for (int j = 0; j < kSkvWords; ++j) {
                    eb[kSkvAhead - 1][j] = ld ? __ldg(erow + cn * 8 + j) : zero;
                    qb[kSkvAhead - 1][j] = ld ? __ldg(qrow + cn * 8 + j) : zero;
                }
            }
            uint4 f[3][kSkvWords];  // the chunk's three K-slices of this thread's part of the row
#pragma unroll
            for (int jj = 0; jj < kSkvWords; ++jj) {
                f[0][jj] = e[jj];
                features2(e[jj].x, qv[jj].x, f[1][jj].x, f[2][jj].x);
                features2(e[jj].y, qv[jj].y, f[1][jj].y, f[2][jj].y);
                features2(e[jj].z, qv[jj].z, f[1][jj].z, f[2][jj].z);
                features2(e[jj].w, qv[jj].w, f[1][jj].w, f[2][jj].w);
            }
            // Row r of each slice: 16-byte chunk j at position j ^ (r & 7).
            const int sw = r & 7;
#pragma unroll
            for (int b = 0; b < 3; ++b) {
                const int u = 3 * c + b, s = u % kSkvStagesA;
                const uint32_t ph = (uint32_t)(u / kSkvStagesA) & 1u;
                // warp-uniform: every lane waits (bounded), then the warp votes
                if (!__all_sync(0xffffffffu, mbar_wait(smem_addr(&sh->emptyA[s]), ph ^ 1u, p.timeout_ns))) {
                    ok = false;
                    break;
                }
                const uint32_t base = smem_addr(sA + s * kSkvStageA) + r * 128;
#pragma unroll
                for (int jj = 0; jj < kSkvWords; ++jj)
                    sts128(base + (uint32_t)(((kSkvWords * part + jj) ^ sw) << 4), f[b][jj]);
                // each writer makes its stores visible to the tensor core's
                // (async) proxy, then one arrival per warp: 257 arrivals on
                // one barrier per slice were serialised
                fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0) mbar_arrive(smem_addr(&sh->fullA[s]));
            }
            if (!ok) break;
        }
        if (!ok) atomicOr(p.err, kErrTimeout);
        // Epilogue: h = acc + c_q, ReLU, dot with w2 over this CTA's units.
        if (part == 0) {
            const bool done = mbar_wait(smem_addr(&sh->tfull), 0, p.timeout_ns);
            if (!done) atomicOr(p.err, kErrTimeout);
            tc_fence_after();
            // c_q comes from the GEMM launched just before this kernel (whose
            // programmatic dependent it is): wait for that grid here only.
            grid_dep_wait();
            // c_q of the tile's questions for this CTA's units, the GEMM's
            // K-split slabs summed once, staged in the A ring (free: every
            // MMA that read it has completed; 64 KB holds 128 questions).
            // cqs[(q - q0) * 128 + n].
            float *cqs = reinterpret_cast<float *>(sA);
            const int q0 = (int)(m0 / p.K);
            const int64_t last = (m0 + kSkvRows < p.P ? m0 + kSkvRows : p.P) - 1;
            const int nq = m0 < p.P ? (int)(last / p.K) - q0 + 1 : 0;  // <= 128: fits the ring
            const int et = (warp & 3) * 32 + lane;                      // 0..127
            const int64_t slab = (int64_t)p.Q * p.H;
            if (done)
                for (int t = et; t < nq * kSkvHidden; t += kSkvRows) {
                    const float *src = p.cq + (int64_t)(q0 + t / kSkvHidden) * p.H + n0 + t % kSkvHidden;
                    float v = 0.f;
                    for (int z = 0; z < p.cq_splits; ++z) v += src[z * slab];
                    cqs[t] = v;
                }
            asm volatile("bar.sync 1, %0;" ::"r"(kSkvRows) : "memory");  // the four epilogue warps
            if (done) {
                const uint32_t lane_addr = (uint32_t)((warp & 3) * 32) << 16;
                // rows past the last slot (q = 0) read question q0's entries and write
                // nothing; the index is clamped to the staged questions in any case
                const int qq = slot < p.P ? q - q0 : 0;
                const float *cq = cqs + (qq < 0 ? 0 : qq >= nq ? (nq > 0 ? nq - 1 : 0) : qq) * kSkvHidden;
                const float *w2 = p.w2 + n0;
                float part = 0.f;
#pragma unroll 1
                for (int c = 0; c < kSkvHidden / 32; ++c) {
                    uint32_t v[32];
                    tmem_ld_32x32b_x32(tmem + lane_addr + c * 32, v);
                    tmem_ld_wait(v);
#pragma unroll
                    for (int i = 0; i < 32; ++i) {
                        const float h = __uint_as_float(v[i]) + cq[c * 32 + i];
                        part = fmaf(fmaxf(h, 0.f), __ldg(w2 + c * 32 + i), part);
                    }
                }
                if (slot < p.P) p.partial[(int64_t)blockIdx.y * p.P + slot] = part;
            }
        }
    }

    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 1) {
        __syncwarp();
        tmem_dealloc(tmem, kSkvHidden);
    }
}

// One block per question: nu for every slot, the gate, and the first n by
// (nu desc, id asc).  Keys (ordered nu bits << 32 | ~id) sort descending.
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
    const int nb = p.H / kSkvHidden;
    int my_ne = 0, my_g = 0;
    for (int j = threadIdx.x; j < Kp; j += kSelThreads) {
        uint64_t key = 0;
        if (j < K) {
            const int64_t slot = (int64_t)q * K + j;
            int64_t id = p.ids[slot];
            if (id >= p.N) id = -1;  // flagged by k_skv_mlp
            float nu = -__int_as_float(0x7f800000);
            if (id >= 0) {
                float logit = p.b2;
                for (int b = 0; b < nb; ++b) logit += p.partial[(int64_t)b * p.P + slot];
                nu = 1.f / (1.f + expf(-logit));
                ++my_ne;
                if (nu >= p.tau) {
                    key = ((uint64_t)(__float_as_uint(nu) | 0x80000000u) << 32) |
                          (uint64_t)(0xFFFFFFFFu - (uint32_t)id);
                    ++my_g;
                }
            }
            if (p.nu_all) p.nu_all[slot] = nu;
        }
        keys[j] = key;
    }
    if (my_ne) atomicAdd(&nonempty, my_ne);
    if (my_g) atomicAdd(&ngated, my_g);
    __syncthreads();
    // bitonic sort, descending
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
    const double nd = ceil((double)p.rho * (double)nonempty - 1e-3);
    int n = nd < 0.0 ? 0 : (int)nd;
    if (n > nonempty) n = nonempty;
    if (n > ngated) n = ngated;
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
    if (threadIdx.x == 0) p.out_count[q] = n;
}

}  // namespace

size_t skv_mlp_smem_bytes() {
    return 1024 + (size_t)kSkvStagesA * kSkvStageA + (size_t)kSkvStagesB * kSkvStageB + sizeof(SkvShared);
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

cudaError_t launch_skv_mlp(const CUtensorMap &tw, const SkvParams &p, cudaStream_t s) {
    if (p.Q == 0) return cudaSuccess;
    const size_t smem = skv_mlp_smem_bytes();
    cudaError_t e = cudaFuncSetAttribute(k_skv_mlp, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    dim3 grid((unsigned)((p.P + kSkvRows - 1) / kSkvRows), (unsigned)(p.H / kSkvHidden));
    return launch_dependent(k_skv_mlp, grid, kSkvThreads, smem, s, tw, p);
}

cudaError_t launch_skv_select(const SkvParams &p, cudaStream_t s) {
    if (p.Q == 0) return cudaSuccess;
    return launch_dependent(k_skv_select, dim3((unsigned)p.Q), kSelThreads, 0, s, p);
}

}  // namespace skipk
