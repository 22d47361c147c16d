// SKV passage gate (App. B.4 Def. B.4, Eq. skv_score; Alg. 1 "SKV: verify"
// and the TopK after it) on the merged retrieval lists.
//
//  (k_gemm)      per question: c_q = b1 + W1[:, qbar] qbar + W1[:, vbar] vbar
//                for all questions at once, on the tensor cores (k_gemm.cu).
//  k_skv_features per passage slot: F = [e | bf16(e * qbar) | bf16(|e - qbar|)]
//                (3d bf16 in the column order of W1's passage blocks), from
//                the gathered corpus row and qbar; zeros for an empty slot.
//                Runs while the c_q GEMM runs (programmatic dependent).
//  k_skv_mlp     per 128 passage slots x 128 hidden units: the passage part
//                of layer 1 on the tensor cores, both operands by TMA (the
//                feature rows and the matching W1 column blocks) into a
//                six-stage ring; tcgen05.mma (kind::f16, M = N = 128)
//                accumulates in TMEM; the epilogue adds c_q, applies ReLU
//                and the w2 dot for its 128 units and writes one partial
//                logit per slot and hidden block.  (Building the features in
//                shared memory inside this kernel instead, once per hidden
//                block, made the builders and their hand-offs set the pace.)
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
// A stage holds one K-slice of A (64 feature columns of 128 slots) and of B
// (the matching W1 column block for 128 units), both copied by TMA.
constexpr int kSkvStageA = kSkvSlice;
constexpr int kSkvStageB = kSkvSlice;
constexpr int kSkvStages = 6;
constexpr int kSkvThreads = 192;                     // TMA warp, MMA warp, four epilogue warps
constexpr uint32_t kSkvIdesc = idesc_bf16_f32(128, kSkvHidden);
constexpr uint64_t kDrainTimeoutNs = 1000000000ull;  // 1 s for copies in flight
constexpr int kFeatWarps = 8;                        // slots per feature block

struct SkvShared {
    uint64_t full[kSkvStages];   // A and B slices landed (tx bytes)
    uint64_t empty[kSkvStages];  // stage consumed (tcgen05.commit)
    uint64_t tfull;              // accumulator complete
    uint32_t tmem_base;
};

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
// c_q GEMM: it gathers while the GEMM runs and, before it completes, waits
// for the GEMM, so that a kernel waiting for this grid also sees c_q.
__global__ void __launch_bounds__(32 * kFeatWarps) k_skv_features(const SkvParams p, uint16_t *__restrict__ F) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t slot = (int64_t)blockIdx.x * kFeatWarps + warp;
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
        for (int w0 = 0; w0 < nw; w0 += 64) {
            uint4 e[2], qv[2];
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                const int w = w0 + lane + 32 * h;
                e[h] = (id >= 0 && w < nw) ? __ldg(erow + w) : zero;
                qv[h] = (id >= 0 && w < nw) ? __ldg(qrow + w) : zero;
            }
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                const int w = w0 + lane + 32 * h;
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
    grid_dep_wait();
}

__global__ void __launch_bounds__(kSkvThreads, 1)
    k_skv_mlp(const __grid_constant__ CUtensorMap tf, const __grid_constant__ CUtensorMap tw, const SkvParams p) {
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t *sA = smem;
    uint8_t *sB = smem + kSkvStages * kSkvStageA;
    SkvShared *sh = reinterpret_cast<SkvShared *>(sB + kSkvStages * kSkvStageB);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t m0 = (int64_t)blockIdx.x * kSkvRows;
    const int n0 = blockIdx.y * kSkvHidden;
    const int nsl = 3 * (p.d / 64);  // K-slices: 3d / 64

    if (threadIdx.x == 0) {
        for (int s = 0; s < kSkvStages; ++s) {
            mbar_init(smem_addr(&sh->full[s]), 1);
            mbar_init(smem_addr(&sh->empty[s]), 1);
        }
        mbar_init(smem_addr(&sh->tfull), 1);
        mbar_fence_init();
    }
    if (warp == 0 && lane == 0) {
        tma_prefetch_desc(&tf);
        tma_prefetch_desc(&tw);
    }
    if (warp == 1) {
        tmem_alloc(smem_addr(&sh->tmem_base), kSkvHidden);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = sh->tmem_base;

    if (warp == 0) {
        // ------------------------------------------------ TMA: features and W1 blocks
        if (lane == 0) {
            // the features (and through them c_q) come from the kernels before this one
            grid_dep_wait();
            bool ok = true;
            int issued = 0;
            for (int u = 0; u < nsl && ok; ++u) {
                const int s = u % kSkvStages;
                const uint32_t ph = (uint32_t)(u / kSkvStages) & 1u;
                if (!mbar_wait(smem_addr(&sh->empty[s]), ph ^ 1u, p.timeout_ns)) {
                    ok = false;
                    break;
                }
                const uint32_t fb = smem_addr(&sh->full[s]);
                mbar_arrive_expect_tx(fb, kSkvStageA + kSkvStageB);
                tma_load_2d(smem_addr(sA + s * kSkvStageA), &tf, fb, u * 64, (int)m0);
                tma_load_2d(smem_addr(sB + s * kSkvStageB), &tw, fb, 2 * p.d + u * 64, n0);
                ++issued;
            }
            if (!ok) atomicOr(p.err, kErrTimeout);
            // Copies in flight: wait for the last use of each stage to complete.
            for (int s = 0; s < kSkvStages; ++s) {
                const int uses = issued / kSkvStages + (s < issued % kSkvStages ? 1 : 0);
                if (uses == 0) continue;
                if (!mbar_wait(smem_addr(&sh->full[s]), (uint32_t)((uses - 1) & 1), kDrainTimeoutNs))
                    atomicOr(p.err, kErrTimeout);
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------ MMA issuer
        if (lane == 0) {
            bool ok = true;
            for (int u = 0; u < nsl && ok; ++u) {
                const int s = u % kSkvStages;
                if (!mbar_wait(smem_addr(&sh->full[s]), (uint32_t)(u / kSkvStages) & 1u, p.timeout_ns)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint64_t ad = smem_desc_k128(smem_addr(sA + s * kSkvStageA));
                const uint64_t bd = smem_desc_k128(smem_addr(sB + s * kSkvStageB));
#pragma unroll
                for (int kk = 0; kk < 4; ++kk)
                    tc_mma_f16(tmem, ad + (uint64_t)(kk * 2), bd + (uint64_t)(kk * 2), kSkvIdesc, (u | kk) != 0);
                tc_commit(smem_addr(&sh->empty[s]));
            }
            if (!ok) atomicOr(p.err, kErrTimeout);
            // Arrives once every MMA issued has completed (also after a timeout).
            tc_commit(smem_addr(&sh->tfull));
        }
    } else {
        // ------------------------------------------------ epilogue (warps 2..5)
        // Epilogue: h = acc + c_q, ReLU, dot with w2 over this CTA's units.
        const int r = (warp & 3) * 32 + lane;  // TMEM lane = slot row in the tile
        const int64_t slot = m0 + r;
        const int q = slot < p.P ? (int)(slot / p.K) : 0;
        const bool done = mbar_wait(smem_addr(&sh->tfull), 0, p.timeout_ns);
        if (!done) atomicOr(p.err, kErrTimeout);
        tc_fence_after();
        grid_dep_wait();
        // c_q of the tile's questions for this CTA's units, the GEMM's K-split
        // slabs summed once, staged in the A ring (free: every MMA that read it
        // has completed; its 96 KB hold 128 questions).  cqs[(q - q0) * 128 + n].
        float *cqs = reinterpret_cast<float *>(sA);
        const int q0 = (int)(m0 / p.K);
        const int64_t last = (m0 + kSkvRows < p.P ? m0 + kSkvRows : p.P) - 1;
        const int nq = m0 < p.P ? (int)(last / p.K) - q0 + 1 : 0;  // <= 128
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
            // rows past the last slot read question q0's entries and write nothing;
            // the index is clamped to the staged questions in any case
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
    return 1024 + (size_t)kSkvStages * (kSkvStageA + kSkvStageB) + sizeof(SkvShared);
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

cudaError_t launch_skv_mlp(const CUtensorMap &tf, const CUtensorMap &tw, const SkvParams &p, cudaStream_t s) {
    if (p.Q == 0) return cudaSuccess;
    const size_t smem = skv_mlp_smem_bytes();
    cudaError_t e = cudaFuncSetAttribute(k_skv_mlp, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    dim3 grid((unsigned)((p.P + kSkvRows - 1) / kSkvRows), (unsigned)(p.H / kSkvHidden));
    return launch_dependent(k_skv_mlp, grid, kSkvThreads, smem, s, tf, tw, p);
}

cudaError_t launch_skv_select(const SkvParams &p, cudaStream_t s) {
    if (p.Q == 0) return cudaSuccess;
    return launch_dependent(k_skv_select, dim3((unsigned)p.Q), kSelThreads, 0, s, p);
}

}  // namespace skipk
