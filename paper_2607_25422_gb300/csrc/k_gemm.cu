// Small dense bf16 GEMM with fp32 results on the tensor cores (tcgen05 /
// TMEM / TMA, sm_103a), for the two plain products that sit next to the hot
// path:
//  * the QVS projected query U = F_q W_v / sqrt(d_k) of all images at once
//    (App. B.1 Def. B.1: <f_q, W_v v> = <W_v^T f_q, v>), with W_v^T kept by
//    the QVS handle so that both operands are K-major;
//  * the IVF-PQ coarse probe scores S = Q C^T of all regions against every
//    centroid (the inverted file's coarse quantiser, §4.1 "Implementation").
//
//   D[m][n] = alpha * sum_k A[m][k] B[n][k],   A [M x K], B [N x K] bf16
//   row-major (K contiguous), D fp32 row-major with leading dimension ldd.
//
// One CTA computes one 128 x kGemmN tile of D: warp 0 streams K slices of 64
// elements (128 bytes, 128-byte swizzle) of both operands into a four-stage
// shared-memory ring by TMA (rows past M or N are zero-filled by the copy),
// one thread of warp 1 issues tcgen05.mma (kind::f16, M = 128, N = kGemmN)
// into a TMEM accumulator, and warps 2..5 read it back (warp w: TMEM lanes
// 32 (w mod 4) .. + 31, i.e. rows of D) and store their rows, masked at the
// M and N edges.  Every wait is bounded; a wait that gives up sets *err (if
// given) and the roles drain their copies and MMAs before TMEM is freed.
#include "skip_device.cuh"
#include "skip_internal.h"

namespace skipk {
namespace {

constexpr int kStages = 4;
constexpr int kABytes = 128 * 64 * 2;      // 16 KB: 128 rows x 64 elements
constexpr int kBBytes = kGemmN * 64 * 2;   // 8 KB
constexpr int kStageBytes = kABytes + kBBytes;
constexpr int kThreads = 192;
constexpr uint32_t kTmemCols = kGemmN;     // one fp32 accumulator (power of two >= 32)
constexpr uint64_t kDrainTimeoutNs = 1000000000ull;

struct __align__(8) GemmShared {
    uint64_t full[kStages];
    uint64_t empty[kStages];
    uint64_t done;
    uint32_t tmem_base;
};

__global__ void __launch_bounds__(kThreads, 1)
    k_gemm_bf16_f32(const __grid_constant__ CUtensorMap ta, const __grid_constant__ CUtensorMap tb, int M, int N,
                    int K, float alpha, float *__restrict__ D, int64_t ldd, int *err, uint64_t timeout_ns) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    uint8_t *sA = smem;
    uint8_t *sB = smem + kStages * kABytes;
    GemmShared *sh = reinterpret_cast<GemmShared *>(smem + kStages * kStageBytes);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int m0 = blockIdx.x * 128, n0 = blockIdx.y * kGemmN;
    const int KB = (K + 63) / 64;
    constexpr uint32_t kIdesc = idesc_bf16_f32(128, kGemmN);

    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            mbar_init(smem_addr(&sh->full[s]), 1);
            mbar_init(smem_addr(&sh->empty[s]), 1);
        }
        mbar_init(smem_addr(&sh->done), 1);
        mbar_fence_init();
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
    bool ok = true;

    if (warp == 0) {
        if (lane == 0) {
            int issued = 0;
            for (int kb = 0; kb < KB; ++kb) {
                const int s = kb % kStages;
                const uint32_t ph = (uint32_t)(kb / kStages) & 1u;
                if (!mbar_wait(smem_addr(&sh->empty[s]), ph ^ 1u, timeout_ns)) {
                    ok = false;
                    break;
                }
                const uint32_t fb = smem_addr(&sh->full[s]);
                mbar_arrive_expect_tx(fb, kStageBytes);
                tma_load_2d(smem_addr(sA + s * kABytes), &ta, fb, kb * 64, m0);
                tma_load_2d(smem_addr(sB + s * kBBytes), &tb, fb, kb * 64, n0);
                ++issued;
            }
            // copies in flight: the last load issued on every stage
            for (int s = 0; s < kStages; ++s) {
                const int uses = issued / kStages + (s < issued % kStages ? 1 : 0);
                if (uses && !mbar_wait(smem_addr(&sh->full[s]), (uint32_t)((uses - 1) & 1), kDrainTimeoutNs))
                    ok = false;
            }
            if (!ok && err) atomicOr(err, kErrTimeout);
        }
    } else if (warp == 1) {
        if (lane == 0) {
            for (int kb = 0; kb < KB; ++kb) {
                const int s = kb % kStages;
                const uint32_t ph = (uint32_t)(kb / kStages) & 1u;
                if (!mbar_wait(smem_addr(&sh->full[s]), ph, timeout_ns)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint64_t ad = smem_desc_k128(smem_addr(sA + s * kABytes));
                const uint64_t bd = smem_desc_k128(smem_addr(sB + s * kBBytes));
#pragma unroll
                for (int kk = 0; kk < 4; ++kk)
                    tc_mma_f16(tmem, ad + (uint64_t)(kk * 2), bd + (uint64_t)(kk * 2), kIdesc, (kb | kk) != 0);
                tc_commit(smem_addr(&sh->empty[s]));
            }
            // Arrives once every MMA issued above has completed (also after a
            // give-up, so that nothing is outstanding when TMEM is freed).
            tc_commit(smem_addr(&sh->done));
            if (!ok && err) atomicOr(err, kErrTimeout);
        }
    } else {
        const int sub = warp & 3;
        const bool got = mbar_wait(smem_addr(&sh->done), 0, ok ? timeout_ns : kDrainTimeoutNs);
        if (__all_sync(0xffffffffu, got)) {
            tc_fence_after();
            const int row = m0 + sub * 32 + lane;
            float *drow = D + (int64_t)row * ldd;
#pragma unroll 1
            for (int c = 0; c < kGemmN; c += 32) {
                uint32_t v[32];
                tmem_ld_32x32b_x32(tmem + ((uint32_t)(sub * 32) << 16) + (uint32_t)c, v);
                tmem_ld_wait(v);
                if (row < M) {
                    const int nc = N - (n0 + c);
                    if (nc >= 32 && (ldd & 3) == 0) {
                        float4 *o = reinterpret_cast<float4 *>(drow + n0 + c);
#pragma unroll
                        for (int j = 0; j < 8; ++j)
                            o[j] = make_float4(alpha * __uint_as_float(v[4 * j]), alpha * __uint_as_float(v[4 * j + 1]),
                                               alpha * __uint_as_float(v[4 * j + 2]),
                                               alpha * __uint_as_float(v[4 * j + 3]));
                    } else {
#pragma unroll
                        for (int j = 0; j < 32; ++j)
                            if (j < nc) drow[n0 + c + j] = alpha * __uint_as_float(v[j]);
                    }
                }
            }
        } else if (lane == 0 && err) {
            atomicOr(err, kErrTimeout);
        }
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

size_t gemm_smem_bytes() { return 1024 + (size_t)kStages * kStageBytes + sizeof(GemmShared); }

cudaError_t launch_gemm_bf16_f32(const CUtensorMap &ta, const CUtensorMap &tb, int M, int N, int K, float alpha,
                                 float *D, int64_t ldd, int *err, uint64_t timeout_ns, cudaStream_t s) {
    if (M <= 0 || N <= 0) return cudaSuccess;
    if (K <= 0 || (K & 7) != 0) return cudaErrorInvalidValue;
    const size_t smem = gemm_smem_bytes();
    cudaError_t e = cudaFuncSetAttribute(k_gemm_bf16_f32, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    dim3 grid((unsigned)((M + 127) / 128), (unsigned)((N + kGemmN - 1) / kGemmN));
    k_gemm_bf16_f32<<<grid, kThreads, smem, s>>>(ta, tb, M, N, K, alpha, D, ldd, err, timeout_ns);
    return cudaGetLastError();
}

}  // namespace skipk
