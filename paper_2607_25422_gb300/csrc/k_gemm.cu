// Small dense bf16 GEMM with fp32 results on the tensor cores (tcgen05 /
// TMEM / TMA, sm_103a), for the two plain products that sit next to the hot
// path:
//  * the QVS projected query U = F_q W_v / sqrt(d_k) of all images at once
//    (App. B.1 Def. B.1: <f_q, W_v v> = <W_v^T f_q, v>), with W_v^T kept by
//    the QVS handle so that both operands are K-major;
//  * the IVF-PQ coarse probe scores S = Q C^T of all regions against every
//    centroid (the inverted file's coarse quantiser, §4.1 "Implementation").
//
//   D[m][n] = alpha * (sum_k A[m][k] B[n][k] + sum_k A2[m][k] B2[n][k]) + bias[n]
//   A [M x K], B [N x K], A2 [M x K2], B2 [N x K2] bf16 row-major (K
//   contiguous; the second product and the bias are optional), D fp32
//   row-major with leading dimension ldd.  The SKV gate's per-question half
//   of layer 1 is such a sum (its qbar and vbar column blocks of W1).
//
// Split K (splits > 1, for products with few output tiles): CTA z of a
// tile takes the z-th share of the K slices (both products counted
// together) and writes its partial tile to D + z * split_stride; the caller
// sums the `splits` slabs (the bias goes into slab 0 only).
//
// One CTA computes one 128 x BN tile of D (BN = 64, or 32 when that leaves
// too few tiles to occupy the GPU): warp 0 streams K slices of 64 elements
// (128 bytes, 128-byte swizzle) of both operands into an eight-stage
// shared-memory ring by TMA (rows past M or N are zero-filled by the copy),
// one thread of warp 1 issues tcgen05.mma (kind::f16, M = 128, N = BN)
// into a TMEM accumulator, and warps 2..5 read it back (warp w: TMEM lanes
// 32 (w mod 4) .. + 31, i.e. rows of D) and store their rows, masked at the
// M and N edges.  Every wait is bounded; a wait that gives up sets *err (if
// given) and the roles drain their copies and MMAs before TMEM is freed.
#include <algorithm>

#include "skip_device.cuh"
#include "skip_internal.h"

namespace skipk {
namespace {

constexpr int kStages = 8;
constexpr int kABytes = 128 * 64 * 2;      // 16 KB: 128 rows x 64 elements
constexpr int kThreads = 192;
constexpr uint64_t kDrainTimeoutNs = 1000000000ull;

template <int BN>
struct GemmGeom {
    static constexpr int kBBytes = BN * 64 * 2;
    static constexpr int kStageBytes = kABytes + kBBytes;
    static constexpr uint32_t kTmemCols = BN;  // one fp32 accumulator (power of two >= 32)
};

struct __align__(8) GemmShared {
    uint64_t full[kStages];
    uint64_t empty[kStages];
    uint64_t done;
    uint32_t tmem_base;
};

template <int BN>
__global__ void __launch_bounds__(kThreads, 1)
    k_gemm_bf16_f32(const __grid_constant__ CUtensorMap ta, const __grid_constant__ CUtensorMap tb,
                    const __grid_constant__ CUtensorMap ta2, const __grid_constant__ CUtensorMap tb2, int M, int N,
                    int K, int K2, float alpha, const float *__restrict__ bias, float *__restrict__ D, int64_t ldd,
                    int64_t split_stride, int *err, uint64_t timeout_ns) {
    constexpr int kBBytes = GemmGeom<BN>::kBBytes;
    constexpr int kStageBytes = GemmGeom<BN>::kStageBytes;
    constexpr uint32_t kTmemCols = GemmGeom<BN>::kTmemCols;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    uint8_t *sA = smem;
    uint8_t *sB = smem + kStages * kABytes;
    GemmShared *sh = reinterpret_cast<GemmShared *>(smem + kStages * kStageBytes);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int m0 = blockIdx.x * 128, n0 = blockIdx.y * BN;
    const int KB1 = (K + 63) / 64;
    const int KBall = KB1 + (K2 + 63) / 64;
    // this CTA's share of the K slices [kb0, kb0 + KB)
    const int kb0 = (int)((int64_t)blockIdx.z * KBall / gridDim.z);
    const int KB = (int)((int64_t)(blockIdx.z + 1) * KBall / gridDim.z) - kb0;
    if (blockIdx.z > 0) {
        D += (int64_t)blockIdx.z * split_stride;
        bias = nullptr;
    }
    constexpr uint32_t kIdesc = idesc_bf16_f32(128, BN);

    // A kernel launched as this one's programmatic dependent may start now:
    // it waits for this grid's results itself (griddepcontrol.wait).
    grid_dep_launch();
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
        if (K2 > 0) {
            tma_prefetch_desc(&ta2);
            tma_prefetch_desc(&tb2);
        }
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
                const int kg = kb0 + kb;  // slice index over both products
                const bool first = kg < KB1;
                const int x = (first ? kg : kg - KB1) * 64;
                tma_load_2d(smem_addr(sA + s * kABytes), first ? &ta : &ta2, fb, x, m0);
                tma_load_2d(smem_addr(sB + s * kBBytes), first ? &tb : &tb2, fb, x, n0);
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
            for (int c = 0; c < BN; c += 32) {
                uint32_t v[32];
                tmem_ld_32x32b_x32(tmem + ((uint32_t)(sub * 32) << 16) + (uint32_t)c, v);
                tmem_ld_wait(v);
                if (KB == 0) {
                    // an empty share of K (more splits than slices): zeros
#pragma unroll
                    for (int j = 0; j < 32; ++j) v[j] = 0u;
                }
                if (bias) {
#pragma unroll
                    for (int j = 0; j < 32; ++j) {
                        const int n = n0 + c + j;
                        v[j] = __float_as_uint(alpha * __uint_as_float(v[j]) + (n < N ? __ldg(bias + n) : 0.f));
                    }
                } else {
#pragma unroll
                    for (int j = 0; j < 32; ++j) v[j] = __float_as_uint(alpha * __uint_as_float(v[j]));
                }
                if (row < M) {
                    const int nc = N - (n0 + c);
                    if (nc >= 32 && (ldd & 3) == 0) {
                        float4 *o = reinterpret_cast<float4 *>(drow + n0 + c);
#pragma unroll
                        for (int j = 0; j < 8; ++j)
                            o[j] = make_float4(__uint_as_float(v[4 * j]), __uint_as_float(v[4 * j + 1]),
                                               __uint_as_float(v[4 * j + 2]), __uint_as_float(v[4 * j + 3]));
                    } else {
#pragma unroll
                        for (int j = 0; j < 32; ++j)
                            if (j < nc) drow[n0 + c + j] = __uint_as_float(v[j]);
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

template <int BN>
size_t gemm_smem_bytes() {
    return 1024 + (size_t)kStages * GemmGeom<BN>::kStageBytes + sizeof(GemmShared);
}

template <int BN>
cudaError_t launch_bn(const CUtensorMap &ta, const CUtensorMap &tb, const CUtensorMap &ta2, const CUtensorMap &tb2,
                      int M, int N, int K, int K2, float alpha, const float *bias, float *D, int64_t ldd, int splits,
                      int64_t split_stride, int *err, uint64_t timeout_ns, cudaStream_t s) {
    const size_t smem = gemm_smem_bytes<BN>();
    cudaError_t e = cudaFuncSetAttribute(k_gemm_bf16_f32<BN>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    dim3 grid((unsigned)((M + 127) / 128), (unsigned)((N + BN - 1) / BN), (unsigned)splits);
    k_gemm_bf16_f32<BN><<<grid, kThreads, smem, s>>>(ta, tb, ta2, tb2, M, N, K, K2, alpha, bias, D, ldd,
                                                     split_stride, err, timeout_ns);
    return cudaGetLastError();
}

}  // namespace

int gemm_tile_n(int M, int N, int sms) {
    const int64_t tiles64 = (int64_t)((M + 127) / 128) * ((N + 63) / 64);
    return tiles64 * 2 <= sms ? 32 : 64;
}

int gemm_splits(int M, int N, int K, int tile_n, int sms) {
    const int64_t tiles = (int64_t)((M + 127) / 128) * ((N + tile_n - 1) / tile_n);
    const int kb = (K + 63) / 64;
    // at least two K slices per split; no more splits than fill the SMs once
    return (int)std::max<int64_t>(1, std::min<int64_t>(std::min<int64_t>(kb / 2, 16), sms / std::max<int64_t>(1, tiles)));
}

cudaError_t launch_gemm2_bf16_f32(const CUtensorMap &ta, const CUtensorMap &tb, const CUtensorMap *ta2,
                                  const CUtensorMap *tb2, int tile_n, int M, int N, int K, int K2, float alpha,
                                  const float *bias, float *D, int64_t ldd, int *err, uint64_t timeout_ns,
                                  cudaStream_t s, int splits, int64_t split_stride) {
    if (M <= 0 || N <= 0) return cudaSuccess;
    if (K <= 0 || (K & 7) != 0 || K2 < 0 || (K2 & 7) != 0 || (K2 > 0 && (!ta2 || !tb2))) return cudaErrorInvalidValue;
    if (splits < 1 || splits > 64 || (splits > 1 && split_stride < (int64_t)M * ldd)) return cudaErrorInvalidValue;
    const CUtensorMap &a2 = K2 > 0 ? *ta2 : ta, &b2 = K2 > 0 ? *tb2 : tb;
    if (tile_n == 32)
        return launch_bn<32>(ta, tb, a2, b2, M, N, K, K2, alpha, bias, D, ldd, splits, split_stride, err, timeout_ns, s);
    if (tile_n == 64)
        return launch_bn<64>(ta, tb, a2, b2, M, N, K, K2, alpha, bias, D, ldd, splits, split_stride, err, timeout_ns, s);
    return cudaErrorInvalidValue;
}

cudaError_t launch_gemm_bf16_f32(const CUtensorMap &ta, const CUtensorMap &tb, int tile_n, int M, int N, int K,
                                 float alpha, float *D, int64_t ldd, int *err, uint64_t timeout_ns, cudaStream_t s,
                                 int splits, int64_t split_stride) {
    return launch_gemm2_bf16_f32(ta, tb, nullptr, nullptr, tile_n, M, N, K, 0, alpha, nullptr, D, ldd, err, timeout_ns,
                                 s, splits, split_stride);
}

}  // namespace skipk
