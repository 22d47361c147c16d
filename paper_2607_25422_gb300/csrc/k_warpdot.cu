// Warp-dot score + fused top-k for small region batches (latency mode).
//
// Step: per-region MIPS top-k (paper App. B.2 Def. B.2, MIPS(q_r, D; k_r);
// §3.3 Eq. rcsr).  For a handful of region queries the contraction has too
// little reuse for the tensor cores, and the kernel is bound by streaming the
// corpus from HBM, so each lane owns one corpus row at a time: it reads the
// row in 128-byte lines with 16-byte vector loads, widens bf16 (or e4m3 times
// the row scale) to fp32 and accumulates the dot products with all queries of
// the batch, whose fp32 copies sit in shared memory and are read as warp-wide
// broadcasts.  Scores never leave registers: each warp keeps, per query, a
// sorted top-k list and a threshold (the current k-th score); a warp ballot
// finds the rare rows that beat it.  Rows are visited in increasing id order,
// so "beats" is a strict score comparison and ties keep the lower id.  At the
// end the block merges its warps' lists into one list per query.
#include "skip_device.cuh"
#include "skip_internal.h"

namespace skipk {
namespace {

template <int RMAX>
__device__ __forceinline__ void fma_queries(float (&acc)[RMAX], const float *q, float x) {
    if constexpr (RMAX % 4 == 0) {
#pragma unroll
        for (int r = 0; r < RMAX; r += 4) {
            const float4 v = *reinterpret_cast<const float4 *>(q + r);
            acc[r + 0] = fmaf(v.x, x, acc[r + 0]);
            acc[r + 1] = fmaf(v.y, x, acc[r + 1]);
            acc[r + 2] = fmaf(v.z, x, acc[r + 2]);
            acc[r + 3] = fmaf(v.w, x, acc[r + 3]);
        }
    } else {
#pragma unroll
        for (int r = 0; r < RMAX; ++r) acc[r] = fmaf(q[r], x, acc[r]);
    }
}

// One 16-byte vector of a bf16 row: 8 elements starting at element j.
template <int RMAX>
__device__ __forceinline__ void dot_vec_bf16(float (&acc)[RMAX], const float *sq, int j, uint4 v) {
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int t = 0; t < 4; ++t) {
        fma_queries<RMAX>(acc, sq + (j + 2 * t) * RMAX, __uint_as_float(w[t] << 16));
        fma_queries<RMAX>(acc, sq + (j + 2 * t + 1) * RMAX, __uint_as_float(w[t] & 0xFFFF0000u));
    }
}

// One 16-byte vector of an e4m3 row: 16 elements starting at element j.
template <int RMAX>
__device__ __forceinline__ void dot_vec_e4m3(float (&acc)[RMAX], const float *sq, int j, uint4 v) {
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int t = 0; t < 4; ++t) {
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            const __nv_fp8x2_storage_t pair = (__nv_fp8x2_storage_t)((w[t] >> (16 * h)) & 0xFFFFu);
            const __half2 hv = __half2(__nv_cvt_fp8x2_to_halfraw2(pair, __NV_E4M3));
            const float2 f = __half22float2(hv);
            const int e = j + 4 * t + 2 * h;
            fma_queries<RMAX>(acc, sq + e * RMAX, f.x);
            fma_queries<RMAX>(acc, sq + (e + 1) * RMAX, f.y);
        }
    }
}

template <int RMAX, bool E4M3>
__global__ void __launch_bounds__(kWarpDotThreads) k_warpdot_score_topk(WarpDotParams p) {
    extern __shared__ float4 smem_f4[];
    float *sq = reinterpret_cast<float *>(smem_f4);  // [d][RMAX], fp32 queries
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int d = p.d;

    for (int idx = tid; idx < d * RMAX; idx += blockDim.x) {
        const int j = idx / RMAX, r = idx % RMAX;
        float v = 0.0f;
        if (r < p.nq) v = __uint_as_float((uint32_t)p.regions[(int64_t)r * d + j] << 16);
        sq[idx] = v;
    }
    __syncthreads();

    // Contiguous corpus rows for this block, then for this warp.
    const int64_t per_cta = (p.N + gridDim.x - 1) / gridDim.x;
    const int64_t c0 = (int64_t)blockIdx.x * per_cta;
    const int64_t c1 = min(p.N, c0 + per_cta);
    const int64_t span = c1 > c0 ? c1 - c0 : 0;
    const int64_t per_w = (span + kWarpDotWarps - 1) / kWarpDotWarps;
    const int64_t w0 = c0 + (int64_t)warp * per_w;
    const int64_t w1 = min(c1, w0 + per_w);

    uint64_t *wl = p.warp_lists + ((int64_t)(blockIdx.x * kWarpDotWarps + warp) * p.nq) * p.k;
    float thr[RMAX];
    int nfill[RMAX];
#pragma unroll
    for (int r = 0; r < RMAX; ++r) {
        thr[r] = -__int_as_float(0x7f800000);
        nfill[r] = 0;
    }

    const int64_t row_bytes = (int64_t)d * (E4M3 ? 1 : 2);
    const int nvec = (int)(row_bytes / 16);
    constexpr int kElemsPerVec = E4M3 ? 16 : 8;

    for (int64_t b = w0; b < w1; b += 32) {
        const int64_t row = b + lane;
        const bool valid = row < w1;
        const uint4 *src = reinterpret_cast<const uint4 *>(p.corpus + (valid ? row : b) * row_bytes);
        float acc[RMAX];
#pragma unroll
        for (int r = 0; r < RMAX; ++r) acc[r] = 0.0f;

        for (int v0 = 0; v0 < nvec; v0 += 8) {
            uint4 buf[8];
#pragma unroll
            for (int t = 0; t < 8; ++t)
                buf[t] = (valid && v0 + t < nvec) ? __ldg(src + v0 + t) : make_uint4(0, 0, 0, 0);
#pragma unroll
            for (int t = 0; t < 8; ++t) {
                if (v0 + t < nvec) {
                    const int j = (v0 + t) * kElemsPerVec;
                    if constexpr (E4M3)
                        dot_vec_e4m3<RMAX>(acc, sq, j, buf[t]);
                    else
                        dot_vec_bf16<RMAX>(acc, sq, j, buf[t]);
                }
            }
        }
        if constexpr (E4M3) {
            const float sc = valid ? __ldg(p.scale + row) : 0.0f;
#pragma unroll
            for (int r = 0; r < RMAX; ++r) acc[r] *= sc;
        }

#pragma unroll
        for (int r = 0; r < RMAX; ++r) {
            if (r >= p.nq) break;
            unsigned m = __ballot_sync(0xffffffffu, valid && acc[r] > thr[r]);
            while (m) {
                const int l = __ffs(m) - 1;
                m &= m - 1;
                const float sv = __shfl_sync(0xffffffffu, acc[r], l);
                if (sv > thr[r]) {
                    uint64_t kth = 0;
                    int nn = nfill[r];
                    if (lane == 0) kth = sorted_insert(wl + (int64_t)r * p.k, nn, p.k, make_key(sv, (uint32_t)(b + l)));
                    kth = __shfl_sync(0xffffffffu, kth, 0);
                    nfill[r] = __shfl_sync(0xffffffffu, nn, 0);
                    thr[r] = kth ? key_score(kth) : -__int_as_float(0x7f800000);
                }
            }
        }
    }

    // Empty slots of short lists.
#pragma unroll
    for (int r = 0; r < RMAX; ++r) {
        if (r >= p.nq) break;
        for (int t = nfill[r] + lane; t < p.k; t += 32) wl[(int64_t)r * p.k + t] = 0ull;
    }
    __syncthreads();

    // Block merge: one list per query from the block's warps.
    for (int r = warp; r < p.nq; r += kWarpDotWarps) {
        const uint64_t *base =
            p.warp_lists + ((int64_t)blockIdx.x * kWarpDotWarps * p.nq + r) * p.k;
        uint64_t *out = p.lists + (int64_t)blockIdx.x * p.list_g_stride + (int64_t)(p.q0 + r) * p.k;
        warp_merge_topk<1>(base, (int64_t)p.nq * p.k, kWarpDotWarps, p.k, p.k,
                           [&](int i, uint64_t key) { out[i] = key; });
    }
}

template <int RMAX, bool E4M3>
cudaError_t launch_one(const WarpDotParams &p, int grid, cudaStream_t s) {
    const size_t smem = (size_t)p.d * RMAX * sizeof(float);
    auto kern = k_warpdot_score_topk<RMAX, E4M3>;
    if (smem > 48 * 1024) {
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
    }
    kern<<<grid, kWarpDotThreads, smem, s>>>(p);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_warpdot(const WarpDotParams &p, bool e4m3, int grid, cudaStream_t s) {
    const int rmax = p.nq <= 1 ? 1 : p.nq <= 2 ? 2 : p.nq <= 4 ? 4 : 8;
    if (p.nq > 8 || p.nq < 1) return cudaErrorInvalidValue;
    if (e4m3) {
        switch (rmax) {
            case 1: return launch_one<1, true>(p, grid, s);
            case 2: return launch_one<2, true>(p, grid, s);
            case 4: return launch_one<4, true>(p, grid, s);
            default: return launch_one<8, true>(p, grid, s);
        }
    }
    switch (rmax) {
        case 1: return launch_one<1, false>(p, grid, s);
        case 2: return launch_one<2, false>(p, grid, s);
        case 4: return launch_one<4, false>(p, grid, s);
        default: return launch_one<8, false>(p, grid, s);
    }
}

}  // namespace skipk
