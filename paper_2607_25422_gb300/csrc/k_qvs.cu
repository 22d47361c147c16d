// QVS, question-guided visual token pruning (App. B.1 Def. B.1, Eq.
// qvs_score; Alg. 1 "QVS: prune").  With f_v linear,
//   logit_i = <f_q, W_v v_i + b_v> / sqrt(d_k) + <w_b, v_i> = <u, v_i> + c,
//   u = W_v^T f_q / sqrt(d_k) + w_b,  c = <f_q, b_v> / sqrt(d_k),
// so the per-token work is one inner product (the scan reads every token
// once: HBM-bound), and the ranking by s = sigmoid(logit) is the ranking by
// the logit.
//
//  k_qvs_u       u and c for eight images per block (W_v read once per eight).
//  k_qvs_logits  one warp per token, 16-byte loads, u in shared memory.
//  k_qvs_select  per image: (logit, ~index) keys sorted descending in shared
//                memory, the first n kept; their sigmoid scores and (optional)
//                the kept token rows copied out.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <algorithm>

#include "skip_device.cuh"
#include "skip_internal.h"

namespace skipk {
namespace {

constexpr int kUImgs = 8, kUThreads = 128;

__global__ void __launch_bounds__(kUThreads) k_qvs_u(const QvsParams p) {
    extern __shared__ float fq_smem[];  // [kUImgs][dk]
    auto fqs = [&](int u, int k) -> float & { return fq_smem[u * p.dk + k]; };
    const int b0 = blockIdx.y * kUImgs;
    const int j = blockIdx.x * kUThreads + threadIdx.x;
    const __nv_bfloat16 *fq = reinterpret_cast<const __nv_bfloat16 *>(p.fq);
    for (int e = threadIdx.x; e < kUImgs * p.dk; e += kUThreads) {
        const int u = e / p.dk, k = e - u * p.dk;
        fqs(u, k) = b0 + u < p.B ? __bfloat162float(fq[(int64_t)(b0 + u) * p.dk + k]) : 0.f;
    }
    __syncthreads();
    const float inv = rsqrtf((float)p.dk);
    if (j < p.d) {
        const __nv_bfloat16 *wv = reinterpret_cast<const __nv_bfloat16 *>(p.wv);
        float acc[kUImgs];
#pragma unroll
        for (int u = 0; u < kUImgs; ++u) acc[u] = 0.f;
        for (int k = 0; k < p.dk; ++k) {
            const float w = __bfloat162float(wv[(int64_t)k * p.d + j]);
#pragma unroll
            for (int u = 0; u < kUImgs; ++u) acc[u] = fmaf(w, fqs(u, k), acc[u]);
        }
        const float wbj = p.wb[j];
#pragma unroll
        for (int u = 0; u < kUImgs; ++u)
            if (b0 + u < p.B) p.u[(int64_t)(b0 + u) * p.d + j] = acc[u] * inv + wbj;
    }
    if (blockIdx.x == 0 && threadIdx.x < 32) {  // c = <f_q, b_v> / sqrt(d_k), one warp per image in turn
        for (int u = 0; u < kUImgs && b0 + u < p.B; ++u) {
            float s = 0.f;
            if (p.bv)
                for (int k = threadIdx.x; k < p.dk; k += 32) s = fmaf(fqs(u, k), p.bv[k], s);
#pragma unroll
            for (int o = 16; o; o >>= 1) s += __shfl_xor_sync(0xFFFFFFFFu, s, o);
            if (threadIdx.x == 0) p.c[b0 + u] = s * inv;
        }
    }
}

constexpr int kLogThreads = 256;

__global__ void __launch_bounds__(kLogThreads) k_qvs_logits(const QvsParams p) {
    extern __shared__ float us[];  // [d]
    const int b = blockIdx.y;
    for (int t = threadIdx.x; t < p.d; t += kLogThreads) us[t] = p.u[(int64_t)b * p.d + t];
    __syncthreads();
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nw = p.d / 8;  // 16-byte words per token
    const float cb = p.c[b];
    for (int i = blockIdx.x * (kLogThreads / 32) + warp; i < p.L; i += gridDim.x * (kLogThreads / 32)) {
        const uint4 *row = reinterpret_cast<const uint4 *>(p.tokens) + ((int64_t)b * p.L + i) * nw;
        float s = 0.f;
        for (int w = lane; w < nw; w += 32) {
            const uint4 x = __ldg(row + w);
            const uint32_t xv[4] = {x.x, x.y, x.z, x.w};
#pragma unroll
            for (int h = 0; h < 4; ++h) {
                const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(&xv[h]));
                s = fmaf(f.x, us[w * 8 + 2 * h], s);
                s = fmaf(f.y, us[w * 8 + 2 * h + 1], s);
            }
        }
#pragma unroll
        for (int o = 16; o; o >>= 1) s += __shfl_xor_sync(0xFFFFFFFFu, s, o);
        if (lane == 0) p.logits[(int64_t)b * p.L + i] = s + cb;
    }
}

constexpr int kSelThreads = 512;

__global__ void __launch_bounds__(kSelThreads) k_qvs_select(const QvsParams p) {
    __shared__ uint64_t keys[kQvsMaxL];
    const int b = blockIdx.x;
    int Lp = 2;
    while (Lp < p.L) Lp <<= 1;
    for (int i = threadIdx.x; i < Lp; i += kSelThreads) {
        uint64_t key = 0;
        if (i < p.L) key = ((uint64_t)ord_of_score(p.logits[(int64_t)b * p.L + i]) << 32) | (uint32_t)(0xFFFFFFFFu - i);
        keys[i] = key;
    }
    __syncthreads();
    for (int size = 2; size <= Lp; size <<= 1)
        for (int stride = size >> 1; stride > 0; stride >>= 1) {
            for (int t = threadIdx.x; t < Lp / 2; t += kSelThreads) {
                const int lo = 2 * t - (t & (stride - 1));
                const int hi = lo + stride;
                const bool desc = (lo & size) == 0;
                const uint64_t x = keys[lo], y = keys[hi];
                if ((x < y) == desc) {
                    keys[lo] = y;
                    keys[hi] = x;
                }
            }
            __syncthreads();
        }
    for (int r = threadIdx.x; r < p.n; r += kSelThreads) {
        const uint64_t key = keys[r];
        p.out_idx[(int64_t)b * p.n + r] = (int32_t)(0xFFFFFFFFu - (uint32_t)key);
        p.out_score[(int64_t)b * p.n + r] = 1.f / (1.f + expf(-score_of_ord((uint32_t)(key >> 32))));
    }
    if (p.out_tokens) {
        const int nw = p.d / 8;
        for (int e = threadIdx.x; e < p.n * nw; e += kSelThreads) {
            const int r = e / nw, w = e - r * nw;
            const int i = (int)(0xFFFFFFFFu - (uint32_t)keys[r]);
            reinterpret_cast<uint4 *>(p.out_tokens)[((int64_t)b * p.n + r) * nw + w] =
                __ldg(reinterpret_cast<const uint4 *>(p.tokens) + ((int64_t)b * p.L + i) * nw + w);
        }
    }
}

}  // namespace

cudaError_t launch_qvs_u(const QvsParams &p, cudaStream_t s) {
    if (p.B == 0) return cudaSuccess;
    const size_t smem = (size_t)kUImgs * p.dk * sizeof(float);
    cudaError_t e = cudaFuncSetAttribute(k_qvs_u, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    dim3 grid((unsigned)((p.d + kUThreads - 1) / kUThreads), (unsigned)((p.B + kUImgs - 1) / kUImgs));
    k_qvs_u<<<grid, kUThreads, smem, s>>>(p);
    return cudaGetLastError();
}

cudaError_t launch_qvs_logits(const QvsParams &p, int sms, cudaStream_t s) {
    if (p.B == 0) return cudaSuccess;
    // Enough blocks for about four per SM; each covers a strided share of an image's tokens.
    const int per_img = std::max(1, std::min((p.L + 7) / 8, (4 * sms + p.B - 1) / p.B));
    dim3 grid((unsigned)per_img, (unsigned)p.B);
    k_qvs_logits<<<grid, kLogThreads, (size_t)p.d * sizeof(float), s>>>(p);
    return cudaGetLastError();
}

cudaError_t launch_qvs_select(const QvsParams &p, cudaStream_t s) {
    if (p.B == 0) return cudaSuccess;
    k_qvs_select<<<p.B, kSelThreads, 0, s>>>(p);
    return cudaGetLastError();
}

}  // namespace skipk
