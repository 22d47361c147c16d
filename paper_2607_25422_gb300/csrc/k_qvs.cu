// QVS, question-guided visual token pruning (App. B.1 Def. B.1, Eq.
// qvs_score; Alg. 1 "QVS: prune").  With f_v linear,
//   logit_i = <f_q, W_v v_i + b_v> / sqrt(d_k) + <w_b, v_i> = <u, v_i> + c,
//   u = W_v^T f_q / sqrt(d_k) + w_b,  c = <f_q, b_v> / sqrt(d_k),
// so the per-token work is one inner product (the scan reads every token
// once: HBM-bound), and the ranking by s = sigmoid(logit) is the ranking by
// the logit.
//
//  k_gemm        W_v^T f_q / sqrt(d_k) for all images at once: the library's
//                tensor-core GEMM (k_gemm.cu) on F_q [B x d_k] and the handle's
//                copy of W_v^T [d x d_k] (k_transpose_bf16, once per handle).
//  k_qvs_logits  u = that + w_b in shared memory and c by one warp; one warp
//                per four tokens at a time, 16-byte loads.
//  k_qvs_select  per image: (logit, ~index) keys sorted descending in shared
//                memory, the first n kept with their sigmoid scores.
//  k_qvs_gather  (optional) the kept token rows copied out, a warp per row.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <algorithm>

#include "skip_device.cuh"
#include "skip_internal.h"

namespace skipk {
namespace {

constexpr int kLogThreads = 256;

__global__ void __launch_bounds__(kLogThreads) k_qvs_logits(const QvsParams p) {
    extern __shared__ float us[];  // [d]
    __shared__ float cbs;
    const int b = blockIdx.y;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    // u = W_v^T f_q / sqrt(d_k) (the library GEMM) + w_b; c = <f_q, b_v> / sqrt(d_k)
    for (int t = threadIdx.x; t < p.d; t += kLogThreads) us[t] = p.u[(int64_t)b * p.d + t] + p.wb[t];
    if (warp == 0) {
        const __nv_bfloat16 *fq = reinterpret_cast<const __nv_bfloat16 *>(p.fq) + (int64_t)b * p.dk;
        float c = 0.f;
        for (int k = lane; k < p.dk; k += 32) c = fmaf(__bfloat162float(fq[k]), p.bv[k], c);
#pragma unroll
        for (int o = 16; o; o >>= 1) c += __shfl_xor_sync(0xFFFFFFFFu, c, o);
        if (lane == 0) cbs = c * rsqrtf((float)p.dk);
    }
    __syncthreads();
    const int nw = p.d / 8;  // 16-byte words per token
    const float cb = cbs;
    // Four tokens per warp at a time: their loads are issued together.
    constexpr int kT = 4;
    const int wstep = gridDim.x * (kLogThreads / 32);
    for (int i0 = blockIdx.x * (kLogThreads / 32) + warp; i0 < p.L; i0 += kT * wstep) {
        float s[kT];
#pragma unroll
        for (int t = 0; t < kT; ++t) s[t] = 0.f;
        for (int w = lane; w < nw; w += 32) {
            uint4 x[kT];
#pragma unroll
            for (int t = 0; t < kT; ++t) {
                const int i = i0 + t * wstep;
                x[t] = i < p.L ? __ldg(reinterpret_cast<const uint4 *>(p.tokens) + ((int64_t)b * p.L + i) * nw + w)
                               : make_uint4(0, 0, 0, 0);
            }
            float uu[8];
#pragma unroll
            for (int e = 0; e < 8; ++e) uu[e] = us[w * 8 + e];
#pragma unroll
            for (int t = 0; t < kT; ++t) {
                const uint32_t xv[4] = {x[t].x, x[t].y, x[t].z, x[t].w};
#pragma unroll
                for (int h = 0; h < 4; ++h) {
                    const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(&xv[h]));
                    s[t] = fmaf(f.x, uu[2 * h], s[t]);
                    s[t] = fmaf(f.y, uu[2 * h + 1], s[t]);
                }
            }
        }
#pragma unroll
        for (int t = 0; t < kT; ++t) {
#pragma unroll
            for (int o = 16; o; o >>= 1) s[t] += __shfl_xor_sync(0xFFFFFFFFu, s[t], o);
            const int i = i0 + t * wstep;
            if (lane == 0 && i < p.L) p.logits[(int64_t)b * p.L + i] = s[t] + cb;
        }
    }
}

constexpr int kSelThreads = 512;

// One bitonic step on a register pair held by lanes (lane, lane ^ j): the
// lower lane keeps the larger key when `desc`, else the smaller.
__device__ __forceinline__ uint64_t bitonic_lane_step(uint64_t v, int pos, int j, bool desc) {
    const uint64_t o = __shfl_xor_sync(0xFFFFFFFFu, v, j);
    const bool lower = (pos & j) == 0;
    const bool keep_max = lower == desc;
    return keep_max ? (v > o ? v : o) : (v < o ? v : o);
}

// Sorts keys[0, n) descending (n a power of two, 64 <= n <= kQvsMaxL, block of
// kSelThreads threads).  Strides below 32 run inside warps on registers,
// one key per lane; larger strides through shared memory.
__device__ void bitonic_desc(uint64_t *keys, int n) {
    const int lane = threadIdx.x & 31;
    for (int size = 2; size <= n; size <<= 1) {
        int stride = size >> 1;
        for (; stride >= 32; stride >>= 1) {
            for (int t = threadIdx.x; t < n / 2; t += kSelThreads) {
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
        // strides 16 .. 1: each warp sorts its 32-key runs in registers
        for (int base = (threadIdx.x & ~31); base < n; base += kSelThreads) {
            const int pos = base + lane;
            uint64_t v = keys[pos];
            const bool desc = (pos & size) == 0;
            for (int j = stride; j > 0; j >>= 1) v = bitonic_lane_step(v, pos, j, desc);
            keys[pos] = v;
        }
        __syncthreads();
    }
}

__global__ void __launch_bounds__(kSelThreads) k_qvs_select(const QvsParams p) {
    __shared__ uint64_t keys[kQvsMaxL];
    const int b = blockIdx.x;
    int Lp = 64;
    while (Lp < p.L) Lp <<= 1;
    for (int i = threadIdx.x; i < Lp; i += kSelThreads) {
        uint64_t key = 0;
        if (i < p.L) key = ((uint64_t)ord_of_score(p.logits[(int64_t)b * p.L + i]) << 32) | (uint32_t)(0xFFFFFFFFu - i);
        keys[i] = key;
    }
    __syncthreads();
    bitonic_desc(keys, Lp);
    for (int r = threadIdx.x; r < p.n; r += kSelThreads) {
        const uint64_t key = keys[r];
        p.out_idx[(int64_t)b * p.n + r] = (int32_t)(0xFFFFFFFFu - (uint32_t)key);
        p.out_score[(int64_t)b * p.n + r] = 1.f / (1.f + expf(-score_of_ord((uint32_t)(key >> 32))));
    }
}

// Kept token rows: one block per (rank, image), 16-byte copies.
constexpr int kGatherWarps = 8;

__global__ void __launch_bounds__(32 * kGatherWarps) k_qvs_gather(const QvsParams p) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int r = blockIdx.x * kGatherWarps + warp, b = blockIdx.y;
    if (r >= p.n) return;
    const int i = p.out_idx[(int64_t)b * p.n + r];
    const int nw = p.d / 8;
    const uint4 *src = reinterpret_cast<const uint4 *>(p.tokens) + ((int64_t)b * p.L + i) * nw;
    uint4 *dst = reinterpret_cast<uint4 *>(p.out_tokens) + ((int64_t)b * p.n + r) * nw;
    // four 16-byte words per lane in flight
    for (int w0 = 0; w0 < nw; w0 += 128) {
        uint4 x[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int w = w0 + lane + 32 * u;
            if (w < nw) x[u] = __ldg(src + w);
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int w = w0 + lane + 32 * u;
            if (w < nw) dst[w] = x[u];
        }
    }
}

// W^T of a bf16 matrix W [rows x cols] (row-major) into wt [cols x ldt]
// (ldt >= rows) through 32 x 32 tiles in shared memory: both the reads and
// the writes are coalesced.
__global__ void __launch_bounds__(256) k_transpose_bf16(const uint16_t *__restrict__ w, int rows, int cols,
                                                        uint16_t *__restrict__ wt, int ldt) {
    __shared__ uint16_t tile[32][33];
    const int c0 = blockIdx.x * 32, r0 = blockIdx.y * 32;
    const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;  // 8 rows of threads
    for (int y = ty; y < 32; y += 8) {
        const int r = r0 + y, c = c0 + tx;
        if (r < rows && c < cols) tile[y][tx] = w[(int64_t)r * cols + c];
    }
    __syncthreads();
    for (int y = ty; y < 32; y += 8) {
        const int c = c0 + y, r = r0 + tx;
        if (r < rows && c < cols) wt[(int64_t)c * ldt + r] = tile[tx][y];
    }
}

}  // namespace

cudaError_t launch_transpose_bf16(const uint16_t *w, int rows, int cols, uint16_t *wt, int ldt, cudaStream_t s) {
    if (rows <= 0 || cols <= 0) return cudaSuccess;
    if (ldt < rows) return cudaErrorInvalidValue;
    k_transpose_bf16<<<dim3((unsigned)((cols + 31) / 32), (unsigned)((rows + 31) / 32)), 256, 0, s>>>(w, rows, cols,
                                                                                                     wt, ldt);
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
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess || !p.out_tokens || p.n == 0) return e;
    k_qvs_gather<<<dim3((unsigned)((p.n + kGatherWarps - 1) / kGatherWarps), (unsigned)p.B), 32 * kGatherWarps, 0, s>>>(p);
    return cudaGetLastError();
}

}  // namespace skipk
