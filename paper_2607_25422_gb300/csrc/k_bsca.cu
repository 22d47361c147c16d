// BSCA, bipartite sparse cross-attention (App. B.3 Def. B.3, Eq. bsca_edges
// and bsca_attn; §3.3 "BSCA"; Alg. 1 "BSCA: graph" and "BSCA: fuse").  Two
// passes, as the paper's kernel: the first computes the compatibility of
// every (visual token, chunk) pair of a question and the question's edge
// threshold; the second attends each visual token over its surviving edges
// only.
//
//  k_bsca_graph   one block per question: the chunks' h_k rows normalised in
//                 shared memory; a warp per visual token computes its cosines
//                 (written to the workspace); then tau_e = the m-th largest
//                 cosine of the question by a 4 x 8-bit radix select on the
//                 order-preserving integers of the values.
//  k_bsca_attend  a warp per visual token: its neighbours are the chunks with
//                 cos >= tau_e; e_ij = <q_i, k_j> / sqrt(d_h) with an online
//                 softmax; each lane accumulates a strided share of the d_o
//                 output values of sum_j softmax_j * W_V k_j.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "skip_device.cuh"
#include "skip_internal.h"

namespace skipk {
namespace {

constexpr int kGraphThreads = 256;

__device__ __forceinline__ float bf16_at(const uint16_t *p, int64_t i) {
    return __uint_as_float((uint32_t)p[i] << 16);
}

__global__ void __launch_bounds__(kGraphThreads) k_bsca_graph(const BscaParams p) {
    extern __shared__ float hks[];  // [R][dp] normalised chunk projections
    __shared__ uint32_t hist[256];
    __shared__ uint32_t sel_prefix;
    __shared__ int sel_rank;
    const int q = blockIdx.x;
    const int i0 = p.vis_offsets[q], P = p.vis_offsets[q + 1] - i0;
    const int j0 = p.chunk_offsets[q], R = p.chunk_offsets[q + 1] - j0;
    if (P < 0 || R < 0 || R > kBscaMaxR) {
        if (threadIdx.x == 0) {
            atomicOr(p.err, kErrConfig);
            p.tau[q] = __int_as_float(0x7f800000);  // no edges
        }
        return;
    }
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    // normalised h_k rows, a warp per chunk
    for (int j = warp; j < R; j += kGraphThreads / 32) {
        const uint16_t *row = p.hk + (int64_t)(j0 + j) * p.dp;
        float ss = 0.f;
        for (int t = lane; t < p.dp; t += 32) {
            const float x = bf16_at(row, t);
            ss = fmaf(x, x, ss);
        }
#pragma unroll
        for (int o = 16; o; o >>= 1) ss += __shfl_xor_sync(0xFFFFFFFFu, ss, o);
        const float inv = ss > 0.f ? 1.f / sqrtf(ss) : 0.f;
        for (int t = lane; t < p.dp; t += 32) hks[j * p.dp + t] = bf16_at(row, t) * inv;
    }
    __syncthreads();
    // cosines, a warp per visual token
    for (int i = warp; i < P; i += kGraphThreads / 32) {
        const uint16_t *row = p.hv + (int64_t)(i0 + i) * p.dp;
        float x[kBscaMaxDp / 32];
        float ss = 0.f;
#pragma unroll
        for (int u = 0; u < kBscaMaxDp / 32; ++u) {
            const int t = lane + 32 * u;
            x[u] = t < p.dp ? bf16_at(row, t) : 0.f;
            ss = fmaf(x[u], x[u], ss);
        }
#pragma unroll
        for (int o = 16; o; o >>= 1) ss += __shfl_xor_sync(0xFFFFFFFFu, ss, o);
        const float inv = ss > 0.f ? 1.f / sqrtf(ss) : 0.f;
        float *crow = p.cos + (int64_t)(i0 + i) * kBscaMaxR;
        for (int j = 0; j < R; ++j) {
            float s = 0.f;
#pragma unroll
            for (int u = 0; u < kBscaMaxDp / 32; ++u) {
                const int t = lane + 32 * u;
                if (t < p.dp) s = fmaf(x[u], hks[j * p.dp + t], s);
            }
#pragma unroll
            for (int o = 16; o; o >>= 1) s += __shfl_xor_sync(0xFFFFFFFFu, s, o);
            if (lane == 0) crow[j] = s * inv;
        }
    }
    __syncthreads();
    // tau_e: the m-th largest of the P * R cosines
    const int64_t total = (int64_t)P * R;
    const double md = ceil((double)p.dbar * (double)P - 1e-3);
    const int64_t m = md < 0.0 ? 0 : (int64_t)md;
    if (m < 1 || total == 0) {
        if (threadIdx.x == 0) p.tau[q] = __int_as_float(0x7f800000);
        return;
    }
    if (m >= total) {
        if (threadIdx.x == 0) p.tau[q] = -__int_as_float(0x7f800000);
        return;
    }
    if (threadIdx.x == 0) {
        sel_prefix = 0;
        sel_rank = (int)m;
    }
    for (int pass = 0; pass < 4; ++pass) {
        const int shift = 24 - 8 * pass;
        for (int b = threadIdx.x; b < 256; b += kGraphThreads) hist[b] = 0;
        __syncthreads();
        const uint32_t prefix = sel_prefix;
        for (int64_t e = threadIdx.x; e < total; e += kGraphThreads) {
            const int i = (int)(e / R), j = (int)(e - (int64_t)i * R);
            const uint32_t o = ord_of_score(p.cos[(int64_t)(i0 + i) * kBscaMaxR + j]);
            const bool match = pass == 0 || (o >> (shift + 8)) == prefix;
            if (match) atomicAdd(&hist[(o >> shift) & 0xFFu], 1u);
        }
        __syncthreads();
        if (threadIdx.x == 0) {
            int r = sel_rank;
            int d = 255;
            for (; d > 0; --d) {
                if ((int)hist[d] >= r) break;
                r -= (int)hist[d];
            }
            sel_rank = r;
            sel_prefix = (prefix << 8) | (uint32_t)d;
        }
        __syncthreads();
    }
    if (threadIdx.x == 0) p.tau[q] = score_of_ord(sel_prefix);
}

constexpr int kAttWarps = 8;

__global__ void __launch_bounds__(32 * kAttWarps) k_bsca_attend(const BscaParams p) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t i = (int64_t)blockIdx.x * kAttWarps + warp;
    if (i >= p.Nv) return;
    // the question holding token i: vis_offsets[q] <= i < vis_offsets[q + 1]
    int lo = 0, hi = p.Q - 1;
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (p.vis_offsets[mid] <= i) lo = mid;
        else hi = mid - 1;
    }
    const int q = lo;
    const int j0 = p.chunk_offsets[q];
    int R = p.chunk_offsets[q + 1] - j0;
    if (R < 0 || R > kBscaMaxR) R = 0;  // flagged by k_bsca_graph
    const float tau = p.tau[q];
    const float *crow = p.cos + i * kBscaMaxR;
    // neighbour masks: lane l looks at chunks l and l + 32
    const bool n0 = lane < R && crow[lane] >= tau;
    const bool n1 = lane + 32 < R && crow[lane + 32] >= tau;
    uint64_t nb = (uint64_t)__ballot_sync(0xFFFFFFFFu, n0) | ((uint64_t)__ballot_sync(0xFFFFFFFFu, n1) << 32);
    if (p.degree && lane == 0) p.degree[i] = __popcll(nb);
    if (p.edges && lane == 0) p.edges[i] = nb;
    // q_i in registers (lane t holds elements t, t + 32, ...)
    float qv[kBscaMaxDh / 32];
#pragma unroll
    for (int u = 0; u < kBscaMaxDh / 32; ++u) {
        const int t = lane + 32 * u;
        qv[u] = t < p.dh ? bf16_at(p.qh, i * p.dh + t) : 0.f;
    }
    const float scale = rsqrtf((float)p.dh);
    float mx = -__int_as_float(0x7f800000), den = 0.f;
    float acc[kBscaMaxDo / 64][2];
    const int npair = p.dout / 2;  // lane owns pairs lane, lane + 32, ...
#pragma unroll
    for (int u = 0; u < kBscaMaxDo / 64; ++u) acc[u][0] = acc[u][1] = 0.f;
    while (nb) {
        const int j = __ffsll((long long)nb) - 1;
        nb &= nb - 1;
        const uint16_t *kr = p.kh + (int64_t)(j0 + j) * p.dh;
        float s = 0.f;
#pragma unroll
        for (int u = 0; u < kBscaMaxDh / 32; ++u) {
            const int t = lane + 32 * u;
            if (t < p.dh) s = fmaf(qv[u], bf16_at(kr, t), s);
        }
#pragma unroll
        for (int o = 16; o; o >>= 1) s += __shfl_xor_sync(0xFFFFFFFFu, s, o);
        const float e = s * scale;
        // online softmax: rescale what is accumulated when the maximum grows
        const float nm = fmaxf(mx, e);
        const float c = expf(mx - nm), w = expf(e - nm);
        den = den * c + w;
        mx = nm;
        const __nv_bfloat162 *vr = reinterpret_cast<const __nv_bfloat162 *>(p.vh + (int64_t)(j0 + j) * p.dout);
#pragma unroll
        for (int u = 0; u < kBscaMaxDo / 64; ++u) {
            const int pr = lane + 32 * u;
            if (pr < npair) {
                const float2 v = __bfloat1622float2(vr[pr]);
                acc[u][0] = fmaf(w, v.x, acc[u][0] * c);
                acc[u][1] = fmaf(w, v.y, acc[u][1] * c);
            }
        }
    }
    const float inv = den > 0.f ? 1.f / den : 0.f;
    float2 *orow = reinterpret_cast<float2 *>(p.out + i * p.dout);
#pragma unroll
    for (int u = 0; u < kBscaMaxDo / 64; ++u) {
        const int pr = lane + 32 * u;
        if (pr < npair) orow[pr] = make_float2(acc[u][0] * inv, acc[u][1] * inv);
    }
}

}  // namespace

cudaError_t launch_bsca(const BscaParams &p, cudaStream_t s) {
    if (p.Q == 0) return cudaSuccess;
    const size_t smem = (size_t)kBscaMaxR * p.dp * sizeof(float);
    cudaError_t e = cudaFuncSetAttribute(k_bsca_graph, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    k_bsca_graph<<<p.Q, kGraphThreads, smem, s>>>(p);
    e = cudaGetLastError();
    if (e != cudaSuccess || p.Nv == 0) return e;
    k_bsca_attend<<<(unsigned)((p.Nv + kAttWarps - 1) / kAttWarps), 32 * kAttWarps, 0, s>>>(p);
    return cudaGetLastError();
}

}  // namespace skipk
