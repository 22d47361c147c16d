// BSCA, bipartite sparse cross-attention (App. B.3 Def. B.3, Eq. bsca_edges
// and bsca_attn; §3.3 "BSCA"; Alg. 1 "BSCA: graph" and "BSCA: fuse").  Two
// passes, as the paper's kernel: the first computes the compatibility of
// every (visual token, chunk) pair of a question and the question's edge
// threshold; the second attends each visual token over its surviving edges
// only.
//
//  k_bsca_graph   one block per question: the chunks' h_k rows normalised in
//                 shared memory (rows padded against bank conflicts); a warp
//                 per visual token, a lane per chunk, computes its cosines
//                 (written to the workspace); then tau_e = the m-th largest
//                 cosine of the question by a 4 x 8-bit radix select on the
//                 order-preserving integers of the values (a histogram per
//                 warp, increments aggregated over lanes with equal digits).
//  k_bsca_attend  a warp per visual token: its neighbours are the chunks with
//                 cos >= tau_e; e_ij = <q_i, k_j> / sqrt(d_h) and the softmax
//                 weights first (one per lane), then sum_j w_j W_V k_j 256
//                 output values at a time.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "skip_device.cuh"
#include "skip_internal.h"

namespace skipk {
namespace {

constexpr int kGraphThreads = 512;

__device__ __forceinline__ float bf16_at(const uint16_t *p, int64_t i) {
    return __uint_as_float((uint32_t)p[i] << 16);
}

__global__ void __launch_bounds__(kGraphThreads) k_bsca_graph(const BscaParams p) {
    // shared: hks [R][dp + 1] normalised chunk rows | hvs [warps][dp] | cs [P * R] cosines
    extern __shared__ float sm[];
    __shared__ uint32_t hist[kGraphThreads / 32][256];
    __shared__ uint32_t sel_prefix;
    __shared__ int sel_rank;
    const int q = blockIdx.x;
    const int i0 = p.vis_offsets[q], P = p.vis_offsets[q + 1] - i0;
    const int j0 = p.chunk_offsets[q], R = p.chunk_offsets[q + 1] - j0;
    if (P < 0 || R < 0 || R > kBscaMaxR || (int64_t)P * R > kBscaMaxPairs) {
        if (threadIdx.x == 0) {
            atomicOr(p.err, kErrConfig);
            p.tau[q] = __int_as_float(0x7f800000);  // no edges
        }
        return;
    }
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int ld = p.dp + 1;  // padded row: lanes reading different rows hit different banks
    float *hks = sm;
    float *hvs = sm + kBscaMaxR * ld + warp * p.dp;
    float *cs = sm + kBscaMaxR * ld + (kGraphThreads / 32) * p.dp;
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
        for (int t = lane; t < p.dp; t += 32) hks[j * ld + t] = bf16_at(row, t) * inv;
    }
    __syncthreads();
    // cosines: a warp per visual token, a lane per chunk (two rounds if R > 32);
    // the next token's h_v row is loaded while this one is scored
    float nx[kBscaMaxDp / 32];
    int i = warp;
    if (i < P) {
#pragma unroll
        for (int u = 0; u < kBscaMaxDp / 32; ++u) {
            const int t = lane + 32 * u;
            nx[u] = t < p.dp ? bf16_at(p.hv, (int64_t)(i0 + i) * p.dp + t) : 0.f;
        }
    }
    for (; i < P; i += kGraphThreads / 32) {
        float ss = 0.f;
#pragma unroll
        for (int u = 0; u < kBscaMaxDp / 32; ++u) {
            const int t = lane + 32 * u;
            if (t < p.dp) hvs[t] = nx[u];
            ss = fmaf(nx[u], nx[u], ss);
        }
        const int inext = i + kGraphThreads / 32;
        if (inext < P) {
#pragma unroll
            for (int u = 0; u < kBscaMaxDp / 32; ++u) {
                const int t = lane + 32 * u;
                nx[u] = t < p.dp ? bf16_at(p.hv, (int64_t)(i0 + inext) * p.dp + t) : 0.f;
            }
        }
#pragma unroll
        for (int o = 16; o; o >>= 1) ss += __shfl_xor_sync(0xFFFFFFFFu, ss, o);
        const float inv = ss > 0.f ? 1.f / sqrtf(ss) : 0.f;
        __syncwarp();
        float *crow = p.cos + (int64_t)(i0 + i) * kBscaMaxR;
        for (int j = lane; j < R; j += 32) {
            const float *kr = hks + j * ld;
            float s0 = 0.f, s1 = 0.f;
            int t = 0;
            for (; t + 1 < p.dp; t += 2) {
                s0 = fmaf(hvs[t], kr[t], s0);
                s1 = fmaf(hvs[t + 1], kr[t + 1], s1);
            }
            if (t < p.dp) s0 = fmaf(hvs[t], kr[t], s0);
            const float c = (s0 + s1) * inv;
            crow[j] = c;
            cs[i * R + j] = c;
        }
        __syncwarp();
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
    // 4 x 8-bit radix select; a histogram per warp, increments aggregated over
    // lanes with equal digits
    for (int pass = 0; pass < 4; ++pass) {
        const int shift = 24 - 8 * pass;
        for (int b = lane; b < 256; b += 32) hist[warp][b] = 0;
        __syncthreads();
        const uint32_t prefix = sel_prefix;
        for (int64_t base = 0; base < total; base += kGraphThreads) {
            const int64_t e = base + threadIdx.x;
            bool match = false;
            uint32_t digit = 0;
            if (e < total) {
                const uint32_t o = ord_of_score(cs[e]);
                match = pass == 0 || (o >> (shift + 8)) == prefix;
                digit = (o >> shift) & 0xFFu;
            }
            const uint32_t act = __ballot_sync(0xFFFFFFFFu, match);
            if (match) {
                const uint32_t same = __match_any_sync(act, digit);
                if ((same & ((1u << lane) - 1u)) == 0u) atomicAdd(&hist[warp][digit], (uint32_t)__popc(same));
            }
        }
        __syncthreads();
        if (warp == 0) {  // the digit holding the rank: counts of digits 255 - 32 l ... in lane l
            int r = sel_rank;
            int d = 255, found = -1;
            for (int blk = 0; blk < 8 && found < 0; ++blk) {
                const int dd = 255 - blk * 32 - lane;
                uint32_t c = 0;
                for (int w = 0; w < kGraphThreads / 32; ++w) c += hist[w][dd];
                // inclusive prefix over lanes (descending digits)
                uint32_t pre = c;
#pragma unroll
                for (int o = 1; o < 32; o <<= 1) {
                    const uint32_t v = __shfl_up_sync(0xFFFFFFFFu, pre, o);
                    if (lane >= o) pre += v;
                }
                const uint32_t hit = __ballot_sync(0xFFFFFFFFu, (int)pre >= r);
                if (hit) {
                    const int l = __ffs(hit) - 1;
                    const uint32_t before = __shfl_sync(0xFFFFFFFFu, pre - c, l);
                    d = 255 - blk * 32 - l;
                    r -= (int)before;
                    found = 1;
                } else {
                    r -= (int)__shfl_sync(0xFFFFFFFFu, pre, 31);
                }
            }
            if (lane == 0) {
                sel_rank = r;
                sel_prefix = (prefix << 8) | (uint32_t)d;
            }
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
    // logits of the neighbours: lane l keeps those of the l-th and (l+32)-th
    float e0 = -__int_as_float(0x7f800000), e1 = e0;
    int cnt = 0;
    for (uint64_t m = nb; m; m &= m - 1, ++cnt) {
        const int j = __ffsll((long long)m) - 1;
        const uint16_t *kr = p.kh + (int64_t)(j0 + j) * p.dh;
        float s = 0.f;
#pragma unroll
        for (int u = 0; u < kBscaMaxDh / 32; ++u) {
            const int t = lane + 32 * u;
            if (t < p.dh) s = fmaf(qv[u], bf16_at(kr, t), s);
        }
#pragma unroll
        for (int o = 16; o; o >>= 1) s += __shfl_xor_sync(0xFFFFFFFFu, s, o);
        if (cnt == lane) e0 = s * scale;
        if (cnt == lane + 32) e1 = s * scale;
    }
    // softmax weights
    float mx = fmaxf(e0, e1);
#pragma unroll
    for (int o = 16; o; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xFFFFFFFFu, mx, o));
    const float w0 = lane < cnt ? expf(e0 - mx) : 0.f, w1 = lane + 32 < cnt ? expf(e1 - mx) : 0.f;
    float den = w0 + w1;
#pragma unroll
    for (int o = 16; o; o >>= 1) den += __shfl_xor_sync(0xFFFFFFFFu, den, o);
    const float inv = den > 0.f ? 1.f / den : 0.f;
    // out_i = sum_j w_j W_V k_j, 256 values (8 per lane) at a time
    const int npair = p.dout / 2;
    float2 *orow = reinterpret_cast<float2 *>(p.out + i * p.dout);
    for (int c0 = 0; c0 < npair; c0 += 128) {
        float2 acc[4] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
        int k = 0;
        for (uint64_t m = nb; m; m &= m - 1, ++k) {
            const int j = __ffsll((long long)m) - 1;
            const float w = __shfl_sync(0xFFFFFFFFu, k < 32 ? w0 : w1, k & 31);
            const __nv_bfloat162 *vr = reinterpret_cast<const __nv_bfloat162 *>(p.vh + (int64_t)(j0 + j) * p.dout);
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int pr = c0 + lane + 32 * u;
                if (pr < npair) {
                    const float2 v = __bfloat1622float2(vr[pr]);
                    acc[u].x = fmaf(w, v.x, acc[u].x);
                    acc[u].y = fmaf(w, v.y, acc[u].y);
                }
            }
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int pr = c0 + lane + 32 * u;
            if (pr < npair) orow[pr] = make_float2(acc[u].x * inv, acc[u].y * inv);
        }
    }
}

}  // namespace

cudaError_t launch_bsca(const BscaParams &p, cudaStream_t s) {
    if (p.Q == 0) return cudaSuccess;
    const size_t smem = ((size_t)kBscaMaxR * (p.dp + 1) + (size_t)(kGraphThreads / 32) * p.dp + kBscaMaxPairs) *
                        sizeof(float);
    cudaError_t e = cudaFuncSetAttribute(k_bsca_graph, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    k_bsca_graph<<<p.Q, kGraphThreads, smem, s>>>(p);
    e = cudaGetLastError();
    if (e != cudaSuccess || p.Nv == 0) return e;
    k_bsca_attend<<<(unsigned)((p.Nv + kAttWarps - 1) / kAttWarps), 32 * kAttWarps, 0, s>>>(p);
    return cudaGetLastError();
}

}  // namespace skipk
