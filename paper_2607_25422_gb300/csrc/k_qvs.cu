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
//                copy of W_v^T [d x d_k] (k_transpose_bf16, once per handle),
//                K split over up to four CTAs per tile (partial slabs).
//  k_qvs_logits  u = the slabs' sum + w_b in shared memory, c by all warps;
//                one warp per eight tokens, each token's row requested whole
//                (2 KB at a time, 16-byte loads), two tokens per round.
//  k_qvs_rank    rank of every token = the number of the image's keys
//                (logit, ~index) above its own, counted against all the
//                image's keys in shared memory (many blocks per image, a warp
//                per eight tokens); a token with rank < n is written at its
//                rank with its sigmoid score, and (optionally) its row copied
//                out: the block's kept rows spread over all its warps, two
//                rows in flight a warp.  The same order as a descending sort.
// The logits and rank kernels are programmatic dependents of the kernel
// before them: they launch while it drains and wait for its results.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <algorithm>

#include "skip_device.cuh"
#include "skip_internal.h"

namespace skipk {
namespace {

constexpr int kLogThreads = 256;
constexpr int kLogTok = 8;  // tokens per warp in flight

// (At most 64 registers a thread, four blocks an SM: with 80 registers only
// three fit, and 576 blocks took two waves.)
__global__ void __launch_bounds__(kLogThreads, 4) k_qvs_logits(const QvsParams p) {
    extern __shared__ float us[];  // [d]
    __shared__ float cpart[kLogThreads / 32];
    const int b = blockIdx.y;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    // The tokens are inputs of the call, not results of the GEMM before this
    // kernel: while that GEMM still runs (this kernel is its programmatic
    // dependent), pull this warp's token rows into L2, one 128-byte line per
    // lane and step.
    {
        const int lines = p.d / 64;  // 128-byte lines per token row
        const int ws = gridDim.x * (kLogThreads / 32);
        for (int i = blockIdx.x * (kLogThreads / 32) + warp; i < p.L; i += ws) {
            const char *row = reinterpret_cast<const char *>(p.tokens) + ((int64_t)b * p.L + i) * p.d * 2;
            for (int l = lane; l < lines; l += 32) asm volatile("prefetch.global.L2 [%0];" ::"l"(row + l * 128) : "memory");
        }
    }
    grid_dep_wait();
    // u = W_v^T f_q / sqrt(d_k) (the GEMM's partial slabs) + w_b; c = <f_q, b_v> / sqrt(d_k)
    const int64_t slab = (int64_t)p.B * p.d;
    for (int t = threadIdx.x; t < p.d; t += kLogThreads) {
        float v = p.wb[t];
        for (int z = 0; z < p.u_splits; ++z) v += p.u[z * slab + (int64_t)b * p.d + t];
        us[t] = v;
    }
    {
        // c = <f_q, b_v> / sqrt(d_k): every warp a share, summed in shared memory
        const __nv_bfloat16 *fq = reinterpret_cast<const __nv_bfloat16 *>(p.fq) + (int64_t)b * p.dk;
        float c = 0.f;
        for (int k = threadIdx.x; k < p.dk; k += kLogThreads) c = fmaf(__bfloat162float(fq[k]), p.bv[k], c);
#pragma unroll
        for (int o = 16; o; o >>= 1) c += __shfl_xor_sync(0xFFFFFFFFu, c, o);
        if (lane == 0) cpart[warp] = c;
    }
    __syncthreads();
    const int nw = p.d / 8;  // 16-byte words per token
    float cb = 0.f;
#pragma unroll
    for (int w = 0; w < kLogThreads / 32; ++w) cb += cpart[w];
    cb *= rsqrtf((float)p.dk);
    // kLogTok tokens per warp; each token's row is requested whole (2 KB at a
    // time: four 16-byte words a lane), two tokens per round.
    constexpr int kT = kLogTok;
    const int wstep = gridDim.x * (kLogThreads / 32);
    const float4 *us4 = reinterpret_cast<const float4 *>(us);
    const uint4 *tok = reinterpret_cast<const uint4 *>(p.tokens);
    for (int i0 = blockIdx.x * (kLogThreads / 32) + warp; i0 < p.L; i0 += kT * wstep) {
        float s[kT];
#pragma unroll
        for (int t = 0; t < kT; ++t) s[t] = 0.f;
        for (int c0 = 0; c0 < nw; c0 += 128) {
#pragma unroll
            for (int t0 = 0; t0 < kT; t0 += 2) {
                uint4 x[2][4];
#pragma unroll
                for (int tt = 0; tt < 2; ++tt) {
                    const int i = i0 + (t0 + tt) * wstep;
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        const int w = c0 + lane + 32 * j;
                        x[tt][j] = (i < p.L && w < nw) ? __ldg(tok + ((int64_t)b * p.L + i) * nw + w)
                                                       : make_uint4(0, 0, 0, 0);
                    }
                }
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    const int w = c0 + lane + 32 * j;
                    if (w >= nw) break;
                    const float4 ua = us4[2 * w], ub = us4[2 * w + 1];
                    const float uu[8] = {ua.x, ua.y, ua.z, ua.w, ub.x, ub.y, ub.z, ub.w};
#pragma unroll
                    for (int tt = 0; tt < 2; ++tt) {
                        const uint32_t xv[4] = {x[tt][j].x, x[tt][j].y, x[tt][j].z, x[tt][j].w};
#pragma unroll
                        for (int h = 0; h < 4; ++h) {
                            const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(&xv[h]));
                            s[t0 + tt] = fmaf(f.x, uu[2 * h], s[t0 + tt]);
                            s[t0 + tt] = fmaf(f.y, uu[2 * h + 1], s[t0 + tt]);
                        }
                    }
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

constexpr int kRankWarps = 8;
constexpr int kRankTok = 8;  // tokens per warp (576 blocks for 64 images: one wave at five an SM)

__global__ void __launch_bounds__(32 * kRankWarps) k_qvs_rank(const QvsParams p) {
    extern __shared__ uint64_t keys[];  // [L]: (ord(logit), ~index) of every token of the image
    __shared__ int2 kept[kRankWarps * kRankTok];  // (token, rank) of this block's kept tokens
    __shared__ int nkept;
    const int b = blockIdx.y;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) nkept = 0;
    grid_dep_wait();
    const float *lg = p.logits + (int64_t)b * p.L;
    for (int i = threadIdx.x; i < p.L; i += 32 * kRankWarps)
        keys[i] = ((uint64_t)ord_of_score(lg[i]) << 32) | (uint32_t)(0xFFFFFFFFu - i);
    __syncthreads();
    const int i0 = (blockIdx.x * kRankWarps + warp) * kRankTok;
    if (i0 < p.L) {
        uint64_t mine[kRankTok];
        int cnt[kRankTok];
#pragma unroll
        for (int t = 0; t < kRankTok; ++t) {
            mine[t] = i0 + t < p.L ? keys[i0 + t] : ~0ull;  // past L: rank 0 of nothing, never written
            cnt[t] = 0;
        }
        // Keys are distinct (the index is in the low word), so a token's rank
        // is its position in the descending order.
        for (int j = lane; j < p.L; j += 32) {
            const uint64_t kj = keys[j];
#pragma unroll
            for (int t = 0; t < kRankTok; ++t) cnt[t] += kj > mine[t] ? 1 : 0;
        }
#pragma unroll
        for (int t = 0; t < kRankTok; ++t) cnt[t] = __reduce_add_sync(0xFFFFFFFFu, cnt[t]);
#pragma unroll
        for (int t = 0; t < kRankTok; ++t) {
            const int i = i0 + t, r = cnt[t];
            if (i >= p.L || r >= p.n) continue;  // warp-uniform
            if (lane == 0) {
                p.out_idx[(int64_t)b * p.n + r] = i;
                p.out_score[(int64_t)b * p.n + r] = 1.f / (1.f + expf(-score_of_ord((uint32_t)(mine[t] >> 32))));
                if (p.out_tokens) kept[atomicAdd(&nkept, 1)] = make_int2(i, r);
            }
        }
    }
    if (!p.out_tokens) return;
    __syncthreads();
    // The kept rows, spread over all the block's warps, two rows in flight a
    // warp (a row is four 16-byte words a lane at a time).
    const int nw = p.d / 8;  // 16-byte words per token
    const uint4 *src0 = reinterpret_cast<const uint4 *>(p.tokens) + (int64_t)b * p.L * nw;
    uint4 *dst0 = reinterpret_cast<uint4 *>(p.out_tokens) + (int64_t)b * p.n * nw;
    const int m = nkept;
    for (int e = 2 * warp; e < m; e += 2 * kRankWarps) {
        const int2 a = kept[e];
        const int2 c = e + 1 < m ? kept[e + 1] : make_int2(-1, -1);
        for (int w0 = 0; w0 < nw; w0 += 128) {
            uint4 x[2][4];
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int w = w0 + lane + 32 * u;
                if (w < nw) {
                    x[0][u] = __ldg(src0 + (int64_t)a.x * nw + w);
                    if (c.x >= 0) x[1][u] = __ldg(src0 + (int64_t)c.x * nw + w);
                }
            }
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int w = w0 + lane + 32 * u;
                if (w < nw) {
                    dst0[(int64_t)a.y * nw + w] = x[0][u];
                    if (c.x >= 0) dst0[(int64_t)c.y * nw + w] = x[1][u];
                }
            }
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

cudaError_t launch_qvs_logits(const QvsParams &p, int sms, cudaStream_t s) {
    if (p.B == 0) return cudaSuccess;
    if (p.u_splits < 1) return cudaErrorInvalidValue;
    // Enough blocks that every warp loads its tokens in one round (kLogTok
    // per warp), but no more than about four per SM: each block first builds
    // u (the GEMM's slabs summed) and c, so more blocks per image repeat that
    // work (at 18 blocks per image, 4 tokens per warp, the step was 8% slower).
    const int one_round = (p.L + kLogTok * (kLogThreads / 32) - 1) / (kLogTok * (kLogThreads / 32));
    const int per_img = std::max(1, std::min(one_round, (4 * sms + p.B - 1) / p.B));
    dim3 grid((unsigned)per_img, (unsigned)p.B);
    return launch_dependent(k_qvs_logits, grid, kLogThreads, (size_t)p.d * sizeof(float), s, p);
}

cudaError_t launch_qvs_select(const QvsParams &p, cudaStream_t s) {
    if (p.B == 0 || p.L == 0) return cudaSuccess;
    const size_t smem = (size_t)p.L * sizeof(uint64_t);  // <= 32 KB: no opt-in needed
    const int per_img = (p.L + kRankWarps * kRankTok - 1) / (kRankWarps * kRankTok);
    return launch_dependent(k_qvs_rank, dim3((unsigned)per_img, (unsigned)p.B), 32 * kRankWarps, smem, s, p);
}

}  // namespace skipk
