// BSCA, bipartite sparse cross-attention (App. B.3 Def. B.3, Eq. bsca_edges
// and bsca_attn; §3.3 "BSCA"; Alg. 1 "BSCA: graph" and "BSCA: fuse").  Two
// stages, as the paper's kernel: the first computes the compatibility of
// every (visual token, chunk) pair of a question and the question's edge
// threshold; the second attends each visual token over its surviving edges
// only.
//
//  k_bsca_cos     blocks (question, slice of its tokens): the question's h_k
//                 rows normalised in shared memory (rows padded against bank
//                 conflicts); a warp per four visual tokens, a lane per
//                 chunk, computes their cosines into the workspace and counts
//                 each in the question's histogram.
//  k_bsca_select  one block per question: tau_e = the m-th largest cosine of
//                 the question: the bin that holds it from a 4,096-bin
//                 histogram k_bsca_cos filled as it wrote the cosines, then
//                 the rank inside that bin by counting over its few values
//                 (a crowded bin falls back to a 4 x 8-bit radix select on
//                 order-preserving integers).
//  k_bsca_attend  blocks (question, slice of its tokens), a warp per visual
//                 token: its neighbours are the chunks with cos >= tau_e;
//                 e_ij = <q_i, k_j> / sqrt(d_h) for four neighbours at a time
//                 (their rows read together, the four sums reduced across the
//                 warp together), the normalised softmax weights (one per
//                 lane), then sum_j w_j W_V k_j with four neighbours' rows in
//                 flight.
// Slices: the host sizes them from the mean tokens per question; a question
// with more tokens is covered by the same blocks looping.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <algorithm>

#include "skip_device.cuh"
#include "skip_internal.h"

namespace skipk {
namespace {

constexpr int kCosThreads = 256;
constexpr int kSelThreads = 512;
constexpr int kAttWarps = 4;

__device__ __forceinline__ float bf16_at(const uint16_t *p, int64_t i) {
    return __uint_as_float((uint32_t)p[i] << 16);
}

// 8 bf16 (16 bytes) as floats.
__device__ __forceinline__ void bf16x8(const uint4 &u, float (&f)[8]) {
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int h = 0; h < 4; ++h) {
        f[2 * h] = __uint_as_float(w[h] << 16);
        f[2 * h + 1] = __uint_as_float(w[h] & 0xFFFF0000u);
    }
}

__device__ __forceinline__ bool question_ok(int P, int R) {
    return P >= 0 && R >= 0 && R <= kBscaMaxR && (int64_t)P * R <= kBscaMaxPairs;
}

// Tokens [ib, ie) of a question's P for slice s of S.
__device__ __forceinline__ void slice_of(int P, int s, int S, int &ib, int &ie) {
    const int per = (P + S - 1) / S;
    ib = min(P, s * per);
    ie = min(P, ib + per);
}

// Histogram bin of a cosine: kBscaBins equal bins over [-1, 1], a
// non-decreasing function of the value (the same float operations wherever
// it is evaluated).
__device__ __forceinline__ int cos_bin(float c) {
    const int b = __float2int_rd((c + 1.f) * (float)(kBscaBins / 2));
    return min(max(b, 0), kBscaBins - 1);
}

__global__ void __launch_bounds__(kCosThreads) k_bsca_cos(const BscaParams p, int S) {
    // shared: hks [R][dp + 1] normalised chunk rows | hv4 [warps][dp] x 4 tokens
    extern __shared__ float sm[];
    const int q = blockIdx.x / S, sl = blockIdx.x - q * S;
    const int i0 = p.vis_offsets[q], P = p.vis_offsets[q + 1] - i0;
    const int j0 = p.chunk_offsets[q], R = p.chunk_offsets[q + 1] - j0;
    if (!question_ok(P, R)) {
        if (sl == 0 && threadIdx.x == 0) atomicOr(p.err, kErrConfig);
        return;
    }
    int ib, ie;
    slice_of(P, sl, S, ib, ie);
    if (ib >= ie || R == 0) return;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    constexpr int kWarps = kCosThreads / 32;
    const int ld = p.dp + 1;  // padded row: lanes reading different rows hit different banks
    float *hks = sm;
    // normalised h_k rows, a warp per chunk
    for (int j = warp; j < R; j += kWarps) {
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
    // four visual tokens per warp at a time, a lane per chunk (two rounds if
    // R > 32): the tokens' h_v rows are kept interleaved (hv4[t] holds the
    // four values of dimension t), so one broadcast float4 read and one read
    // of the chunk row serve four products
    float4 *hv4 = reinterpret_cast<float4 *>(sm + kBscaMaxR * ld) + warp * p.dp;
    for (int ia = ib + 4 * warp; ia < ie; ia += 4 * kWarps) {
        float inv[4];
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const int i = ia + k;
            float x[kBscaMaxDp / 32];
            float ss = 0.f;
#pragma unroll
            for (int u = 0; u < kBscaMaxDp / 32; ++u) {
                const int t = lane + 32 * u;
                x[u] = (i < ie && t < p.dp) ? bf16_at(p.hv, (int64_t)(i0 + i) * p.dp + t) : 0.f;
                ss = fmaf(x[u], x[u], ss);
            }
#pragma unroll
            for (int o = 16; o; o >>= 1) ss += __shfl_xor_sync(0xFFFFFFFFu, ss, o);
            inv[k] = ss > 0.f ? 1.f / sqrtf(ss) : 0.f;
#pragma unroll
            for (int u = 0; u < kBscaMaxDp / 32; ++u) {
                const int t = lane + 32 * u;
                if (t < p.dp) reinterpret_cast<float *>(hv4 + t)[k] = x[u];
            }
        }
        __syncwarp();
        for (int j = lane; j < R; j += 32) {
            const float *kr = hks + j * ld;
            float s0 = 0.f, s1 = 0.f, s2 = 0.f, s3 = 0.f;
            for (int t = 0; t < p.dp; ++t) {
                const float kv = kr[t];
                const float4 h = hv4[t];
                s0 = fmaf(h.x, kv, s0);
                s1 = fmaf(h.y, kv, s1);
                s2 = fmaf(h.z, kv, s2);
                s3 = fmaf(h.w, kv, s3);
            }
            const float sv[4] = {s0, s1, s2, s3};
#pragma unroll
            for (int k = 0; k < 4; ++k)
                if (ia + k < ie) {
                    const float c = sv[k] * inv[k];
                    p.cos[(int64_t)(i0 + ia + k) * kBscaMaxR + j] = c;
                    atomicAdd(p.hist + (int64_t)q * kBscaBins + cos_bin(c), 1u);
                }
        }
        __syncwarp();
    }
}

constexpr int kCandCap = 2048;  // values of the threshold's bin resolved exactly

// The m-th largest of cs[0, total) by a 4 x 8-bit radix select on the
// order-preserving integers (a histogram per warp, increments aggregated
// over lanes with equal digits); all threads of the block call it.
__device__ float radix_select(const float *cs, int64_t total, int64_t m, uint32_t (*hist)[256]) {
    __shared__ uint32_t sel_prefix;
    __shared__ int sel_rank;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) {
        sel_prefix = 0;
        sel_rank = (int)m;
    }
    for (int pass = 0; pass < 4; ++pass) {
        const int shift = 24 - 8 * pass;
        for (int b = lane; b < 256; b += 32) hist[warp][b] = 0;
        __syncthreads();
        const uint32_t prefix = sel_prefix;
        for (int64_t base = 0; base < total; base += kSelThreads) {
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
                for (int w = 0; w < kSelThreads / 32; ++w) c += hist[w][dd];
                uint32_t pre = c;  // inclusive prefix over lanes (descending digits)
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
    return score_of_ord(sel_prefix);
}

// tau_e of one question from the histogram k_bsca_cos built: the bin B that
// holds the m-th largest cosine (a block-wide scan of the bin counts from the
// top), then the values of bin B gathered and the one of the right rank
// among them found by counting; a bin of more than kCandCap values falls
// back to the radix select over all the question's cosines.  The histogram
// row is cleared for the next call.
__global__ void __launch_bounds__(kSelThreads) k_bsca_select(const BscaParams p) {
    extern __shared__ float cs[];  // fallback: the question's P * R cosines
    __shared__ uint32_t hs[kBscaBins];
    __shared__ uint32_t hist[kSelThreads / 32][256];
    __shared__ float cand[kCandCap];
    __shared__ uint32_t wsum[kSelThreads / 32];
    __shared__ int s_bin, s_rank, s_cnt, s_found;
    __shared__ float s_tau;
    grid_dep_wait();  // the cosines and histograms of k_bsca_cos
    const int q = blockIdx.x;
    const int i0 = p.vis_offsets[q], P = p.vis_offsets[q + 1] - i0;
    const int R = p.chunk_offsets[q + 1] - p.chunk_offsets[q];
    const float kInf = __int_as_float(0x7f800000);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    uint32_t *hrow = p.hist + (int64_t)q * kBscaBins;
    for (int b = threadIdx.x; b < kBscaBins; b += kSelThreads) {
        hs[b] = hrow[b];
        hrow[b] = 0u;
    }
    if (!question_ok(P, R)) {
        if (threadIdx.x == 0) p.tau[q] = kInf;  // no edges (flagged by k_bsca_cos)
        return;
    }
    const int64_t total = (int64_t)P * R;
    const double md = ceil((double)p.dbar * (double)P - 1e-3);
    const int64_t m = md < 0.0 ? 0 : (int64_t)md;
    if (m < 1 || total == 0) {
        if (threadIdx.x == 0) p.tau[q] = kInf;
        return;
    }
    if (m >= total) {
        if (threadIdx.x == 0) p.tau[q] = -kInf;
        return;
    }
    if (threadIdx.x == 0) {
        s_bin = -1;
        s_cnt = 0;
        s_found = 0;
    }
    __syncthreads();
    // thread t owns the kBscaBins / kSelThreads bins just below those of
    // thread t - 1, counted from the top
    constexpr int kPer = kBscaBins / kSelThreads;
    const int top = kBscaBins - 1 - kPer * (int)threadIdx.x;
    uint32_t mine = 0;
#pragma unroll
    for (int u = 0; u < kPer; ++u) mine += hs[top - u];
    uint32_t incl = mine;  // inclusive scan over the warp's lanes
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const uint32_t v = __shfl_up_sync(0xFFFFFFFFu, incl, o);
        if (lane >= o) incl += v;
    }
    if (lane == 31) wsum[warp] = incl;
    __syncthreads();
    uint32_t above = incl - mine;  // values in the bins above this thread's
    for (int w = 0; w < warp; ++w) above += wsum[w];
    if (above < (uint64_t)m && above + mine >= (uint64_t)m) {
        uint32_t acc = above;
        for (int u = 0; u < kPer; ++u) {
            const int b = top - u;
            if (acc + hs[b] >= (uint64_t)m) {
                s_bin = b;
                s_rank = (int)(m - acc);  // 1-based rank inside bin b, descending
                break;
            }
            acc += hs[b];
        }
    }
    __syncthreads();
    const int B = s_bin, r = s_rank;
    if (B >= 0 && hs[B] <= (uint32_t)kCandCap) {
        for (int row = warp; row < P; row += kSelThreads / 32)
            for (int j = lane; j < R; j += 32) {
                const float c = p.cos[(int64_t)(i0 + row) * kBscaMaxR + j];
                if (cos_bin(c) == B) {
                    const int pos = atomicAdd(&s_cnt, 1);
                    if (pos < kCandCap) cand[pos] = c;
                }
            }
        __syncthreads();
        const int n = min(s_cnt, kCandCap);
        for (int a = threadIdx.x; a < n; a += kSelThreads) {
            const float v = cand[a];
            int before = 0;  // position of a in the descending order, ties by slot
            for (int e = 0; e < n; ++e) {
                const float x = cand[e];
                before += (x > v) || (x == v && e < a);
            }
            if (before == r - 1) {
                s_tau = v;
                s_found = 1;
            }
        }
        __syncthreads();
        if (s_found) {
            if (threadIdx.x == 0) p.tau[q] = s_tau;
            return;
        }
    }
    // a crowded bin (or counts that do not add up): the radix select over
    // all the cosines
    for (int row = warp; row < P; row += kSelThreads / 32)
        for (int j = lane; j < R; j += 32) cs[row * R + j] = p.cos[(int64_t)(i0 + row) * kBscaMaxR + j];
    __syncthreads();
    const float t = radix_select(cs, total, m, hist);
    if (threadIdx.x == 0) p.tau[q] = t;
}

// Output columns: slot u of a lane covers columns 8 * (lane + 32 u) .. + 7
// (one 16-byte row read); kAttSlots slots cover 512 columns per pass.
constexpr int kAttSlots = 2;
constexpr int kAttGroup = 4;  // neighbours whose rows are read together

__global__ void __launch_bounds__(32 * kAttWarps) k_bsca_attend(const BscaParams p, int S) {
    grid_dep_wait();  // the thresholds (and, through k_bsca_select, the cosines)
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int q = blockIdx.x / S, sl = blockIdx.x - q * S;
    const int i0 = p.vis_offsets[q], P = p.vis_offsets[q + 1] - i0;
    const int j0 = p.chunk_offsets[q];
    int R = p.chunk_offsets[q + 1] - j0;
    if (P < 0) return;              // flagged by k_bsca_cos
    if (!question_ok(P, R)) R = 0;  // no edges, zero output
    int ib, ie;
    slice_of(P, sl, S, ib, ie);
    const float tau = p.tau[q];
    const float scale = rsqrtf((float)p.dh);
    const float kInf = __int_as_float(0x7f800000);
    const bool vvec = p.dout % 8 == 0 && ((uintptr_t)p.vh & 15) == 0 && ((uintptr_t)p.out & 15) == 0;
    const bool kq4 = p.dh % 4 == 0 && ((uintptr_t)p.kh & 7) == 0 && ((uintptr_t)p.qh & 7) == 0;
    for (int li = ib + warp; li < ie; li += kAttWarps) {
        const int64_t i = i0 + li;
        // this token's cosines and W_Q v row (lane t holds elements t, t + 32, ...)
        const float *crow = p.cos + i * kBscaMaxR;
        const bool n0 = lane < R && crow[lane] >= tau;
        const bool n1 = lane + 32 < R && crow[lane + 32] >= tau;
        // lane l holds elements 4 (l + 32 v) .. + 3 of q_i (kq4: d_h % 4 == 0,
        // 8-byte aligned rows), else elements l + 32 u
        float qv[kBscaMaxDh / 32];
        if (kq4) {
#pragma unroll
            for (int v = 0; v < kBscaMaxDh / 128; ++v) {
                const int t = 4 * (lane + 32 * v);
                uint2 x = make_uint2(0u, 0u);
                if (t < p.dh) x = *reinterpret_cast<const uint2 *>(p.qh + i * p.dh + t);
                qv[4 * v] = __uint_as_float(x.x << 16);
                qv[4 * v + 1] = __uint_as_float(x.x & 0xFFFF0000u);
                qv[4 * v + 2] = __uint_as_float(x.y << 16);
                qv[4 * v + 3] = __uint_as_float(x.y & 0xFFFF0000u);
            }
        } else {
#pragma unroll
            for (int u = 0; u < kBscaMaxDh / 32; ++u) {
                const int t = lane + 32 * u;
                qv[u] = t < p.dh ? bf16_at(p.qh, i * p.dh + t) : 0.f;
            }
        }
        const uint64_t nb =
            (uint64_t)__ballot_sync(0xFFFFFFFFu, n0) | ((uint64_t)__ballot_sync(0xFFFFFFFFu, n1) << 32);
        if (p.degree && lane == 0) p.degree[i] = __popcll(nb);
        if (p.edges && lane == 0) p.edges[i] = nb;
        // logits of the neighbours, kAttGroup rows read together: lane l keeps
        // those of the l-th and (l+32)-th neighbour
        float e0 = -kInf, e1 = -kInf;
        int cnt = 0;
        for (uint64_t mm = nb; mm;) {
            int jj[kAttGroup];
#pragma unroll
            for (int g = 0; g < kAttGroup; ++g) {
                jj[g] = mm ? __ffsll((long long)mm) - 1 : -1;
                if (mm) mm &= mm - 1;
            }
            float sg[kAttGroup];
            if (kq4) {
                uint2 x[kAttGroup][kBscaMaxDh / 128];
#pragma unroll
                for (int g = 0; g < kAttGroup; ++g) {
                    const uint16_t *kr = p.kh + (int64_t)(j0 + (jj[g] >= 0 ? jj[g] : 0)) * p.dh;
#pragma unroll
                    for (int v = 0; v < kBscaMaxDh / 128; ++v) {
                        const int t = 4 * (lane + 32 * v);
                        x[g][v] = (jj[g] >= 0 && t < p.dh) ? *reinterpret_cast<const uint2 *>(kr + t)
                                                           : make_uint2(0u, 0u);
                    }
                }
#pragma unroll
                for (int g = 0; g < kAttGroup; ++g) {
                    float acc = 0.f;
#pragma unroll
                    for (int v = 0; v < kBscaMaxDh / 128; ++v) {
                        acc = fmaf(qv[4 * v], __uint_as_float(x[g][v].x << 16), acc);
                        acc = fmaf(qv[4 * v + 1], __uint_as_float(x[g][v].x & 0xFFFF0000u), acc);
                        acc = fmaf(qv[4 * v + 2], __uint_as_float(x[g][v].y << 16), acc);
                        acc = fmaf(qv[4 * v + 3], __uint_as_float(x[g][v].y & 0xFFFF0000u), acc);
                    }
                    sg[g] = acc;
                }
            } else {
#pragma unroll
                for (int g = 0; g < kAttGroup; ++g) {
                    const uint16_t *kr = p.kh + (int64_t)(j0 + (jj[g] >= 0 ? jj[g] : 0)) * p.dh;
                    float acc = 0.f;
#pragma unroll
                    for (int u = 0; u < kBscaMaxDh / 32; ++u) {
                        const int t = lane + 32 * u;
                        if (jj[g] >= 0 && t < p.dh) acc = fmaf(qv[u], bf16_at(kr, t), acc);
                    }
                    sg[g] = acc;
                }
            }
#pragma unroll
            for (int o = 16; o; o >>= 1)
#pragma unroll
                for (int g = 0; g < kAttGroup; ++g) sg[g] += __shfl_xor_sync(0xFFFFFFFFu, sg[g], o);
#pragma unroll
            for (int g = 0; g < kAttGroup; ++g)
                if (jj[g] >= 0) {
                    if (cnt == lane) e0 = sg[g] * scale;
                    if (cnt == lane + 32) e1 = sg[g] * scale;
                    ++cnt;
                }
        }
        // softmax weights, normalised
        float mx = fmaxf(e0, e1);
#pragma unroll
        for (int o = 16; o; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xFFFFFFFFu, mx, o));
        float w0 = lane < cnt ? expf(e0 - mx) : 0.f, w1 = lane + 32 < cnt ? expf(e1 - mx) : 0.f;
        float den = w0 + w1;
#pragma unroll
        for (int o = 16; o; o >>= 1) den += __shfl_xor_sync(0xFFFFFFFFu, den, o);
        const float inv = den > 0.f ? 1.f / den : 0.f;
        w0 *= inv;
        w1 *= inv;
        float *orow = p.out + i * p.dout;
        // out_i = sum_j w_j W_V k_j, kAttGroup rows in flight
        if (vvec) {
            for (int c0 = 0; c0 < p.dout; c0 += 8 * 32 * kAttSlots) {
                float acc[kAttSlots][8];
#pragma unroll
                for (int u = 0; u < kAttSlots; ++u)
#pragma unroll
                    for (int h = 0; h < 8; ++h) acc[u][h] = 0.f;
                int k = 0;
                for (uint64_t mm = nb; mm;) {
                    int jj[kAttGroup];
                    float ww[kAttGroup];
#pragma unroll
                    for (int g = 0; g < kAttGroup; ++g) {
                        jj[g] = mm ? __ffsll((long long)mm) - 1 : -1;
                        if (mm) mm &= mm - 1;
                        const int kk = k + g;
                        const float wv = __shfl_sync(0xFFFFFFFFu, kk < 32 ? w0 : w1, kk & 31);
                        ww[g] = jj[g] >= 0 ? wv : 0.f;
                    }
                    k += kAttGroup;
                    uint4 x[kAttGroup][kAttSlots];
#pragma unroll
                    for (int g = 0; g < kAttGroup; ++g) {
                        const uint4 *r4 = reinterpret_cast<const uint4 *>(
                            p.vh + (int64_t)(j0 + (jj[g] >= 0 ? jj[g] : 0)) * p.dout + c0);
#pragma unroll
                        for (int u = 0; u < kAttSlots; ++u) {
                            const bool in = jj[g] >= 0 && c0 + 8 * (lane + 32 * u) < p.dout;
                            x[g][u] = in ? r4[lane + 32 * u] : make_uint4(0u, 0u, 0u, 0u);
                        }
                    }
#pragma unroll
                    for (int g = 0; g < kAttGroup; ++g)
#pragma unroll
                        for (int u = 0; u < kAttSlots; ++u) {
                            float f[8];
                            bf16x8(x[g][u], f);
#pragma unroll
                            for (int h = 0; h < 8; ++h) acc[u][h] = fmaf(ww[g], f[h], acc[u][h]);
                        }
                }
#pragma unroll
                for (int u = 0; u < kAttSlots; ++u) {
                    const int col = c0 + 8 * (lane + 32 * u);
                    if (col < p.dout) {
                        float4 *o4 = reinterpret_cast<float4 *>(orow + col);
                        o4[0] = make_float4(acc[u][0], acc[u][1], acc[u][2], acc[u][3]);
                        o4[1] = make_float4(acc[u][4], acc[u][5], acc[u][6], acc[u][7]);
                    }
                }
            }
        } else {
            // d_o not a multiple of 8, or unaligned rows: two columns per step
            // (the loop runs the same number of times in every lane: the
            // shuffle needs the whole warp)
            const int npair = p.dout / 2;
            float2 *o2 = reinterpret_cast<float2 *>(orow);
            for (int pr0 = 0; pr0 < npair; pr0 += 32) {
                const int pr = pr0 + lane;
                float2 acc = make_float2(0.f, 0.f);
                int k = 0;
                for (uint64_t mm = nb; mm; mm &= mm - 1, ++k) {
                    const int j = __ffsll((long long)mm) - 1;
                    const float w = __shfl_sync(0xFFFFFFFFu, k < 32 ? w0 : w1, k & 31);
                    if (pr < npair) {
                        const float2 v = __bfloat1622float2(
                            reinterpret_cast<const __nv_bfloat162 *>(p.vh + (int64_t)(j0 + j) * p.dout)[pr]);
                        acc.x = fmaf(w, v.x, acc.x);
                        acc.y = fmaf(w, v.y, acc.y);
                    }
                }
                if (pr < npair) o2[pr] = acc;
            }
        }
    }
}

}  // namespace

// Launch as the programmatic dependent of the previous kernel in the stream
// (its launch overlaps that kernel's tail; it waits for its results).
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

cudaError_t launch_bsca(const BscaParams &p, cudaStream_t s) {
    if (p.Q == 0) return cudaSuccess;
    // slices per question from the mean tokens per question: about 32 tokens
    // per cosine block, one token per warp of an attention block
    const int64_t mean = (p.Nv + p.Q - 1) / p.Q;
    const int S1 = (int)std::min<int64_t>(64, std::max<int64_t>(1, (mean + 31) / 32));
    const int S3 = (int)std::min<int64_t>(64, std::max<int64_t>(1, (mean + kAttWarps - 1) / kAttWarps));
    const size_t smem1 = ((size_t)kBscaMaxR * (p.dp + 1) + (size_t)(kCosThreads / 32) * p.dp * 4) * sizeof(float);
    cudaError_t e = cudaFuncSetAttribute(k_bsca_cos, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem1);
    if (e != cudaSuccess) return e;
    k_bsca_cos<<<(unsigned)(p.Q * S1), kCosThreads, smem1, s>>>(p, S1);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    const size_t smem2 = (size_t)kBscaMaxPairs * sizeof(float);
    e = cudaFuncSetAttribute(k_bsca_select, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem2);
    if (e != cudaSuccess) return e;
    if ((e = launch_dependent(k_bsca_select, dim3((unsigned)p.Q), kSelThreads, smem2, s, p)) != cudaSuccess) {
        // the select clears the histograms; without it they must be cleared here
        cudaMemsetAsync(p.hist, 0, (size_t)p.Q * kBscaBins * sizeof(uint32_t), s);
        return e;
    }
    if (p.Nv == 0) return e;
    return launch_dependent(k_bsca_attend, dim3((unsigned)(p.Q * S3)), 32 * kAttWarps, (size_t)0, s, p, S3);
}

}  // namespace skipk
