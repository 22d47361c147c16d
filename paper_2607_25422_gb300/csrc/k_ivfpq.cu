// IVF-PQ approximate variant of the per-region search (the index of §4.1
// "Implementation" / App. I.4: inverted lists over inner-product centroids,
// product-quantised residual codes, asymmetric scoring).
//
// Build (after the coarse assignment, which runs on the exact MIPS path with
// the centroids as the corpus and the corpus rows as queries, k = 1):
//   k_pq_encode     residual x - c_list, nearest of 256 codewords per
//                   sub-space (fp32, ties to the lower codeword); a block of
//                   128 rows shares each sub-space's codebook in shared memory,
//                   read as 16-byte broadcasts.
//   k_ivf_count / k_ivf_offsets / k_ivf_scatter
//                   counting sort of the rows into their lists (order inside
//                   a list is arbitrary: the search breaks ties by id).
//   k_ivf_interleave
//                   the codes of each list regrouped into blocks of 32
//                   entries, byte m of entry j at [m][j] inside its block, so
//                   that one lane reads one sub-space of 32 entries at once.
// Search (after the coarse top-nprobe, again on the exact MIPS path):
//   k_ivfpq_scan    one region per CTA at a time: the region's lookup table
//                   T[j][m] = <q_m, p_{m,j}> in shared memory (a row holds
//                   the sub-spaces of codeword j, so lane m % 32 always reads
//                   bank m % 32: no conflicts), then each warp scores blocks
//                   of 32 entries: lane m adds T[code_{e,m}][m] for the 32
//                   entries e, and a butterfly reduce-scatter leaves lane e
//                   with <q, c_l> + sum_m T[code_{e,m}][m]; candidates above
//                   the running k-th key go to a shared buffer that is sorted
//                   and cut back to k when it fills.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <algorithm>

#include "skip_device.cuh"
#include "skip_internal.h"

namespace skipk {
namespace {

// ---------------------------------------------------------------- encode

constexpr int kEncRows = 128;

// DSB: the sub-space width rounded up to 4, 8, 12, 16, 24 or 32; the
// codebook copy in shared memory and the residual are zero past ds, so the
// padded sum adds exact zeros after the same terms in the same order.
template <int DSB>
__global__ void __launch_bounds__(kEncRows) k_pq_encode(const IvfParams p, const int64_t *row_list,
                                                         uint8_t *codes) {
    extern __shared__ float4 cbs4[];  // [256][DSB / 4]: codebook of one sub-space
    float *cbs = reinterpret_cast<float *>(cbs4);
    const int64_t i = (int64_t)blockIdx.x * kEncRows + threadIdx.x;
    const bool valid = i < p.N;
    const int ds = p.ds;
    int64_t l = valid ? row_list[i] : 0;
    if (l < 0 || l >= p.C) l = 0;  // flagged by k_ivf_count
    const __nv_bfloat16 *x = reinterpret_cast<const __nv_bfloat16 *>(p.rows) + (valid ? i : 0) * (int64_t)p.d;
    const __nv_bfloat16 *c = reinterpret_cast<const __nv_bfloat16 *>(p.centroids) + l * (int64_t)p.d;
    for (int m = 0; m < p.M; ++m) {
        __syncthreads();
        for (int e = threadIdx.x; e < 256 * DSB; e += kEncRows) {
            const int j = e / DSB, t = e - j * DSB;
            cbs[e] = t < ds ? p.codebook[((int64_t)m * 256 + j) * ds + t] : 0.f;
        }
        __syncthreads();
        float r[DSB];
#pragma unroll
        for (int t = 0; t < DSB; ++t)
            r[t] = t < ds ? __bfloat162float(x[m * ds + t]) - __bfloat162float(c[m * ds + t]) : 0.f;
        int best = 0;
        float bd = __int_as_float(0x7f800000);
        for (int j = 0; j < 256; ++j) {
            float dist = 0.f;
#pragma unroll
            for (int q = 0; q < DSB / 4; ++q) {
                const float4 v = cbs4[j * (DSB / 4) + q];
                const float e0 = r[4 * q] - v.x, e1 = r[4 * q + 1] - v.y;
                const float e2 = r[4 * q + 2] - v.z, e3 = r[4 * q + 3] - v.w;
                dist = fmaf(e0, e0, dist);
                dist = fmaf(e1, e1, dist);
                dist = fmaf(e2, e2, dist);
                dist = fmaf(e3, e3, dist);
            }
            if (dist < bd) {
                bd = dist;
                best = j;
            }
        }
        if (valid) codes[i * p.M + m] = (uint8_t)best;
    }
}

// ---------------------------------------------------------------- lists

__global__ void k_ivf_count(const int64_t *row_list, int64_t N, int C, int64_t *counts, int *err) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < N; i += (int64_t)gridDim.x * blockDim.x) {
        const int64_t l = row_list[i];
        if (l < 0 || l >= C) {
            atomicOr(err, kErrConfig);
            continue;
        }
        atomicAdd(reinterpret_cast<unsigned long long *>(counts + l), 1ull);
    }
}

// Exclusive scan of counts [C] into offsets [C+1] (one block), and the
// scatter cursors set to the list starts.
__global__ void __launch_bounds__(1024) k_ivf_offsets(const int64_t *counts, int C, int64_t *offsets,
                                                      int64_t *cursor) {
    __shared__ int64_t part[1024];
    const int t = threadIdx.x;
    const int per = (C + 1023) / 1024;
    const int lo = min(C, t * per), hi = min(C, lo + per);
    int64_t s = 0;
    for (int l = lo; l < hi; ++l) s += counts[l];
    part[t] = s;
    __syncthreads();
    for (int o = 1; o < 1024; o <<= 1) {
        const int64_t v = t >= o ? part[t - o] : 0;
        __syncthreads();
        part[t] += v;
        __syncthreads();
    }
    int64_t run = part[t] - s;  // exclusive prefix of this thread's range
    for (int l = lo; l < hi; ++l) {
        offsets[l] = run;
        cursor[l] = run;
        run += counts[l];
    }
    if (t == 1023) offsets[C] = part[1023];
}

__global__ void k_ivf_scatter(const int64_t *row_list, const uint8_t *codes_rows, int64_t N, int C, int M,
                              int64_t *cursor, int32_t *ids, uint8_t *codes) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < N; i += (int64_t)gridDim.x * blockDim.x) {
        const int64_t l = row_list[i];
        if (l < 0 || l >= C) continue;
        const int64_t pos = (int64_t)atomicAdd(reinterpret_cast<unsigned long long *>(cursor + l), 1ull);
        ids[pos] = (int32_t)i;
        const uint4 *src = reinterpret_cast<const uint4 *>(codes_rows + i * M);
        uint4 *dst = reinterpret_cast<uint4 *>(codes + pos * M);
        for (int w = 0; w < M / 16; ++w) dst[w] = src[w];
    }
}

// Where byte m of entry j (0 <= j < 32) sits inside its block of 32 entries
// (M * 32 bytes).  The scan's lane l = m % 32 of pass pp = m / 32 owns the
// 32 bytes of sub-space m, in the order s = j ^ l (the order its
// reduce-scatter wants), and loads them as two 16-byte halves; each half of
// a pass is stored contiguously over the pass's lanes, so that one
// warp-wide load reads 16 * Mq contiguous bytes (Mq = sub-spaces in the pass).
__device__ __forceinline__ int64_t il_offset(int M, int m, int j) {
    const int pp = m >> 5, l = m & 31, mq = min(32, M - (pp << 5));
    const int sl = j ^ l;
    return ((int64_t)pp << 10) + (sl >> 4) * (mq << 4) + (l << 4) + (sl & 15);
}

// Entry e of the list order lies in list l (off[l] <= e < off[l + 1]) at
// position j = e - off[l]: block boff[l] + j / 32, entry j % 32 there.
// il_out set: rows -> il, else il -> rows.  Offsets are validated on the
// host before this runs.
__global__ void k_ivf_interleave(const int64_t *off, const int64_t *boff, int C, int64_t N, int M,
                                 const uint8_t *rows_in, uint8_t *rows_out, const uint8_t *il_in, uint8_t *il_out) {
    for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < N; e += (int64_t)gridDim.x * blockDim.x) {
        int lo = 0, hi = C - 1;  // the largest l with off[l] <= e
        while (lo < hi) {
            const int mid = (lo + hi + 1) >> 1;
            if (off[mid] <= e) lo = mid;
            else hi = mid - 1;
        }
        const int64_t j = e - off[lo];
        const int64_t blk = (boff[lo] + (j >> 5)) * M * 32;
        const int jj = (int)(j & 31);
        if (il_out) {
            for (int m = 0; m < M; ++m) il_out[blk + il_offset(M, m, jj)] = rows_in[e * M + m];
        } else {
            for (int m = 0; m < M; ++m) rows_out[e * M + m] = il_in[blk + il_offset(M, m, jj)];
        }
    }
}

// cbT[(j * ds + t) * Mp + m] = codebook[(m * 256 + j) * ds + t], 0 for m >= M:
// the lookup-table build reads one codeword coordinate of 32 sub-spaces per
// warp-wide load.
__global__ void k_pq_codebook_t(const float *cb, int M, int ds, int Mp, float *cbT) {
    const int64_t n = (int64_t)256 * ds * Mp;
    for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < n; e += (int64_t)gridDim.x * blockDim.x) {
        const int m = (int)(e % Mp);
        const int64_t jt = e / Mp;  // j * ds + t
        const int j = (int)(jt / ds), t = (int)(jt % ds);
        cbT[e] = m < M ? cb[((int64_t)m * 256 + j) * ds + t] : 0.f;
    }
}

// ---------------------------------------------------------------- search

constexpr int kScanWarps = 8;
constexpr int kScanThreads = kScanWarps * 32;
constexpr int kScanBpw = 4;                        // blocks of 32 entries per warp per round
constexpr int kScanRound = kScanWarps * kScanBpw;  // blocks per round
constexpr int kCandBuf = 2048;
static_assert(kCandBuf - kScanRound * 32 >= 1024, "a round must fit behind a cut to k <= 1024 keys");
static_assert(kScanBpw % 2 == 0, "blocks alternate between two register sets");

// Sorts keys[0, n) descending in place (n a power of two, >= 2).
__device__ void block_sort_desc(uint64_t *keys, int n) {
    for (int size = 2; size <= n; size <<= 1)
        for (int stride = size >> 1; stride > 0; stride >>= 1) {
            for (int t = threadIdx.x; t < n / 2; t += blockDim.x) {
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
}

// Coarse probe of a small centroid set: region r's C centroid scores
// (a GEMM's row) sorted by (score desc, id asc) in shared memory; the first
// nprobe are the probed lists.
__global__ void __launch_bounds__(256) k_ivf_probe_select(const float *scores, int C, int nprobe,
                                                          int64_t *probe_ids, float *probe_sc) {
    extern __shared__ uint64_t pkeys[];  // [n], n = C rounded up to a power of two
    const int r = blockIdx.x;
    int n = 2;
    while (n < C) n <<= 1;
    const float *sr = scores + (int64_t)r * C;
    for (int c = threadIdx.x; c < n; c += blockDim.x) pkeys[c] = c < C ? make_key(sr[c], (uint32_t)c) : 0ull;
    __syncthreads();
    block_sort_desc(pkeys, n);
    for (int i = threadIdx.x; i < nprobe; i += blockDim.x) {
        int64_t id;
        float sc;
        key_decode(pkeys[i], id, sc);
        probe_ids[(int64_t)r * nprobe + i] = id;
        probe_sc[(int64_t)r * nprobe + i] = sc;
    }
}

// One step of the butterfly reduce-scatter.  Slot i of lane l holds entry
// i ^ l (the index stores each sub-space's bytes in that order), so the
// lane keeps slots [0, O) and adds the partner's slots [O, 2 O), which hold
// the same entries: no lane-dependent register choice.
template <int O>
__device__ __forceinline__ void reduce_step(float (&a)[32]) {
#pragma unroll
    for (int i = 0; i < O; ++i) a[i] += __shfl_xor_sync(0xFFFFFFFFu, a[i + O], O);
}

// Lane l returns the sum over all lanes of their entry-l partial sums
// (31 shuffles for 32 sums).
__device__ __forceinline__ float warp_reduce_scatter(float (&a)[32]) {
    reduce_step<16>(a);
    reduce_step<8>(a);
    reduce_step<4>(a);
    reduce_step<2>(a);
    reduce_step<1>(a);
    return a[0];
}

// The probe whose blocks hold block b of the region (pref[pi] <= b <
// pref[pi + 1]), searched forward from probe pi: a warp's blocks only grow.
__device__ __forceinline__ int advance_probe(const int *pref, int nprobe, int pi, int b) {
    while (pi + 1 < nprobe && pref[pi + 1] <= b) ++pi;
    return pi;
}

// Lane l of pass pp loads the 32 bytes of sub-space m = 32 pp + l of block b
// (held by probe pi), as laid out by il_offset.
template <int NP>
__device__ __forceinline__ void load_block(const uint8_t *codes, const int *pref, const int *pblk, int M, int lane,
                                           int pi, int b, uint4 (&cw)[NP][2]) {
    const uint8_t *blk = codes + (int64_t)(pblk[pi] + (b - pref[pi])) * (M * 32);
#pragma unroll
    for (int pp = 0; pp < NP; ++pp) {
        const int mq = min(32, M - pp * 32);  // sub-spaces in this pass
        if (lane < mq) {
            const uint8_t *src = blk + (pp << 10) + (lane << 4);
            cw[pp][0] = __ldg(reinterpret_cast<const uint4 *>(src));
            cw[pp][1] = __ldg(reinterpret_cast<const uint4 *>(src + (mq << 4)));
        }
    }
}

// The lookup table is kept in slabs of 256 rows x 64 floats: sub-space
// m = 32 pp + l sits in slab pp / 2, column 32 (pp % 2) + l, so the byte
// offset of (codeword c, pass pp, lane l) inside its slab is
// c * 256 + 128 (pp % 2) + 4 l, which one byte permute builds from the code
// word and the lane's constant.
constexpr int kSlab = 256 * 64;

// Lane l's partial sums over its sub-spaces for the 32 entries of a block
// (slot e holds entry e ^ l), reduced so that lane l returns entry l's
// sum_m T[code_{l,m}][m].
template <int NP>
__device__ __forceinline__ float score_block(const float *T, const uint4 (&cw)[NP][2], int M, int lane,
                                             const uint32_t (&y)[2]) {
    float a[32];
#pragma unroll
    for (int pp = 0; pp < NP; ++pp) {
        const char *Ts = reinterpret_cast<const char *>(T + (pp >> 1) * kSlab);
        const uint32_t w[8] = {cw[pp][0].x, cw[pp][0].y, cw[pp][0].z, cw[pp][0].w,
                               cw[pp][1].x, cw[pp][1].y, cw[pp][1].z, cw[pp][1].w};
        if (pp * 32 + lane < M) {
#pragma unroll
            for (int e = 0; e < 32; ++e) {
                // bytes [0, 0, code byte e, byte 0 of y]: c * 256 + 128 (pp % 2) + 4 l
                const uint32_t off = __byte_perm(w[e >> 2], y[pp & 1], 0x7604u | ((e & 3) << 4));
                const float v = *reinterpret_cast<const float *>(Ts + off);
                a[e] = pp == 0 ? v : a[e] + v;
            }
        } else if (pp == 0) {
#pragma unroll
            for (int e = 0; e < 32; ++e) a[e] = 0.f;
        }
    }
    return warp_reduce_scatter(a);
}

template <int NP>
__global__ void __launch_bounds__(kScanThreads, NP <= 2 ? 2 : 1)
    k_ivfpq_scan(const IvfParams p, const uint16_t *regions, int R, const int64_t *probe_ids,
                 const float *probe_scores, int nprobe, int k, int G, uint64_t *out_keys) {
    constexpr int kSlabs = (NP + 1) / 2;
    extern __shared__ __align__(16) uint8_t sm[];
    float *T = reinterpret_cast<float *>(sm);                          // [kSlabs][256][64]
    uint64_t *cand = reinterpret_cast<uint64_t *>(T + kSlab * kSlabs);  // [kCandBuf]
    int *pref = reinterpret_cast<int *>(cand + kCandBuf);              // [nprobe + 1] prefix of block counts
    int *pstart = pref + (nprobe + 1);                                 // [nprobe] first entry of the list
    int *pblk = pstart + nprobe;                                       // [nprobe] first block of the list
    int *plen = pblk + nprobe;                                         // [nprobe] entries of the list
    float *pscore = reinterpret_cast<float *>(plen + nprobe);          // [nprobe] <q, c_l>
    __shared__ int cnt;
    __shared__ uint64_t tau;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int M = p.M, ds = p.ds;
    constexpr int Mp = 32 * NP;
    constexpr int kLutUnroll = NP == 2 ? 3 : 2;  // codebook loads in flight per lane: 32 x this
    // item it: part g of region r (its blocks [TB g / G, TB (g + 1) / G))
    for (int it = blockIdx.x; it < R * G; it += gridDim.x) {
        const int r = it / G, g = it - r * G;
        for (int t = threadIdx.x; t < nprobe; t += kScanThreads) {
            const int64_t l = probe_ids[(int64_t)r * nprobe + t];
            const bool ok = l >= 0 && l < p.C;
            pstart[t] = ok ? (int)p.offsets[l] : 0;
            plen[t] = ok ? (int)(p.offsets[l + 1] - p.offsets[l]) : 0;
            pblk[t] = ok ? (int)p.boff[l] : 0;
            pref[t + 1] = ok ? (int)(p.boff[l + 1] - p.boff[l]) : 0;
            pscore[t] = probe_scores[(int64_t)r * nprobe + t];
        }
        if (threadIdx.x == 0) {
            pref[0] = 0;
            cnt = 0;
            tau = 0;
        }
        // lookup table T[c][m] = <q_m, p_{m,c}>: the warps of pass pp = warp % NP
        // fill its rows c, 32 rows at a time, lane m reading cbT[c][t][m].
        {
            const __nv_bfloat16 *q = reinterpret_cast<const __nv_bfloat16 *>(regions) + (int64_t)r * p.d;
            const int pp = warp % NP, m = pp * 32 + lane;
            const int nw = (kScanWarps - pp + NP - 1) / NP;  // warps sharing pass pp
            float *Tw = T + (pp >> 1) * kSlab + (pp & 1) * 32 + lane;  // row c at Tw[c * 64]
            for (int c0 = warp / NP; c0 < 256; c0 += 32 * nw) {
                float acc[32];
#pragma unroll
                for (int i = 0; i < 32; ++i) acc[i] = 0.f;
#pragma unroll kLutUnroll
                for (int t = 0; t < ds; ++t) {
                    const float qv = m < M ? __bfloat162float(q[m * ds + t]) : 0.f;
                    const float *pc = p.cbT + ((int64_t)c0 * ds + t) * Mp + m;
#pragma unroll
                    for (int i = 0; i < 32; ++i)
                        if (c0 + i * nw < 256) acc[i] = fmaf(qv, __ldg(pc + (int64_t)i * nw * ds * Mp), acc[i]);
                }
#pragma unroll
                for (int i = 0; i < 32; ++i)
                    if (c0 + i * nw < 256) Tw[(c0 + i * nw) * 64] = acc[i];
            }
        }
        __syncthreads();
        if (threadIdx.x < 32) {  // inclusive scan of pref[1..nprobe], one warp
            int carry = 0;
            for (int b = 0; b < nprobe; b += 32) {
                const int t = b + (int)threadIdx.x;
                int v = t < nprobe ? pref[t + 1] : 0;
#pragma unroll
                for (int o = 1; o < 32; o <<= 1) {
                    const int u = __shfl_up_sync(0xFFFFFFFFu, v, o);
                    if ((int)threadIdx.x >= o) v += u;
                }
                if (t < nprobe) pref[t + 1] = v + carry;
                carry += __shfl_sync(0xFFFFFFFFu, v, 31);
            }
        }
        __syncthreads();
        const int TB = pref[nprobe];  // blocks of 32 entries over the probed lists
        // the buffer is cut back to k once it holds more than max(k, 512) keys
        // (a first cut after one round sets tau early); a round adds at most
        // kScanRound * 32, so it never overflows
        const int cut_at = min(max(k, 512), kCandBuf - kScanRound * 32);
        const int lo = (int)((int64_t)TB * g / G), hi = (int)((int64_t)TB * (g + 1) / G);
        const uint32_t y[2] = {(uint32_t)lane * 4u, (uint32_t)lane * 4u + 128u};
        // this warp scores blocks warp, warp + kScanWarps, ...; the next
        // block's codes are loaded (into the other register set) while the
        // current one is scored
        // lane l's entry of block b joins the candidates when its key beats
        // tau; one atomic per warp reserves the slots
        auto consider = [&](int b, int pi, float part) {
            const int pos = (b - pref[pi]) * 32 + lane;  // entry of the list
            uint64_t key = 0;
            if (pos < plen[pi]) {
                const float sc = pscore[pi] + part;
                const uint64_t tk = tau;
                if (ord_of_score(sc) >= (uint32_t)(tk >> 32)) {
                    const uint64_t kk = make_key(sc, (uint32_t)p.ids[pstart[pi] + pos]);
                    if (kk > tk) key = kk;
                }
            }
            const unsigned want = __ballot_sync(0xFFFFFFFFu, key != 0);
            if (want) {
                int at = 0;
                if (lane == 0) at = atomicAdd(&cnt, __popc(want));
                at = __shfl_sync(0xFFFFFFFFu, at, 0) + __popc(want & ((1u << lane) - 1u));
                if (key) cand[at] = key;  // at < kCandBuf: at most kScanRound * 32 are added per round
            }
        };
        int b = lo + warp, pi = 0;
        uint4 cw[NP][2], nx[NP][2];
        if (b < hi) {
            pi = advance_probe(pref, nprobe, 0, b);
            load_block<NP>(p.codes, pref, pblk, M, lane, pi, b, cw);
        }
        for (int base = lo; base < hi; base += kScanRound) {
#pragma unroll 1
            for (int i = 0; i < kScanBpw; i += 2) {
                const int b1 = b + kScanWarps;
                int p1 = pi;
                if (b1 < hi) {
                    p1 = advance_probe(pref, nprobe, pi, b1);
                    load_block<NP>(p.codes, pref, pblk, M, lane, p1, b1, nx);
                }
                if (b < hi) consider(b, pi, score_block<NP>(T, cw, M, lane, y));
                const int b2 = b1 + kScanWarps;
                int p2 = p1;
                if (b2 < hi) {
                    p2 = advance_probe(pref, nprobe, p1, b2);
                    load_block<NP>(p.codes, pref, pblk, M, lane, p2, b2, cw);
                }
                if (b1 < hi) consider(b1, p1, score_block<NP>(T, nx, M, lane, y));
                b = b2;
                pi = p2;
            }
            __syncthreads();
            if (cnt > cut_at) {
                int n = 2;
                while (n < cnt) n <<= 1;
                for (int t = cnt + threadIdx.x; t < n; t += kScanThreads) cand[t] = 0;
                __syncthreads();
                block_sort_desc(cand, n);
                if (threadIdx.x == 0) {
                    cnt = min(cnt, k);
                    if (cnt == k) tau = cand[k - 1];
                }
                __syncthreads();
            }
        }
        // final cut
        int n = 2;
        while (n < max(cnt, k)) n <<= 1;
        for (int t = cnt + threadIdx.x; t < n; t += kScanThreads) cand[t] = 0;
        __syncthreads();
        block_sort_desc(cand, n);
        for (int t = threadIdx.x; t < k; t += kScanThreads) out_keys[((int64_t)g * R + r) * k + t] = cand[t];
        __syncthreads();
    }
}

}  // namespace

namespace {
template <int DSB>
void launch_encode_dsb(const IvfParams &p, const int64_t *row_list, uint8_t *codes, cudaStream_t s) {
    k_pq_encode<DSB><<<(unsigned)((p.N + kEncRows - 1) / kEncRows), kEncRows, (size_t)256 * DSB * sizeof(float), s>>>(
        p, row_list, codes);
}
}  // namespace

cudaError_t launch_pq_encode(const IvfParams &p, const int64_t *row_list, uint8_t *codes, cudaStream_t s) {
    if (p.N == 0) return cudaSuccess;
    if (p.ds <= 4) launch_encode_dsb<4>(p, row_list, codes, s);
    else if (p.ds <= 8) launch_encode_dsb<8>(p, row_list, codes, s);
    else if (p.ds <= 12) launch_encode_dsb<12>(p, row_list, codes, s);
    else if (p.ds <= 16) launch_encode_dsb<16>(p, row_list, codes, s);
    else if (p.ds <= 24) launch_encode_dsb<24>(p, row_list, codes, s);
    else if (p.ds <= 32) launch_encode_dsb<32>(p, row_list, codes, s);
    else return cudaErrorInvalidValue;
    return cudaGetLastError();
}

cudaError_t launch_ivf_lists(const IvfParams &p, const int64_t *row_list, const uint8_t *codes_rows,
                             int64_t *counts, int64_t *cursor, int64_t *offsets, int32_t *ids, uint8_t *codes,
                             int *err, int sms, cudaStream_t s) {
    cudaError_t e = cudaMemsetAsync(counts, 0, sizeof(int64_t) * p.C, s);
    if (e != cudaSuccess) return e;
    const int grid = std::max(1, std::min<int>((int)((p.N + 255) / 256), sms * 8));
    if (p.N > 0) k_ivf_count<<<grid, 256, 0, s>>>(row_list, p.N, p.C, counts, err);
    k_ivf_offsets<<<1, 1024, 0, s>>>(counts, p.C, offsets, cursor);
    if (p.N > 0) k_ivf_scatter<<<grid, 256, 0, s>>>(row_list, codes_rows, p.N, p.C, p.M, cursor, ids, codes);
    return cudaGetLastError();
}

cudaError_t launch_ivf_interleave(const IvfParams &p, const uint8_t *rows, uint8_t *il, int sms, cudaStream_t s) {
    if (p.N == 0) return cudaSuccess;
    const int grid = std::max(1, std::min<int>((int)((p.N + 255) / 256), sms * 8));
    k_ivf_interleave<<<grid, 256, 0, s>>>(p.offsets, p.boff, p.C, p.N, p.M, rows, nullptr, nullptr, il);
    return cudaGetLastError();
}

cudaError_t launch_ivf_deinterleave(const IvfParams &p, uint8_t *rows, int sms, cudaStream_t s) {
    if (p.N == 0) return cudaSuccess;
    const int grid = std::max(1, std::min<int>((int)((p.N + 255) / 256), sms * 8));
    k_ivf_interleave<<<grid, 256, 0, s>>>(p.offsets, p.boff, p.C, p.N, p.M, nullptr, rows, p.codes, nullptr);
    return cudaGetLastError();
}

cudaError_t launch_pq_codebook_t(const float *codebook, int M, int ds, float *cbT, cudaStream_t s) {
    const int Mp = ivf_padded_m(M);
    const int64_t n = (int64_t)256 * ds * Mp;
    k_pq_codebook_t<<<(unsigned)std::min<int64_t>((n + 255) / 256, 4096), 256, 0, s>>>(codebook, M, ds, Mp, cbT);
    return cudaGetLastError();
}

cudaError_t launch_ivf_probe_select(const float *scores, int R, int C, int nprobe, int64_t *probe_ids,
                                    float *probe_sc, cudaStream_t s) {
    if (R == 0) return cudaSuccess;
    if (C < 1 || C > kIvfCoarseMaxC || nprobe < 1 || nprobe > C) return cudaErrorInvalidValue;
    int n = 2;
    while (n < C) n <<= 1;
    k_ivf_probe_select<<<R, 256, (size_t)n * sizeof(uint64_t), s>>>(scores, C, nprobe, probe_ids, probe_sc);
    return cudaGetLastError();
}

size_t ivfpq_scan_smem(int M, int nprobe) {
    const int slabs = (ivf_padded_m(M) / 32 + 1) / 2;
    return (size_t)kSlab * 4 * slabs + (size_t)kCandBuf * 8 + (size_t)(nprobe + 1) * 4 + (size_t)nprobe * 16 + 16;
}

namespace {
template <int NP>
cudaError_t scan_slots(int M, int nprobe, int sms, int *slots) {
    const size_t smem = ivfpq_scan_smem(M, nprobe);
    cudaError_t e = cudaFuncSetAttribute(k_ivfpq_scan<NP>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    int per_sm = 0;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k_ivfpq_scan<NP>, kScanThreads, smem);
    *slots = sms * std::max(per_sm, 1);
    return e;
}

template <int NP>
cudaError_t launch_scan_np(const IvfParams &p, const uint16_t *regions, int R, const int64_t *probe_ids,
                           const float *probe_scores, int nprobe, int k, int G, uint64_t *out_keys, int sms,
                           cudaStream_t s) {
    int slots = 0;
    cudaError_t e = scan_slots<NP>(p.M, nprobe, sms, &slots);
    if (e != cudaSuccess) return e;
    const int grid = std::max(1, std::min(R * G, slots));
    k_ivfpq_scan<NP><<<grid, kScanThreads, ivfpq_scan_smem(p.M, nprobe), s>>>(p, regions, R, probe_ids, probe_scores,
                                                                              nprobe, k, G, out_keys);
    return cudaGetLastError();
}

// Exact re-rank of an IVF-PQ shortlist (an option beyond the paper's FAISS
// IVF-PQ, the usual "refine" step): per region, the ks candidates the scan
// kept by s^ (keys [R x ks], descending, 0 = none) are scored exactly,
// s(r, i) = sum_j q_{r,j} x_{i,j} in fp32 from the bf16 corpus rows, and the
// k best by (s desc, id asc) are written as keys [R x k].  One block per
// region: a warp per candidate row (16-byte loads, the query in shared memory
// as fp32), then a bitonic sort of the keys in shared memory.
constexpr int kRefineThreads = 256;
constexpr int kRefineMax = 1024;

__global__ void __launch_bounds__(kRefineThreads) k_ivf_refine(const uint16_t *__restrict__ rows, int64_t N, int d,
                                                                const uint16_t *__restrict__ regions,
                                                                const uint64_t *__restrict__ cand, int ks, int k,
                                                                uint64_t *__restrict__ out) {
    extern __shared__ float qf[];                       // [d]
    __shared__ uint64_t keys[kRefineMax];
    const int r = blockIdx.x;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    for (int j = threadIdx.x; j < d; j += kRefineThreads)
        qf[j] = __uint_as_float((uint32_t)regions[(int64_t)r * d + j] << 16);
    int n2 = 1;
    while (n2 < ks) n2 <<= 1;
    for (int t = threadIdx.x; t < n2; t += kRefineThreads) keys[t] = 0ull;
    __syncthreads();
    const int nw = d / 8;  // 16-byte words per row
    for (int t = warp; t < ks; t += kRefineThreads / 32) {
        const uint64_t ck = cand[(int64_t)r * ks + t];
        if (ck == 0ull) continue;  // warp-uniform
        const int64_t id = (int64_t)(0xFFFFFFFFu - (uint32_t)ck);
        if (id < 0 || id >= N) continue;
        const uint4 *row = reinterpret_cast<const uint4 *>(rows + id * (int64_t)d);
        float acc = 0.f;
        for (int w = lane; w < nw; w += 32) {
            const uint4 x = __ldg(row + w);
            const uint32_t xv[4] = {x.x, x.y, x.z, x.w};
#pragma unroll
            for (int h = 0; h < 4; ++h) {
                acc = fmaf(__uint_as_float(xv[h] << 16), qf[8 * w + 2 * h], acc);
                acc = fmaf(__uint_as_float(xv[h] & 0xFFFF0000u), qf[8 * w + 2 * h + 1], acc);
            }
        }
#pragma unroll
        for (int o = 16; o; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
        if (lane == 0) keys[t] = make_key(acc, (uint32_t)id);
    }
    __syncthreads();
    for (int size = 2; size <= n2; size <<= 1)
        for (int stride = size >> 1; stride > 0; stride >>= 1) {
            for (int t = threadIdx.x; t < n2 / 2; t += kRefineThreads) {
                const int lo = 2 * t - (t & (stride - 1)), hi = lo + stride;
                const bool desc = (lo & size) == 0;
                const uint64_t a = keys[lo], b = keys[hi];
                if ((a < b) == desc) {
                    keys[lo] = b;
                    keys[hi] = a;
                }
            }
            __syncthreads();
        }
    for (int t = threadIdx.x; t < k; t += kRefineThreads) out[(int64_t)r * k + t] = t < n2 ? keys[t] : 0ull;
}

}  // namespace

cudaError_t launch_ivf_refine(const uint16_t *rows, int64_t N, int d, const uint16_t *regions, int R,
                              const uint64_t *cand, int ks, int k, uint64_t *out, cudaStream_t s) {
    if (R <= 0) return cudaSuccess;
    if (ks < 1 || ks > kRefineMax || k < 1 || k > ks || d % 8 != 0) return cudaErrorInvalidValue;
    k_ivf_refine<<<R, kRefineThreads, (size_t)d * sizeof(float), s>>>(rows, N, d, regions, cand, ks, k, out);
    return cudaGetLastError();
}

cudaError_t ivfpq_scan_split(int M, int nprobe, int R, int sms, int requested, int *G) {
    if (requested > 0) {
        *G = requested;
        return cudaSuccess;
    }
    int slots = 0;
    cudaError_t e;
    switch (ivf_padded_m(M) / 32) {
    case 1: e = scan_slots<1>(M, nprobe, sms, &slots); break;
    case 2: e = scan_slots<2>(M, nprobe, sms, &slots); break;
    case 3: e = scan_slots<3>(M, nprobe, sms, &slots); break;
    case 4: e = scan_slots<4>(M, nprobe, sms, &slots); break;
    default: return cudaErrorInvalidValue;
    }
    if (e != cudaSuccess) return e;
    // Each part rebuilds its region's lookup table and warms up its own
    // threshold, which costs more than an uneven last wave saves: split only
    // while the items would not fill half the resident CTAs.
    int g = 1;
    while (g < kIvfMaxSplit / 2 && (int64_t)R * g * 2 <= slots) g *= 2;
    *G = g;
    return cudaSuccess;
}

cudaError_t launch_ivfpq_scan(const IvfParams &p, const uint16_t *regions, int R, const int64_t *probe_ids,
                              const float *probe_scores, int nprobe, int k, int G, uint64_t *out_keys, int sms,
                              cudaStream_t s) {
    if (R == 0) return cudaSuccess;
    if (G < 1 || G > kIvfMaxSplit) return cudaErrorInvalidValue;
    switch (ivf_padded_m(p.M) / 32) {
    case 1: return launch_scan_np<1>(p, regions, R, probe_ids, probe_scores, nprobe, k, G, out_keys, sms, s);
    case 2: return launch_scan_np<2>(p, regions, R, probe_ids, probe_scores, nprobe, k, G, out_keys, sms, s);
    case 3: return launch_scan_np<3>(p, regions, R, probe_ids, probe_scores, nprobe, k, G, out_keys, sms, s);
    case 4: return launch_scan_np<4>(p, regions, R, probe_ids, probe_scores, nprobe, k, G, out_keys, sms, s);
    default: return cudaErrorInvalidValue;
    }
}

}  // namespace skipk
