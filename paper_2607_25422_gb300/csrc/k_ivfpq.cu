// IVF-PQ approximate variant of the per-region search (the index of §4.1
// "Implementation" / App. I.4: inverted lists over inner-product centroids,
// product-quantised residual codes, asymmetric scoring).
//
// Build (after the coarse assignment, which runs on the exact MIPS path with
// the centroids as the corpus and the corpus rows as queries, k = 1):
//   k_pq_encode     residual x - c_list, nearest of 256 codewords per
//                   sub-space (fp32, ties to the lower codeword); a block of
//                   128 rows shares each sub-space's codebook in shared memory.
//   k_ivf_count / k_ivf_offsets / k_ivf_scatter
//                   counting sort of the rows into their lists (order inside
//                   a list is arbitrary: the search breaks ties by id).
// Search (after the coarse top-nprobe, again on the exact MIPS path):
//   k_ivfpq_scan    one region per CTA at a time: the region's lookup table
//                   T[m][j] = <q_m, p_{m,j}> in shared memory, then every code
//                   of its probed lists scored as <q, c_l> + sum_m T[m][code_m];
//                   candidates above the running k-th key go to a shared
//                   buffer that is sorted and cut back to k when it fills.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <algorithm>

#include "skip_device.cuh"
#include "skip_internal.h"

namespace skipk {
namespace {

// ---------------------------------------------------------------- encode

constexpr int kEncRows = 128;

__global__ void __launch_bounds__(kEncRows) k_pq_encode(const IvfParams p, const int64_t *row_list,
                                                         uint8_t *codes) {
    extern __shared__ float cbs[];  // [256][ds] codebook of one sub-space
    const int64_t i = (int64_t)blockIdx.x * kEncRows + threadIdx.x;
    const bool valid = i < p.N;
    const int ds = p.ds;
    int64_t l = valid ? row_list[i] : 0;
    if (l < 0 || l >= p.C) l = 0;  // flagged by k_ivf_count
    const __nv_bfloat16 *x = reinterpret_cast<const __nv_bfloat16 *>(p.rows) + (valid ? i : 0) * (int64_t)p.d;
    const __nv_bfloat16 *c = reinterpret_cast<const __nv_bfloat16 *>(p.centroids) + l * (int64_t)p.d;
    for (int m = 0; m < p.M; ++m) {
        __syncthreads();
        for (int e = threadIdx.x; e < 256 * ds; e += kEncRows) cbs[e] = p.codebook[(int64_t)m * 256 * ds + e];
        __syncthreads();
        float r[kIvfMaxDs];
#pragma unroll
        for (int t = 0; t < kIvfMaxDs; ++t)
            r[t] = t < ds ? __bfloat162float(x[m * ds + t]) - __bfloat162float(c[m * ds + t]) : 0.f;
        int best = 0;
        float bd = __int_as_float(0x7f800000);
        for (int j = 0; j < 256; ++j) {
            const float *pj = cbs + j * ds;
            float dist = 0.f;
#pragma unroll
            for (int t = 0; t < kIvfMaxDs; ++t) {
                if (t < ds) {
                    const float e = r[t] - pj[t];
                    dist = fmaf(e, e, dist);
                }
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

// ---------------------------------------------------------------- search

constexpr int kScanThreads = 256;
constexpr int kCandBuf = 2048;

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

__global__ void __launch_bounds__(kScanThreads) k_ivfpq_scan(const IvfParams p, const uint16_t *regions, int R,
                                                             const int64_t *probe_ids, const float *probe_scores,
                                                             int nprobe, int k, uint64_t *out_keys) {
    extern __shared__ __align__(16) uint8_t sm[];
    float *T = reinterpret_cast<float *>(sm);                       // [M][256]
    uint64_t *cand = reinterpret_cast<uint64_t *>(T + p.M * 256);   // [kCandBuf]
    int64_t *pref = reinterpret_cast<int64_t *>(cand + kCandBuf);   // [nprobe + 1]
    int64_t *pstart = pref + (nprobe + 1);                          // [nprobe] list start
    float *pscore = reinterpret_cast<float *>(pstart + nprobe);     // [nprobe]
    float *qf = pscore + nprobe;                                    // [d]
    __shared__ int cnt;
    __shared__ uint64_t tau;
    const int ds = p.ds;
    for (int r = blockIdx.x; r < R; r += gridDim.x) {
        // query, probes and the prefix of their list lengths
        for (int t = threadIdx.x; t < p.d; t += kScanThreads)
            qf[t] = __bfloat162float(reinterpret_cast<const __nv_bfloat16 *>(regions)[(int64_t)r * p.d + t]);
        for (int t = threadIdx.x; t < nprobe; t += kScanThreads) {
            const int64_t l = probe_ids[(int64_t)r * nprobe + t];
            const bool ok = l >= 0 && l < p.C;
            pstart[t] = ok ? p.offsets[l] : 0;
            pref[t + 1] = ok ? p.offsets[l + 1] - p.offsets[l] : 0;
            pscore[t] = probe_scores[(int64_t)r * nprobe + t];
        }
        if (threadIdx.x == 0) {
            pref[0] = 0;
            cnt = 0;
            tau = 0;
        }
        __syncthreads();
        if (threadIdx.x < 32) {  // inclusive scan of pref[1..nprobe], one warp
            int64_t carry = 0;
            for (int b = 0; b < nprobe; b += 32) {
                const int t = b + (int)threadIdx.x;
                int64_t v = t < nprobe ? pref[t + 1] : 0;
#pragma unroll
                for (int o = 1; o < 32; o <<= 1) {
                    const int64_t u = __shfl_up_sync(0xFFFFFFFFu, v, o);
                    if ((int)threadIdx.x >= o) v += u;
                }
                if (t < nprobe) pref[t + 1] = v + carry;
                carry += __shfl_sync(0xFFFFFFFFu, v, 31);
            }
        }
        // lookup table
        for (int e = threadIdx.x; e < p.M * 256; e += kScanThreads) {
            const int m = e >> 8;
            const float *pj = p.codebook + (int64_t)e * ds;
            const float *qm = qf + m * ds;
            float s = 0.f;
            for (int t = 0; t < ds; ++t) s = fmaf(qm[t], pj[t], s);
            T[e] = s;
        }
        __syncthreads();
        const int64_t total = pref[nprobe];
        for (int64_t base = 0; base < total; base += kScanThreads) {
            const int64_t v = base + threadIdx.x;
            if (v < total) {
                int lo = 0, hi = nprobe - 1;  // the probe holding slot v: pref[pi] <= v < pref[pi + 1]
                while (lo < hi) {
                    const int mid = (lo + hi + 1) >> 1;
                    if (pref[mid] <= v) lo = mid;
                    else hi = mid - 1;
                }
                const int64_t e = pstart[lo] + (v - pref[lo]);
                const uint4 *code = reinterpret_cast<const uint4 *>(p.codes + e * p.M);
                // four independent sums (one per 32-bit word of a 16-byte chunk)
                float acc[4] = {0.f, 0.f, 0.f, 0.f};
                for (int w = 0; w < p.M / 16; ++w) {
                    const uint4 cw = __ldg(code + w);
                    const uint32_t ws[4] = {cw.x, cw.y, cw.z, cw.w};
#pragma unroll
                    for (int h = 0; h < 4; ++h)
#pragma unroll
                        for (int b = 0; b < 4; ++b)
                            acc[h] += T[((w * 16 + h * 4 + b) << 8) + ((ws[h] >> (8 * b)) & 0xFFu)];
                }
                const float s = pscore[lo] + ((acc[0] + acc[1]) + (acc[2] + acc[3]));
                const uint64_t key = make_key(s, (uint32_t)p.ids[e]);
                if (key > tau) {
                    const int pos = atomicAdd(&cnt, 1);
                    cand[pos] = key;  // pos < kCandBuf: at most kScanThreads are added per round
                }
            }
            __syncthreads();
            if (cnt > kCandBuf - kScanThreads) {
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
        for (int t = threadIdx.x; t < k; t += kScanThreads) out_keys[(int64_t)r * k + t] = cand[t];
        __syncthreads();
    }
}

}  // namespace

cudaError_t launch_pq_encode(const IvfParams &p, const int64_t *row_list, uint8_t *codes, cudaStream_t s) {
    if (p.N == 0) return cudaSuccess;
    const size_t smem = (size_t)256 * p.ds * sizeof(float);
    k_pq_encode<<<(unsigned)((p.N + kEncRows - 1) / kEncRows), kEncRows, smem, s>>>(p, row_list, codes);
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

size_t ivfpq_scan_smem(int M, int d, int nprobe) {
    return (size_t)M * 256 * 4 + (size_t)kCandBuf * 8 + (size_t)(2 * nprobe + 1) * 8 + (size_t)nprobe * 4 +
           (size_t)d * 4 + 16;
}

cudaError_t launch_ivfpq_scan(const IvfParams &p, const uint16_t *regions, int R, const int64_t *probe_ids,
                              const float *probe_scores, int nprobe, int k, uint64_t *out_keys, int sms,
                              cudaStream_t s) {
    if (R == 0) return cudaSuccess;
    const size_t smem = ivfpq_scan_smem(p.M, p.d, nprobe);
    cudaError_t e = cudaFuncSetAttribute(k_ivfpq_scan, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    int per_sm = 0;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k_ivfpq_scan, kScanThreads, smem);
    if (e != cudaSuccess) return e;
    const int grid = std::max(1, std::min(R, sms * std::max(per_sm, 1)));
    k_ivfpq_scan<<<grid, kScanThreads, smem, s>>>(p, regions, R, probe_ids, probe_scores, nprobe, k, out_keys);
    return cudaGetLastError();
}

}  // namespace skipk
