// Pieces shared by the tensor-core score kernels (bf16 and e4m3 corpora):
// the work item of a persistent CTA, the per-row top-k set kept by the
// epilogue, and register helpers for the 32-column chunks it scans.
#pragma once

#include "skip_device.cuh"
#include "skip_internal.h"

namespace skipk {
namespace tc {

struct Item {
    int mb;
    int g;
    int64_t t0, t1;
};

__device__ __forceinline__ Item item_of(const TcParams &p, int v, int rank) {
    Item it;
    it.g = v / p.QG;
    it.mb = (v - it.g * p.QG) * p.CL + rank;
    it.t0 = (int64_t)it.g * p.tiles / p.G;
    it.t1 = (int64_t)(it.g + 1) * p.tiles / p.G;
    return it;
}

// A row's running top-k is an unsorted set of up to k keys (slot t at
// L[t * ls]) plus the slot of its smallest key.  A key that beats the
// smallest replaces it and the smallest is found again with k independent
// loads, which overlap, instead of a shift loop whose loads depend on each
// other.  The set is sorted once, when the chunk is done.
struct RowTopK {
    int n = 0;          // keys held
    int min_slot = 0;   // slot of the smallest key once n == k
    uint64_t min_key = 0;
};

__device__ __forceinline__ void topk_rescan(uint64_t *L, int ls, int k, RowTopK &st) {
    // Four independent running minima, combined at the end: the compare
    // chain is k/4 deep instead of k.  Keys are distinct, so the slot found
    // does not depend on the order of the compares.
    uint64_t m0 = ~0ull, m1 = ~0ull, m2 = ~0ull, m3 = ~0ull;
    int s0 = 0, s1 = 0, s2 = 0, s3 = 0;
    int t = 0;
#pragma unroll 2
    for (; t + 4 <= k; t += 4) {
        const uint64_t x0 = L[t * ls], x1 = L[(t + 1) * ls], x2 = L[(t + 2) * ls], x3 = L[(t + 3) * ls];
        if (x0 < m0) { m0 = x0; s0 = t; }
        if (x1 < m1) { m1 = x1; s1 = t + 1; }
        if (x2 < m2) { m2 = x2; s2 = t + 2; }
        if (x3 < m3) { m3 = x3; s3 = t + 3; }
    }
    for (; t < k; ++t) {
        const uint64_t x = L[t * ls];
        if (x < m0) { m0 = x; s0 = t; }
    }
    if (m1 < m0) { m0 = m1; s0 = s1; }
    if (m3 < m2) { m2 = m3; s2 = s3; }
    if (m2 < m0) { m0 = m2; s0 = s2; }
    st.min_key = m0;
    st.min_slot = s0;
}

// The same over a contiguous set in global memory (slot t at L[t], k even,
// L 16-byte aligned): 16 keys per batch as eight 16-byte loads, two batches
// in flight, so a rescan costs a few round trips to L2 instead of one per
// eight keys.
__device__ __forceinline__ void topk_rescan_contig(const uint64_t *L, int k, RowTopK &st) {
    uint64_t m0 = ~0ull, m1 = ~0ull;
    int s0 = 0, s1 = 0;
    const ulonglong2 *V = reinterpret_cast<const ulonglong2 *>(L);
    const int pairs = k >> 1;
    int t = 0;
#pragma unroll 2
    for (; t + 8 <= pairs; t += 8) {
        ulonglong2 x[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) x[u] = V[t + u];
#pragma unroll
        for (int u = 0; u < 8; ++u) {
            if (x[u].x < m0) { m0 = x[u].x; s0 = 2 * (t + u); }
            if (x[u].y < m1) { m1 = x[u].y; s1 = 2 * (t + u) + 1; }
        }
    }
    for (; t < pairs; ++t) {
        const ulonglong2 x = V[t];
        if (x.x < m0) { m0 = x.x; s0 = 2 * t; }
        if (x.y < m1) { m1 = x.y; s1 = 2 * t + 1; }
    }
    if (m1 < m0) { m0 = m1; s0 = s1; }
    st.min_key = m0;
    st.min_slot = s0;
}

// The caller has checked that key beats the smallest key (or n < k).
__device__ __forceinline__ void topk_add(uint64_t *L, int ls, int k, RowTopK &st, uint64_t key) {
    const bool contig = ls == 1 && (k & 1) == 0 && ((uintptr_t)L & 15) == 0;
    if (st.n < k) {
        L[st.n * ls] = key;
        if (++st.n == k) {
            if (contig)
                topk_rescan_contig(L, k, st);
            else
                topk_rescan(L, ls, k, st);
        }
    } else {
        L[st.min_slot * ls] = key;
        if (contig)
            topk_rescan_contig(L, k, st);
        else
            topk_rescan(L, ls, k, st);
    }
}

// Sorts the held keys descending (insertion sort, once per chunk).
__device__ __forceinline__ void topk_sort(uint64_t *L, int ls, int n) {
    for (int i = 1; i < n; ++i) {
        const uint64_t x = L[i * ls];
        int j = i - 1;
        while (j >= 0 && L[j * ls] < x) {
            L[(j + 1) * ls] = L[j * ls];
            --j;
        }
        L[(j + 1) * ls] = x;
    }
}

// Sorts the first n <= W keys (W = 16 or 32) of a list in global memory
// descending, through registers (a bitonic network; empty slots are 0 and
// sort last).
template <int W>
__device__ __forceinline__ void sortw_desc_in_place(uint64_t *L, int n) {
    uint64_t r[W];
#pragma unroll
    for (int i = 0; i < W; ++i) r[i] = i < n ? L[i] : 0ull;
#pragma unroll
    for (int size = 2; size <= W; size <<= 1)
#pragma unroll
        for (int stride = size >> 1; stride > 0; stride >>= 1)
#pragma unroll
            for (int i = 0; i < W; ++i) {
                const int j = i ^ stride;
                if (j > i) {
                    const bool desc = (i & size) == 0;  // blocks alternate; the last stage is one block
                    const uint64_t a = r[i], b = r[j];
                    if ((a < b) == desc) {
                        r[i] = b;
                        r[j] = a;
                    }
                }
            }
#pragma unroll
    for (int i = 0; i < W; ++i)
        if (i < n) L[i] = r[i];
}

// The largest float below x (x itself for -inf): "s > below(x)" is "s >= x".
__device__ __forceinline__ float float_below(float x) {
    const uint32_t b = __float_as_uint(x);
    if (b == 0xFF800000u) return x;
    if ((b & 0x7FFFFFFFu) == 0u) return __uint_as_float(0x80000001u);
    return __uint_as_float((b & 0x80000000u) ? b + 1u : b - 1u);
}

// v[j] for a run-time j without indexing the register array (5 levels of
// selects), so that v stays in registers.
__device__ __forceinline__ uint32_t select32(const uint32_t (&v)[32], int j) {
    uint32_t a[16];
#pragma unroll
    for (int i = 0; i < 16; ++i) a[i] = (j & 16) ? v[i + 16] : v[i];
#pragma unroll
    for (int i = 0; i < 8; ++i) a[i] = (j & 8) ? a[i + 8] : a[i];
#pragma unroll
    for (int i = 0; i < 4; ++i) a[i] = (j & 4) ? a[i + 4] : a[i];
#pragma unroll
    for (int i = 0; i < 2; ++i) a[i] = (j & 2) ? a[i + 2] : a[i];
    return (j & 1) ? a[1] : a[0];
}

// Three-input maximum (one instruction on sm_100 and later).
__device__ __forceinline__ float fmax3f(float a, float b, float c) {
    float d;
    asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
    return d;
}

__device__ __forceinline__ float fmax32(const uint32_t (&v)[32]) {
    float m[11];
#pragma unroll
    for (int j = 0; j < 10; ++j)
        m[j] = fmax3f(__uint_as_float(v[j]), __uint_as_float(v[j + 10]), __uint_as_float(v[j + 20]));
    m[10] = fmaxf(__uint_as_float(v[30]), __uint_as_float(v[31]));
    const float a = fmax3f(m[0], m[1], m[2]), b = fmax3f(m[3], m[4], m[5]), c = fmax3f(m[6], m[7], m[8]);
    const float e = fmaxf(m[9], m[10]);
    return fmaxf(fmax3f(a, b, c), e);
}

}  // namespace tc
}  // namespace skipk
