// Cross-partition merge (per region) and region-to-question merge with
// deduplication (per question).
//
// Per region (paper App. B.2 Def. B.2, MIPS(q_r, D; k_r)): the score kernels
// leave, for every region row, one sorted top-k list per corpus partition
// they scanned.  The exact top-k over the whole corpus is the top-k of the
// union of those lists, because every member of the global top-k is a
// member of its own partition's top-k.  One warp merges one row.
//
// Per question (§3.3 "deduplicate the union of K_r"; Def. B.2
// K = Dedup(union_i K_{r_i}); Alg. 1 Dedup step): the lists of the question's
// regions are pooled, each id keeps its maximum score, and the first K by
// (score desc, id asc) are written, padded with (-1, -inf).  One block per
// question.  The pool is sorted by (id asc, score desc) so that the first
// entry of every id run carries the id's maximum; those entries are then
// sorted by the ranking key.  When a question's pool exceeds the shared
// memory capacity, regions are folded in chunks: the running top-K already
// holds every id's best score that can still reach the output, since an id
// that fell below the running K-th score can only return with a larger one.
#include "skip_device.cuh"
#include "skip_internal.h"

namespace skipk {
namespace {

constexpr int kMergeWarps = 4;

template <int LPL>
__global__ void __launch_bounds__(kMergeWarps * 32)
    k_merge_lists(const uint64_t *__restrict__ lists, int G, int64_t g_stride, int len, int R, int k,
                  uint64_t *__restrict__ reg_keys, int64_t *__restrict__ reg_ids,
                  float *__restrict__ reg_scores, uint32_t *__restrict__ tau) {
    grid_dep_wait();
    grid_dep_launch();
    const int warp = threadIdx.x >> 5;
    const int row = blockIdx.x * kMergeWarps + warp;
    if (row >= R) return;
    const uint64_t *base = lists + (int64_t)row * len;
    uint64_t *kout = reg_keys ? reg_keys + (int64_t)row * k : nullptr;
    int64_t *iout = reg_ids ? reg_ids + (int64_t)row * k : nullptr;
    float *sout = reg_scores ? reg_scores + (int64_t)row * k : nullptr;
    warp_merge_topk<LPL>(base, g_stride, G, len, k, [&](int i, uint64_t key) {
        if (kout) kout[i] = key;
        // the k-th key's upper 32 bits are the order-preserving integer of its score
        if (tau && i == k - 1 && key != 0ull) atomicMax(tau + row, (uint32_t)(key >> 32));
        if (iout) {
            int64_t id;
            float s;
            key_decode(key, id, s);
            iout[i] = id;
            sout[i] = s;
        }
    });
}

constexpr int kQThreads = 512;
constexpr int kQCap = 4096;  // pooled candidates per pass (32 KB per array)
constexpr uint64_t kNone = ~0ull;

// Block-wide bitonic sort of s[0..n2) (n2 a power of two), ascending.
// One bitonic compare-exchange between lanes pos and pos ^ j of a warp's
// 32-key run (j < 32), blocks of `size` keys alternately ascending and
// descending.
__device__ __forceinline__ uint64_t bitonic_lane_step_asc(uint64_t v, int pos, int j, int size) {
    const uint64_t o = __shfl_xor_sync(0xFFFFFFFFu, v, j);
    const bool up = (pos & size) == 0;
    const bool lower = (pos & j) == 0;
    return lower == up ? (v < o ? v : o) : (v > o ? v : o);
}

// Sorts s[0, n2) ascending (n2 a power of two).  Strides of 32 and more go
// through shared memory with a block barrier each; the strides below 32 of
// every stage run inside warps on registers (one 32-key run per warp at a
// time): of the 45 stages of a 512-key sort, 15 need a block barrier.
__device__ void block_bitonic_sort_asc(uint64_t *s, int n2) {
    auto smem_stage = [&](int size, int stride) {
        for (int i = threadIdx.x; i < (n2 >> 1); i += blockDim.x) {
            const int lo = 2 * i - (i & (stride - 1));
            const int hi = lo + stride;
            const bool up = (lo & size) == 0;
            const uint64_t a = s[lo], b = s[hi];
            if ((a > b) == up) {
                s[lo] = b;
                s[hi] = a;
            }
        }
    };
    if (n2 < 64) {
        for (int size = 2; size <= n2; size <<= 1)
            for (int stride = size >> 1; stride > 0; stride >>= 1) {
                __syncthreads();
                smem_stage(size, stride);
            }
        __syncthreads();
        return;
    }
    const int lane = threadIdx.x & 31;
    __syncthreads();
    // sizes 2 .. 32: whole 32-key runs in registers
    for (int base = threadIdx.x & ~31; base < n2; base += blockDim.x) {
        const int pos = base + lane;
        uint64_t v = s[pos];
        for (int size = 2; size <= 32; size <<= 1)
            for (int j = size >> 1; j > 0; j >>= 1) v = bitonic_lane_step_asc(v, pos, j, size);
        s[pos] = v;
    }
    for (int size = 64; size <= n2; size <<= 1) {
        for (int stride = size >> 1; stride >= 32; stride >>= 1) {
            __syncthreads();
            smem_stage(size, stride);
        }
        __syncthreads();
        for (int base = threadIdx.x & ~31; base < n2; base += blockDim.x) {
            const int pos = base + lane;
            uint64_t v = s[pos];
            for (int j = 16; j > 0; j >>= 1) v = bitonic_lane_step_asc(v, pos, j, size);
            s[pos] = v;
        }
    }
    __syncthreads();
}

__device__ __forceinline__ int pow2_at_least(int n) {
    int p = 1;
    while (p < n) p <<= 1;
    return p;
}

// (id asc, score desc) ordering key of a ranking key; empty slots sort last.
__device__ __forceinline__ uint64_t id_major(uint64_t key) {
    if (key == 0) return kNone;
    const uint64_t id = (uint64_t)key_id(key);
    const uint32_t ord = (uint32_t)(key >> 32);
    return (id << 32) | (uint64_t)(0xFFFFFFFFu - ord);
}

__device__ __forceinline__ uint64_t rank_of_id_major(uint64_t im) {
    const uint32_t id = (uint32_t)(im >> 32);
    const uint32_t ord = 0xFFFFFFFFu - (uint32_t)im;
    return ((uint64_t)ord << 32) | (uint64_t)(0xFFFFFFFFu - id);
}

__global__ void __launch_bounds__(kQThreads)
    k_question_merge(const uint64_t *__restrict__ reg_keys, int k, const int32_t *__restrict__ offsets,
                     int R, int K, int64_t *__restrict__ out_ids, float *__restrict__ out_scores,
                     int *__restrict__ err) {
    extern __shared__ uint64_t qsmem[];
    grid_dep_wait();
    grid_dep_launch();
    uint64_t *pool = qsmem;            // [kQCap] id-major keys
    uint64_t *ranked = qsmem + kQCap;  // [kQCap] ranking keys, negated for the ascending sort
    __shared__ int s_kept;
    const int q = blockIdx.x;
    // Offsets outside [0, R] or decreasing are clamped (and flagged) so that
    // no read leaves the region lists.
    const int o0 = offsets[q], o1 = offsets[q + 1];
    const int r0 = min(max(o0, 0), R);
    const int r1 = min(max(o1, r0), R);
    if ((r0 != o0 || r1 != o1) && threadIdx.x == 0) atomicOr(err, kErrConfig);
    int nrun = 0;  // running top-K, kept as ranking keys in ranked[0..nrun) (descending)
    int r = r0;
    do {
        const int nreg = min(r1 - r, (kQCap - nrun) / k);
        const int n = nrun + nreg * k;
        for (int i = threadIdx.x; i < nrun; i += blockDim.x) pool[i] = id_major(ranked[i]);
        for (int i = threadIdx.x; i < nreg * k; i += blockDim.x)
            pool[nrun + i] = id_major(reg_keys[(int64_t)r * k + i]);
        const int n2 = pow2_at_least(n > 1 ? n : 1);
        for (int i = n + threadIdx.x; i < n2; i += blockDim.x) pool[i] = kNone;
        if (threadIdx.x == 0) s_kept = 0;
        block_bitonic_sort_asc(pool, n2);
        // First entry of every id run = that id with its maximum score.
        for (int i = threadIdx.x; i < n; i += blockDim.x) {
            const uint64_t v = pool[i];
            if (v == kNone) continue;
            if (i > 0 && (pool[i - 1] >> 32) == (v >> 32)) continue;
            const int at = atomicAdd(&s_kept, 1);
            ranked[at] = ~rank_of_id_major(v);  // ascending sort of ~key = descending by key
        }
        __syncthreads();
        const int m = s_kept;
        const int m2 = pow2_at_least(m > 1 ? m : 1);
        for (int i = m + threadIdx.x; i < m2; i += blockDim.x) ranked[i] = kNone;
        block_bitonic_sort_asc(ranked, m2);
        nrun = min(m, K);
        for (int i = threadIdx.x; i < nrun; i += blockDim.x) ranked[i] = ~ranked[i];
        __syncthreads();
        r += nreg;
    } while (r < r1);

    for (int i = threadIdx.x; i < K; i += blockDim.x) {
        int64_t id = -1;
        float s = -__int_as_float(0x7f800000);
        if (i < nrun) key_decode(ranked[i], id, s);
        out_ids[(int64_t)q * K + i] = id;
        out_scores[(int64_t)q * K + i] = s;
    }
}

// Both merges in one launch, for batches whose questions' pooled region
// lists fit in shared memory (R k <= kQCap): one block per question; its
// warps merge the question's region rows (k-way over the G partition
// lists, as k_merge_lists) straight into the block's pool, then the block
// deduplicates and ranks the pool as k_question_merge does.  One launch
// and one hand-off fewer for the small batches.
template <int LPL>
__global__ void __launch_bounds__(kQThreads)
    k_merge_regions_questions(const uint64_t *__restrict__ lists, int G, int64_t g_stride, int k,
                              const int32_t *__restrict__ offsets, int R, int K, int64_t *__restrict__ out_ids,
                              float *__restrict__ out_scores, int *__restrict__ err) {
    extern __shared__ uint64_t qsmem[];
    grid_dep_wait();
    grid_dep_launch();
    uint64_t *pool = qsmem;            // [kQCap] id-major keys
    uint64_t *ranked = qsmem + kQCap;  // [kQCap] ranking keys, negated for the ascending sort
    __shared__ int s_kept;
    const int q = blockIdx.x;
    const int warp = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
    const int o0 = offsets[q], o1 = offsets[q + 1];
    const int r0 = min(max(o0, 0), R);
    const int r1 = min(max(o1, r0), R);
    if ((r0 != o0 || r1 != o1) && threadIdx.x == 0) atomicOr(err, kErrConfig);
    const int nreg = r1 - r0, n = nreg * k;  // n <= R k <= kQCap (checked at launch)
    for (int j = warp; j < nreg; j += nwarps)
        warp_merge_topk<LPL>(lists + (int64_t)(r0 + j) * k, g_stride, G, k, k,
                             [&](int i, uint64_t key) { pool[j * k + i] = id_major(key); });
    const int n2 = pow2_at_least(n > 1 ? n : 1);
    for (int i = n + threadIdx.x; i < n2; i += blockDim.x) pool[i] = kNone;
    if (threadIdx.x == 0) s_kept = 0;
    block_bitonic_sort_asc(pool, n2);  // starts with a block barrier
    // First entry of every id run = that id with its maximum score.
    for (int i = threadIdx.x; i < n; i += blockDim.x) {
        const uint64_t v = pool[i];
        if (v == kNone) continue;
        if (i > 0 && (pool[i - 1] >> 32) == (v >> 32)) continue;
        const int at = atomicAdd(&s_kept, 1);
        ranked[at] = ~rank_of_id_major(v);
    }
    __syncthreads();
    const int m = s_kept;
    const int m2 = pow2_at_least(m > 1 ? m : 1);
    for (int i = m + threadIdx.x; i < m2; i += blockDim.x) ranked[i] = kNone;
    block_bitonic_sort_asc(ranked, m2);
    const int nrun = min(m, K);
    for (int i = threadIdx.x; i < K; i += blockDim.x) {
        int64_t id = -1;
        float sc = -__int_as_float(0x7f800000);
        if (i < nrun) key_decode(~ranked[i], id, sc);
        out_ids[(int64_t)q * K + i] = id;
        out_scores[(int64_t)q * K + i] = sc;
    }
}

}  // namespace


cudaError_t launch_merge_lists_len(const uint64_t *lists, int G, int64_t g_stride, int len, int R, int k,
                                   uint64_t *reg_keys, int64_t *reg_ids, float *reg_scores, uint32_t *tau,
                                   cudaStream_t s, bool pdl) {
    if (R <= 0) return cudaSuccess;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)((R + kMergeWarps - 1) / kMergeWarps), 1, 1);
    cfg.blockDim = dim3(kMergeWarps * 32, 1, 1);
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl ? 1 : 0;
    if (G <= 32)
        return cudaLaunchKernelEx(&cfg, k_merge_lists<1>, lists, G, g_stride, len, R, k, reg_keys, reg_ids,
                                  reg_scores, tau);
    if (G <= 64)
        return cudaLaunchKernelEx(&cfg, k_merge_lists<2>, lists, G, g_stride, len, R, k, reg_keys, reg_ids,
                                  reg_scores, tau);
    if (G <= 128)
        return cudaLaunchKernelEx(&cfg, k_merge_lists<4>, lists, G, g_stride, len, R, k, reg_keys, reg_ids,
                                  reg_scores, tau);
    if (G <= 256)
        return cudaLaunchKernelEx(&cfg, k_merge_lists<8>, lists, G, g_stride, len, R, k, reg_keys, reg_ids,
                                  reg_scores, tau);
    if (G <= 512)
        return cudaLaunchKernelEx(&cfg, k_merge_lists<16>, lists, G, g_stride, len, R, k, reg_keys, reg_ids,
                                  reg_scores, tau);
    return cudaErrorInvalidValue;
}

cudaError_t launch_merge_lists(const uint64_t *lists, int G, int64_t g_stride, int R, int k,
                               uint64_t *reg_keys, int64_t *reg_ids, float *reg_scores,
                               cudaStream_t s, bool pdl) {
    return launch_merge_lists_len(lists, G, g_stride, k, R, k, reg_keys, reg_ids, reg_scores, nullptr, s, pdl);
}

int question_merge_capacity() { return kQCap; }

cudaError_t launch_merge_regions_questions(const uint64_t *lists, int G, int64_t g_stride, int R, int k,
                                           const int32_t *offsets, int Q, int K, int64_t *out_ids,
                                           float *out_scores, int *err, cudaStream_t s, bool pdl) {
    if (Q <= 0) return cudaSuccess;
    if ((int64_t)R * k > kQCap || K > kQCap || G > 512) return cudaErrorInvalidValue;
    const int smem = 2 * kQCap * (int)sizeof(uint64_t);
    auto kern = G <= 32 ? k_merge_regions_questions<1> : G <= 64 ? k_merge_regions_questions<2>
              : G <= 128 ? k_merge_regions_questions<4> : G <= 256 ? k_merge_regions_questions<8>
                         : k_merge_regions_questions<16>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)Q, 1, 1);
    cfg.blockDim = dim3(kQThreads, 1, 1);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl ? 1 : 0;
    return cudaLaunchKernelEx(&cfg, kern, lists, G, g_stride, k, offsets, R, K, out_ids, out_scores, err);
}

cudaError_t launch_question_merge(const uint64_t *reg_keys, int k, const int32_t *offsets, int Q,
                                  int R, int K, int64_t *out_ids, float *out_scores, int *err,
                                  cudaStream_t s, bool pdl) {
    if (Q <= 0) return cudaSuccess;
    if (K + k > kQCap) return cudaErrorInvalidValue;
    const int smem = 2 * kQCap * (int)sizeof(uint64_t);
    cudaError_t e = cudaFuncSetAttribute(k_question_merge, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)Q, 1, 1);
    cfg.blockDim = dim3(kQThreads, 1, 1);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl ? 1 : 0;
    return cudaLaunchKernelEx(&cfg, k_question_merge, reg_keys, k, offsets, R, K, out_ids, out_scores, err);
}

}  // namespace skipk
