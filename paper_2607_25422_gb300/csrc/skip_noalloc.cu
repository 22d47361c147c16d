// Per-region retrieval for callers that must not allocate device memory.
//
// Some callers cannot call cudaMalloc: code that runs inside a host
// application or framework that owns every device allocation (all memory
// must come from its pool, so a library that allocates on its own breaks
// the caller's memory accounting), and latency-critical serving loops that
// cannot afford the device-wide synchronisation that cudaMalloc/cudaFree
// may cause.  For them this entry point takes the corpus as a plain device
// pointer (no handle, whose creation copies and allocates) and keeps its
// scratch -- the per-warp and per-block candidate lists of the warp-dot
// score kernel, read back by the list merge kernel -- in one file-scope
// __device__ array of kNoAllocScratchBytes.  It calls no cudaMalloc,
// cudaFree or other allocating routine.
//
// The array exists once per device that loads this library and stays
// allocated until the process exits.  Host code cannot use the array's name
// as a device address, so the first call on each device looks the address
// up with cudaGetSymbolAddress (with that device current) and caches it;
// make that first call before any stream capture.  All calls on a device
// share the one array and it keeps the previous call's contents: the kernels
// write every slot they later read, so nothing needs clearing, but calls
// whose work overlaps on the GPU (different streams without ordering) race
// on the array.
#include <algorithm>
#include <mutex>

#include "../../include/skip_retrieve.h"
#include "skip_internal.h"

using namespace skipk;

namespace {

constexpr size_t kNoAllocScratchBytes = (size_t)16 << 20;  // 16 MiB per device
constexpr int kMaxDevices = 64;

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

std::mutex g_noalloc_mutex;
void *g_noalloc_ptr[kMaxDevices];  // device address of the array, per device

size_t round256(size_t v) { return (v + 255) / 256 * 256; }

bool aligned(const void *p, uintptr_t a) { return ((uintptr_t)p & (a - 1)) == 0; }

}  // namespace

extern "C" {

skip_status_t skip_retrieve_regions_noalloc(const void *corpus_rows, int64_t N, int32_t d,
                                            skip_dtype_t dtype, const float *row_scale,
                                            const void *regions, int32_t R_total, int32_t k_region,
                                            int64_t *reg_ids, float *reg_scores, void *stream) {
    if (!corpus_rows || N < 1 || N >= (1LL << 31) || d < 16 || d % 16 != 0 || d > 4096) return SKIP_EINVAL;
    if (dtype != SKIP_BF16 && dtype != SKIP_E4M3) return SKIP_EINVAL;
    if ((dtype == SKIP_E4M3) != (row_scale != nullptr)) return SKIP_EINVAL;
    if (R_total < 0 || k_region < 1 || k_region > SKIP_MAX_K_REGION || (int64_t)k_region > N) return SKIP_EINVAL;
    if (R_total > 0 && (!regions || !reg_ids || !reg_scores)) return SKIP_EINVAL;
    // The score kernel reads corpus rows as 16-byte vectors (d % 16 == 0 keeps
    // every row on that boundary once the first one is), the row scales as
    // fp32, the regions as 16-bit words; the merge writes int64 ids and fp32
    // scores.  A misaligned pointer is refused here, before any launch.
    if (!aligned(corpus_rows, 16) || (row_scale && !aligned(row_scale, 4))) return SKIP_EINVAL;
    if (R_total > 0 && (!aligned(regions, 2) || !aligned(reg_ids, 8) || !aligned(reg_scores, 4)))
        return SKIP_EINVAL;
    if (R_total == 0) return SKIP_OK;

    int dev = 0, major = 0, minor = 0, sms = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) {
        cudaGetLastError();
        return SKIP_EUNSUPPORTED;
    }
    cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
    cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (major != 10 || minor != 3 || dev >= kMaxDevices) return SKIP_EUNSUPPORTED;

    // Scratch: one list per (block, region row) and one per (warp, region of
    // the current group of eight); sizes beyond the array are rejected.
    // Blocks of the score kernel: one per SM, at most 512, and no more than
    // the corpus has 256-row slices (so small corpora need little scratch).
    const int grid = (int)std::max<int64_t>(1, std::min<int64_t>(std::min(sms, 512), (N + 255) / 256));
    const size_t lists_bytes = round256((size_t)grid * R_total * k_region * sizeof(uint64_t));
    const size_t wl_bytes = (size_t)grid * kWarpDotWarps * 8 * k_region * sizeof(uint64_t);
    if (lists_bytes + wl_bytes > kNoAllocScratchBytes) return SKIP_EUNSUPPORTED;

    void *base = nullptr;
    {
        std::lock_guard<std::mutex> lock(g_noalloc_mutex);
        if (!g_noalloc_ptr[dev]) {
            void *p = nullptr;
            if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || !p) {
                cudaGetLastError();
                return SKIP_ECUDA;
            }
            g_noalloc_ptr[dev] = p;
        }
        base = g_noalloc_ptr[dev];
    }
    uint64_t *lists = reinterpret_cast<uint64_t *>(base);
    uint64_t *wl = reinterpret_cast<uint64_t *>(reinterpret_cast<char *>(base) + lists_bytes);
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    const uint16_t *q = reinterpret_cast<const uint16_t *>(regions);
    for (int q0 = 0; q0 < R_total; q0 += 8) {
        WarpDotParams p;
        p.corpus = reinterpret_cast<const uint8_t *>(corpus_rows);
        p.scale = row_scale;
        p.N = N;
        p.d = d;
        p.regions = q + (size_t)q0 * d;
        p.nq = std::min(8, R_total - q0);
        p.k = k_region;
        p.warp_lists = wl;
        p.lists = lists;
        p.list_g_stride = (int64_t)R_total * k_region;
        p.q0 = q0;
        if (launch_warpdot(p, dtype == SKIP_E4M3, grid, s) != cudaSuccess) return SKIP_ECUDA;
    }
    if (launch_merge_lists(lists, grid, (int64_t)R_total * k_region, R_total, k_region, nullptr, reg_ids,
                           reg_scores, s) != cudaSuccess)
        return SKIP_ECUDA;
    return SKIP_OK;
}

}  // extern "C"
