// Tensor-core score + fused top-k for an e4m3 corpus (sm_103a).
//
// Step: per-region MIPS top-k (paper App. B.2 Def. B.2, MIPS(q_r, D; k_r);
// §3.3 Eq. rcsr) when the corpus rows are OCP e4m3 with one fp32 scale per
// row: s(r, i) = scale_i * sum_j q_rj * e4m3_ij.  The region queries stay
// bf16, and kind::f16 MMAs take both operands in one 16-bit type, so every
// e4m3 corpus tile is widened to bf16 in shared memory first; e4m3 values
// are exactly representable in bf16, so the widening loses nothing.  The
// row scale multiplies the fp32 accumulator in the epilogue, before the
// filter (scales differ from row to row).
//
// Pipelines: a raw ring of e4m3 slices (256 corpus rows x 128 elements, 128-
// byte swizzle, filled by TMA from one producer thread) that runs ahead to
// keep HBM busy -- this path is bound by corpus bytes -- and a ring of MMA
// operand stages (128 region rows x 64 and 256 corpus rows x 64, bf16, the
// region part by TMA from a second producer thread, the corpus part written
// by eight converter warps: cvt e4m3x2 -> f16x2, then an exact re-bias of the
// exponent to bf16).  Writes by the converter threads are made visible to
// the tensor core (async proxy) with fence.proxy.async before they arrive
// on the stage's barrier.
//
// Warps (480 threads): 0 region producer, 1 TMEM owner and MMA issuer,
// 2..5 epilogue (as in the bf16 kernel), 6 corpus producer, 7..14 converters.
// Single-CTA MMA (M = 128 region rows, N = 256 corpus rows).  Every wait is
// bounded; a wait that gives up sets the error word, and before exit each
// producer waits (at most a second) for its copies in flight and the MMA
// thread for its MMAs, so TMEM is freed with nothing outstanding.
#include "skip_device.cuh"
#include "skip_internal.h"
#include "tc_common.cuh"

namespace skipk {
namespace {

using namespace tc;

constexpr int kABytes = kTcTileM * kTcTileK * 2;  // 16 KB
constexpr int kBBytes = kTcTileN * kTcTileK * 2;  // 32 KB (bf16)
constexpr int kRawK = 128;                        // e4m3 elements per raw slice row
constexpr int kRawBytes = kTcTileN * kRawK;       // 32 KB
constexpr uint32_t kTmemCols = 512;
constexpr uint64_t kDrainTimeoutNs = 1000000000ull;
constexpr uint32_t kIdesc = idesc_bf16_f32(kTcTileM, kTcTileN);
constexpr int kMaxRing = 4;
constexpr int kThreads = 480;
constexpr int kConvWarp0 = 7;
constexpr int kConvWarps = 8;

struct __align__(8) Fp8Shared {
    uint64_t full[kMaxRing];    // operand stage ready: region TMA bytes + converter arrivals
    uint64_t empty[kMaxRing];   // operand stage consumed (tcgen05.commit)
    uint64_t rfull[kMaxRing];   // raw slice loaded (TMA bytes)
    uint64_t rempty[kMaxRing];  // raw slice read by every converter warp
    uint64_t tfull[2];
    uint64_t tempty[2];
    uint64_t drain;
    uint32_t tmem_base;
};

// Two e4m3 values that came out of cvt as f16x2 -> bf16x2.  Every e4m3 value
// is a normal f16 (or zero) whose mantissa has 3 significant bits, so moving
// the exponent from bias 15 to bias 127 is exact: bf16 = (f16 magnitude >> 3)
// + (112 << 7), zero stays zero, the sign is kept.
__device__ __forceinline__ uint32_t f16x2_to_bf16x2(uint32_t h) {
    const uint32_t mag = h & 0x7FFF7FFFu;
    const uint32_t b = ((mag >> 3) & 0x0FFF0FFFu) + 0x38003800u;
    const uint32_t nz = __vcmpne2(mag, 0u);
    return (b & nz) | (h & 0x80008000u);
}

__device__ __forceinline__ uint32_t e4m3x2_to_bf16x2(uint32_t pair16) {
    const __half2_raw h = __nv_cvt_fp8x2_to_halfraw2((__nv_fp8x2_storage_t)(pair16 & 0xFFFFu), __NV_E4M3);
    const uint32_t hv = (uint32_t)h.x | ((uint32_t)h.y << 16);
    return f16x2_to_bf16x2(hv);
}

// 16 e4m3 bytes (elements 0..15) -> lo = bf16 elements 0..7, hi = 8..15.
__device__ __forceinline__ void widen16(uint4 in, uint4 &lo, uint4 &hi) {
    lo.x = e4m3x2_to_bf16x2(in.x);
    lo.y = e4m3x2_to_bf16x2(in.x >> 16);
    lo.z = e4m3x2_to_bf16x2(in.y);
    lo.w = e4m3x2_to_bf16x2(in.y >> 16);
    hi.x = e4m3x2_to_bf16x2(in.z);
    hi.y = e4m3x2_to_bf16x2(in.z >> 16);
    hi.z = e4m3x2_to_bf16x2(in.w);
    hi.w = e4m3x2_to_bf16x2(in.w >> 16);
}

__device__ __forceinline__ uint4 lds128(uint32_t addr) {
    uint4 v;
    asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(addr));
    return v;
}

__device__ __forceinline__ void sts128(uint32_t addr, uint4 v) {
    asm volatile("st.shared.v4.u32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w)
                 : "memory");
}

__device__ __forceinline__ void fence_proxy_async_smem() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// Scores of columns id0 .. id0 + 31 times their rows' scales; columns past N
// become -inf.
__device__ __forceinline__ void scale32(uint32_t (&v)[32], const float *__restrict__ scale, int64_t id0,
                                        int64_t N) {
    if (id0 + 32 <= N) {
        const float4 *s4 = reinterpret_cast<const float4 *>(scale + id0);
#pragma unroll
        for (int q = 0; q < 8; ++q) {
            const float4 f = __ldg(s4 + q);
            v[4 * q + 0] = __float_as_uint(__uint_as_float(v[4 * q + 0]) * f.x);
            v[4 * q + 1] = __float_as_uint(__uint_as_float(v[4 * q + 1]) * f.y);
            v[4 * q + 2] = __float_as_uint(__uint_as_float(v[4 * q + 2]) * f.z);
            v[4 * q + 3] = __float_as_uint(__uint_as_float(v[4 * q + 3]) * f.w);
        }
    } else {
#pragma unroll
        for (int j = 0; j < 32; ++j)
            v[j] = id0 + j < N ? __float_as_uint(__uint_as_float(v[j]) * __ldg(scale + id0 + j)) : 0xFF800000u;
    }
}

__global__ void __launch_bounds__(kThreads, 1)
    k_tc_fp8_score_topk(const __grid_constant__ CUtensorMap tq, const __grid_constant__ CUtensorMap traw,
                        const TcParams p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    const int S = p.stages, RS = p.raw_stages;
    uint8_t *sA = smem;
    uint8_t *sB = sA + S * kABytes;
    uint8_t *sR = sB + S * kBBytes;
    uint64_t *slists = reinterpret_cast<uint64_t *>(sR + RS * kRawBytes);
    const size_t list_bytes = p.list_in_smem ? (size_t)kTcTileM * p.k * 8 : 0;
    Fp8Shared *sh = reinterpret_cast<Fp8Shared *>(reinterpret_cast<uint8_t *>(slists) + list_bytes);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int items = p.QG * p.G;
    const int KR = (p.d + kRawK - 1) / kRawK;  // raw slices per tile
    const int KB = 2 * KR;                     // operand slices per tile

    if (threadIdx.x == 0) {
        for (int s = 0; s < S; ++s) {
            mbar_init(smem_addr(&sh->full[s]), 1 + kConvWarps);
            mbar_init(smem_addr(&sh->empty[s]), 1);
        }
        for (int r = 0; r < RS; ++r) {
            mbar_init(smem_addr(&sh->rfull[r]), 1);
            mbar_init(smem_addr(&sh->rempty[r]), kConvWarps);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(smem_addr(&sh->tfull[b]), 1);
            mbar_init(smem_addr(&sh->tempty[b]), 4);
        }
        mbar_init(smem_addr(&sh->drain), 1);
        mbar_fence_init();
    }
    if (warp == 0 && lane == 0) {
        tma_prefetch_desc(&tq);
        tma_prefetch_desc(&traw);
    }
    if (warp == 1) {
        tmem_alloc(smem_addr(&sh->tmem_base), kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = sh->tmem_base;

    if (warp == 0) {
        // ------------------------------------------------ region (A) producer
        if (lane == 0) {
            int s = 0;
            uint32_t ph = 0;
            int64_t issued = 0;
            bool ok = true;
            for (int v = blockIdx.x; v < items && ok; v += gridDim.x) {
                const Item it = item_of(p, v, 0);
                for (int64_t t = it.t0; t < it.t1 && ok; ++t)
                    for (int kb = 0; kb < KB; ++kb) {
                        if (!mbar_wait(smem_addr(&sh->empty[s]), ph ^ 1u, p.timeout_ns)) {
                            ok = false;
                            break;
                        }
                        const uint32_t fb = smem_addr(&sh->full[s]);
                        mbar_arrive_expect_tx(fb, kABytes);
                        tma_load_2d(smem_addr(sA + s * kABytes), &tq, fb, kb * kTcTileK, it.mb * kTcTileM);
                        ++issued;
                        if (++s == S) {
                            s = 0;
                            ph ^= 1u;
                        }
                    }
            }
            if (!ok) atomicOr(p.err, kErrTimeout);
            for (int st = 0; st < S; ++st) {
                const int64_t uses = issued / S + (st < issued % S ? 1 : 0);
                if (uses && !mbar_wait(smem_addr(&sh->full[st]), (uint32_t)((uses - 1) & 1), kDrainTimeoutNs))
                    atomicOr(p.err, kErrTimeout);
            }
        }
    } else if (warp == 6) {
        // ------------------------------------------------ corpus (raw e4m3) producer
        if (lane == 0) {
            int r = 0;
            uint32_t rph = 0;
            int64_t issued = 0;
            bool ok = true;
            for (int v = blockIdx.x; v < items && ok; v += gridDim.x) {
                const Item it = item_of(p, v, 0);
                for (int64_t t = it.t0; t < it.t1 && ok; ++t)
                    for (int kr = 0; kr < KR; ++kr) {
                        if (!mbar_wait(smem_addr(&sh->rempty[r]), rph ^ 1u, p.timeout_ns)) {
                            ok = false;
                            break;
                        }
                        const uint32_t rb = smem_addr(&sh->rfull[r]);
                        mbar_arrive_expect_tx(rb, kRawBytes);
                        tma_load_2d(smem_addr(sR + r * kRawBytes), &traw, rb, kr * kRawK, (int)(t * kTcTileN));
                        ++issued;
                        if (++r == RS) {
                            r = 0;
                            rph ^= 1u;
                        }
                    }
            }
            if (!ok) atomicOr(p.err, kErrTimeout);
            for (int st = 0; st < RS; ++st) {
                const int64_t uses = issued / RS + (st < issued % RS ? 1 : 0);
                if (uses && !mbar_wait(smem_addr(&sh->rfull[st]), (uint32_t)((uses - 1) & 1), kDrainTimeoutNs))
                    atomicOr(p.err, kErrTimeout);
            }
        }
    } else if (warp >= kConvWarp0) {
        // ------------------------------------------------ converters
        // Warp cw widens rows [32 cw, 32 cw + 32) of every raw slice; in each
        // step lanes 8i..8i+7 take eight consecutive rows at one 16-byte
        // chunk, so the swizzled reads and writes hit eight different bank
        // groups.
        const int cw = warp - kConvWarp0;
        const int lrow = lane & 7, rc = lane >> 3;
        int s = 0, r = 0;
        uint32_t ph = 0, rph = 0;
        bool ok = true;
        for (int v = blockIdx.x; v < items && ok; v += gridDim.x) {
            const Item it = item_of(p, v, 0);
            for (int64_t t = it.t0; t < it.t1 && ok; ++t)
                for (int kr = 0; kr < KR && ok; ++kr) {
                    if (!mbar_wait(smem_addr(&sh->rfull[r]), rph, p.timeout_ns)) {
                        ok = false;
                        break;
                    }
                    const uint32_t raw = smem_addr(sR + r * kRawBytes);
                    for (int h = 0; h < 2; ++h) {
                        if (!mbar_wait(smem_addr(&sh->empty[s]), ph ^ 1u, p.timeout_ns)) {
                            ok = false;
                            break;
                        }
                        const uint32_t bt = smem_addr(sB + s * kBBytes);
#pragma unroll
                        for (int i = 0; i < 4; ++i) {
                            const int row = 32 * cw + 8 * i + lrow;
                            const int sw = row & 7;
                            const uint4 in = lds128(raw + row * 128 + (((4 * h + rc) ^ sw) << 4));
                            uint4 lo, hi;
                            widen16(in, lo, hi);
                            sts128(bt + row * 128 + (((2 * rc) ^ sw) << 4), lo);
                            sts128(bt + row * 128 + (((2 * rc + 1) ^ sw) << 4), hi);
                        }
                        fence_proxy_async_smem();
                        __syncwarp();
                        if (lane == 0) mbar_arrive(smem_addr(&sh->full[s]));
                        if (++s == S) {
                            s = 0;
                            ph ^= 1u;
                        }
                    }
                    if (!ok) break;
                    __syncwarp();
                    if (lane == 0) mbar_arrive(smem_addr(&sh->rempty[r]));
                    if (++r == RS) {
                        r = 0;
                        rph ^= 1u;
                    }
                }
        }
        if (!ok && lane == 0) atomicOr(p.err, kErrTimeout);
    } else if (warp == 1) {
        // ------------------------------------------------ MMA issuer
        if (lane == 0) {
            int s = 0;
            uint32_t ph = 0, lt = 0;
            bool ok = true;
            for (int v = blockIdx.x; v < items && ok; v += gridDim.x) {
                const Item it = item_of(p, v, 0);
                for (int64_t t = it.t0; t < it.t1 && ok; ++t, ++lt) {
                    const uint32_t buf = lt & 1u, use = lt >> 1;
                    if (!mbar_wait(smem_addr(&sh->tempty[buf]), (use & 1u) ^ 1u, p.timeout_ns)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t dt = tmem + buf * kTcTileN;
                    for (int kb = 0; kb < KB; ++kb) {
                        if (!mbar_wait(smem_addr(&sh->full[s]), ph, p.timeout_ns)) {
                            ok = false;
                            break;
                        }
                        tc_fence_after();
                        const uint64_t ad = smem_desc_k128(smem_addr(sA + s * kABytes));
                        const uint64_t bd = smem_desc_k128(smem_addr(sB + s * kBBytes));
#pragma unroll
                        for (int kk = 0; kk < kTcTileK / 16; ++kk)
                            tc_mma_f16(dt, ad + (uint64_t)(kk * 2), bd + (uint64_t)(kk * 2), kIdesc, (kb | kk) != 0);
                        tc_commit(smem_addr(&sh->empty[s]));
                        if (++s == S) {
                            s = 0;
                            ph ^= 1u;
                        }
                    }
                    if (!ok) break;
                    tc_commit(smem_addr(&sh->tfull[buf]));
                }
            }
            if (!ok) atomicOr(p.err, kErrTimeout);
            tc_commit(smem_addr(&sh->drain));
            if (!mbar_wait(smem_addr(&sh->drain), 0, kDrainTimeoutNs)) atomicOr(p.err, kErrTimeout);
        }
    } else {
        // ------------------------------------------------ epilogue (warps 2..5)
        const int sub = warp & 3;
        const int rib = sub * 32 + lane;
        const uint32_t lane_addr = (uint32_t)(sub * 32) << 16;
        const float kNegInf = -__int_as_float(0x7f800000);
        uint32_t lt = 0;
        bool ok = true;
        for (int v = blockIdx.x; v < items && ok; v += gridDim.x) {
            const Item it = item_of(p, v, 0);
            const int row = it.mb * kTcTileM + rib;
            const bool row_valid = it.mb < p.MB && row < p.R;
            uint64_t *glist = p.lists + ((int64_t)it.g * p.R_pad + row) * p.k;
            uint64_t *L = p.list_in_smem ? slists + rib : glist;
            const int ls = p.list_in_smem ? kTcTileM : 1;
            RowTopK top;
            float thr = kNegInf, gthr = kNegInf;
            uint32_t published = 0;
            uint32_t *tau = p.tau + row;
            // The shared threshold is read one tile ahead, off the critical path.
            uint32_t tau_next = row_valid ? *reinterpret_cast<volatile uint32_t *>(tau) : 0u;
            auto scan32 = [&](uint32_t (&vv)[32], uint32_t id0) {
                if (!row_valid) return;
                const float mx = fmax32(vv);
                if (!(mx > thr && mx >= gthr)) return;
                uint32_t m = 0;
#pragma unroll
                for (int j = 0; j < 32; ++j) {
                    const float sj = __uint_as_float(vv[j]);
                    m |= (sj > thr && sj >= gthr ? 1u : 0u) << j;
                }
                while (m) {
                    const int j = __ffs(m) - 1;
                    m &= m - 1;
                    const float sj = __uint_as_float(select32(vv, j));
                    if (sj > thr) {
                        topk_add(L, ls, p.k, top, make_key(sj, id0 + j));
                        if (top.n == p.k) thr = key_score(top.min_key);
                    }
                }
            };
            for (int64_t t = it.t0; t < it.t1; ++t, ++lt) {
                const uint32_t buf = lt & 1u, use = lt >> 1;
                if (!mbar_wait(smem_addr(&sh->tfull[buf]), use & 1u, p.timeout_ns)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                if (row_valid) {
                    const uint32_t mine = top.n == p.k ? ord_of_score(thr) : 0u;
                    if (mine > published) {
                        atomicMax(tau, mine);
                        published = mine;
                    }
                    if (tau_next > published) gthr = score_of_ord(tau_next);
                    tau_next = *reinterpret_cast<volatile uint32_t *>(tau);
                }
                const int64_t n0 = t * kTcTileN;
#pragma unroll 1
                for (int c = 0; c < kTcTileN / 64; ++c) {
                    uint32_t v0[32], v1[32];
                    const uint32_t taddr = tmem + lane_addr + buf * kTcTileN + c * 64;
                    tmem_ld_32x32b_x32(taddr, v0);
                    tmem_ld_32x32b_x32(taddr + 32, v1);
                    tmem_ld_wait(v0);
                    regs_after_wait(v1);
                    if (c == kTcTileN / 64 - 1) {
                        tc_fence_before();
                        __syncwarp();
                        if (lane == 0) mbar_arrive(smem_addr(&sh->tempty[buf]));
                    }
                    const int64_t id0 = n0 + c * 64;
                    if (row_valid) {
                        scale32(v0, p.scale, id0, p.N);
                        scale32(v1, p.scale, id0 + 32, p.N);
                    }
                    scan32(v0, (uint32_t)id0);
                    scan32(v1, (uint32_t)(id0 + 32));
                }
            }
            if (row_valid) {
                topk_sort(L, ls, top.n);
                for (int t = 0; t < p.k; ++t) glist[t] = t < top.n ? L[t * ls] : 0ull;
            }
        }
        if (!ok && lane == 0) atomicOr(p.err, kErrTimeout);
    }

    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 1) {
        __syncwarp();
        tmem_dealloc(tmem, kTmemCols);
    }
}

size_t smem_bytes(int stages, int raw_stages, int k, bool list_in_smem) {
    return 1024 + (size_t)stages * (kABytes + kBBytes) + (size_t)raw_stages * kRawBytes +
           (list_in_smem ? (size_t)kTcTileM * k * 8 : 0) + sizeof(Fp8Shared);
}

}  // namespace

void tc_fp8_pick_layout(int k, int max_smem, int *stages, int *raw_stages, bool *list_in_smem) {
    // Prefer the deepest raw ring (bytes in flight from HBM), then lists in
    // shared memory; two operand stages suffice because the converters, not
    // the tensor core, set the pace.
    for (int rs = 3; rs >= 2; --rs)
        if (smem_bytes(2, rs, k, true) <= (size_t)max_smem) {
            *stages = 2;
            *raw_stages = rs;
            *list_in_smem = true;
            return;
        }
    *stages = 2;
    *raw_stages = 3;
    *list_in_smem = false;
}

cudaError_t launch_tc_fp8(const CUtensorMap &tq, const CUtensorMap &traw, const TcParams &p, int grid,
                          cudaStream_t s) {
    const size_t smem = smem_bytes(p.stages, p.raw_stages, p.k, p.list_in_smem != 0);
    cudaError_t e = cudaFuncSetAttribute(k_tc_fp8_score_topk, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    k_tc_fp8_score_topk<<<grid, kThreads, smem, s>>>(tq, traw, p);
    return cudaGetLastError();
}

}  // namespace skipk
