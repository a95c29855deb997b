// frt_selftest.cu — unit probes of the building blocks the attention kernel relies on,
// exported for the GPU tests (include/frt_selftest.h):
//   * one 128x128x128 bf16 tile through TMA (128-byte swizzle) + tcgen05.mma into TMEM +
//     tcgen05.ld, with B either K-major or MN-major (the QK^T and PV operand layouts), and
//     optionally A staged in TMEM (the tcgen05.mma A-from-TMEM form);
//   * a bounded mbarrier wait that nothing satisfies, which must end with FRT_ERR_TIMEOUT
//     in the stream's status block while the context stays usable.
#include <cstring>

#include "../../include/frt.h"
#include "../../include/frt_selftest.h"
#include "frt_internal.h"
#include "frt_ptx.cuh"

using namespace frt;

namespace {

constexpr int kTile = 128;
constexpr int kTileBytes = kTile * kTile * 2;  // 32 KB
constexpr int kSmem = 2 * kTileBytes + 1024 + 256 + 32768;  // + slack for descriptor variants

struct TestBars {
    uint64_t full;
    uint64_t mma;
    uint32_t tmem;
    int abort_flag;
};

__global__ void __launch_bounds__(128, 1)
umma_tile_kernel(const __grid_constant__ CUtensorMap a_map, const __grid_constant__ CUtensorMap b_map,
                 float* c, int b_mn_major, int lbo_b, int sbo_b, int a_from_tmem, int* status) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                               ~uintptr_t(1023));
    const uint32_t sA = smem_u32(smem);
    const uint32_t sB = sA + kTileBytes;
    TestBars* bars = reinterpret_cast<TestBars*>(smem + 2 * kTileBytes);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint64_t lim = 1000000000ull;
    volatile int* abort = &bars->abort_flag;
    if (threadIdx.x == 0) {
        mbar_init(smem_u32(&bars->full), 1);
        mbar_init(smem_u32(&bars->mma), 1);
        bars->abort_flag = 0;
        fence_mbar_init();
        fence_proxy_async_smem();
    }
    if (warp == 0) {
        tmem_alloc(smem_u32(&bars->tmem), 256);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = bars->tmem;
    bool ok = true;
    if (threadIdx.x == 0) {
        const uint32_t fb = smem_u32(&bars->full);
        mbar_arrive_expect_tx(fb, 2 * kTileBytes);
        for (int cb = 0; cb < 2; ++cb) {
            tma_load_2d(sA + cb * (kTile * 128), &a_map, fb, cb * 64, 0);
            tma_load_2d(sB + cb * (kTile * 128), &b_map, fb, cb * 64, 0);
        }
    }
    if (!mbar_wait(smem_u32(&bars->full), 0, lim, abort)) ok = false;
    ok = __all_sync(0xffffffffu, ok);
    if (ok && a_from_tmem) {
        // thread t = row t of A: read it from the swizzled tile, store packed bf16 pairs
        // into TMEM columns [128, 192) of lane t
        const int row = threadIdx.x;
        uint32_t regs[64];
        for (int ch = 0; ch < 16; ++ch) {
            const int cb = ch >> 3, cc = ch & 7;
            const uint4 v = *reinterpret_cast<const uint4*>(smem + cb * (kTile * 128) + row * 128 +
                                                            ((cc ^ (row & 7)) << 4));
            regs[4 * ch + 0] = v.x; regs[4 * ch + 1] = v.y;
            regs[4 * ch + 2] = v.z; regs[4 * ch + 3] = v.w;
        }
        const uint32_t lane_off = uint32_t(warp * 32) << 16;
        uint32_t r32[32];
        for (int h = 0; h < 2; ++h) {
            for (int i = 0; i < 32; ++i) r32[i] = regs[32 * h + i];
            tmem_st32(tmem + lane_off + 128 + 32 * h, r32);
        }
        tmem_st_wait();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (ok && threadIdx.x == 0) {
        const uint32_t idesc = idesc_bf16_f32(kTile, kTile, b_mn_major != 0);
        for (int k = 0; k < kTile / 16; ++k) {
            const uint32_t aoff = (k >> 2) * (kTile * 128) + (k & 3) * 32;
            const uint32_t boff = b_mn_major ? k * (16 * 128) : aoff;
            const uint64_t bd = b_mn_major ? sdesc_sw128(sB + boff, lbo_b, sbo_b)
                                           : sdesc_sw128(sB + boff, 16, 1024);
            if (a_from_tmem)
                umma_ts(tmem, tmem + 128 + k * 8, bd, idesc, k > 0);
            else
                umma_ss(tmem, sdesc_sw128(sA + aoff, 16, 1024), bd, idesc, k > 0);
        }
        umma_commit(smem_u32(&bars->mma));
    }
    if (ok && !mbar_wait(smem_u32(&bars->mma), 0, lim, abort)) ok = false;
    ok = __all_sync(0xffffffffu, ok);
    if (ok) {
        tc_fence_after();
        const int row = warp * 32 + lane;
        const uint32_t lane_off = uint32_t(warp * 32) << 16;
        for (int cc = 0; cc < 4; ++cc) {
            uint32_t r[32];
            tmem_ld32(tmem + lane_off + cc * 32, r);
            tmem_ld_wait();
            for (int i = 0; i < 32; ++i) c[row * kTile + cc * 32 + i] = __uint_as_float(r[i]);
        }
    } else if (lane == 0) {
        atomicExch(status, 1);
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 0) tmem_dealloc(tmem, 256);
}

// ----------------------------------------------------------------------------------------
// CTA pair: one M=256 x N=128 x K=128 tile with tcgen05.mma.cta_group::2. CTA r of the
// pair holds rows [128 r, 128 r + 128) of A and rows [64 r, 64 r + 64) of B (the N
// half); the leader (rank 0) issues the MMAs; each CTA reads its 128 rows of D.
// ----------------------------------------------------------------------------------------
constexpr int kPairA = 128 * 128 * 2;
constexpr int kPairB = 64 * 128 * 2;
constexpr int kPairSmem = kPairA + kPairB + 1024;

// pv = 1: the P.V form of the attention's pair MMA instead: A (256 x 128, K-major) is
// staged in TMEM (CTA r its 128 rows, packed bf16 pairs in columns [128, 192)) and B is
// the [128 (K), 128 (N)] row-major matrix read MN-major, CTA r holding the N columns
// [64 r, 64 r + 64): C = A B.
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(128, 1)
umma_pair_kernel(const __grid_constant__ CUtensorMap a_map, const __grid_constant__ CUtensorMap b_map,
                 float* c, uint32_t* taddrs, int* status, int pv) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                               ~uintptr_t(1023));
    const uint32_t sA = smem_u32(smem), sB = sA + kPairA;
    __shared__ uint64_t full, done;
    __shared__ uint32_t tbase;
    __shared__ int abort_flag;
    const uint32_t rank = cluster_ctarank();
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint64_t lim = 1000000000ull;
    if (threadIdx.x == 0) {
        mbar_init(smem_u32(&full), 1);
        mbar_init(smem_u32(&done), 1);
        abort_flag = 0;
        fence_mbar_init();
    }
    if (warp == 0) {
        tmem_alloc_pair(smem_u32(&tbase), 256);
        tmem_relinquish_pair();
    }
    tc_fence_before();
    cluster_sync_all();
    tc_fence_after();
    const uint32_t tmem = tbase;
    if (threadIdx.x == 0) taddrs[rank] = tmem;
    if (threadIdx.x == 0) {
        const uint32_t full_leader = mapa_shared(smem_u32(&full), 0);
        if (rank == 0) mbar_arrive_expect_tx(smem_u32(&full), 2 * (kPairA + kPairB));
        for (int cb = 0; cb < 2; ++cb)
            tma_load_2d_pair(sA + cb * (128 * 128), &a_map, full_leader, cb * 64, int(rank) * 128);
        if (pv)   // this CTA's 64 N columns of all 128 K rows: one 128-byte-wide box
            tma_load_2d_pair(sB, &b_map, full_leader, int(rank) * 64, 0);
        else
            for (int cb = 0; cb < 2; ++cb)
                tma_load_2d_pair(sB + cb * (64 * 128), &b_map, full_leader, cb * 64, int(rank) * 64);
    }
    // every CTA waits for the pair's loads (they complete on the leader's barrier), then
    // in the P.V form stages its A rows in TMEM
    bool got = true;
    if (pv) {
        if (rank == 0) got = mbar_wait(smem_u32(&full), 0, lim, &abort_flag);
        cluster_sync_all();   // the leader has seen every byte of both CTAs land
        got = __all_sync(0xffffffffu, got);
        const int row = threadIdx.x;
        uint32_t regs[64];
        for (int ch = 0; ch < 16; ++ch) {
            const int cb = ch >> 3, cc = ch & 7;
            const uint4 v = *reinterpret_cast<const uint4*>(smem + cb * (128 * 128) + row * 128 +
                                                            ((cc ^ (row & 7)) << 4));
            regs[4 * ch + 0] = v.x; regs[4 * ch + 1] = v.y;
            regs[4 * ch + 2] = v.z; regs[4 * ch + 3] = v.w;
        }
        const uint32_t lane_off = uint32_t(warp * 32) << 16;
        uint32_t r32[32];
        for (int h = 0; h < 2; ++h) {
            for (int i = 0; i < 32; ++i) r32[i] = regs[32 * h + i];
            tmem_st32(tmem + lane_off + 128 + 32 * h, r32);
        }
        tmem_st_wait();
        tc_fence_before();
        cluster_sync_all();   // both CTAs' A rows are in TMEM
        tc_fence_after();
    }
    if (threadIdx.x == 0 && rank == 0) {
        if (!pv) got = mbar_wait(smem_u32(&full), 0, lim, &abort_flag);
        if (got) {
            tc_fence_after();
            const uint32_t idesc = idesc_bf16_f32(256, 128, pv != 0);
            for (int k = 0; k < 8; ++k) {
                if (pv) {
                    umma_ts_pair(tmem, tmem + 128 + k * 8, sdesc_sw128(sB + k * (16 * 128), 16384, 1024),
                                 idesc, k > 0);
                } else {
                    const uint32_t aoff = (k >> 2) * (128 * 128) + (k & 3) * 32;
                    const uint32_t boff = (k >> 2) * (64 * 128) + (k & 3) * 32;
                    umma_ss_pair(tmem, sdesc_sw128(sA + aoff, 16, 1024),
                                 sdesc_sw128(sB + boff, 16, 1024), idesc, k > 0);
                }
            }
            umma_commit_pair(smem_u32(&done), 0x3);
        }
    }
    bool ok = __all_sync(0xffffffffu, mbar_wait(smem_u32(&done), 0, lim, &abort_flag));
    if (ok) {
        tc_fence_after();
        const int row = warp * 32 + lane;
        const uint32_t lane_off = uint32_t(warp * 32) << 16;
        for (int cc = 0; cc < 4; ++cc) {
            uint32_t r[32];
            tmem_ld32(tmem + lane_off + cc * 32, r);
            tmem_ld_wait();
            for (int i = 0; i < 32; ++i)
                c[(size_t(rank) * 128 + row) * 128 + cc * 32 + i] = __uint_as_float(r[i]);
        }
    } else if (lane == 0) {
        atomicExch(status, 1);
    }
    // both CTAs are done with TMEM and with each other's shared memory
    tc_fence_before();
    cluster_sync_all();
    tc_fence_after();
    if (warp == 0) tmem_dealloc_pair(tmem, 256);
}

__global__ void wait_timeout_kernel(DeviceStatus* st, unsigned long long limit_ns) {
    __shared__ uint64_t bar;
    __shared__ int abort_flag;
    if (threadIdx.x == 0) {
        mbar_init(smem_u32(&bar), 1);  // expects one arrival that never comes
        abort_flag = 0;
        fence_mbar_init();
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        if (!mbar_wait(smem_u32(&bar), 0, limit_ns, &abort_flag)) {
            volatile DeviceStatus* s = st;
            if (s->code == 0) {
                s->block = blockIdx.x;
                s->role = 99;
                s->where = 0;
                __threadfence_system();
                s->code = FRT_ERR_TIMEOUT;
            }
        }
    }
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

int map_2d(CUtensorMap* m, const void* ptr, int rows, int box_rows) {
    void* fp = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fp, 12000, cudaEnableDefault,
                                         &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess)
        return 1;
    auto fn = reinterpret_cast<EncodeTiledFn>(fp);
    cuuint64_t dims[2] = {128, cuuint64_t(rows)};
    cuuint64_t strides[1] = {256};
    cuuint32_t box[2] = {64, cuuint32_t(box_rows)};
    cuuint32_t es[2] = {1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides, box,
              es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS
               ? 0
               : 2;
}

int map_128x128(CUtensorMap* m, const void* ptr) {
    void* fp = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fp, 12000, cudaEnableDefault,
                                         &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess)
        return 1;
    auto fn = reinterpret_cast<EncodeTiledFn>(fp);
    cuuint64_t dims[2] = {128, 128};
    cuuint64_t strides[1] = {256};
    cuuint32_t box[2] = {64, 128};
    cuuint32_t es[2] = {1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides, box,
              es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS
               ? 0
               : 2;
}

}  // namespace

extern "C" int frt_selftest_umma_tile(const void* a, const void* b, float* c, int b_mn_major,
                                      int lbo_b, int sbo_b, int a_from_tmem, int* dev_status,
                                      void* cuda_stream) {
    if (!a || !b || !c || !dev_status) return -1;
    // keep every descriptor variant inside the CTA's shared memory
    if (lbo_b < 16 || sbo_b < 16 || lbo_b > 16384 || sbo_b > 16384) return -1;
    CUtensorMap am, bm;
    if (map_128x128(&am, a) || map_128x128(&bm, b)) return -2;
    cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
    if (cudaFuncSetAttribute(umma_tile_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             kSmem) != cudaSuccess)
        return -3;
    umma_tile_kernel<<<1, 128, kSmem, st>>>(am, bm, c, b_mn_major, lbo_b, sbo_b, a_from_tmem,
                                            dev_status);
    return cudaGetLastError() == cudaSuccess ? 0 : -4;
}

extern "C" int frt_selftest_umma_pair(const void* a, const void* b, float* c, unsigned* taddrs,
                                      int* dev_status, void* cuda_stream) {
    if (!a || !b || !c || !taddrs || !dev_status) return -1;
    CUtensorMap am, bm;
    if (map_2d(&am, a, 256, 128) || map_2d(&bm, b, 128, 64)) return -2;
    if (cudaFuncSetAttribute(umma_pair_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             kPairSmem) != cudaSuccess)
        return -3;
    umma_pair_kernel<<<2, 128, kPairSmem, static_cast<cudaStream_t>(cuda_stream)>>>(
        am, bm, c, taddrs, dev_status, 0);
    return cudaGetLastError() == cudaSuccess ? 0 : -4;
}

extern "C" int frt_selftest_umma_pair_pv(const void* a, const void* b, float* c, unsigned* taddrs,
                                         int* dev_status, void* cuda_stream) {
    if (!a || !b || !c || !taddrs || !dev_status) return -1;
    CUtensorMap am, bm;
    if (map_2d(&am, a, 256, 128) || map_2d(&bm, b, 128, 128)) return -2;
    if (cudaFuncSetAttribute(umma_pair_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             kPairSmem + kPairB) != cudaSuccess)
        return -3;
    umma_pair_kernel<<<2, 128, kPairSmem + kPairB, static_cast<cudaStream_t>(cuda_stream)>>>(
        am, bm, c, taddrs, dev_status, 1);
    return cudaGetLastError() == cudaSuccess ? 0 : -4;
}

// Defined in frt_host.cu: status block of a stream (device pointer).
extern "C" void* frt_internal_status_dev(frt_stream_t* s);

extern "C" frt_status frt_selftest_wait_timeout(frt_stream_t* s, long long limit_ns,
                                               void* cuda_stream) {
    if (!s || limit_ns <= 0 || limit_ns > 100000000LL) return FRT_ERR_INVALID_ARG;
    void* st = frt_internal_status_dev(s);
    if (!st) return FRT_ERR_STATE;
    wait_timeout_kernel<<<1, 32, 0, static_cast<cudaStream_t>(cuda_stream)>>>(
        static_cast<DeviceStatus*>(st), static_cast<unsigned long long>(limit_ns));
    return cudaGetLastError() == cudaSuccess ? FRT_OK : FRT_ERR_CUDA;
}
