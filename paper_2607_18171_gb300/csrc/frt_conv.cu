// frt_conv.cu — streaming causal 3D convolution on the sm_103a tensor cores.
//
// The second stage of the paper's video pipelines is a streaming VAE decoder (App. A.3:
// the DiT -> VAE template, whose (V, V, 1) self-edge is the decoder's state carried from
// one batch to the next). Its building block is a causal 3D convolution over a chunk of
// frames whose first kt - 1 temporal taps reach into a cache of the previous chunk's
// last frames. For output frame t, pixel (h, w), channel o:
//     y = bias[o] + sum over taps (dt, dh, dw) and input channels c of
//         w[tap][o][c] * x_ext[t + dt][h + dh - kh/2][w + dw - kw/2][c]
// with x_ext = (cache frames, chunk frames) and zero outside the frame.
//
// As an implicit GEMM: M = output pixels, N = Cout, K = taps x Cin. An M tile is 8 rows x
// 16 columns of one output frame; for each tap the A tile is a TMA box of the input
// frame (64 channels x 16 x 8) moved by the tap's offset: out-of-frame pixels arrive as
// zeros, which is the spatial padding. The temporal tap picks the cache or the chunk
// tensor map. B is the tap's [Cout, Cin] weight slice. Persistent kernel, 192 threads:
//   warp 0      TMA producer (A box + B box per k-block of 64 channels, 4-stage ring);
//   warp 1      TMEM allocator + single-thread tcgen05.mma issuer (M 128, N = BN, K 16);
//   warps 2-5   epilogue (one thread per output pixel of the tile; bias added, pixels
//               outside the frame not stored).
// The accumulator is double-buffered in TMEM (2 x BN columns). With enough tiles, two
// CTAs of a cluster work as a pair on two pixel tiles with tcgen05.mma.cta_group::2 (M =
// 256): each holds its own A and half of the weight tile, which cuts the bytes each SM
// must take in per FLOP — what bounds this kernel. A second, small kernel
// writes the next cache (last kt - 1 frames of (cache, chunk)) into the other half of a
// ping-pong pair, so no launch reads what it writes.
#include <algorithm>
#include <cstring>
#include <mutex>
#include <new>

#include "../../include/frt.h"
#include "frt_internal.h"
#include "frt_ptx.cuh"

namespace frt {
namespace {

constexpr int kThreads = 192;
constexpr int kBM = 128;         // output pixels per tile: 8 rows x 16 columns
constexpr int kTileW = 16;
constexpr int kTileH = 8;
constexpr int kBK = 64;          // input channels per k-block (one 128-byte swizzle row)
constexpr int kMaxStages = 6;
constexpr int kTimeoutCode = 6;  // FRT_ERR_TIMEOUT
constexpr int kMaxTaps = 64;

struct ConvParams {
    CUtensorMap x_map;      // 4D (Cin, W, H, F) bf16 over the chunk, box (64, 16, 8, 1)
    CUtensorMap c_map;      // 4D (Cin, W, H, kt - 1) over the cache (unused when kt == 1)
    CUtensorMap w_map;      // 3D (Cin, Cout, taps) bf16 over the weights, box (64, BN, 1)
    const float* bias;      // [Cout]
    void* y;                // [F, H, W, Cout] fp32 or bf16
    int y_bf16;
    int cin, cout, kt, kh, kw, H, W, F;
    int tiles_w, tiles_h, tiles_n, n_tiles;
    unsigned long long wait_limit_ns;
    DeviceStatus* status;
};

template <int BN, bool PAIR>
struct CCfg {
    static constexpr int CM = PAIR ? 2 : 1;
    static constexpr int A_BYTES = kBM * kBK * 2;
    static constexpr int B_BYTES = (BN / CM) * kBK * 2;
    static constexpr int STAGE = A_BYTES + B_BYTES;
    static constexpr int STAGES = PAIR ? 6 : 4;
    static constexpr int SMEM = STAGES * STAGE + 1024;
    static constexpr uint32_t IDESC = idesc_bf16_f32(kBM * CM, BN, false);
    static constexpr uint32_t TMEM_COLS = (2 * BN <= 256) ? 256 : 512;
};

struct CBars {
    uint64_t full[kMaxStages];
    uint64_t empty[kMaxStages];
    uint64_t acc_full[2];
    uint64_t acc_empty[2];
    uint64_t drain;
    uint32_t tmem_base;
    int abort_flag;
};

__device__ __forceinline__ void report(DeviceStatus* st, volatile int* abort, int role, int where) {
    *abort = 1;
    if (st != nullptr) {
        volatile DeviceStatus* s = st;
        if (s->code == 0) {
            s->block = blockIdx.x;
            s->role = 300 + role;
            s->where = where;
            __threadfence_system();
            s->code = kTimeoutCode;
        }
    }
}

// tile index -> (frame, tile row, tile column, N tile); N tiles vary fastest so CTAs
// launched together share the input window. With pairs, tile t covers pixel tiles
// 2 m and 2 m + 1 (one per CTA, `rank`) of the same N tile.
__device__ __forceinline__ void tile_coords(const ConvParams& p, int t, int cm, int rank, int& f,
                                            int& th, int& tw, int& tn) {
    tn = t % p.tiles_n;
    int m = (t / p.tiles_n) * cm + rank;
    tw = m % p.tiles_w;
    m /= p.tiles_w;
    th = m % p.tiles_h;
    f = m / p.tiles_h;
}

template <int BN, bool PAIR>
__global__ void __launch_bounds__(kThreads, 1) conv_kernel(const __grid_constant__ ConvParams p) {
    using C = CCfg<BN, PAIR>;
    constexpr int CM = C::CM;
    constexpr int kStages = C::STAGES;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                               ~uintptr_t(1023));
    __shared__ CBars bars;
    const uint32_t sbase = smem_u32(smem);
    volatile int* abort = &bars.abort_flag;
    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const int nkb = p.cin / kBK;
    const int taps = p.kt * p.kh * p.kw;
    const int nk = taps * nkb;
    const uint64_t lim = p.wait_limit_ns;
    const int rank = PAIR ? int(cluster_ctarank()) : 0;
    const bool leader = rank == 0;
    const int c_first = blockIdx.x / CM;
    const int c_stride = gridDim.x / CM;

    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            mbar_init(smem_u32(&bars.full[s]), 1);
            mbar_init(smem_u32(&bars.empty[s]), 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(smem_u32(&bars.acc_full[b]), 1);
            mbar_init(smem_u32(&bars.acc_empty[b]), 128 * CM);
        }
        mbar_init(smem_u32(&bars.drain), 1);
        bars.abort_flag = 0;
        fence_mbar_init();
    }
    if (warp == 1) {
        if (PAIR) {
            tmem_alloc_pair(smem_u32(&bars.tmem_base), C::TMEM_COLS);
            tmem_relinquish_pair();
        } else {
            tmem_alloc(smem_u32(&bars.tmem_base), C::TMEM_COLS);
            tmem_relinquish();
        }
    }
    tc_fence_before();
    __syncthreads();
    if (PAIR) cluster_sync_all();
    tc_fence_after();
    const uint32_t tmem = bars.tmem_base;

    if (warp == 0) {
        // ==================================== TMA producer ===================================
        if (lane == 0) {
            tma_prefetch_map(&p.x_map);
            if (p.kt > 1) tma_prefetch_map(&p.c_map);
            tma_prefetch_map(&p.w_map);
            int it = 0;
            bool ok = true;
            for (int t = c_first; t < p.n_tiles && ok; t += c_stride) {
                int f, th, tw, tn;
                tile_coords(p, t, CM, rank, f, th, tw, tn);
                for (int kk = 0; kk < nk; ++kk) {
                    const int s = it % kStages;
                    if (it >= kStages &&
                        !mbar_wait(smem_u32(&bars.empty[s]), ((it / kStages) - 1) & 1, lim, abort)) {
                        report(p.status, abort, 0, it);
                        ok = false;
                        break;
                    }
                    const int tap = kk / nkb;
                    const int kb = kk - tap * nkb;
                    const int dt = tap / (p.kh * p.kw);
                    const int rem = tap - dt * p.kh * p.kw;
                    const int dh = rem / p.kw;
                    const int dw = rem - dh * p.kw;
                    const int src = f + dt - (p.kt - 1);      // frame of (cache, chunk) - cache
                    const uint32_t dst = sbase + s * C::STAGE;
                    const int cx = tw * kTileW + dw - p.kw / 2;
                    const int cy = th * kTileH + dh - p.kh / 2;
                    const CUtensorMap* amap = src < 0 ? &p.c_map : &p.x_map;
                    const int az = src < 0 ? src + p.kt - 1 : src;
                    if (PAIR) {
                        const uint32_t fb = mapa_shared(smem_u32(&bars.full[s]), 0);
                        if (leader) mbar_arrive_expect_tx(smem_u32(&bars.full[s]), 2 * C::STAGE);
                        tma_load_4d_pair(dst, amap, fb, kb * kBK, cx, cy, az);
                        tma_load_3d_pair(dst + C::A_BYTES, &p.w_map, fb, kb * kBK,
                                         tn * BN + rank * (BN / 2), tap);
                    } else {
                        const uint32_t fb = smem_u32(&bars.full[s]);
                        mbar_arrive_expect_tx(fb, C::STAGE);
                        tma_load_4d(dst, amap, fb, kb * kBK, cx, cy, az);
                        tma_load_3d(dst + C::A_BYTES, &p.w_map, fb, kb * kBK, tn * BN, tap);
                    }
                    ++it;
                }
            }
            if (leader)
                for (int i = (it > kStages ? it - kStages : 0); i < it; ++i)
                    mbar_wait_drain(smem_u32(&bars.full[i % kStages]), (i / kStages) & 1, lim);
        }
    } else if (warp == 1) {
        // ======================= MMA issuer (one thread of the leader) =======================
        if (lane == 0 && leader) {
            const uint64_t da0 = sdesc_sw128(sbase, 16, 1024);
            const uint64_t db0 = sdesc_sw128(sbase + C::A_BYTES, 16, 1024);
            int it = 0;
            int tl = 0;
            bool ok = true;
            for (int t = c_first; t < p.n_tiles && ok; t += c_stride, ++tl) {
                const int b = tl & 1;
                if (tl >= 2 &&
                    !mbar_wait(smem_u32(&bars.acc_empty[b]), ((tl >> 1) - 1) & 1, lim, abort)) {
                    report(p.status, abort, 1, -1 - tl);
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t d = tmem + uint32_t(b * BN);
                for (int kk = 0; kk < nk; ++kk, ++it) {
                    const int s = it % kStages;
                    if (!mbar_wait(smem_u32(&bars.full[s]), (it / kStages) & 1, lim, abort)) {
                        report(p.status, abort, 1, it);
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint64_t so = uint64_t((s * C::STAGE) >> 4);
#pragma unroll
                    for (int k = 0; k < kBK / 16; ++k) {
                        if (PAIR)
                            umma_ss_pair(d, da0 + so + uint64_t(2 * k), db0 + so + uint64_t(2 * k),
                                         C::IDESC, (kk > 0 || k > 0) ? 1u : 0u);
                        else
                            umma_ss(d, da0 + so + uint64_t(2 * k), db0 + so + uint64_t(2 * k),
                                    C::IDESC, (kk > 0 || k > 0) ? 1u : 0u);
                    }
                    if (PAIR) umma_commit_pair(smem_u32(&bars.empty[s]), 0x3);
                    else umma_commit(smem_u32(&bars.empty[s]));
                }
                if (ok) {
                    if (PAIR) umma_commit_pair(smem_u32(&bars.acc_full[b]), 0x3);
                    else umma_commit(smem_u32(&bars.acc_full[b]));
                }
            }
            if (PAIR) umma_commit_pair(smem_u32(&bars.drain), 0x1);
            else umma_commit(smem_u32(&bars.drain));
            mbar_wait_drain(smem_u32(&bars.drain), 0, lim);
        }
    } else {
        // ====================================== epilogue =====================================
        const int sub = warp & 3;
        const int row = sub * 32 + lane;                 // pixel of the tile: 16 per row
        const uint32_t lane_off = uint32_t(sub * 32) << 16;
        int tl = 0;
        for (int t = c_first; t < p.n_tiles; t += c_stride, ++tl) {
            const int b = tl & 1;
            int f, th, tw, tn;
            tile_coords(p, t, CM, rank, f, th, tw, tn);
            const bool got = mbar_wait(smem_u32(&bars.acc_full[b]), (tl >> 1) & 1, lim, abort);
            if (!__all_sync(0xffffffffu, got)) {
                if (!got) report(p.status, abort, 2, tl);
                break;
            }
            tc_fence_after();
            const int h = th * kTileH + (row >> 4);
            const int w = tw * kTileW + (row & 15);
            const bool live = f < p.F && h < p.H && w < p.W;
            const size_t obase = ((size_t(f) * p.H + h) * p.W + w) * p.cout + size_t(tn) * BN;
#pragma unroll 1
            for (int c = 0; c < BN / 32; ++c) {
                uint32_t r[32];
                tmem_ld32(tmem + lane_off + uint32_t(b * BN + c * 32), r);
                tmem_ld_wait();
                if (live) {
                    const float4* bp = reinterpret_cast<const float4*>(p.bias + tn * BN + c * 32);
                    float v[32];
#pragma unroll
                    for (int i = 0; i < 8; ++i) {
                        const float4 bb = __ldg(bp + i);
                        v[4 * i] = __uint_as_float(r[4 * i]) + bb.x;
                        v[4 * i + 1] = __uint_as_float(r[4 * i + 1]) + bb.y;
                        v[4 * i + 2] = __uint_as_float(r[4 * i + 2]) + bb.z;
                        v[4 * i + 3] = __uint_as_float(r[4 * i + 3]) + bb.w;
                    }
                    if (p.y_bf16) {
                        uint4* o = reinterpret_cast<uint4*>(static_cast<uint16_t*>(p.y) + obase + c * 32);
#pragma unroll
                        for (int i = 0; i < 4; ++i)
                            o[i] = make_uint4(pack_bf16x2(v[8 * i], v[8 * i + 1]), pack_bf16x2(v[8 * i + 2], v[8 * i + 3]),
                                              pack_bf16x2(v[8 * i + 4], v[8 * i + 5]), pack_bf16x2(v[8 * i + 6], v[8 * i + 7]));
                    } else {
                        float4* o = reinterpret_cast<float4*>(static_cast<float*>(p.y) + obase + c * 32);
#pragma unroll
                        for (int i = 0; i < 8; ++i)
                            o[i] = make_float4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
                    }
                }
                __syncwarp();
            }
            tc_fence_before();
            if (PAIR) mbar_arrive_cluster(mapa_shared(smem_u32(&bars.acc_empty[b]), 0));
            else mbar_arrive(smem_u32(&bars.acc_empty[b]));
        }
    }
    __syncwarp();
    tc_fence_before();
    __syncthreads();
    if (PAIR) cluster_sync_all();
    tc_fence_after();
    if (warp == 1) {
        if (PAIR) tmem_dealloc_pair(tmem, C::TMEM_COLS);
        else tmem_dealloc(tmem, C::TMEM_COLS);
    }
}

// next cache = last kt - 1 frames of (cache, chunk), written to the other ping-pong half
__global__ void cache_shift_kernel(const uint4* __restrict__ cache, const uint4* __restrict__ x,
                                   uint4* __restrict__ next, long long frame_vec, int keep, int F) {
    const long long total = frame_vec * keep;
    for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < total;
         i += (long long)gridDim.x * blockDim.x) {
        const int j = int(i / frame_vec);          // frame of the next cache
        const long long r = i - (long long)j * frame_vec;
        const int src = j + F;                     // frame of (cache, chunk)
        next[i] = src < keep ? cache[(long long)src * frame_vec + r]
                             : x[(long long)(src - keep) * frame_vec + r];
    }
}

template <int BN, bool PAIR>
cudaError_t launch_conv(ConvParams p, cudaStream_t st) {
    using C = CCfg<BN, PAIR>;
    static bool attr = false;
    if (!attr) {
        cudaError_t e = cudaFuncSetAttribute(conv_kernel<BN, PAIR>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
        if (e != cudaSuccess) return e;
        attr = true;
    }
    const int units = std::min(p.n_tiles, num_sms() / C::CM);
    if (!PAIR) {
        conv_kernel<BN, false><<<units, kThreads, C::SMEM, st>>>(p);
        return cudaGetLastError();
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(unsigned(units * 2));
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = C::SMEM;
    cfg.stream = st;
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = 2;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, conv_kernel<BN, true>, p);
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
    static EncodeTiledFn fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void* q = nullptr;
        cudaDriverEntryPointQueryResult r;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &q, 12000,
                                             cudaEnableDefault, &r) == cudaSuccess &&
            r == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(q);
    });
    return fn;
}

bool encode(CUtensorMap* map, const void* base, int rank, const cuuint64_t* dims,
            const cuuint32_t* box) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return false;
    cuuint64_t strides[3];
    cuuint64_t acc = dims[0] * 2;
    for (int i = 0; i + 1 < rank; ++i) {
        strides[i] = acc;
        acc *= dims[i + 1];
    }
    cuuint32_t estr[4] = {1, 1, 1, 1};
    return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, rank, const_cast<void*>(base), dims, strides,
              box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Output-channel tile and pairing. Cost of one k-block on an SM ~ the larger of its MMA
// time (BN / 2 cycles per 16-deep MMA, four of them) and the time to receive its operand
// bytes at the ~40 bytes/cycle an SM takes in with all SMs loading (A 16 KB, plus its
// share of the BN x 64 weight slice); every tile has the same number of k-blocks, and
// tiles run in rounds over the SMs (or SM pairs), so the launch costs rounds x that.
// The cheapest of the widths dividing Cout wins; pairs need at least two pixel tiles.
int choose_bn(int cout, long long m_tiles, bool& pair) {
    const int cands[4] = {256, 192, 128, 64};
    const long long sms = num_sms();
    int best = 0;
    double best_t = 1e30;
    for (int pr = 0; pr < 2; ++pr) {
        if (pr == 1 && m_tiles < 2) continue;
        const int cm = pr ? 2 : 1;
        const long long units = sms / cm;
        const long long mt = (m_tiles + cm - 1) / cm;
        for (int bn : cands) {
            if (cout % bn) continue;
            const long long tiles = mt * (cout / bn);
            const double rounds = double((tiles + units - 1) / units);
            const double mma = 4.0 * bn / 2.0;
            const double bytes = 16384.0 + double(bn / cm) * 128.0;
            const double t = rounds * std::max(mma, bytes / 40.0);
            if (t < best_t - 1e-9) {
                best_t = t;
                best = bn;
                pair = pr == 1;
            }
        }
    }
    return best;
}

}  // namespace
}  // namespace frt

using namespace frt;

struct frt_conv {
    int cin, cout, kt, kh, kw, H, W, F;
    int out_dtype = FRT_OUT_F32;
    cudaStream_t cs = nullptr;
    bool configured = false;
    void* cache[2] = {nullptr, nullptr};   // ping-pong [kt - 1, H, W, Cin] bf16
    int cur = 0;
    size_t frame_bytes = 0;
    DeviceStatus* status_host = nullptr;
    DeviceStatus* status_dev = nullptr;
    long long chunks = 0;
    unsigned long long wait_limit_ns = 2000000000ull;
};

namespace {
frt_status cfail(frt_status st, const char* msg) {
    set_last_error(msg);
    return st;
}
bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
void free_conv(frt_conv_t* c) {
    for (int i = 0; i < 2; ++i)
        if (c->cache[i]) cudaFree(c->cache[i]);
    if (c->status_host) cudaFreeHost(c->status_host);
    c->cache[0] = c->cache[1] = nullptr;
    c->status_host = c->status_dev = nullptr;
}
}  // namespace

extern "C" {

frt_conv_t* frt_conv_create(int cin, int cout, int kt, int kh, int kw, int grid_h, int grid_w,
                            int frames_per_chunk) {
    if (cin < 64 || cin % 64 || cout < 64 || cout % 64 || kt < 1 || kt > 4 || kh < 1 || kh > 7 ||
        kw < 1 || kw > 7 || kh % 2 == 0 || kw % 2 == 0 || grid_h < 1 || grid_w < 1 ||
        frames_per_chunk < 1 || kt * kh * kw > kMaxTaps || (long long)grid_h * grid_w > (1LL << 24)) {
        set_last_error("need Cin, Cout multiples of 64, 1 <= kt <= 4, odd kh, kw <= 7, positive sizes");
        return nullptr;
    }
    auto* c = new (std::nothrow) frt_conv;
    if (!c) {
        set_last_error("host allocation failed");
        return nullptr;
    }
    c->cin = cin;
    c->cout = cout;
    c->kt = kt;
    c->kh = kh;
    c->kw = kw;
    c->H = grid_h;
    c->W = grid_w;
    c->F = frames_per_chunk;
    c->frame_bytes = size_t(grid_h) * grid_w * cin * 2;
    return c;
}

frt_status frt_conv_configure(frt_conv_t* c, int out_dtype, void* cuda_stream) {
    if (!c) return cfail(FRT_ERR_INVALID_ARG, "NULL conv handle");
    if (out_dtype != FRT_OUT_F32 && out_dtype != FRT_OUT_BF16)
        return cfail(FRT_ERR_INVALID_ARG, "unknown out_dtype");
    cudaError_t e;
    if (!c->configured) {
        const size_t bytes = std::max<size_t>(1, size_t(c->kt - 1)) * c->frame_bytes;
        for (int i = 0; i < 2; ++i)
            if ((e = cudaMalloc(&c->cache[i], bytes)) != cudaSuccess ||
                (e = cudaMemset(c->cache[i], 0, bytes)) != cudaSuccess) {
                free_conv(c);
                return cfail(e == cudaErrorMemoryAllocation ? FRT_ERR_OOM : FRT_ERR_CUDA,
                             "frame cache allocation failed");
            }
        if ((e = cudaHostAlloc(reinterpret_cast<void**>(&c->status_host), sizeof(DeviceStatus),
                               cudaHostAllocMapped)) != cudaSuccess ||
            (e = cudaHostGetDevicePointer(reinterpret_cast<void**>(&c->status_dev), c->status_host,
                                          0)) != cudaSuccess) {
            free_conv(c);
            return cfail(FRT_ERR_CUDA, "status allocation failed");
        }
        std::memset(c->status_host, 0, sizeof(DeviceStatus));
        if ((e = cudaDeviceSynchronize()) != cudaSuccess) return cfail(FRT_ERR_CUDA, "sync failed");
    }
    c->out_dtype = out_dtype;
    c->cs = static_cast<cudaStream_t>(cuda_stream);
    c->configured = true;
    return FRT_OK;
}

frt_status frt_conv_step(frt_conv_t* c, const void* x, const void* w, const void* bias, void* y) {
    if (!c) return cfail(FRT_ERR_INVALID_ARG, "NULL conv handle");
    if (!c->configured) return cfail(FRT_ERR_STATE, "conv not configured");
    if (c->status_host && c->status_host->code != 0)
        return cfail(static_cast<frt_status>(c->status_host->code),
                     "a device wait gave up earlier; reset the conv");
    if (!x || !w || !bias || !y || !aligned16(x) || !aligned16(w) || !aligned16(bias) ||
        !aligned16(y))
        return cfail(FRT_ERR_INVALID_ARG, "x, w, bias, y must be non-NULL and 16-byte aligned");
    ConvParams p;
    std::memset(&p, 0, sizeof(p));
    p.cin = c->cin;
    p.cout = c->cout;
    p.kt = c->kt;
    p.kh = c->kh;
    p.kw = c->kw;
    p.H = c->H;
    p.W = c->W;
    p.F = c->F;
    p.tiles_w = (c->W + kTileW - 1) / kTileW;
    p.tiles_h = (c->H + kTileH - 1) / kTileH;
    const long long m_tiles = (long long)c->F * p.tiles_w * p.tiles_h;
    bool pair = false;
    const int bn = choose_bn(c->cout, m_tiles, pair);
    if (bn == 0) return cfail(FRT_ERR_UNSUPPORTED, "Cout has no supported tile width");
    p.tiles_n = c->cout / bn;
    const long long m_units = pair ? (m_tiles + 1) / 2 : m_tiles;
    if (m_units * p.tiles_n >= (1LL << 31)) return cfail(FRT_ERR_UNSUPPORTED, "too many tiles");
    p.n_tiles = int(m_units * p.tiles_n);
    const cuuint32_t abox[4] = {64, kTileW, kTileH, 1};
    const cuuint64_t xdims[4] = {cuuint64_t(c->cin), cuuint64_t(c->W), cuuint64_t(c->H),
                                 cuuint64_t(c->F)};
    const cuuint64_t cdims[4] = {cuuint64_t(c->cin), cuuint64_t(c->W), cuuint64_t(c->H),
                                 cuuint64_t(std::max(1, c->kt - 1))};
    const cuuint64_t wdims[3] = {cuuint64_t(c->cin), cuuint64_t(c->cout),
                                 cuuint64_t(c->kt * c->kh * c->kw)};
    const cuuint32_t wbox[3] = {64, cuuint32_t(pair ? bn / 2 : bn), 1};
    if (!encode(&p.x_map, x, 4, xdims, abox) || !encode(&p.c_map, c->cache[c->cur], 4, cdims, abox) ||
        !encode(&p.w_map, w, 3, wdims, wbox))
        return cfail(FRT_ERR_CUDA, "tensor map encoding failed");
    p.bias = static_cast<const float*>(bias);
    p.y = y;
    p.y_bf16 = c->out_dtype == FRT_OUT_BF16;
    p.wait_limit_ns = c->wait_limit_ns;
    p.status = c->status_dev;
    cudaError_t e;
    switch (bn * 2 + (pair ? 1 : 0)) {
        case 513: e = launch_conv<256, true>(p, c->cs); break;
        case 512: e = launch_conv<256, false>(p, c->cs); break;
        case 385: e = launch_conv<192, true>(p, c->cs); break;
        case 384: e = launch_conv<192, false>(p, c->cs); break;
        case 257: e = launch_conv<128, true>(p, c->cs); break;
        case 256: e = launch_conv<128, false>(p, c->cs); break;
        case 129: e = launch_conv<64, true>(p, c->cs); break;
        default: e = launch_conv<64, false>(p, c->cs); break;
    }
    if (e != cudaSuccess) return cfail(FRT_ERR_CUDA, cudaGetErrorString(e));
    if (c->kt > 1) {
        const int keep = c->kt - 1;
        const long long frame_vec = (long long)(c->frame_bytes / 16);
        const long long total = frame_vec * keep;
        const int blocks = int(std::min<long long>((total + 255) / 256, 4LL * num_sms()));
        cache_shift_kernel<<<blocks, 256, 0, c->cs>>>(static_cast<const uint4*>(c->cache[c->cur]),
                                                       static_cast<const uint4*>(x),
                                                       static_cast<uint4*>(c->cache[c->cur ^ 1]),
                                                       frame_vec, keep, c->F);
        if ((e = cudaGetLastError()) != cudaSuccess)
            return cfail(FRT_ERR_CUDA, cudaGetErrorString(e));
        c->cur ^= 1;
    }
    c->chunks += 1;
    return FRT_OK;
}

frt_status frt_conv_cache(const frt_conv_t* c, const void** cache) {
    if (!c || !cache) return cfail(FRT_ERR_INVALID_ARG, "NULL argument");
    if (!c->configured) return cfail(FRT_ERR_STATE, "conv not configured");
    *cache = c->cache[c->cur];
    return FRT_OK;
}

frt_status frt_conv_sync(frt_conv_t* c) {
    if (!c) return cfail(FRT_ERR_INVALID_ARG, "NULL conv handle");
    if (!c->configured) return FRT_OK;
    cudaError_t e = cudaStreamSynchronize(c->cs);
    if (e != cudaSuccess) return cfail(FRT_ERR_CUDA, cudaGetErrorString(e));
    if (c->status_host && c->status_host->code != 0)
        return cfail(static_cast<frt_status>(c->status_host->code),
                     "a device-side bounded wait gave up");
    return FRT_OK;
}

frt_status frt_conv_reset(frt_conv_t* c) {
    if (!c) return cfail(FRT_ERR_INVALID_ARG, "NULL conv handle");
    if (!c->configured) return FRT_OK;
    cudaError_t e = cudaStreamSynchronize(c->cs);
    const size_t bytes = std::max<size_t>(1, size_t(c->kt - 1)) * c->frame_bytes;
    for (int i = 0; i < 2 && e == cudaSuccess; ++i) e = cudaMemset(c->cache[i], 0, bytes);
    if (e != cudaSuccess) return cfail(FRT_ERR_CUDA, cudaGetErrorString(e));
    std::memset(c->status_host, 0, sizeof(DeviceStatus));
    c->cur = 0;
    c->chunks = 0;
    return FRT_OK;
}

void frt_conv_destroy(frt_conv_t* c) {
    if (!c) return;
    if (c->configured) cudaStreamSynchronize(c->cs);
    free_conv(c);
    delete c;
}

}  // extern "C"
