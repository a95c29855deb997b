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
// As an implicit GEMM: M = output pixels, N = Cout, K = taps x Cin. An M tile is 16 rows
// x 8 columns of one output frame. For each temporal tap and 64-channel block, ONE TMA
// box brings in the tile's halo, (16 + kh - 1) x (8 + kw - 1) input pixels (out-of-frame
// pixels arrive as zeros: the spatial padding), and all kh x kw spatial taps read their
// A operand from it: the operand of tap (dh, dw) is the same 128-byte-swizzled halo seen
// from a start address moved by (dh * halo_w + dw) pixel rows, with 8-row groups (one
// tile row) halo_w * 128 bytes apart. tcgen05 applies the swizzle to absolute shared-
// memory addresses, so any whole-row start is valid once the halo sits at a 1024-byte
// boundary. This brings each input pixel into the SM about 1.4 times per temporal tap
// and channel block instead of kh x kw times. B is the tap's [Cout, Cin] weight slice.
// Persistent kernel, 256 threads:
//   warp 0      TMA producer of the halo ring;
//   warp 6      TMA producer of the weight ring (one slice per spatial tap);
//   warp 1      TMEM allocator + tcgen05.mma issuer (M 128, N = BN, K 16): a converged
//               warp whose lane 0 issues; it touches no mbarrier in its loops;
//   warp 7      observer: waits on the halo, weight and accumulator barriers in the
//               issuer's order and hands each off to it through a named barrier;
//   warps 2-5   epilogue: one thread per output pixel of the tile adds the bias and
//               writes its 128-byte slice of each column unit (32 fp32 or 64 bf16
//               channels) into a 128-byte-swizzled staging slab, which one TMA tensor
//               store writes to y (pixels outside the frame are clipped by the store);
//               per-thread stores of whole pixel rows would touch 32 rows per warp
//               instruction.
// The accumulator is double-buffered in TMEM (2 x BN columns). With enough tiles, two
// CTAs of a cluster work as a pair on two pixel tiles with tcgen05.mma.cta_group::2 (M =
// 256): each holds its own halo and half of the weight slice, which halves the weight
// bytes each SM takes in per FLOP — with the halo, the larger share of what bounds this
// kernel. The next cache (last kt - 1 frames of (cache, chunk)) is written into the other
// half of a ping-pong pair by the epilogue warps of every CTA, a slice each, while they
// wait for their first accumulator; no launch reads what it writes.
#include <algorithm>
#include <cstring>
#include <mutex>
#include <new>

#include "../../include/frt.h"
#include "frt_internal.h"
#include "frt_ptx.cuh"

namespace frt {
namespace {

constexpr int kThreads = 256;
// Named barrier of the issuer / observer hand-off (warps 1 and 7); id 1 serves the
// epilogue warps, id 0 is __syncthreads.
constexpr int kBarHandoff = 4;
constexpr int kBM = 128;         // output pixels per tile: 16 rows x 8 columns
constexpr int kTileW = 8;        // one 8-row operand group = one tile row
constexpr int kTileH = 16;
constexpr int kBK = 64;          // input channels per k-block (one 128-byte swizzle row)
constexpr int kMaxStages = 8;
constexpr int kTimeoutCode = 6;  // FRT_ERR_TIMEOUT
constexpr int kSmemBudget = 225 * 1024;  // dynamic shared memory of the kernel
constexpr int kSlab = kBM * 128;         // epilogue staging: 128 rows of 128 bytes
// How long the first part of a split tile waits, with its own sum done, for the other
// parts before it writes itself out instead (they usually land within a few us).
constexpr unsigned long long kPartWaitNs = 20000;

struct ConvParams {
    CUtensorMap x_map;      // 4D (Cin, W, H, F) bf16 over the chunk, box (64, halo_w, halo_h, 1)
    CUtensorMap c_map;      // the same over the cache (unused when kt == 1)
    CUtensorMap w_map;      // 3D (Cin, Cout, taps) bf16 over the weights, box (64, BN / pair, tb)
    CUtensorMap y_map;      // 4D (Cout, W, H, F) fp32 or bf16 over y, box (32 | 64, 8, 16, 1)
    const float* bias;      // [Cout]
    void* y;                // [F, H, W, Cout] fp32 or bf16
    int y_bf16;
    int cin, cout, kt, kh, kw, H, W, F;
    int tiles_w, tiles_h, tiles_n, n_tiles;
    int halo_w, halo_h;     // 8 + kw - 1, 16 + kh - 1 input pixels
    int halo_tx;            // bytes one halo box delivers: halo_w * halo_h * 128
    int a_bytes;            // halo ring stage (halo_tx rounded up to 1024)
    int a_stages, b_stages;
    int tb;                 // spatial taps per weight-ring stage: kw (one kernel row) or 1
    int b_stage;            // weight-ring stage bytes: tb * (BN / pair) * 128
    unsigned long long wait_limit_ns;
    DeviceStatus* status;
    // next cache = frames [F, F + keep) of (cache, chunk), in 16-byte vectors (keep = 0:
    // no cache)
    const uint4* shift_cache;
    const uint4* shift_x;
    uint4* shift_next;
    long long shift_frame_vec;   // vectors per frame
    int shift_keep;              // kt - 1
    // Work split over the grid's units (a CTA, or a CTA pair): the K loop of tile t is
    // its halos, global steps [t * nhalo, (t + 1) * nhalo). Split: unit u takes the steps
    // [u * total / units, (u + 1) * total / units), so a tile may be shared by
    // consecutive units, each adding a part of its K sum. Not split: unit u takes the
    // whole tiles [u * n_tiles / units, (u + 1) * n_tiles / units).
    long long total;             // n_tiles * nhalo
    int split;
    // split tiles: each part is written to part[slot][rank][BN / 4][128] (float4, slot
    // 2u for the first item of unit u's range, 2u + 1 for its last), and the part that
    // arrives last at counters[t * pair + rank] adds all parts in step order
    float4* part;
    int* counters;               // zero between launches: the adding part resets it
    long long part_cap;          // float4s in part, entries in counters (the FRT_DEBUG
    long long ctr_cap;           // build checks every derived index against them)
    int part_mode;               // 0 as built; 1 no watch; 2 no watch, no wait (self-test)
};

template <int BN, bool PAIR>
struct CCfg {
    static constexpr int CM = PAIR ? 2 : 1;
    static constexpr int B_BYTES = (BN / CM) * kBK * 2;
    static constexpr uint32_t IDESC = idesc_bf16_f32(kBM * CM, BN, false);
    static constexpr uint32_t TMEM_COLS = (2 * BN <= 256) ? 256 : 512;
};

struct CBars {
    uint64_t a_full[kMaxStages];
    uint64_t a_empty[kMaxStages];
    uint64_t b_full[kMaxStages];
    uint64_t b_empty[kMaxStages];
    uint64_t acc_full[2];
    uint64_t acc_empty[2];
    uint64_t drain;
    uint64_t part_full;     // a split tile's part copied into the (idle) rings
    float4 bias[64];        // epilogue: the current tile's bias slice (BN <= 256)
    uint32_t tmem_base;
    int abort_flag;
    int last_part;          // epilogue: broadcast word of the split-tile protocol
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

// First global step of unit u's share.
__device__ __forceinline__ long long unit_start(const ConvParams& p, int u, int units, int nhalo) {
    return p.split ? (long long)u * p.total / units : (long long)u * p.n_tiles / units * nhalo;
}

// Split: the unit whose share holds global step s (the largest u with unit_start <= s).
__device__ __forceinline__ int unit_of(const ConvParams& p, long long s, int units) {
    return int(((s + 1) * units - 1) / p.total);
}

// Workspace slot of unit u's part of the split tile that starts at step ts: the tile is
// the unit's first item if its share starts inside the tile, else its last.
__device__ __forceinline__ int part_slot(const ConvParams& p, int u, long long ts, int units,
                                         int nhalo) {
    return 2 * u + (unit_start(p, u, units, nhalo) < ts ? 1 : 0);
}

// The items of a unit's share in order: tile t, halos [h0, h1) of its K loop.
struct Items {
    long long s, s1;
    int nhalo;
    int t, h0, h1;
    __device__ __forceinline__ bool next() {
        if (s >= s1) return false;
        t = int(s / nhalo);
        const long long ts = (long long)t * nhalo;
        const long long te = ts + nhalo;
        h0 = int(s - ts);
        h1 = int((s1 < te ? s1 : te) - ts);
        s = ts + h1;
        return true;
    }
};

// Split tiles sum their parts in one order, whoever adds them: the parts that continue
// the tile (1, 2, ..., n - 1, in step order) and then the part that starts it (0):
// ((part 1 + part 2) + ...) + part 0. Its starting part is its unit's last item, so it
// usually completes last, and this order lets that unit add the others while its own
// MMAs still run.
//
// sum_parts: TMEM columns [dst, dst + BN) of this thread's lane become the sum, in that
// order, of NO parts read from L2 (src[0..NO), this thread's row of each) and, at
// position own of the order, this CTA's own part already in dst (own = -1: none). The
// parts are read in batches of 16 16-byte loads per thread: an L2 round trip here
// is about a microsecond, so one 32-column batch at a time would cost one per batch.
// (Not inlined: its loads would otherwise be allocated together with the callers' live
// state, and the epilogue would spill.)
template <int NO, int BN>
__device__ __noinline__ void sum_parts(uint32_t dst, const float4* const (&src)[4], int own) {
    constexpr int CPB = (2 / NO) > 0 ? 2 / NO : 1;   // 32-column chunks per batch
#pragma unroll 1
    for (int c0 = 0; c0 < BN; c0 += 32 * CPB) {
        float4 q[CPB][NO][8];
#pragma unroll
        for (int cb = 0; cb < CPB; ++cb)
            if (c0 + cb * 32 < BN)
#pragma unroll
                for (int o = 0; o < NO; ++o)
#pragma unroll
                    for (int i = 0; i < 8; ++i)
                        q[cb][o][i] = __ldcg(src[o] + size_t((c0 + cb * 32) / 4 + i) * kBM);
#pragma unroll
        for (int cb = 0; cb < CPB; ++cb) {
            if (c0 + cb * 32 >= BN) break;
            uint32_t r[32];
            if (own >= 0) {
                tmem_ld32(dst + uint32_t(c0 + cb * 32), r);
                tmem_ld_wait();
            }
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                const float4 mine = make_float4(__uint_as_float(r[4 * i]), __uint_as_float(r[4 * i + 1]),
                                                __uint_as_float(r[4 * i + 2]), __uint_as_float(r[4 * i + 3]));
                float4 sum = own == 0 ? mine : q[cb][0][i];
#pragma unroll
                for (int k = 1; k <= NO; ++k) {
                    if (own < 0 && k == NO) break;          // NO positions without an own part
                    // position k of the order: the own part, else global part k or k - 1
                    const float4 a = q[cb][k < NO ? k : NO - 1][i];
                    const float4 b = q[cb][k - 1][i];
                    const float4 v = k == own ? mine : ((own < 0 || k < own) ? a : b);
                    sum.x += v.x;
                    sum.y += v.y;
                    sum.z += v.z;
                    sum.w += v.w;
                }
                r[4 * i] = __float_as_uint(sum.x);
                r[4 * i + 1] = __float_as_uint(sum.y);
                r[4 * i + 2] = __float_as_uint(sum.z);
                r[4 * i + 3] = __float_as_uint(sum.w);
            }
            tmem_st32(dst + uint32_t(c0 + cb * 32), r);
        }
    }
    tmem_st_wait();
}

template <int BN, bool PAIR>
__global__ void __launch_bounds__(kThreads, 1) conv_kernel(const __grid_constant__ ConvParams p) {
    using C = CCfg<BN, PAIR>;
    constexpr int CM = C::CM;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                               ~uintptr_t(1023));
    __shared__ CBars bars;
    const uint32_t sA = smem_u32(smem);
    const uint32_t sB = sA + uint32_t(p.a_stages * p.a_bytes);
    const uint32_t sStg = sB + uint32_t(p.b_stages * p.b_stage);   // 1024-aligned
    volatile int* abort = &bars.abort_flag;
    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const int nkb = p.cin / kBK;
    const int nhalo = p.kt * nkb;              // halos (k-block groups) per tile
    const int sp = p.kh * p.kw;                // spatial taps per halo
    const int ngrp = sp / p.tb;                // weight-ring stages per halo
    const uint64_t lim = p.wait_limit_ns;
    const int rank = PAIR ? int(cluster_ctarank()) : 0;
    const bool leader = rank == 0;
    const int unit = blockIdx.x / CM;
    const int units = gridDim.x / CM;
    const long long s_begin = unit_start(p, unit, units, nhalo);
    const long long s_end = unit_start(p, unit + 1, units, nhalo);

    if (threadIdx.x == 0) {
        for (int s = 0; s < p.a_stages; ++s) {
            mbar_init(smem_u32(&bars.a_full[s]), 1);
            mbar_init(smem_u32(&bars.a_empty[s]), 1);
        }
        for (int s = 0; s < p.b_stages; ++s) {
            mbar_init(smem_u32(&bars.b_full[s]), 1);
            mbar_init(smem_u32(&bars.b_empty[s]), 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(smem_u32(&bars.acc_full[b]), 1);
            mbar_init(smem_u32(&bars.acc_empty[b]), 128 * CM);
        }
        mbar_init(smem_u32(&bars.drain), 1);
        mbar_init(smem_u32(&bars.part_full), 1);
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

    // Every loop below keeps its ring slot and phase in counters that wrap, and advances
    // coordinates and descriptors by additions: the single issuing threads must not spend
    // the tensor pipe's time on integer divisions between MMAs or copies.
    if (warp == 0) {
        // ================================ halo producer (TMA) ================================
        if (lane == 0) {
            tma_prefetch_map(&p.x_map);
            if (p.kt > 1) tma_prefetch_map(&p.c_map);
            int s = 0;
            uint32_t ph = 0;
            int ia = 0;
            bool ok = true;
            Items it{s_begin, s_end, nhalo, 0, 0, 0};
            while (ok && it.next()) {
                int f, th, tw, tn;
                tile_coords(p, it.t, CM, rank, f, th, tw, tn);
                const int cx = tw * kTileW - p.kw / 2;
                const int cy = th * kTileH - p.kh / 2;
                // halo hi = (temporal tap hi / nkb, channel block hi % nkb)
                int src = f - (p.kt - 1) + it.h0 / nkb;  // frame of (cache, chunk) - cache
                int kb = it.h0 % nkb;
                for (int hi = it.h0; hi < it.h1; ++hi, ++ia) {
                    if (ia >= p.a_stages && !mbar_test_wait(smem_u32(&bars.a_empty[s]), ph ^ 1) &&
                        !mbar_wait(smem_u32(&bars.a_empty[s]), ph ^ 1, lim, abort)) {
                        report(p.status, abort, 0, ia);
                        ok = false;
                        break;
                    }
                    const CUtensorMap* amap = src < 0 ? &p.c_map : &p.x_map;
                    const int az = src < 0 ? src + p.kt - 1 : src;
                    const uint32_t dst = sA + uint32_t(s * p.a_bytes);
                    if (PAIR) {
                        if (leader) mbar_arrive_expect_tx(smem_u32(&bars.a_full[s]), 2 * p.halo_tx);
                        tma_load_4d_pair(dst, amap, mapa_shared(smem_u32(&bars.a_full[s]), 0),
                                         kb * kBK, cx, cy, az);
                    } else {
                        mbar_arrive_expect_tx(smem_u32(&bars.a_full[s]), p.halo_tx);
                        tma_load_4d(dst, amap, smem_u32(&bars.a_full[s]), kb * kBK, cx, cy, az);
                    }
                    if (++s == p.a_stages) {
                        s = 0;
                        ph ^= 1;
                    }
                    if (++kb == nkb) {
                        kb = 0;
                        ++src;
                    }
                }
            }
            if (leader)
                for (int i = (ia > p.a_stages ? ia - p.a_stages : 0); i < ia; ++i)
                    mbar_wait_drain(smem_u32(&bars.a_full[i % p.a_stages]), (i / p.a_stages) & 1, lim);
        }
    } else if (warp == 6) {
        // ================================ weight producer (TMA) ==============================
        if (lane == 0) {
            tma_prefetch_map(&p.w_map);
            int s = 0;
            uint32_t ph = 0;
            int ib = 0;
            bool ok = true;
            Items it{s_begin, s_end, nhalo, 0, 0, 0};
            while (ok && it.next()) {
                const int n0 = (it.t % p.tiles_n) * BN + rank * (BN / CM);
                int kb = it.h0 % nkb;
                int tap0 = (it.h0 / nkb) * sp;            // first tap of this temporal tap
                for (int hi = it.h0; hi < it.h1 && ok; ++hi) {
                    for (int g = 0; g < ngrp; ++g, ++ib) {
                        if (ib >= p.b_stages && !mbar_test_wait(smem_u32(&bars.b_empty[s]), ph ^ 1) &&
                            !mbar_wait(smem_u32(&bars.b_empty[s]), ph ^ 1, lim, abort)) {
                            report(p.status, abort, 3, ib);
                            ok = false;
                            break;
                        }
                        const uint32_t dst = sB + uint32_t(s * p.b_stage);
                        const int tap = tap0 + g * p.tb;
                        if (PAIR) {
                            if (leader) mbar_arrive_expect_tx(smem_u32(&bars.b_full[s]), 2 * p.b_stage);
                            tma_load_3d_pair(dst, &p.w_map, mapa_shared(smem_u32(&bars.b_full[s]), 0),
                                             kb * kBK, n0, tap);
                        } else {
                            mbar_arrive_expect_tx(smem_u32(&bars.b_full[s]), p.b_stage);
                            tma_load_3d(dst, &p.w_map, smem_u32(&bars.b_full[s]), kb * kBK, n0, tap);
                        }
                        if (++s == p.b_stages) {
                            s = 0;
                            ph ^= 1;
                        }
                    }
                    if (++kb == nkb) {
                        kb = 0;
                        tap0 += sp;
                    }
                }
            }
            if (leader)
                for (int i = (ib > p.b_stages ? ib - p.b_stages : 0); i < ib; ++i)
                    mbar_wait_drain(smem_u32(&bars.b_full[i % p.b_stages]), (i / p.b_stages) & 1, lim);
        }
    } else if (warp == 1) {
        // ============ MMA issuer (a converged warp of the leader; lane 0 issues) ============
        // The warp never touches an mbarrier in its loops: the observer warp (warp 7) waits
        // for every barrier the next MMAs need and meets it at the hand-off named barrier.
        // (A shared-memory access by the issuing thread behind queued MMAs waits behind
        // their operand reads, ~400 cycles per weight stage measured; a named barrier reads
        // no shared memory.) Both warps pass the same barriers in the same order whatever
        // happens, so neither can strand the other.
        if (leader) {
            const uint32_t lead = lane == 0 ? 1u : 0u;
            auto handoff = [&]() {
                named_bar_sync(kBarHandoff, 64);
                tc_fence_after();
            };
            // descriptors are linear in the 16-byte start address (addresses stay below
            // 256 KB, so the 14-bit field never carries): tap (dh, dw) of halo stage sa
            // is da0 + sa * a_step + dh * halo_w * 8 + dw, k-step k adds 2 k
            const uint64_t da0 = sdesc_sw128(sA, 16, uint32_t(p.halo_w * 128));
            const uint64_t db0 = sdesc_sw128(sB, 16, 1024);
            const uint32_t a_step = uint32_t(p.a_bytes >> 4);
            const uint32_t row_skip = uint32_t((p.halo_w - p.kw) * 8);
            const uint32_t b_step = uint32_t(p.b_stage >> 4);
            int sa = 0, sb = 0;
            int tl = 0;
            Items it{s_begin, s_end, nhalo, 0, 0, 0};
            for (; it.next(); ++tl) {
                const int b = tl & 1;
                if (tl >= 2) handoff();                      // accumulator b drained
                const uint32_t d = tmem + uint32_t(b * BN);
                uint32_t accumulate = 0;
                for (int hi = it.h0; hi < it.h1; ++hi) {
                    handoff();                               // halo stage sa landed
                    uint64_t da = da0 + uint64_t(uint32_t(sa) * a_step);
                    // a weight stage holds tb consecutive taps of one kernel row: one
                    // hand-off per tb * 4 MMAs
                    for (int dh = 0; dh < p.kh; ++dh, da += row_skip) {
                        for (int dw = 0; dw < p.kw; dw += p.tb) {
                            handoff();                       // weight stage sb landed
                            uint64_t db = db0 + uint64_t(uint32_t(sb) * b_step);
                            for (int u = 0; u < p.tb; ++u, da += 8, db += uint64_t(C::B_BYTES >> 4)) {
#pragma unroll
                                for (int k = 0; k < kBK / 16; ++k) {
                                    if (PAIR)
                                        umma_ss_pair_if(lead, d, da + uint64_t(2 * k),
                                                        db + uint64_t(2 * k), C::IDESC, accumulate);
                                    else
                                        umma_ss_if(lead, d, da + uint64_t(2 * k), db + uint64_t(2 * k),
                                                   C::IDESC, accumulate);
                                    accumulate = 1;
                                }
                            }
                            if (PAIR) umma_commit_pair_if(lead, smem_u32(&bars.b_empty[sb]), 0x3);
                            else umma_commit_if(lead, smem_u32(&bars.b_empty[sb]));
                            if (++sb == p.b_stages) sb = 0;
                        }
                    }
                    if (PAIR) umma_commit_pair_if(lead, smem_u32(&bars.a_empty[sa]), 0x3);
                    else umma_commit_if(lead, smem_u32(&bars.a_empty[sa]));
                    if (++sa == p.a_stages) sa = 0;
                }
                if (PAIR) umma_commit_pair_if(lead, smem_u32(&bars.acc_full[b]), 0x3);
                else umma_commit_if(lead, smem_u32(&bars.acc_full[b]));
            }
            if (PAIR) umma_commit_pair_if(lead, smem_u32(&bars.drain), 0x1);
            else umma_commit_if(lead, smem_u32(&bars.drain));
            mbar_wait_drain(smem_u32(&bars.drain), 0, lim);
        }
    } else if (warp == 7) {
        // ======== observer (leader): waits for what the issuer's next MMAs need ========
        // After a wait gives up (or another role raised the abort flag) the remaining
        // hand-offs pass without waiting; the issuer then finishes on stale operands, which
        // the recorded error status marks as void.
        if (leader) {
            bool ok = true;
            auto observe = [&](uint32_t bar, uint32_t parity, int role, int where) {
                if (ok) {
                    ok = __all_sync(0xffffffffu, mbar_wait(bar, parity, lim, abort));
                    if (!ok && lane == 0) report(p.status, abort, role, where);
                }
                named_bar_sync(kBarHandoff, 64);
            };
            int sa = 0, sb = 0;
            uint32_t pa = 0, pb = 0;
            int ia = 0, ib = 0;
            int tl = 0;
            Items it{s_begin, s_end, nhalo, 0, 0, 0};
            for (; it.next(); ++tl) {
                const int b = tl & 1;
                if (tl >= 2) observe(smem_u32(&bars.acc_empty[b]), ((tl >> 1) - 1) & 1, 1, -1 - tl);
                for (int hi = it.h0; hi < it.h1; ++hi, ++ia) {
                    observe(smem_u32(&bars.a_full[sa]), pa, 1, ia);
                    for (int dh = 0; dh < p.kh; ++dh)
                        for (int dw = 0; dw < p.kw; dw += p.tb, ++ib) {
                            observe(smem_u32(&bars.b_full[sb]), pb, 4, ib);
                            if (++sb == p.b_stages) {
                                sb = 0;
                                pb ^= 1;
                            }
                        }
                    if (++sa == p.a_stages) {
                        sa = 0;
                        pa ^= 1;
                    }
                }
            }
        }
    } else {
        // ====================================== epilogue =====================================
        const int sub = warp & 3;
        const int row = sub * 32 + lane;                 // pixel of the tile: 8 per row
        const uint32_t lane_off = uint32_t(sub * 32) << 16;
        const uint32_t sw = uint32_t(row & 7);
        const bool est = threadIdx.x == 64;              // issues the tile's TMA stores
        const int ucols = p.y_bf16 ? 64 : 32;            // output channels per unit
        if (p.shift_keep > 0) {
            // this CTA's slice of the next cache, while the first tile's MMAs run
            const long long nvec = p.shift_frame_vec * p.shift_keep;
            const long long per = (nvec + gridDim.x - 1) / gridDim.x;
            const long long lo = per * blockIdx.x;
            const long long hi = lo + per < nvec ? lo + per : nvec;
            for (long long i = lo + (threadIdx.x - 64); i < hi; i += 128) {
                const int j = int(i / p.shift_frame_vec);
                const long long r = i - (long long)j * p.shift_frame_vec;
                const int src = j + p.F;                     // frame of (cache, chunk)
                p.shift_next[i] = src < p.shift_keep
                                      ? __ldg(p.shift_cache + (long long)src * p.shift_frame_vec + r)
                                      : __ldg(p.shift_x + (long long)(src - p.shift_keep) * p.shift_frame_vec + r);
            }
        }
        int tl = 0;
        uint32_t part_phase = 0;                          // parity of bars.part_full
        Items it{s_begin, s_end, nhalo, 0, 0, 0};
        for (; it.next(); ++tl) {
            const int b = tl & 1;
            int f, th, tw, tn;
            tile_coords(p, it.t, CM, rank, f, th, tw, tn);
            // the tile's bias slice, read once (the barriers below pass before its use, and
            // the previous tile's last use precedes a barrier every thread has passed)
            if (row < BN / 4) bars.bias[row] = __ldg(reinterpret_cast<const float4*>(p.bias + tn * BN) + row);
            const uint32_t acc = tmem + lane_off + uint32_t(b * BN);
            const uint32_t acc2 = tmem + lane_off + uint32_t((b ^ 1) * BN);   // the idle buffer
            // A split tile: its parts come from units first .. first + n_parts - 1 (part
            // k = unit - first covers the k-th piece of its halo steps) and are summed as
            // ((part 1 + ... + part n-1) + part 0).
            const bool split = it.h0 != 0 || it.h1 != nhalo;
            int n_parts = 1, first = unit;
            long long ts = 0;
            int* ctr = nullptr;
            if (split) {
                ts = (long long)it.t * nhalo;
                first = unit_of(p, ts, units);
                n_parts = unit_of(p, ts + nhalo - 1, units) - first + 1;
                ctr = p.counters + size_t(it.t) * CM + rank;
            }
            const int kpart = unit - first;
            if (n_parts > 3) {                               // excluded by the plan
                if (est) report(p.status, abort, 5, it.t);
                break;
            }
#ifdef FRT_DEBUG
            // every workspace row and counter a split tile touches lies inside the
            // allocations; a tile that fails records FRT_ERR_BOUNDS and the epilogue
            // stops (the abort flag ends the other roles' waits)
            if (split) {
                bool bad = n_parts < 2 || kpart < 0 || kpart >= n_parts ||
                           (long long)(it.t + 1) * CM > p.ctr_cap;
                for (int k = 0; k < n_parts && !bad; ++k)
                    bad = (long long)(part_slot(p, first + k, ts, units, nhalo) * CM + rank + 1) *
                              (BN / 4) * kBM > p.part_cap;
                if (bad) {
                    if (est) {
                        *abort = 1;
                        record_status(p.status, kStatusBounds, 307, it.t);
                    }
                    break;
                }
            }
#endif
            auto part_row = [&](int k) {                     // this thread's row of part k
                return p.part + (size_t(part_slot(p, first + k, ts, units, nhalo)) * CM + rank) *
                                    (BN / 4) * kBM + row;
            };
            auto other = [&](int j) -> const float4* {       // j-th other part in sum order
                const int k = kpart == 0 ? j + 1 : (j < kpart - 1 ? j + 1 : (j < n_parts - 2 ? j + 2 : 0));
                return part_row(k);
            };
            // TMEM dst = the sum of the other parts and, at position own of the order (-1:
            // none), this CTA's part already in dst
            auto sum_into = [&](uint32_t dst, int own) {
                const int no = n_parts - 1;
                // the plan gives every unit at least half a tile of steps: <= 3 parts
                const float4* src[4];
#pragma unroll
                for (int o = 0; o < 4; ++o) src[o] = o < no ? other(o) : nullptr;
                if (no == 1) sum_parts<1, BN>(dst, src, own);
                else sum_parts<2, BN>(dst, src, own);
            };
            // Part 0 is this unit's last item. While its MMAs run, watch the tile's arrival
            // word (part k sets bit k): every other part that has arrived is added into the
            // idle buffer at once, so that part 0 adds itself at the end with no round trip
            // through memory. With at most two other parts their sum is the same in either
            // arrival order (two-operand addition commutes). The watch ends when this
            // CTA's accumulator is ready; parts still missing then get a bounded wait
            // (below), and past it everything goes the write-and-arrive way. No wait here
            // needs another CTA to be resident to end.
            const int others = (1 << n_parts) - 2;           // bits of parts 1 .. n-1
            int loaded = 0;                                   // parts summed into acc2
            auto take = [&](int fresh) {                      // add newly arrived parts
                __threadfence();
                const float4* src[4] = {nullptr, nullptr, nullptr, nullptr};
                if (fresh == 6) {                             // parts 1 and 2 together
                    src[0] = part_row(1);
                    src[1] = part_row(2);
                    sum_parts<2, BN>(acc2, src, -1);
                } else {                                      // one part: the first, or added
                    src[0] = part_row((fresh & 2) ? 1 : 2);
                    sum_parts<1, BN>(acc2, src, loaded != 0 ? 0 : -1);
                }
                loaded |= fresh;
            };
            if (split && kpart == 0 && p.part_mode == 0) {
                const uint64_t t0 = globaltimer_ns();
                for (;;) {
                    if (est) {
                        int st = ld_acquire_gpu(ctr) & others;
                        if (mbar_test_wait(smem_u32(&bars.acc_full[b]), (tl >> 1) & 1)) st |= 1 << 16;
                        else if (*abort != 0 || globaltimer_ns() - t0 > lim) st |= 1 << 17;
                        bars.last_part = st;
                    }
                    named_bar_sync(1, 128);
                    const int st = *reinterpret_cast<volatile int*>(&bars.last_part);
                    named_bar_sync(1, 128);
                    if ((st >> 16) != 0) break;                // accumulator ready: bulk path
                    const int fresh = st & others & ~loaded;
                    if (fresh != 0) take(fresh);
                    if (loaded == others) break;
                    __nanosleep(500);
                }
            }
            const bool got = mbar_wait(smem_u32(&bars.acc_full[b]), (tl >> 1) & 1, lim, abort);
            // all four warps go on or stop together: the staging below synchronises them
            if (!named_bar_and(1, 128, got)) {
                if (!got) report(p.status, abort, 2, tl);
                break;
            }
            tc_fence_after();
            bool early_ready = false;
            if (split && kpart == 0 && p.part_mode != 2) {
                // Part 0, accumulator ready: the parts still missing are usually a few
                // microseconds from arriving (a unit whose whole share lies inside this tile
                // ends when this one does). Give them kPartWaitNs, taking each as it lands;
                // reading one part then is cheaper than writing this one and having the
                // last arrival read them all. Past that, write and arrive as below.
                // This is the unit's last item, so its MMAs are done and the halo and
                // weight rings are idle: a part that lands now is brought in by bulk copies
                // (16 KB per 32 columns) and added from shared memory, which keeps many
                // more bytes in flight than loads into registers can.
                const uint32_t ring_bytes = uint32_t(p.a_stages * p.a_bytes + p.b_stages * p.b_stage);
                const bool bulk = ring_bytes >= uint32_t(kBM * BN * 4);
                const uint64_t t0 = globaltimer_ns();
                bool bad = false;
                while (loaded != others && !bad) {
                    if (est) {
                        int st = ld_acquire_gpu(ctr) & others;
                        if (*abort != 0 || globaltimer_ns() - t0 > kPartWaitNs) st |= 1 << 16;
                        bars.last_part = st;
                    }
                    named_bar_sync(1, 128);
                    const int st = *reinterpret_cast<volatile int*>(&bars.last_part);
                    named_bar_sync(1, 128);
                    const int fresh = st & others & ~loaded;
                    if (fresh != 0 && !bulk) take(fresh);
                    for (int k = 1; bulk && k < n_parts; ++k) {
                        if ((fresh & (1 << k)) == 0) continue;
                        const float4* blk = p.part + (size_t(part_slot(p, first + k, ts, units, nhalo)) * CM + rank) *
                                                         (BN / 4) * kBM;
                        if (est) {
                            fence_proxy_async_global();
                            mbar_arrive_expect_tx(smem_u32(&bars.part_full), uint32_t(kBM * BN * 4));
                            for (int c = 0; c < BN; c += 32)
                                bulk_load(sA + uint32_t(c * kBM * 4), blk + size_t(c / 4) * kBM,
                                          uint32_t(32 * kBM * 4), smem_u32(&bars.part_full));
                        }
                        const bool in = __all_sync(0xffffffffu, mbar_wait(smem_u32(&bars.part_full), part_phase, lim, abort));
                        part_phase ^= 1;
                        if (!named_bar_and(1, 128, in)) {
                            if (est) report(p.status, abort, 6, it.t);
                            bad = true;
                            break;
                        }
                        // acc2 = that part (the first taken) or acc2 + it (two-operand sums
                        // commute, so the arrival order does not matter)
#pragma unroll 1
                        for (int c = 0; c < BN; c += 32) {
                            uint32_t r[32];
                            if (loaded != 0) {
                                tmem_ld32(acc2 + uint32_t(c), r);
                                tmem_ld_wait();
                            }
#pragma unroll
                            for (int i = 0; i < 8; ++i) {
                                const uint4 q = ld_shared_v4(sA + uint32_t(((c / 4 + i) * kBM + row) * 16));
                                if (loaded != 0) {
                                    r[4 * i] = __float_as_uint(__uint_as_float(r[4 * i]) + __uint_as_float(q.x));
                                    r[4 * i + 1] = __float_as_uint(__uint_as_float(r[4 * i + 1]) + __uint_as_float(q.y));
                                    r[4 * i + 2] = __float_as_uint(__uint_as_float(r[4 * i + 2]) + __uint_as_float(q.z));
                                    r[4 * i + 3] = __float_as_uint(__uint_as_float(r[4 * i + 3]) + __uint_as_float(q.w));
                                } else {
                                    r[4 * i] = q.x;
                                    r[4 * i + 1] = q.y;
                                    r[4 * i + 2] = q.z;
                                    r[4 * i + 3] = q.w;
                                }
                            }
                            tmem_st32(acc2 + uint32_t(c), r);
                        }
                        tmem_st_wait();
                        loaded |= 1 << k;
                        named_bar_sync(1, 128);               // the ring is read before the next copy
                    }
                    if ((st >> 16) != 0) break;
                    if (loaded != others && !bad) __nanosleep(256);
                }
                if (bad) break;
                early_ready = loaded == others;
                if (early_ready && est) *ctr = 0;             // parts 1 .. n-1 arrived, 0 did not
            }
            if (split && !early_ready) {
                // any other case: the part is written out and counted, and the one that
                // completes the count adds them all
                bool adder;
                {
                    float4* mine = part_row(kpart);
#pragma unroll 1
                    for (int c = 0; c < BN; c += 32) {
                        uint32_t r[32];
                        tmem_ld32(acc + uint32_t(c), r);
                        tmem_ld_wait();
#pragma unroll
                        for (int i = 0; i < 8; ++i)
                            mine[size_t(c / 4 + i) * kBM] =
                                make_float4(__uint_as_float(r[4 * i]), __uint_as_float(r[4 * i + 1]),
                                            __uint_as_float(r[4 * i + 2]), __uint_as_float(r[4 * i + 3]));
                    }
                    named_bar_sync(1, 128);
                    if (est) {
                        // publishes the part (every thread's stores precede the barrier)
                        const int bit = 1 << kpart;
                        const int old = atom_add_acq_rel_gpu(ctr, bit);
                        const int last = old + bit == (1 << n_parts) - 1;
                        if (last) *ctr = 0;                  // every part has arrived
                        bars.last_part = last;
                    }
                    named_bar_sync(1, 128);
                    adder = *reinterpret_cast<volatile int*>(&bars.last_part) != 0;
                    named_bar_sync(1, 128);
                }
                if (!adder) {
                    tc_fence_before();
                    if (PAIR) mbar_arrive_cluster(mapa_shared(smem_u32(&bars.acc_empty[b]), 0));
                    else mbar_arrive(smem_u32(&bars.acc_empty[b]));
                    continue;
                }
                __threadfence();                             // the other parts are visible
                sum_into(acc, kpart == 0 ? n_parts - 1 : kpart - 1);
            }
            // On the unit's last item the rings are idle: every column unit gets its own
            // slab there and the stores go out together, instead of one slab in turn.
            const bool wide = it.s >= s_end &&
                              p.a_stages * p.a_bytes + p.b_stages * p.b_stage >= (BN / ucols) * kSlab;
#pragma unroll 1
            for (int u = 0; u < BN / ucols; ++u) {
                // the unit's 32 words per thread are computed before the slab is claimed,
                // so the previous store's read of the slab overlaps this work
                uint32_t o[32];
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    if (h == 1 && !p.y_bf16) break;
                    const int c = u * ucols + h * 32;    // first column of this TMEM load
                    uint32_t r[32];
                    tmem_ld32(acc + uint32_t(c), r);
                    tmem_ld_wait();
                    float v[32];
#pragma unroll
                    for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
                    if (early_ready) {                       // (parts 1 .. n-1) + part 0
                        tmem_ld32(acc2 + uint32_t(c), r);
                        tmem_ld_wait();
#pragma unroll
                        for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]) + v[i];
                    }
#pragma unroll
                    for (int i = 0; i < 8; ++i) {
                        const float4 bb = bars.bias[c / 4 + i];
                        v[4 * i] += bb.x;
                        v[4 * i + 1] += bb.y;
                        v[4 * i + 2] += bb.z;
                        v[4 * i + 3] += bb.w;
                    }
                    if (p.y_bf16) {
#pragma unroll
                        for (int i = 0; i < 16; ++i) o[16 * h + i] = pack_bf16x2(v[2 * i], v[2 * i + 1]);
                    } else {
#pragma unroll
                        for (int i = 0; i < 32; ++i) o[i] = __float_as_uint(v[i]);
                    }
                }
                const uint32_t slab = wide ? sA + uint32_t(u * kSlab) : sStg;
                if (!wide) {
                    if (est) bulk_wait_read<0>();        // the previous store has read the slab
                    named_bar_sync(1, 128);
                }
                const uint32_t rbu = slab + uint32_t(row * 128);
#pragma unroll
                for (int i = 0; i < 8; ++i)
                    st_shared_v4(rbu + ((uint32_t(i) ^ sw) << 4), o[4 * i], o[4 * i + 1], o[4 * i + 2],
                                 o[4 * i + 3]);
                if (!wide) {
                    fence_proxy_async_smem();
                    named_bar_sync(1, 128);
                    if (est && f < p.F) {
                        tma_store_4d(&p.y_map, sStg, tn * BN + u * ucols, tw * kTileW, th * kTileH, f);
                        bulk_commit();
                    }
                }
            }
            if (wide) {
                fence_proxy_async_smem();
                named_bar_sync(1, 128);
                if (est && f < p.F) {
                    for (int u = 0; u < BN / ucols; ++u)
                        tma_store_4d(&p.y_map, sA + uint32_t(u * kSlab), tn * BN + u * ucols, tw * kTileW,
                                     th * kTileH, f);
                    bulk_commit();
                }
            }
            tc_fence_before();
            if (PAIR) mbar_arrive_cluster(mapa_shared(smem_u32(&bars.acc_empty[b]), 0));
            else mbar_arrive(smem_u32(&bars.acc_empty[b]));
        }
        // the stores have read their slabs before the CTA exits (their writes complete
        // with the grid)
        if (est) bulk_wait_read<0>();
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

template <int BN, bool PAIR>
cudaError_t launch_conv(ConvParams p, int units, cudaStream_t st) {
    using C = CCfg<BN, PAIR>;
    const int smem = p.a_stages * p.a_bytes + p.b_stages * p.b_stage + kSlab + 1024;
    static int attr[kMaxDevices] = {};   // per device: the largest size set so far
    const int dev = device_slot();
    if (dev < 0 || smem > attr[dev]) {
        cudaError_t e = cudaFuncSetAttribute(conv_kernel<BN, PAIR>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
        if (e != cudaSuccess) return e;
        if (dev >= 0) attr[dev] = smem;
    }
    if (!PAIR) {
        conv_kernel<BN, false><<<units, kThreads, smem, st>>>(p);
        return cudaGetLastError();
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(unsigned(units * 2));
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = smem;
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
            const cuuint32_t* box, bool f32 = false) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return false;
    cuuint64_t strides[3];
    cuuint64_t acc = dims[0] * (f32 ? 4 : 2);
    for (int i = 0; i + 1 < rank; ++i) {
        strides[i] = acc;
        acc *= dims[i + 1];
    }
    cuuint32_t estr[4] = {1, 1, 1, 1};
    return fn(map, f32 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, rank,
              const_cast<void*>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
              CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Ring plan for one tile shape: a weight stage holds a whole kernel row of taps (tb = kw)
// when three such stages fit beside the halo ring, else one tap; three halos in flight
// when that leaves room for three weight stages, else two. Returns false if even two
// halo and two weight stages do not fit.
bool plan_rings(int a_bytes, int b_bytes, int kw, int& tb, int& a_stages, int& b_stages) {
    const int room = kSmemBudget - 1024 - kSlab;
    tb = 1;
    a_stages = 2;
    bool found = false;
    for (int t : {kw, 1})
        for (int as = 3; as >= 2 && !found; --as)
            if (room - as * a_bytes >= 3 * t * b_bytes) {
                tb = t;
                a_stages = as;
                found = true;
            }
    b_stages = std::min(kMaxStages, (room - a_stages * a_bytes) / (tb * b_bytes));
    return b_stages >= 2;
}

int g_conv_part_mode = 0;   // self-test override (frt_selftest_conv_part_mode)

// Launch plan of one chunk: tile width, pairing, rings, units and whether tiles are split.
struct ConvPlan {
    int bn = 0;
    bool pair = false;
    int tb = 1, a_stages = 2, b_stages = 2;
    int tiles_n = 0, n_tiles = 0;
    int units = 0;             // CTAs, or CTA pairs
    bool split = false;
    long long total = 0;       // n_tiles * halos per tile
};

// Cycles per spatial tap (four MMAs of K 16 and their share of the ring hand-offs),
// fitted to clock traces and timings of this kernel on GB300: single CTAs are bound by
// shared-memory operand reads (A, B and the weight copies), about 3.5 cycles per output
// channel of the tile, with a floor of about 450; CTA pairs read half of B each and
// take about 570 cycles per tap up to BN 192. A weight stage of one tap adds about 300.
double tap_cycles(int bn, bool pair, int tb, int kw) {
    const double t = pair ? std::max(570.0, 2.3 * bn) : std::max(450.0, 3.5 * bn);
    return t + (tb == 1 && kw > 1 ? 300.0 : 0.0);
}

// Cycles a split tile's last part spends beyond its MMAs: writing its part, reading the
// others and the store (measured 1-2 us at the VAE sizes).
constexpr double kSplitCycles = 3000.0;

// split_mode: 0 automatic, 1 whole tiles only, 2 split whenever units do not divide the
// tiles evenly. units_req: 0 = every SM (or SM pair), else at most that many units.
// bn_req / pair_req: 0 = automatic tile. Returns false if nothing fits.
bool plan_conv(int cin, int cout, int kt, int kh, int kw, int H, int W, int F, bool y_bf16,
               int bn_req, int pair_req, int split_mode, int units_req, int sms, ConvPlan& out) {
    const int halo_w = kTileW + kw - 1, halo_h = kTileH + kh - 1;
    const int a_bytes = (halo_w * halo_h * kBK * 2 + 1023) & ~1023;
    const long long m_tiles =
        (long long)F * ((W + kTileW - 1) / kTileW) * ((H + kTileH - 1) / kTileH);
    const int nhalo = kt * (cin / kBK);
    const int sp = kh * kw;
    const int cands[5] = {256, 192, 128, 96, 64};
    double best_t = 1e300;
    bool found = false;
    for (int pr = 0; pr < 2; ++pr) {
        if (bn_req != 0 && pr != pair_req) continue;
        if (pr == 1 && m_tiles < 2 && bn_req == 0) continue;
        const int cm = pr ? 2 : 1;
        const long long m_units = (m_tiles + cm - 1) / cm;
        long long all = sms / cm;
        if (units_req > 0) all = std::min<long long>(all, units_req);
        for (int bn : cands) {
            if (bn_req != 0 && bn != bn_req) continue;
            if (cout % bn || (y_bf16 && bn % 64)) continue;
            ConvPlan c;
            c.bn = bn;
            c.pair = pr == 1;
            if (!plan_rings(a_bytes, (bn / cm) * kBK * 2, kw, c.tb, c.a_stages, c.b_stages)) continue;
            c.tiles_n = cout / bn;
            if (m_units * c.tiles_n >= (1LL << 31)) continue;
            c.n_tiles = int(m_units * c.tiles_n);
            c.total = (long long)c.n_tiles * nhalo;
            const double halo = sp * tap_cycles(bn, c.pair, c.tb, kw);
            // whole tiles in rounds over the units
            const long long uw = std::min<long long>(all, c.n_tiles);
            const double t_whole = double((c.n_tiles + uw - 1) / uw) * nhalo * halo;
            // split: every unit takes an equal share of the halo steps, at least half a
            // tile's, so that a tile has at most three parts
            const long long us = std::min<long long>(all, c.total / ((nhalo + 1) / 2));
            const double t_split = double((c.total + us - 1) / us) * halo + kSplitCycles;
            const bool uneven = c.n_tiles % uw != 0 || uw < all;
            c.split = split_mode == 2 ? (c.n_tiles % us != 0 || us > c.n_tiles)
                    : split_mode == 1 ? false
                                      : (uneven && t_split < t_whole);
            c.units = int(c.split ? us : uw);
            const double t = c.split ? t_split : t_whole;
            if (t < best_t - 1e-9) {
                best_t = t;
                out = c;
                found = true;
            }
        }
    }
    return found;
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
    int force_bn = 0;      // 0: the cost model picks the tile
    int force_pair = 0;
    int split_mode = 0;    // 0 automatic, 1 whole tiles, 2 split when uneven
    int split_units = 0;   // 0: every SM (or SM pair)
    // split tiles: parts [2 * units][pair][BN][128] fp32 and one arrival counter per
    // tile and pair rank, sized for the current plan
    void* part = nullptr;
    size_t part_bytes = 0;
    int* counters = nullptr;
    size_t n_counters = 0;
};

namespace {
frt_status cfail(frt_status st, const char* msg) {
    set_last_error(msg);
    return st;
}
// A CUDA runtime call of this layer failed (see clear_cuda_error).
frt_status cuda_cfail(frt_status st, const char* msg) {
    clear_cuda_error();
    return cfail(st, msg);
}
bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
void free_conv(frt_conv_t* c) {
    for (int i = 0; i < 2; ++i)
        if (c->cache[i]) cudaFree(c->cache[i]);
    if (c->status_host) cudaFreeHost(c->status_host);
    if (c->part) cudaFree(c->part);
    if (c->counters) cudaFree(c->counters);
    c->cache[0] = c->cache[1] = nullptr;
    c->status_host = c->status_dev = nullptr;
    c->part = nullptr;
    c->counters = nullptr;
    c->part_bytes = c->n_counters = 0;
}

bool conv_plan(const frt_conv_t* c, ConvPlan& pl) {
    return plan_conv(c->cin, c->cout, c->kt, c->kh, c->kw, c->H, c->W, c->F,
                     c->out_dtype == FRT_OUT_BF16, c->force_bn, c->force_pair, c->split_mode,
                     c->split_units, num_sms(), pl);
}

// Size the split workspace for the current plan (grows only; synchronises before it
// frees). Called where the plan can change: configure and the tuning setters.
frt_status ensure_split_scratch(frt_conv_t* c) {
    ConvPlan pl;
    if (!conv_plan(c, pl) || !pl.split) return FRT_OK;     // step reports an unfit plan
    const int cm = pl.pair ? 2 : 1;
    const size_t need = size_t(2) * pl.units * cm * kBM * pl.bn * sizeof(float);
    const size_t n_ctr = size_t(pl.n_tiles) * cm;
    cudaError_t e = cudaSuccess;
    if (need > c->part_bytes || n_ctr > c->n_counters) {
        if ((e = cudaStreamSynchronize(c->cs)) != cudaSuccess) return cuda_cfail(FRT_ERR_CUDA, "sync failed");
    }
    if (need > c->part_bytes) {
        if (c->part) cudaFree(c->part);
        c->part = nullptr;
        c->part_bytes = 0;
        if ((e = cudaMalloc(&c->part, need)) != cudaSuccess)
            return cuda_cfail(e == cudaErrorMemoryAllocation ? FRT_ERR_OOM : FRT_ERR_CUDA,
                              "split workspace allocation failed");
        c->part_bytes = need;
    }
    if (n_ctr > c->n_counters) {
        if (c->counters) cudaFree(c->counters);
        c->counters = nullptr;
        c->n_counters = 0;
        if ((e = cudaMalloc(&c->counters, n_ctr * sizeof(int))) != cudaSuccess ||
            (e = cudaMemset(c->counters, 0, n_ctr * sizeof(int))) != cudaSuccess ||
            (e = cudaDeviceSynchronize()) != cudaSuccess)
            return cuda_cfail(e == cudaErrorMemoryAllocation ? FRT_ERR_OOM : FRT_ERR_CUDA,
                              "split counter allocation failed");
        c->n_counters = n_ctr;
    }
    return FRT_OK;
}
}  // namespace

extern "C" {

frt_conv_t* frt_conv_create(int cin, int cout, int kt, int kh, int kw, int grid_h, int grid_w,
                            int frames_per_chunk) {
    if (cin < 64 || cin % 64 || cout < 64 || cout % 64 || kt < 1 || kt > 4 || kh < 1 || kh > 7 ||
        kw < 1 || kw > 7 || kh % 2 == 0 || kw % 2 == 0 || grid_h < 1 || grid_w < 1 ||
        frames_per_chunk < 1 || (long long)grid_h * grid_w > (1LL << 24)) {
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
                return cuda_cfail(e == cudaErrorMemoryAllocation ? FRT_ERR_OOM : FRT_ERR_CUDA,
                                  "frame cache allocation failed");
            }
        if ((e = cudaHostAlloc(reinterpret_cast<void**>(&c->status_host), sizeof(DeviceStatus),
                               cudaHostAllocMapped)) != cudaSuccess ||
            (e = cudaHostGetDevicePointer(reinterpret_cast<void**>(&c->status_dev), c->status_host,
                                          0)) != cudaSuccess) {
            free_conv(c);
            return cuda_cfail(FRT_ERR_CUDA, "status allocation failed");
        }
        std::memset(c->status_host, 0, sizeof(DeviceStatus));
        if ((e = cudaDeviceSynchronize()) != cudaSuccess) return cuda_cfail(FRT_ERR_CUDA, "sync failed");
    }
    c->out_dtype = out_dtype;
    c->cs = static_cast<cudaStream_t>(cuda_stream);
    c->configured = true;
    return ensure_split_scratch(c);
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
    p.halo_w = kTileW + c->kw - 1;
    p.halo_h = kTileH + c->kh - 1;
    p.halo_tx = p.halo_w * p.halo_h * kBK * 2;
    p.a_bytes = (p.halo_tx + 1023) & ~1023;
    const bool y_bf16 = c->out_dtype == FRT_OUT_BF16;
    if (y_bf16 && c->force_bn % 64)
        return cfail(FRT_ERR_UNSUPPORTED, "a bf16 output needs a tile width that is a multiple of 64");
    ConvPlan pl;
    if (!conv_plan(c, pl))
        return cfail(FRT_ERR_UNSUPPORTED, "no tile width fits Cout and the shared-memory rings");
    const int bn = pl.bn;
    const bool pair = pl.pair;
    const int b_bytes = (pair ? bn / 2 : bn) * kBK * 2;
    p.tb = pl.tb;
    p.a_stages = pl.a_stages;
    p.b_stages = pl.b_stages;
    p.b_stage = p.tb * b_bytes;
    p.tiles_n = pl.tiles_n;
    p.n_tiles = pl.n_tiles;
    p.total = pl.total;
    p.split = pl.split ? 1 : 0;
    if (pl.split) {
        const int cm = pair ? 2 : 1;
        if (size_t(2) * pl.units * cm * kBM * bn * sizeof(float) > c->part_bytes ||
            size_t(pl.n_tiles) * cm > c->n_counters)
            return cfail(FRT_ERR_STATE, "split workspace missing: configure the conv again");
        p.part = static_cast<float4*>(c->part);
        p.counters = c->counters;
        p.part_cap = (long long)(c->part_bytes / sizeof(float4));
        p.ctr_cap = (long long)c->n_counters;
    }
    const cuuint32_t abox[4] = {64, cuuint32_t(p.halo_w), cuuint32_t(p.halo_h), 1};
    const cuuint64_t xdims[4] = {cuuint64_t(c->cin), cuuint64_t(c->W), cuuint64_t(c->H),
                                 cuuint64_t(c->F)};
    const cuuint64_t cdims[4] = {cuuint64_t(c->cin), cuuint64_t(c->W), cuuint64_t(c->H),
                                 cuuint64_t(std::max(1, c->kt - 1))};
    const cuuint64_t wdims[3] = {cuuint64_t(c->cin), cuuint64_t(c->cout),
                                 cuuint64_t(c->kt * c->kh * c->kw)};
    const cuuint32_t wbox[3] = {64, cuuint32_t(pair ? bn / 2 : bn), cuuint32_t(p.tb)};
    const bool y_f32 = c->out_dtype != FRT_OUT_BF16;
    const cuuint64_t ydims[4] = {cuuint64_t(c->cout), cuuint64_t(c->W), cuuint64_t(c->H),
                                 cuuint64_t(c->F)};
    const cuuint32_t ybox[4] = {y_f32 ? 32u : 64u, kTileW, kTileH, 1};
    if (!encode(&p.x_map, x, 4, xdims, abox) || !encode(&p.c_map, c->cache[c->cur], 4, cdims, abox) ||
        !encode(&p.w_map, w, 3, wdims, wbox) || !encode(&p.y_map, y, 4, ydims, ybox, y_f32))
        return cfail(FRT_ERR_CUDA, "tensor map encoding failed");
    p.bias = static_cast<const float*>(bias);
    p.y = y;
    p.y_bf16 = c->out_dtype == FRT_OUT_BF16;
    p.wait_limit_ns = c->wait_limit_ns;
    p.status = c->status_dev;
    p.part_mode = g_conv_part_mode;
    if (c->kt > 1) {
        p.shift_cache = static_cast<const uint4*>(c->cache[c->cur]);
        p.shift_x = static_cast<const uint4*>(x);
        p.shift_next = static_cast<uint4*>(c->cache[c->cur ^ 1]);
        p.shift_frame_vec = (long long)(c->frame_bytes / 16);
        p.shift_keep = c->kt - 1;
    }
    cudaError_t e;
    switch (bn * 2 + (pair ? 1 : 0)) {
        case 513: e = launch_conv<256, true>(p, pl.units, c->cs); break;
        case 512: e = launch_conv<256, false>(p, pl.units, c->cs); break;
        case 385: e = launch_conv<192, true>(p, pl.units, c->cs); break;
        case 384: e = launch_conv<192, false>(p, pl.units, c->cs); break;
        case 257: e = launch_conv<128, true>(p, pl.units, c->cs); break;
        case 256: e = launch_conv<128, false>(p, pl.units, c->cs); break;
        case 193: e = launch_conv<96, true>(p, pl.units, c->cs); break;
        case 192: e = launch_conv<96, false>(p, pl.units, c->cs); break;
        case 129: e = launch_conv<64, true>(p, pl.units, c->cs); break;
        default: e = launch_conv<64, false>(p, pl.units, c->cs); break;
    }
    if (e != cudaSuccess) return cuda_cfail(FRT_ERR_CUDA, cudaGetErrorString(e));
    if (c->kt > 1) c->cur ^= 1;
    c->chunks += 1;
    return FRT_OK;
}

frt_status frt_conv_set_tile(frt_conv_t* c, int bn, int pair) {
    if (!c) return cfail(FRT_ERR_INVALID_ARG, "NULL conv handle");
    if (bn == 0) {
        c->force_bn = 0;
        c->force_pair = 0;
        return FRT_OK;
    }
    if ((bn != 64 && bn != 96 && bn != 128 && bn != 192 && bn != 256) || c->cout % bn != 0 ||
        (pair != 0 && pair != 1))
        return cfail(FRT_ERR_INVALID_ARG, "bn must be 64, 96, 128, 192 or 256 dividing Cout; pair 0 or 1");
    c->force_bn = bn;
    c->force_pair = pair;
    return c->configured ? ensure_split_scratch(c) : FRT_OK;
}

frt_status frt_conv_plan(int cin, int cout, int kt, int kh, int kw, int grid_h, int grid_w,
                         int frames_per_chunk, int out_dtype, int sms, int bn, int pair,
                         int split_mode, int units, int* plan) {
    if (!plan || cin < 64 || cin % 64 || cout < 64 || cout % 64 || kt < 1 || kh < 1 || kw < 1 ||
        grid_h < 1 || grid_w < 1 || frames_per_chunk < 1 || sms < 1 || split_mode < 0 ||
        split_mode > 2 || units < 0)
        return cfail(FRT_ERR_INVALID_ARG, "invalid sizes or modes");
    ConvPlan pl;
    if (!plan_conv(cin, cout, kt, kh, kw, grid_h, grid_w, frames_per_chunk,
                   out_dtype == FRT_OUT_BF16, bn, pair, split_mode, units, sms, pl))
        return cfail(FRT_ERR_UNSUPPORTED, "no tile width fits");
    plan[0] = pl.bn;
    plan[1] = pl.pair ? 1 : 0;
    plan[2] = pl.units;
    plan[3] = pl.split ? 1 : 0;
    plan[4] = pl.n_tiles;
    plan[5] = kt * (cin / kBK);
    return FRT_OK;
}

int frt_selftest_conv_part_mode(int mode) {
    if (mode < 0 || mode > 2) return -1;
    g_conv_part_mode = mode;
    return 0;
}

frt_status frt_conv_set_split(frt_conv_t* c, int mode, int units) {
    if (!c) return cfail(FRT_ERR_INVALID_ARG, "NULL conv handle");
    if (mode < 0 || mode > 2 || units < 0)
        return cfail(FRT_ERR_INVALID_ARG, "mode 0 (automatic), 1 (whole tiles) or 2 (split); units >= 0");
    c->split_mode = mode;
    c->split_units = units;
    return c->configured ? ensure_split_scratch(c) : FRT_OK;
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
    if (e != cudaSuccess) return cuda_cfail(FRT_ERR_CUDA, cudaGetErrorString(e));
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
    // a launch that gave up may have left split tiles half counted
    if (e == cudaSuccess && c->counters) e = cudaMemset(c->counters, 0, c->n_counters * sizeof(int));
    if (e == cudaSuccess) e = cudaDeviceSynchronize();
    if (e != cudaSuccess) return cuda_cfail(FRT_ERR_CUDA, cudaGetErrorString(e));
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
