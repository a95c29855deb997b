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
    const int c_first = blockIdx.x / CM;
    const int c_stride = gridDim.x / CM;

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
            for (int t = c_first; t < p.n_tiles && ok; t += c_stride) {
                int f, th, tw, tn;
                tile_coords(p, t, CM, rank, f, th, tw, tn);
                const int cx = tw * kTileW - p.kw / 2;
                const int cy = th * kTileH - p.kh / 2;
                int src = f - (p.kt - 1);                 // frame of (cache, chunk) - cache
                int kb = 0;
                for (int hi = 0; hi < nhalo; ++hi, ++ia) {
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
            for (int t = c_first; t < p.n_tiles && ok; t += c_stride) {
                const int n0 = (t % p.tiles_n) * BN + rank * (BN / CM);
                int kb = 0, tap0 = 0;                     // tap0 = first tap of this dt
                for (int hi = 0; hi < nhalo && ok; ++hi) {
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
            for (int t = c_first; t < p.n_tiles; t += c_stride, ++tl) {
                const int b = tl & 1;
                if (tl >= 2) handoff();                      // accumulator b drained
                const uint32_t d = tmem + uint32_t(b * BN);
                uint32_t accumulate = 0;
                for (int hi = 0; hi < nhalo; ++hi) {
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
            for (int t = c_first; t < p.n_tiles; t += c_stride, ++tl) {
                const int b = tl & 1;
                if (tl >= 2) observe(smem_u32(&bars.acc_empty[b]), ((tl >> 1) - 1) & 1, 1, -1 - tl);
                for (int hi = 0; hi < nhalo; ++hi, ++ia) {
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
        const uint32_t rb = sStg + uint32_t(row * 128);
        const uint32_t sw = uint32_t(row & 7);
        const bool est = threadIdx.x == 64;              // issues the tile's TMA stores
        const int ucols = p.y_bf16 ? 64 : 32;            // output channels per unit
        if (p.shift_keep > 0) {
            // this CTA's slice of the next cache, while the first tile's MMAs run
            const long long total = p.shift_frame_vec * p.shift_keep;
            const long long per = (total + gridDim.x - 1) / gridDim.x;
            const long long lo = per * blockIdx.x;
            const long long hi = lo + per < total ? lo + per : total;
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
        for (int t = c_first; t < p.n_tiles; t += c_stride, ++tl) {
            const int b = tl & 1;
            int f, th, tw, tn;
            tile_coords(p, t, CM, rank, f, th, tw, tn);
            const bool got = mbar_wait(smem_u32(&bars.acc_full[b]), (tl >> 1) & 1, lim, abort);
            // all four warps go on or stop together: the staging below synchronises them
            if (!named_bar_and(1, 128, got)) {
                if (!got) report(p.status, abort, 2, tl);
                break;
            }
            tc_fence_after();
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
                    tmem_ld32(tmem + lane_off + uint32_t(b * BN + c), r);
                    tmem_ld_wait();
                    const float4* bp = reinterpret_cast<const float4*>(p.bias + tn * BN + c);
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
#pragma unroll
                        for (int i = 0; i < 16; ++i) o[16 * h + i] = pack_bf16x2(v[2 * i], v[2 * i + 1]);
                    } else {
#pragma unroll
                        for (int i = 0; i < 32; ++i) o[i] = __float_as_uint(v[i]);
                    }
                }
                if (est) bulk_wait_read<0>();            // the previous store has read the slab
                named_bar_sync(1, 128);
#pragma unroll
                for (int i = 0; i < 8; ++i)
                    st_shared_v4(rb + ((uint32_t(i) ^ sw) << 4), o[4 * i], o[4 * i + 1], o[4 * i + 2],
                                 o[4 * i + 3]);
                fence_proxy_async_smem();
                named_bar_sync(1, 128);
                if (est && f < p.F) {
                    tma_store_4d(&p.y_map, sStg, tn * BN + u * ucols, tw * kTileW, th * kTileH, f);
                    bulk_commit();
                }
            }
            tc_fence_before();
            if (PAIR) mbar_arrive_cluster(mapa_shared(smem_u32(&bars.acc_empty[b]), 0));
            else mbar_arrive(smem_u32(&bars.acc_empty[b]));
        }
        if (est) bulk_wait<0>();                          // y written before the CTA exits
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
cudaError_t launch_conv(ConvParams p, cudaStream_t st) {
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
    const int units = std::min(p.n_tiles, num_sms() / C::CM);
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

// Output-channel tile and pairing, from a cost model measured on GB300 with this
// kernel: a spatial tap costs its MMA issue time (four MMAs of max(BN / 2, 50) cycles,
// 1.2x that for CTA pairs, whose MMAs issue slower) plus ~350 cycles of ring
// bookkeeping (a shared-memory access by the issuing thread behind queued MMAs costs it
// ~140 cycles), plus ~300 more when a weight stage holds a single tap; every tile has the
// same number of taps and tiles run in rounds over the SMs (or SM pairs), so a launch
// costs rounds x that. The cheapest of the widths dividing Cout wins; pairs need at
// least two pixel tiles. A bf16 output is staged in 64-channel units, so its widths are
// multiples of 64.
int choose_bn(int cout, long long m_tiles, int a_bytes, int kw, bool y_bf16, bool& pair) {
    const int cands[5] = {256, 192, 128, 96, 64};
    const long long sms = num_sms();
    int best = 0;
    double best_t = 1e30;
    for (int pr = 0; pr < 2; ++pr) {
        if (pr == 1 && m_tiles < 2) continue;
        const int cm = pr ? 2 : 1;
        const long long units = sms / cm;
        const long long mt = (m_tiles + cm - 1) / cm;
        for (int bn : cands) {
            if (cout % bn || (y_bf16 && bn % 64)) continue;
            int tb, as, bs;
            if (!plan_rings(a_bytes, (bn / cm) * kBK * 2, kw, tb, as, bs)) continue;
            const long long tiles = mt * (cout / bn);
            const double rounds = double((tiles + units - 1) / units);
            const double mma = 4.0 * std::max(bn / 2.0, 50.0) * (pr ? 1.2 : 1.0);
            const double t = rounds * (350.0 + mma + (tb == 1 && kw > 1 ? 300.0 : 0.0));
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
    int force_bn = 0;      // 0: the cost model picks the tile
    int force_pair = 0;
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
    c->cache[0] = c->cache[1] = nullptr;
    c->status_host = c->status_dev = nullptr;
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
    p.halo_w = kTileW + c->kw - 1;
    p.halo_h = kTileH + c->kh - 1;
    p.halo_tx = p.halo_w * p.halo_h * kBK * 2;
    p.a_bytes = (p.halo_tx + 1023) & ~1023;
    const long long m_tiles = (long long)c->F * p.tiles_w * p.tiles_h;
    bool pair = c->force_pair != 0;
    const bool y_bf16 = c->out_dtype == FRT_OUT_BF16;
    const int bn = c->force_bn != 0 ? c->force_bn
                                    : choose_bn(c->cout, m_tiles, p.a_bytes, c->kw, y_bf16, pair);
    if (bn == 0) return cfail(FRT_ERR_UNSUPPORTED, "Cout has no supported tile width");
    if (y_bf16 && bn % 64)
        return cfail(FRT_ERR_UNSUPPORTED, "a bf16 output needs a tile width that is a multiple of 64");
    const int b_bytes = (pair ? bn / 2 : bn) * kBK * 2;
    if (!plan_rings(p.a_bytes, b_bytes, c->kw, p.tb, p.a_stages, p.b_stages))
        return cfail(FRT_ERR_UNSUPPORTED, "halo and weight rings do not fit");
    p.b_stage = p.tb * b_bytes;
    p.tiles_n = c->cout / bn;
    const long long m_units = pair ? (m_tiles + 1) / 2 : m_tiles;
    if (m_units * p.tiles_n >= (1LL << 31)) return cfail(FRT_ERR_UNSUPPORTED, "too many tiles");
    p.n_tiles = int(m_units * p.tiles_n);
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
    if (c->kt > 1) {
        p.shift_cache = static_cast<const uint4*>(c->cache[c->cur]);
        p.shift_x = static_cast<const uint4*>(x);
        p.shift_next = static_cast<uint4*>(c->cache[c->cur ^ 1]);
        p.shift_frame_vec = (long long)(c->frame_bytes / 16);
        p.shift_keep = c->kt - 1;
    }
    cudaError_t e;
    switch (bn * 2 + (pair ? 1 : 0)) {
        case 513: e = launch_conv<256, true>(p, c->cs); break;
        case 512: e = launch_conv<256, false>(p, c->cs); break;
        case 385: e = launch_conv<192, true>(p, c->cs); break;
        case 384: e = launch_conv<192, false>(p, c->cs); break;
        case 257: e = launch_conv<128, true>(p, c->cs); break;
        case 256: e = launch_conv<128, false>(p, c->cs); break;
        case 193: e = launch_conv<96, true>(p, c->cs); break;
        case 192: e = launch_conv<96, false>(p, c->cs); break;
        case 129: e = launch_conv<64, true>(p, c->cs); break;
        default: e = launch_conv<64, false>(p, c->cs); break;
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
