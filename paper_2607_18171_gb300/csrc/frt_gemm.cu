// frt_gemm.cu — C = A · B^T on the sm_103a tensor cores: bf16 operands (both K-major),
// fp32 accumulation in TMEM, for the linear projections around the chunk attention of a
// DiT block (QKV projection in front of it, output projection after it).
//
// Persistent kernel, one CTA per SM, 352 threads:
//   warp 0      TMA producer: two k-blocks of A (128 x 64 each) and of B (BN x 64 each)
//               per ring stage, 128-byte swizzle, through a shared-memory ring (with K a
//               multiple of 64, one box per operand loads both k-blocks through a 3D view
//               (64, rows, K / 64) of the matrix);
//   warp 1      TMEM allocator + tcgen05.mma issuer (M = 128, N = BN, K = 16 per
//               instruction, eight per stage): a converged warp whose lane 0 issues; it
//               touches no mbarrier in its loop (a shared-memory access by the issuing
//               thread behind queued MMAs stalls it behind their operand reads);
//   warp 10     observer: waits on the stage and accumulator barriers in the issuer's
//               order and hands each off to it through a named barrier;
//   warps 2-9   epilogue: two warps per TMEM lane quarter, each thread one accumulator
//               row (TMEM lane) and one half of every column unit: each 128-byte
//               column unit of the tile (32 fp32 or 64 bf16 columns) is staged in a 128-byte-swizzled shared-memory slab and written
//               by one TMA tensor store (rows past M and columns past N are clipped by
//               the store); per-thread row stores would touch 32 rows per warp
//               instruction.
// The accumulator is double-buffered in TMEM (2 x BN columns), so the epilogue of tile i
// runs while the tensor pipe computes tile i + 1.
// When M spans more than one 128-row tile, two CTAs of a cluster work as a pair on a
// 256 x BN tile with tcgen05.mma.cta_group::2: each holds its own 128 rows of A and one
// half of B in shared memory (the tensor cores of the two SMs read both halves), so each
// SM takes in 32 KB per k-block instead of 48 — what bounds this kernel is how fast
// operands reach an SM. The leader CTA's thread issues the MMAs for both; both CTAs'
// TMA loads complete on the leader's barriers; the leader's commits reach both CTAs; the
// follower's epilogue hands the accumulator back to the leader by a remote arrive.
//
// Epilogues:
//   plain  C row-major, fp32 or bf16 (round to nearest even), rows >= M and columns >= N
//          are not stored;
//   qkv    the QKV projection of a frame chunk: columns [0, d) are q, [d, 2d) k, [2d, 3d)
//          v (d = heads * head_dim). Values are rounded to bf16 first, then q and k are
//          rotated with the same 3D RoPE routine as every other kernel (so the result is
//          bit-identical to a plain bf16 projection followed by the RoPE kernel); q goes
//          to its buffer, k and v straight into the chunk's ring slot of the KV cache.
//
// Every wait is bounded: a role that gives up records FRT_ERR_TIMEOUT in the status
// block, raises the CTA's abort flag, drains its in-flight copies / MMAs and the CTA
// frees TMEM before exiting.
#include "frt_internal.h"
#include "frt_ptx.cuh"

namespace frt {

namespace {

constexpr int kThreads = 352;
constexpr int kEpiThreads = 256;   // warps 2-9
// Named barrier of the issuer / observer hand-off (warps 1 and 10); id 1 serves the
// epilogue warps, id 0 is __syncthreads.
constexpr int kBarHandoff = 4;
constexpr int kBM = 128;
constexpr int kBK = 64;          // one 128-byte swizzle atom of bf16
constexpr int kMaxStages = 6;
constexpr int kKPS = 2;          // k-blocks per ring stage
constexpr int kTimeoutCode = 6;  // FRT_ERR_TIMEOUT

template <int BN, bool PAIR>
struct GCfg {
    static constexpr int CM = PAIR ? 2 : 1;               // CTAs per tile
    static constexpr int A_BYTES = kBM * kBK * 2;         // this CTA's 128 rows of A, one k-block
    static constexpr int B_BYTES = (BN / CM) * kBK * 2;   // this CTA's share of B, one k-block
    static constexpr int STAGE = kKPS * (A_BYTES + B_BYTES);   // [A kb0 | A kb1 | B kb0 | B kb1]
    static constexpr int SLAB = kBM * 128;                // epilogue staging slab
    static constexpr int STAGES = (225 * 1024 - 1024 - SLAB) / STAGE < kMaxStages
                                      ? (225 * 1024 - 1024 - SLAB) / STAGE : kMaxStages;
    static constexpr int SMEM = STAGES * STAGE + SLAB + 1024;   // + alignment slack
    static constexpr uint32_t IDESC = idesc_bf16_f32(kBM * CM, BN, false);
    static constexpr uint32_t TMEM_COLS = 2 * BN <= 256 ? 256 : 512;   // a power of two
};

struct GBars {
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
            s->role = 200 + role;
            s->where = where;
            __threadfence_system();
            s->code = kTimeoutCode;
        }
    }
}

template <int BN, bool PAIR>
__global__ void __launch_bounds__(kThreads, 1) gemm_kernel(const __grid_constant__ GemmParams p) {
    using C = GCfg<BN, PAIR>;
    constexpr int CM = C::CM;
    constexpr int kStages = C::STAGES;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                               ~uintptr_t(1023));
    __shared__ GBars bars;
    __shared__ float2 s_t[kMaxTEntries];
    const uint32_t sbase = smem_u32(smem);
    volatile int* abort = &bars.abort_flag;
    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    // tiles of CM x 128 rows by BN columns; both CTAs of a pair walk the same sequence
    const int ctm = (p.tiles_m + CM - 1) / CM;
    const int n_tiles = ctm * p.tiles_n;
    const int rank = PAIR ? int(cluster_ctarank()) : 0;
    const bool leader = rank == 0;
    const int c_first = blockIdx.x / CM;
    const int c_stride = gridDim.x / CM;
    const int nk = (p.K + kBK - 1) / kBK;
    const uint64_t lim = p.wait_limit_ns;

    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            mbar_init(smem_u32(&bars.full[s]), 1);
            mbar_init(smem_u32(&bars.empty[s]), 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(smem_u32(&bars.acc_full[b]), 1);
            mbar_init(smem_u32(&bars.acc_empty[b]), kEpiThreads * CM);
        }
        mbar_init(smem_u32(&bars.drain), 1);
        bars.abort_flag = 0;
        fence_mbar_init();
    }
    if (p.epi == kEpiQkv && p.rope)
        for (int i = threadIdx.x; i < kMaxTEntries; i += kThreads) s_t[i] = p.ra.t_tab[i];
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
    if (PAIR) cluster_sync_all();   // both CTAs' barriers exist before any cross-CTA signal
    tc_fence_after();
    const uint32_t tmem = bars.tmem_base;

    if (warp == 0) {
        // ==================================== TMA producer ===================================
        if (lane == 0) {
            tma_prefetch_map(&p.a_map);
            tma_prefetch_map(&p.b_map);
            int it = 0;
            bool ok = true;
            for (int t = c_first; t < n_tiles && ok; t += c_stride) {
                const int tm = (t % ctm) * CM + rank;
                const int tn = t / ctm;
                const int brow = tn * BN + rank * (BN / CM);
                for (int kb = 0; kb < nk; kb += kKPS) {
                    const int s = it % kStages;
                    // slot s was last filled by load it - kStages; the MMA that read it
                    // commits empty[s] (in both CTAs of a pair) once per use
                    if (it >= kStages && !mbar_test_wait(smem_u32(&bars.empty[s]), ((it / kStages) - 1) & 1) &&
                        !mbar_wait(smem_u32(&bars.empty[s]), ((it / kStages) - 1) & 1, lim, abort)) {
                        report(p.status, abort, 0, it);
                        ok = false;
                        break;
                    }
                    const uint32_t dst = sbase + s * C::STAGE;
                    const uint32_t dst_b = dst + kKPS * C::A_BYTES;
                    // both k-blocks of the stage; past K (or past the last k-block) the
                    // copies read zeros, and the bytes still count
                    if (PAIR) {
                        // both CTAs' bytes complete on the leader's barrier
                        const uint32_t fb = mapa_shared(smem_u32(&bars.full[s]), 0);
                        if (leader) mbar_arrive_expect_tx(smem_u32(&bars.full[s]), 2 * C::STAGE);
                        if (p.kview3) {
                            tma_load_3d_pair(dst, &p.a_map, fb, 0, tm * kBM, kb);
                            tma_load_3d_pair(dst_b, &p.b_map, fb, 0, brow, kb);
                        } else {
                            for (int h = 0; h < kKPS; ++h) {
                                tma_load_2d_pair(dst + h * C::A_BYTES, &p.a_map, fb, (kb + h) * kBK, tm * kBM);
                                tma_load_2d_pair(dst_b + h * C::B_BYTES, &p.b_map, fb, (kb + h) * kBK, brow);
                            }
                        }
                    } else {
                        const uint32_t fb = smem_u32(&bars.full[s]);
                        mbar_arrive_expect_tx(fb, C::STAGE);
                        if (p.kview3) {
                            tma_load_3d(dst, &p.a_map, fb, 0, tm * kBM, kb);
                            tma_load_3d(dst_b, &p.b_map, fb, 0, brow, kb);
                        } else {
                            for (int h = 0; h < kKPS; ++h) {
                                tma_load_2d(dst + h * C::A_BYTES, &p.a_map, fb, (kb + h) * kBK, tm * kBM);
                                tma_load_2d(dst_b + h * C::B_BYTES, &p.b_map, fb, (kb + h) * kBK, brow);
                            }
                        }
                    }
                    ++it;
                }
            }
            // drain: every issued load lands before the CTA may exit (a pair's loads all
            // complete on the leader's barriers; the follower is held by the closing
            // cluster barrier until the leader has drained)
            if (leader)
                for (int i = (it > kStages ? it - kStages : 0); i < it; ++i)
                    mbar_wait_drain(smem_u32(&bars.full[i % kStages]), (i / kStages) & 1, lim);
        }
    } else if (warp == 1) {
        // ============ MMA issuer (a converged warp of the leader; lane 0 issues) ============
        // The warp never touches an mbarrier in its loop: the observer warp (warp 10) waits
        // for every barrier the next MMAs need and meets it at the hand-off named barrier.
        // (A shared-memory access by the issuing thread behind queued MMAs waits behind
        // their operand reads, ~300 cycles per stage measured; a named barrier reads no
        // shared memory.) Both warps pass the same barriers in the same order whatever
        // happens, so neither can strand the other.
        if (leader) {
            const uint32_t lead = lane == 0 ? 1u : 0u;
            auto handoff = [&]() {
                named_bar_sync(kBarHandoff, 64);
                tc_fence_after();
            };
            // descriptors are linear in the 16-byte start address: a K step of 16 bf16
            // inside the 128-byte swizzle atom adds 32 bytes (2 units)
            const uint64_t da0 = sdesc_sw128(sbase, 16, 1024);
            const uint64_t db0 = sdesc_sw128(sbase + kKPS * C::A_BYTES, 16, 1024);
            int it = 0;
            int tl = 0;
            for (int t = c_first; t < n_tiles; t += c_stride, ++tl) {
                const int b = tl & 1;
                if (tl >= 2) handoff();                      // accumulator b drained
                const uint32_t d = tmem + uint32_t(b * BN);
                for (int kb = 0; kb < nk; kb += kKPS, ++it) {
                    const int s = it % kStages;
                    handoff();                               // stage s landed
                    const uint64_t so = uint64_t((s * C::STAGE) >> 4);
#pragma unroll
                    for (int h = 0; h < kKPS; ++h) {
                        if (kb + h >= nk) break;          // the zero-filled half of the last stage
                        const uint64_t da = da0 + so + uint64_t((h * C::A_BYTES) >> 4);
                        const uint64_t db = db0 + so + uint64_t((h * C::B_BYTES) >> 4);
#pragma unroll
                        for (int k = 0; k < kBK / 16; ++k) {
                            const uint32_t acc = (kb + h > 0 || k > 0) ? 1u : 0u;
                            if (PAIR)
                                umma_ss_pair_if(lead, d, da + uint64_t(2 * k), db + uint64_t(2 * k),
                                                C::IDESC, acc);
                            else
                                umma_ss_if(lead, d, da + uint64_t(2 * k), db + uint64_t(2 * k),
                                           C::IDESC, acc);
                        }
                    }
                    if (PAIR) umma_commit_pair_if(lead, smem_u32(&bars.empty[s]), 0x3);
                    else umma_commit_if(lead, smem_u32(&bars.empty[s]));
                }
                if (PAIR) umma_commit_pair_if(lead, smem_u32(&bars.acc_full[b]), 0x3);
                else umma_commit_if(lead, smem_u32(&bars.acc_full[b]));
            }
            // drain: all issued MMAs complete before TMEM is released
            if (PAIR) umma_commit_pair_if(lead, smem_u32(&bars.drain), 0x1);
            else umma_commit_if(lead, smem_u32(&bars.drain));
            mbar_wait_drain(smem_u32(&bars.drain), 0, lim);
        }
    } else if (warp == 10) {
        // ======== observer (leader): waits for what the issuer's next MMAs need ========
        // After a wait gives up (or another role raised the abort flag) the remaining
        // hand-offs pass without waiting; the issuer then finishes on stale operands, which
        // the recorded error status marks as void.
        if (leader) {
            bool ok = true;
            auto observe = [&](uint32_t bar, uint32_t parity, int where) {
                if (ok) {
                    ok = __all_sync(0xffffffffu, mbar_wait(bar, parity, lim, abort));
                    if (!ok && lane == 0) report(p.status, abort, 1, where);
                }
                named_bar_sync(kBarHandoff, 64);
            };
            int it = 0;
            int tl = 0;
            for (int t = c_first; t < n_tiles; t += c_stride, ++tl) {
                const int b = tl & 1;
                if (tl >= 2) observe(smem_u32(&bars.acc_empty[b]), ((tl >> 1) - 1) & 1, -1 - tl);
                for (int kb = 0; kb < nk; kb += kKPS, ++it)
                    observe(smem_u32(&bars.full[it % kStages]), (it / kStages) & 1, it);
            }
        }
    } else {
        // ====================================== epilogue =====================================
        const int sub = warp & 3;                      // TMEM lane quarter of this warp
        const int half = (warp - 2) >> 2;              // which half of each column unit
        const int row = sub * 32 + lane;
        const uint32_t lane_off = uint32_t(sub * 32) << 16;
        const uint32_t stg = sbase + uint32_t(kStages * C::STAGE);   // 1024-aligned slab
        const uint32_t rb = stg + uint32_t(row * 128);
        const uint32_t sw = uint32_t(row & 7);
        const bool est = threadIdx.x == 64;            // issues the TMA stores
        // slab free (the previous store has read it), then every thread refills it
        auto slab_acquire = [&]() {
            if (est) bulk_wait_read<0>();
            named_bar_sync(1, kEpiThreads);
        };
        auto slab_release = [&](const CUtensorMap* map, int c0, int r0) {
            fence_proxy_async_smem();
            named_bar_sync(1, kEpiThreads);
            if (est) {
                tma_store_2d(map, stg, c0, r0);
                bulk_commit();
            }
        };
        int tl = 0;
        for (int t = c_first; t < n_tiles; t += c_stride, ++tl) {
            const int b = tl & 1;
            const int tm = (t % ctm) * CM + rank;
            const int tn = t / ctm;
            const bool got = mbar_wait(smem_u32(&bars.acc_full[b]), (tl >> 1) & 1, lim, abort);
            // all epilogue warps go on or stop together: the staging below synchronises them
            if (!named_bar_and(1, kEpiThreads, got)) {
                if (!got) report(p.status, abort, 2, tl);
                break;
            }
            tc_fence_after();
            const int grow = tm * kBM + row;
            const bool live = grow < p.M;
            const int n0 = tn * BN;
            if (p.epi == kEpiQkv) {
                const int which = n0 / p.d;                 // 0 q, 1 k, 2 v
                const int cbase = n0 - which * p.d;
                const bool rot = p.rope && which < 2 && live;
                int f = 0, rr = 0, col = 0;
                if (rot) {
                    f = grow / p.ra.tpf;
                    const int rem = grow - f * p.ra.tpf;
                    rr = rem / p.ra.gw;
                    col = rem - rr * p.ra.gw;
                }
#pragma unroll 1
                for (int u = 0; u < BN / 64; ++u) {      // 64 bf16 columns per unit
                    // the unit's values are computed before the slab is claimed, so the
                    // previous store's read of the slab overlaps this work
                    uint32_t wu[1][16];
                    {
                        const int hh = 0;
                        const int c = 2 * u + half;               // this half's 32 columns
                        uint32_t r[32];
                        tmem_ld32(tmem + lane_off + uint32_t(b * BN + c * 32), r);
                        tmem_ld_wait();
                        const int cc = cbase + c * 32;
                        uint32_t (&w)[16] = wu[hh];
#pragma unroll
                        for (int i = 0; i < 16; ++i)
                            w[i] = pack_bf16x2(__uint_as_float(r[2 * i]), __uint_as_float(r[2 * i + 1]));
                        if (rot) {
                            // all 16 (cos, sin) of the chunk first, each one load from an
                            // address chosen without branching (t segment in shared memory,
                            // h and w segments in the stream's table): a branch per pair on
                            // the runtime segment widths serialises one load latency per pair
                            const int pi0 = (cc & (p.head_dim - 1)) >> 1;
                            const int dt2 = p.ra.dt2, dth = p.ra.dt2 + p.ra.dh2;
                            const float2* t_row = s_t + f * dt2;
                            const float2* h_row = p.ra.hw + rr * p.ra.dh2 - dt2;
                            const float2* w_row = p.ra.hw + p.ra.gh * p.ra.dh2 + col * p.ra.dw2 - dth;
                            float2 cs[16];
#pragma unroll
                            for (int i = 0; i < 16; ++i) {
                                const int pi = pi0 + i;
                                const float2* src = pi < dt2 ? t_row + pi : (pi < dth ? h_row + pi : w_row + pi);
                                cs[i] = *src;
                            }
#pragma unroll
                            for (int i = 0; i < 16; ++i) w[i] = rope_pair(w[i], cs[i].x, cs[i].y);
                        }
                    }
                    slab_acquire();
#pragma unroll
                    for (int i = 0; i < 4; ++i)
                        st_shared_v4(rb + ((uint32_t(half * 4 + i) ^ sw) << 4), wu[0][4 * i],
                                     wu[0][4 * i + 1], wu[0][4 * i + 2], wu[0][4 * i + 3]);
                    slab_release(&p.out_map[which], cbase + u * 64, tm * kBM);
                }
            } else {
                const int ucols = p.c_bf16 ? 64 : 32;      // output columns per unit
#pragma unroll 1
                for (int u = 0; u < BN / ucols; ++u) {
                    if (n0 + u * ucols >= p.N) break;       // the same for every thread
                    // this half's 64 bytes of the row (16 words), loaded before the slab
                    // is claimed
                    uint32_t v[16];
                    if (p.c_bf16) {
                        uint32_t r[32];
                        tmem_ld32(tmem + lane_off + uint32_t(b * BN + u * ucols + half * 32), r);
                        tmem_ld_wait();
#pragma unroll
                        for (int i = 0; i < 16; ++i)
                            v[i] = pack_bf16x2(__uint_as_float(r[2 * i]), __uint_as_float(r[2 * i + 1]));
                    } else {
                        tmem_ld16(tmem + lane_off + uint32_t(b * BN + u * ucols + half * 16), v);
                        tmem_ld_wait();
                    }
                    slab_acquire();
#pragma unroll
                    for (int i = 0; i < 4; ++i)
                        st_shared_v4(rb + ((uint32_t(half * 4 + i) ^ sw) << 4), v[4 * i], v[4 * i + 1],
                                     v[4 * i + 2], v[4 * i + 3]);
                    slab_release(&p.out_map[0], n0 + u * ucols, tm * kBM);
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
    if (PAIR) cluster_sync_all();   // the pair is done with TMEM and with each other
    tc_fence_after();
    if (warp == 1) {
        if (PAIR) tmem_dealloc_pair(tmem, C::TMEM_COLS);
        else tmem_dealloc(tmem, C::TMEM_COLS);
    }
}

template <int BN, bool PAIR>
cudaError_t launch(const GemmParams& p, cudaStream_t st) {
    using C = GCfg<BN, PAIR>;
    static bool attr_set[kMaxDevices] = {};   // per device: attributes are per device
    const int dev = device_slot();
    if (dev < 0 || !attr_set[dev]) {
        cudaError_t e = cudaFuncSetAttribute(gemm_kernel<BN, PAIR>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
        if (e != cudaSuccess) return e;
        if (dev >= 0) attr_set[dev] = true;
    }
    const int n_ctiles = ((p.tiles_m + C::CM - 1) / C::CM) * p.tiles_n;
    const int units = n_ctiles < num_sms() / C::CM ? n_ctiles : num_sms() / C::CM;
    if (!PAIR) {
        gemm_kernel<BN, false><<<units, kThreads, C::SMEM, st>>>(p);
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
    return cudaLaunchKernelEx(&cfg, gemm_kernel<BN, true>, p);
}

}  // namespace

// CTAs per tile: a pair (cta_group::2) whenever there are at least two M tiles.
int gemm_cluster_m(int M) { return M > kBM ? 2 : 1; }

// Output columns per tile: the width in {128, 192, 256} with the least rounds of tiles
// over the SMs (or SM pairs) x width, a 128-wide tile weighted 1.5x (measured: an N = 128
// MMA of a CTA pair issues in ~82 cycles for 64 of work and its stage waits are exposed)
// and a 192-wide one 1.15x (measured per round and column against 256-wide tiles: 1.14x
// on a 4680 x 4608 x 1536 projection, 1.21x on 4680 x 1536 x 1536; each A k-block feeds
// fewer columns, so more operand bytes cross into the SMs per FLOP).
// The QKV epilogue needs a width dividing d (a tile never straddles q, k and v); widths
// past N are not considered unless nothing else fits.
int g_force_bn = 0;   // test override (frt_selftest_gemm_force_bn)

int gemm_block_n_for(int M, int N, int epi, int d) {
    if (g_force_bn != 0) return g_force_bn;
    const int cm = gemm_cluster_m(M);
    const long long units = num_sms() / cm;
    const long long ctm = ((M + kBM - 1) / kBM + cm - 1) / cm;
    int best = 128;
    double best_t = 1e30;
    for (int bn : {256, 192, 128}) {
        if (epi == kEpiQkv && d % bn != 0) continue;
        if (bn > 128 && bn > N) continue;
        const long long tiles = ctm * ((N + bn - 1) / bn);
        const double t = double((tiles + units - 1) / units) * bn * (bn == 128 ? 1.5 : (bn == 192 ? 1.15 : 1.0));
        if (t < best_t - 1e-9) {
            best_t = t;
            best = bn;
        }
    }
    return best;
}

cudaError_t launch_gemm(GemmParams p, cudaStream_t st) {
    if (p.M <= 0 || p.N <= 0 || p.K <= 0) return cudaSuccess;
    const int bn = gemm_block_n_for(p.M, p.N, p.epi, p.d);
    p.tiles_m = (p.M + kBM - 1) / kBM;
    p.tiles_n = (p.N + bn - 1) / bn;
    if (gemm_cluster_m(p.M) == 2)
        return bn == 256 ? launch<256, true>(p, st)
                         : (bn == 192 ? launch<192, true>(p, st) : launch<128, true>(p, st));
    return bn == 256 ? launch<256, false>(p, st)
                     : (bn == 192 ? launch<192, false>(p, st) : launch<128, false>(p, st));
}

}  // namespace frt

extern "C" int frt_selftest_gemm_force_bn(int bn) {
    if (bn != 0 && bn != 128 && bn != 192 && bn != 256) return -1;
    frt::g_force_bn = bn;
    return 0;
}
